// aspis_sgd: the model update that follows the aggregation.  Eq. 1
// (Section 2) moves the parameters against the batch gradient with step
// eta_t; the PS of Algorithm 1 uses the aggregate of the chosen copies in its
// place, and the experiments add momentum 0.9 (Appendix A.3), read as
// heavy-ball momentum without dampening:
//     v <- mu * v + g,    w <- w - eta * v,
// each result the exact value rounded once to fp32 (one fused multiply-add).
//
// The update streams g, w and v once and writes w and v: 20 bytes per
// coordinate with momentum, 12 without.  Each thread moves four float4 of
// each array, 16-byte loads on the widest path the pointers allow, so the
// kernel is bound by HBM like a copy.
#include <limits.h>

#include "aspis_internal.cuh"

namespace {

constexpr int kThreads = 256;
constexpr int kUnroll = 4;            // float4 (or floats) per thread and array

__device__ __forceinline__ float4 ld4(const float4 *p) { return __ldcs(p); }
__device__ __forceinline__ void st4(float4 *p, float4 x) { __stcs(p, x); }

template <bool MOM>
__device__ __forceinline__ void step1(float g, float &w, float &v, float eta, float mu)
{
    if constexpr (MOM) {
        v = __fmaf_rn(mu, v, g);
        w = __fmaf_rn(-eta, v, w);
    } else {
        w = __fmaf_rn(-eta, g, w);
    }
}

// n4 float4 of every array from 16-byte aligned pointers; block 0 also takes
// the last d - 4*n4 (< 4) coordinates one by one
template <bool MOM>
__global__ void __launch_bounds__(kThreads)
sgd_vec_kernel(const float *g, float *w, float *v,
               int64_t n4, int64_t d, float eta, float mu)
{
    const float4 *g4 = reinterpret_cast<const float4 *>(g);
    float4 *w4 = reinterpret_cast<float4 *>(w);
    float4 *v4 = reinterpret_cast<float4 *>(v);
    const int64_t base = (int64_t)blockIdx.x * (kThreads * kUnroll) + threadIdx.x;
    float4 gr[kUnroll], wr[kUnroll], vr[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
        const int64_t i = base + (int64_t)u * kThreads;
        if (i < n4) {
            gr[u] = ld4(g4 + i);
            wr[u] = ld4(w4 + i);
            if constexpr (MOM) vr[u] = ld4(v4 + i);
        }
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
        const int64_t i = base + (int64_t)u * kThreads;
        if (i < n4) {
            step1<MOM>(gr[u].x, wr[u].x, vr[u].x, eta, mu);
            step1<MOM>(gr[u].y, wr[u].y, vr[u].y, eta, mu);
            step1<MOM>(gr[u].z, wr[u].z, vr[u].z, eta, mu);
            step1<MOM>(gr[u].w, wr[u].w, vr[u].w, eta, mu);
            st4(w4 + i, wr[u]);
            if constexpr (MOM) st4(v4 + i, vr[u]);
        }
    }
    if (blockIdx.x == 0 && threadIdx.x < d - 4 * n4) {
        const int64_t c = 4 * n4 + threadIdx.x;
        float wc = w[c], vc = MOM ? v[c] : 0.f;
        step1<MOM>(g[c], wc, vc, eta, mu);
        w[c] = wc;
        if constexpr (MOM) v[c] = vc;
    }
}

// any alignment: kUnroll floats per thread, consecutive threads on
// consecutive coordinates
template <bool MOM>
__global__ void __launch_bounds__(kThreads)
sgd_scalar_kernel(const float *g, float *w, float *v,
                  int64_t d, float eta, float mu)
{
    const int64_t base = (int64_t)blockIdx.x * (kThreads * kUnroll) + threadIdx.x;
    float gr[kUnroll], wr[kUnroll], vr[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
        const int64_t c = base + (int64_t)u * kThreads;
        if (c < d) {
            gr[u] = __ldcs(g + c);
            wr[u] = __ldcs(w + c);
            if constexpr (MOM) vr[u] = __ldcs(v + c);
        }
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
        const int64_t c = base + (int64_t)u * kThreads;
        if (c < d) {
            step1<MOM>(gr[u], wr[u], vr[u], eta, mu);
            __stcs(w + c, wr[u]);
            if constexpr (MOM) __stcs(v + c, vr[u]);
        }
    }
}

// true when [a, a + n) and [b, b + n) overlap without being the same range
bool partial_overlap(const void *a, const void *b, int64_t n)
{
    const uintptr_t x = (uintptr_t)a, y = (uintptr_t)b;
    if (!a || !b || x == y) return false;
    return x < y ? y - x < (uint64_t)n : x - y < (uint64_t)n;
}

template <bool MOM>
cudaError_t launch_sgd(const float *g, float *w, float *v, int64_t d, float eta, float mu,
                       cudaStream_t stream)
{
    const bool vec = (uintptr_t)g % 16 == 0 && (uintptr_t)w % 16 == 0 &&
                     (!MOM || (uintptr_t)v % 16 == 0);
    const int64_t per_block = (int64_t)kThreads * kUnroll;
    if (vec) {
        const int64_t n4 = d / 4;
        const int64_t blocks = n4 > 0 ? (n4 + per_block - 1) / per_block : 1;
        sgd_vec_kernel<MOM><<<(unsigned)blocks, kThreads, 0, stream>>>(g, w, v, n4, d, eta, mu);
    } else {
        const int64_t blocks = (d + per_block - 1) / per_block;
        sgd_scalar_kernel<MOM><<<(unsigned)blocks, kThreads, 0, stream>>>(g, w, v, d, eta, mu);
    }
    return cudaGetLastError();
}

}  // namespace

extern "C" aspis_status aspis_sgd(const float *g, float *w, float *v, int64_t d, float eta,
                                  float mu, void *stream)
{
    const bool mom = mu != 0.0f;
    if (d < 0 || (d > 0 && (!g || !w || (mom && !v)))) return ASPIS_E_INVAL;
    if (d == 0) return ASPIS_OK;
    // one block per kThreads * kUnroll coordinates; byte counts fit int64
    if (d / ((int64_t)kThreads * kUnroll) >= INT_MAX || d > INT64_MAX / 4) return ASPIS_E_RANGE;
    const int64_t bytes = d * 4;
    if (partial_overlap(g, w, bytes) || (mom && (partial_overlap(g, v, bytes) ||
                                                 partial_overlap(w, v, bytes))))
        return ASPIS_E_INVAL;
    const cudaError_t e = mom ? launch_sgd<true>(g, w, v, d, eta, mu, (cudaStream_t)stream)
                              : launch_sgd<false>(g, w, nullptr, d, eta, mu, (cudaStream_t)stream);
    return e == cudaSuccess ? ASPIS_OK : ASPIS_E_CUDA;
}
