// aspis_round_tolerant: the round for copies that are not bit-identical.
// The paper's honest copies of a file are equal bit for bit; after
// Algorithm 1 (Section 5) it notes that copies differing by floating-point
// effects can still be handled: in Case 1 the PS averages the honest copies
// of each file, in Case 2 it clusters the copies and averages the largest
// cluster.  Readings of that remark:
//   - copies a, b of a file are close iff |a[c] - b[c]| <= tau at every
//     coordinate c < d, difference and magnitude in fp32 (never close where
//     either value is NaN); "close" replaces "equal" in the graph rule;
//   - clusters are the connected components of "close" among the r slots;
//     the largest wins, ties to the one holding the lower slot; Case 1 takes
//     the slots whose worker is in the clique (none: the file is dropped);
//   - the average of the chosen copies x_s (x0 the first) per coordinate:
//     e_s = 0 where x_s equals x0 bitwise, else fp32(x_s - x0); acc = fp32
//     sum of the e_s in slot order; the mean is x0 when acc == 0, else
//     fp32(x0 + fp32(acc / k)), so identical copies give their value exactly.
// The per-file means are written to a caller buffer and reduced by the same
// median (or mean) kernel as the exact round, over one row per kept file.
//
// Kernels: compare_tol (the exact round's streaming compare with the
// tolerance test in place of XOR), select_tol (one thread per file: union of
// close slot pairs, at most 28 bits), file_mean (streams the chosen copies
// of every kept file once and writes one row per file).
#include "aspis_internal.cuh"

namespace {

using namespace aspis;

constexpr int kThreads = 256;
constexpr int64_t kChunkVec = 4096;        // float4 of each row per compare work item

__device__ __forceinline__ bool far_apart(float a, float b, float tau)
{
    return !(fabsf(__fsub_rn(a, b)) <= tau);
}

__device__ __forceinline__ bool far4(const float4 &a, const float4 &b, float tau)
{
    return far_apart(a.x, b.x, tau) | far_apart(a.y, b.y, tau) | far_apart(a.z, b.z, tau) |
           far_apart(a.w, b.w, tau);
}

// Work item = (file, chunk of kChunkVec float4 per row); U*R float4 loads in
// flight per thread; pair bits ORed in a register, one atomicOr per warp.
template <int R, int U>
__global__ void __launch_bounds__(kThreads)
compare_tol_kernel(const float *__restrict__ copies, int64_t f, int64_t d, int64_t ld, float tau,
                   int64_t nvec, int64_t nchunks, uint32_t *__restrict__ file_neq)
{
    const int64_t ldv = ld >> 2;
    const float4 *base = reinterpret_cast<const float4 *>(copies);
    const int64_t items = f * nchunks;
    const int tail = (int)(d - nvec * 4);
    for (int64_t item = blockIdx.x; item < items; item += gridDim.x) {
        const int64_t i = item / nchunks;
        const int64_t ch = item - i * nchunks;
        const float4 *row = base + i * R * ldv;
        const int64_t v0 = ch * kChunkVec;
        const int64_t v1 = v0 + kChunkVec < nvec ? v0 + kChunkVec : nvec;
        uint32_t neq = 0;
        for (int64_t v = v0 + threadIdx.x; v < v1; v += (int64_t)kThreads * U) {
            float4 x[U][R];
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int64_t vv = v + (int64_t)u * kThreads;
#pragma unroll
                for (int s = 0; s < R; ++s)
                    x[u][s] = vv < v1 ? __ldcs(row + s * ldv + vv) : make_float4(0.f, 0.f, 0.f, 0.f);
            }
#pragma unroll
            for (int u = 0; u < U; ++u) {
                int p = 0;
#pragma unroll
                for (int s = 0; s < R; ++s)
#pragma unroll
                    for (int t = s + 1; t < R; ++t, ++p)
                        neq |= (far4(x[u][s], x[u][t], tau) ? 1u : 0u) << p;
            }
        }
        if (tail && ch == nchunks - 1 && threadIdx.x < (unsigned)tail) {
            const float *rw = copies + i * R * ld;
            const int64_t c = nvec * 4 + threadIdx.x;
            float y[R];
#pragma unroll
            for (int s = 0; s < R; ++s) y[s] = rw[s * ld + c];
            int p = 0;
#pragma unroll
            for (int s = 0; s < R; ++s)
#pragma unroll
                for (int t = s + 1; t < R; ++t, ++p)
                    neq |= (far_apart(y[s], y[t], tau) ? 1u : 0u) << p;
        }
        neq = __reduce_or_sync(0xffffffffu, neq);
        if ((threadIdx.x & 31) == 0 && neq) atomicOr(&file_neq[i], neq);
    }
}

// any alignment: one float per thread and step
template <int R>
__global__ void __launch_bounds__(kThreads)
compare_tol_scalar_kernel(const float *__restrict__ copies, int64_t f, int64_t d, int64_t ld,
                          float tau, int64_t nchunks, uint32_t *__restrict__ file_neq)
{
    const int64_t chunk = kChunkVec * 4;
    for (int64_t item = blockIdx.x; item < f * nchunks; item += gridDim.x) {
        const int64_t i = item / nchunks;
        const int64_t c0 = (item - i * nchunks) * chunk;
        const int64_t c1 = c0 + chunk < d ? c0 + chunk : d;
        const float *rw = copies + i * R * ld;
        uint32_t neq = 0;
        for (int64_t c = c0 + threadIdx.x; c < c1; c += kThreads) {
            float y[R];
#pragma unroll
            for (int s = 0; s < R; ++s) y[s] = __ldcs(rw + s * ld + c);
            int p = 0;
#pragma unroll
            for (int s = 0; s < R; ++s)
#pragma unroll
                for (int t = s + 1; t < R; ++t, ++p)
                    neq |= (far_apart(y[s], y[t], tau) ? 1u : 0u) << p;
        }
        neq = __reduce_or_sync(0xffffffffu, neq);
        if ((threadIdx.x & 31) == 0 && neq) atomicOr(&file_neq[i], neq);
    }
}

// One thread per file: the slots to average (Case 1: clique members; Case
// 2: the largest component of "close"), sel = 0 for kept files, -1 else;
// det->n_sel counts the kept files.
template <int R>
__global__ void __launch_bounds__(kThreads)
select_tol_kernel(const uint32_t *__restrict__ file_neq, aspis_detection *det,
                  const uint8_t *__restrict__ fw, int64_t f, uint8_t *__restrict__ slot_mask,
                  int8_t *__restrict__ sel)
{
    const int64_t i = (int64_t)blockIdx.x * kThreads + threadIdx.x;
    const uint32_t clique = det->clique_mask;
    const bool success = det->success != 0;
    uint32_t m = 0u;
    if (i < f) {
        if (success) {
#pragma unroll
            for (int s = 0; s < R; ++s)
                if ((clique >> fw[i * R + s]) & 1u) m |= 1u << s;
        } else {
            // component of each slot as a slot mask, grown to a fixed point
            // (at most R - 1 rounds: each round adds every neighbour of the set)
            const uint32_t w = file_neq[i];
            uint32_t nb[R];
#pragma unroll
            for (int s = 0; s < R; ++s) nb[s] = 1u << s;
            int p = 0;
#pragma unroll
            for (int s = 0; s < R; ++s)
#pragma unroll
                for (int t = s + 1; t < R; ++t, ++p)
                    if (!((w >> p) & 1u)) {
                        nb[s] |= 1u << t;
                        nb[t] |= 1u << s;
                    }
            int best_size = 0;
#pragma unroll
            for (int s = 0; s < R; ++s) {
                uint32_t comp = nb[s];
#pragma unroll
                for (int round = 0; round < R - 1; ++round) {
                    uint32_t grown = comp;
#pragma unroll
                    for (int t = 0; t < R; ++t)
                        if ((comp >> t) & 1u) grown |= nb[t];
                    comp = grown;
                }
                const int size = __popc(comp);
                // the first slot of each component decides (lowest slot wins ties)
                if ((comp & ((1u << s) - 1u)) == 0u && size > best_size) {
                    best_size = size;
                    m = comp;
                }
            }
        }
        slot_mask[i] = (uint8_t)m;
        sel[i] = m ? 0 : -1;
    }
    const int kept = __syncthreads_count(i < f && m != 0u);
    if (threadIdx.x == 0 && kept) atomicAdd(&det->n_sel, kept);
}

// mean of the values x[s] of the slots s in m (reading above); s0 = the
// lowest slot of m, k = |m|; every index is a compile-time slot
template <int R>
__device__ __forceinline__ float mean_masked(const float (&x)[R], uint32_t m, int s0, int k)
{
    float x0 = x[0];
#pragma unroll
    for (int s = 1; s < R; ++s)
        if (s == s0) x0 = x[s];
    const uint32_t b0 = __float_as_uint(x0);
    float acc = 0.f;
#pragma unroll
    for (int s = 0; s < R; ++s)
        if ((m >> s) & 1u) {
            const float e = __float_as_uint(x[s]) == b0 ? 0.f : __fsub_rn(x[s], x0);
            acc = __fadd_rn(acc, e);
        }
    return acc == 0.f ? x0 : __fadd_rn(x0, __fdiv_rn(acc, (float)k));
}

// Grid-stride over (file, chunk of kThreads * 4 float4 or floats); only the
// chosen copies of a kept file are read, once, and their mean is written to
// means[i * ldm + c].
template <int R, bool VEC>
__global__ void __launch_bounds__(kThreads)
file_mean_kernel(const float *__restrict__ copies, int64_t f, int64_t d, int64_t ld,
                 const uint8_t *__restrict__ slot_mask, float *__restrict__ means, int64_t ldm,
                 int64_t nchunks)
{
    constexpr int kU = 4;
    const int64_t per = (int64_t)kThreads * kU * (VEC ? 4 : 1);
    for (int64_t item = blockIdx.x; item < f * nchunks; item += gridDim.x) {
        const int64_t i = item / nchunks;
        const uint32_t m = slot_mask[i];
        if (!m) continue;
        const int s0 = __ffs(m) - 1, k = __popc(m);
        const int64_t c0 = (item - i * nchunks) * per;
        const float *rw = copies + i * R * ld;
        float *out = means + i * ldm;
#pragma unroll
        for (int u = 0; u < kU; ++u) {
            if constexpr (VEC) {
                const int64_t c = c0 + ((int64_t)u * kThreads + threadIdx.x) * 4;
                if (c + 3 < d) {
                    float4 x4[R];
#pragma unroll
                    for (int s = 0; s < R; ++s)
                        x4[s] = (m >> s) & 1u ? __ldcs(reinterpret_cast<const float4 *>(rw + s * ld + c))
                                              : make_float4(0.f, 0.f, 0.f, 0.f);
                    float a[R];
                    float4 r4;
#pragma unroll
                    for (int s = 0; s < R; ++s) a[s] = x4[s].x;
                    r4.x = mean_masked<R>(a, m, s0, k);
#pragma unroll
                    for (int s = 0; s < R; ++s) a[s] = x4[s].y;
                    r4.y = mean_masked<R>(a, m, s0, k);
#pragma unroll
                    for (int s = 0; s < R; ++s) a[s] = x4[s].z;
                    r4.z = mean_masked<R>(a, m, s0, k);
#pragma unroll
                    for (int s = 0; s < R; ++s) a[s] = x4[s].w;
                    r4.w = mean_masked<R>(a, m, s0, k);
                    __stcs(reinterpret_cast<float4 *>(out + c), r4);
                } else {
                    for (int e = 0; e < 4; ++e) {
                        if (c + e >= d) break;
                        float a[R];
#pragma unroll
                        for (int s = 0; s < R; ++s) a[s] = (m >> s) & 1u ? rw[s * ld + c + e] : 0.f;
                        out[c + e] = mean_masked<R>(a, m, s0, k);
                    }
                }
            } else {
                const int64_t c = c0 + (int64_t)u * kThreads + threadIdx.x;
                if (c < d) {
                    float a[R];
#pragma unroll
                    for (int s = 0; s < R; ++s) a[s] = (m >> s) & 1u ? __ldcs(rw + s * ld + c) : 0.f;
                    out[c] = mean_masked<R>(a, m, s0, k);
                }
            }
        }
    }
}

int64_t grid_for(const void *kernel, int64_t items)
{
    int per_sm = 0;
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, kThreads, 0);
    if (per_sm < 1) per_sm = 1;
    int64_t grid = (int64_t)sm_count() * per_sm;
    return grid < items ? grid : (items > 0 ? items : 1);
}

template <int R, int U>
cudaError_t launch_tolerant(const float *copies, int64_t f, int64_t d, int64_t ld, float tau,
                            uint32_t *file_neq, const uint8_t *fw, int K, uint32_t *adj,
                            aspis_detection *det, uint8_t *slot_mask, int8_t *sel, float *means,
                            int64_t ldm, int mode, float *out, cudaStream_t st)
{
    cudaError_t e;
    const bool vec = (uintptr_t)copies % 16 == 0 && ld % 4 == 0;
    if (vec) {
        const int64_t nvec = d >> 2;
        const int64_t nch = nvec > 0 ? (nvec + kChunkVec - 1) / kChunkVec : 1;
        compare_tol_kernel<R, U><<<(unsigned)grid_for((const void *)compare_tol_kernel<R, U>, f * nch),
                                   kThreads, 0, st>>>(copies, f, d, ld, tau, nvec, nch, file_neq);
    } else {
        const int64_t nch = (d + kChunkVec * 4 - 1) / (kChunkVec * 4);
        compare_tol_scalar_kernel<R><<<(unsigned)grid_for((const void *)compare_tol_scalar_kernel<R>, f * nch),
                                       kThreads, 0, st>>>(copies, f, d, ld, tau, nch, file_neq);
    }
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    if ((e = launch_graph(file_neq, fw, f, R, K, adj, st)) != cudaSuccess) return e;
    if ((e = launch_detect(adj, K, det, st)) != cudaSuccess) return e;
    select_tol_kernel<R><<<(unsigned)((f + kThreads - 1) / kThreads), kThreads, 0, st>>>(
        file_neq, det, fw, f, slot_mask, sel);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    const bool vmean = vec && (uintptr_t)means % 16 == 0 && ldm % 4 == 0;
    if (vmean) {
        const int64_t per = (int64_t)kThreads * 4 * 4;
        const int64_t nch = (d + per - 1) / per;
        file_mean_kernel<R, true><<<(unsigned)grid_for((const void *)file_mean_kernel<R, true>, f * nch),
                                    kThreads, 0, st>>>(copies, f, d, ld, slot_mask, means, ldm, nch);
    } else {
        const int64_t per = (int64_t)kThreads * 4;
        const int64_t nch = (d + per - 1) / per;
        file_mean_kernel<R, false><<<(unsigned)grid_for((const void *)file_mean_kernel<R, false>, f * nch),
                                     kThreads, 0, st>>>(copies, f, d, ld, slot_mask, means, ldm, nch);
    }
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    // one row per file: row i = means[i], kept iff sel[i] == 0
    return launch_aggregate(means, f, 1, d, ldm, sel, det, mode, out, st);
}

}  // namespace

extern "C" aspis_status aspis_round_tolerant(const float *copies, int64_t d, int64_t ld,
                                             const aspis_assignment *a, float tau,
                                             uint32_t *file_neq, uint32_t *adj,
                                             aspis_detection *det, uint8_t *slot_mask,
                                             int8_t *sel, float *means, int64_t ldm, int mode,
                                             float *out, void *stream)
{
    if (!a || !a->dev_file_workers || a->r < 2 || a->K < a->r || a->f < 1) return ASPIS_E_INVAL;
    if (a->K > ASPIS_MAX_K || a->r > ASPIS_MAX_R) return ASPIS_E_RANGE;
    if (!copies || d < 1 || ld < d || !(tau >= 0.0f)) return ASPIS_E_INVAL;
    if (!file_neq || !adj || !det || !slot_mask || !sel || !means || ldm < d || !out) return ASPIS_E_INVAL;
    if (mode != 0 && mode != 1) return ASPIS_E_INVAL;
    if (a->f > ASPIS_MAX_AGG_FILES) return ASPIS_E_RANGE;
    if (ld > (INT64_MAX / 8) / (a->f * a->r) || ldm > (INT64_MAX / 8) / a->f) return ASPIS_E_RANGE;
    cudaStream_t st = (cudaStream_t)stream;
    if (cudaMemsetAsync(file_neq, 0, sizeof(uint32_t) * (size_t)a->f, st) != cudaSuccess)
        return ASPIS_E_CUDA;
    cudaError_t e;
#define ASPIS_TOL(RR, UU)                                                                        \
    e = launch_tolerant<RR, UU>(copies, a->f, d, ld, tau, file_neq, a->dev_file_workers, a->K, adj,  \
                                det, slot_mask, sel, means, ldm, mode, out, st);                    \
    break;
    switch (a->r) {
    case 2: ASPIS_TOL(2, 8)
    case 3: ASPIS_TOL(3, 4)
    case 4: ASPIS_TOL(4, 4)
    case 5: ASPIS_TOL(5, 3)
    case 6: ASPIS_TOL(6, 2)
    case 7: ASPIS_TOL(7, 2)
    default: ASPIS_TOL(8, 2)
    }
#undef ASPIS_TOL
    return e == cudaSuccess ? ASPIS_OK : ASPIS_E_CUDA;
}
