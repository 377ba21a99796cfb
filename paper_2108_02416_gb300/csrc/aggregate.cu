// Step 5 of the PS round: coordinate-wise aggregation of the chosen copies
// (Algorithm 1: median of the majority gradients; mean in Case 1).
//
// Persistent kernel.  A CTA (8 warps) owns a tile of TC consecutive
// coordinates for all n kept files.  The tile is staged in shared memory with
// 16-byte cp.async copies (double-buffered: tile t+grid is in flight while t
// is reduced).  Rows of the tile are TC floats; 16-byte chunks are XOR-
// swizzled by row so that the 32 lanes of a warp, reading 4 coordinates of 8
// consecutive rows, hit 32 different banks.
//
// Thread roles: warp w, lane = (cq = lane & 3, g8 = lane >> 2).  The warp
// covers coordinates 4*(w % CPR) + cq (CPR = TC/4 chunk columns) and file
// group ws*8 + g8 (ws = w / CPR); the WS = 8/CPR warps of one chunk column
// share its 4 coordinates and synchronise among themselves only (a named
// barrier; a plain warp sync when WS == 1).  Each lane visits the files
// i = gf, gf + G, ... (G = 8*WS).
//
// Lower median (exact, IEEE totalOrder via a monotone uint32 key):
//   pass A  convert the lane's values to keys in place; min/max per coordinate
//   pass H  histogram of the keys inside [lo, hi] over kNB equal-width bins;
//           the bin holding the target rank becomes the new [lo, hi]
//   pass C  once at most kCap keys remain in [lo, hi], copy them out and rank
//           them directly.
// A coordinate finishes when its range is one key or after pass C.  The key
// map is a bijection, so the output has the chosen element's exact bits.
#include "aspis_internal.cuh"

namespace aspis {
namespace {

constexpr int kThreads = 256;     // 8 warps
constexpr int kNB = 128;          // histogram bins per pass
constexpr int kLogNB = 7;
constexpr int kCap = 32;          // candidates ranked directly

__device__ __forceinline__ uint32_t to_key(uint32_t u)
{
    return u ^ ((uint32_t)((int32_t)u >> 31) | 0x80000000u);
}

__device__ __forceinline__ uint32_t from_key(uint32_t k)
{
    return k ^ ((uint32_t)((int32_t)~k >> 31) | 0x80000000u);
}

__device__ __forceinline__ void cp_async16(uint32_t saddr, const void *g)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(saddr), "l"(g));
}

__device__ __forceinline__ void cp_async4(uint32_t saddr, const void *g)
{
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;\n" ::"r"(saddr), "l"(g));
}

__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }

template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N)); }

// Sync of the warps sharing one chunk column (ids 1..8; 0 is __syncthreads).
template <int WS>
__device__ __forceinline__ void group_sync(int cw)
{
    if constexpr (WS == 1) {
        __syncwarp();
    } else {
        asm volatile("bar.sync %0, %1;\n" ::"r"(cw + 1), "r"(WS * 32) : "memory");
    }
}

// Two-sum: s + e == a + b exactly (Knuth); no products, so nothing to fuse.
__device__ __forceinline__ void two_sum(float a, float b, float &s, float &e)
{
    s = a + b;
    const float bp = s - a;
    e = (a - (s - bp)) + (b - bp);
}

struct Layout {
    // byte offsets into dynamic shared memory
    size_t tile0, tile1, rows, hist, cand, part, state, total;
};

template <int TC>
__host__ __device__ constexpr int groups_of() { return 8 * (8 / (TC / 4)); }

template <int TC>
__host__ __device__ inline Layout make_layout(int64_t f)
{
    constexpr int G = groups_of<TC>();
    Layout L{};
    size_t o = 0;
    const size_t tile = (size_t)f * TC * 4;
    L.tile0 = o; o += (tile + 127) / 128 * 128;
    L.tile1 = o; o += (tile + 127) / 128 * 128;
    L.rows = o; o += ((size_t)f * 4 + 15) / 16 * 16;
    L.hist = o; o += (size_t)kNB * TC * 4;
    L.cand = o; o += (size_t)TC * kCap * 4;
    L.part = o; o += (size_t)G * TC * 8;        // 8 bytes: float pairs for the mean
    L.state = o; o += (size_t)8 * TC * 4;
    L.total = o;
    return L;
}

template <int TC, bool VEC, int MODE>
__global__ void __launch_bounds__(kThreads, 1)
aggregate_kernel(const float *__restrict__ copies, int64_t f, int r, int64_t d, int64_t ld,
                 const int8_t *__restrict__ sel, aspis_detection *det, float *__restrict__ out)
{
    constexpr int CPR = TC / 4;            // 16-byte chunks per tile row
    constexpr int WS = 8 / CPR;            // warps per chunk column
    constexpr int G = 8 * WS;              // lanes (file groups) per coordinate
    constexpr int RPL = 32 / TC;           // tile rows per 128-byte line
    extern __shared__ __align__(128) unsigned char smem[];
    const Layout L = make_layout<TC>(f);
    uint32_t *tiles[2] = {reinterpret_cast<uint32_t *>(smem + L.tile0),
                          reinterpret_cast<uint32_t *>(smem + L.tile1)};
    int32_t *rows = reinterpret_cast<int32_t *>(smem + L.rows);
    uint32_t *hist = reinterpret_cast<uint32_t *>(smem + L.hist);      // [kNB][TC]
    uint32_t *cand = reinterpret_cast<uint32_t *>(smem + L.cand);      // [TC][kCap]
    uint32_t *part = reinterpret_cast<uint32_t *>(smem + L.part);      // [G][TC] (x2 for mean)
    uint32_t *st = reinterpret_cast<uint32_t *>(smem + L.state);
    uint32_t *s_lo = st, *s_hi = st + TC, *s_krem = st + 2 * TC, *s_cnt = st + 3 * TC;
    uint32_t *s_done = st + 4 * TC, *s_res = st + 5 * TC, *s_ccount = st + 6 * TC;
    __shared__ int warp_tot[kThreads / 32];

    const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
    const int cq = lane & 3, g8 = lane >> 2;
    const int cw = w % CPR, ws = w / CPR;
    const int cc = cw * 4 + cq;            // coordinate within the tile
    const int gf = ws * 8 + g8;            // file group of this lane

    // --- kept files: rows[k] = i*r + sel[i] for the k-th file with sel >= 0
    int n = 0;
    for (int64_t b0 = 0; b0 < f; b0 += kThreads) {
        const int64_t i = b0 + tid;
        const int s = i < f ? (int)sel[i] : -1;
        const unsigned m = __ballot_sync(0xffffffffu, s >= 0);
        if (lane == 0) warp_tot[w] = __popc(m);
        __syncthreads();
        int off = n;
        for (int q = 0; q < w; ++q) off += warp_tot[q];
        int tot = 0;
        for (int q = 0; q < kThreads / 32; ++q) tot += warp_tot[q];
        if (s >= 0) rows[off + __popc(m & ((1u << lane) - 1u))] = (int32_t)(i * r + s);
        n += tot;
        __syncthreads();
    }
    if (n == 0) {
        if (blockIdx.x == 0 && tid == 0) det->status = ASPIS_E_EMPTY;
        return;
    }
    const uint32_t krank = (uint32_t)((n - 1) / 2);

    const int64_t ntiles = (d + TC - 1) / TC;
    // lane's first element offset (in words) and its stride between files
    const int fl = (gf / RPL) & (CPR - 1);
    const int off0 = gf * TC + (((cc >> 2) ^ fl) << 2) + (cc & 3);
    const int stride = G * TC;
    const int nmine = n > gf ? (n - gf + G - 1) / G : 0;

    auto issue = [&](int64_t t, uint32_t *buf) {
        const int64_t c0 = t * TC;
        const uint32_t sbase = (uint32_t)__cvta_generic_to_shared(buf);
        if constexpr (VEC) {
            const int total = n * CPR;
            for (int e = tid; e < total; e += kThreads) {
                const int i = e / CPR, ch = e - i * CPR;
                const int64_t c = c0 + ch * 4;
                if (c < d) {
                    const int sw = ch ^ ((i / RPL) & (CPR - 1));
                    cp_async16(sbase + (uint32_t)(i * TC + sw * 4) * 4u,
                               copies + (int64_t)rows[i] * ld + c);
                }
            }
        } else {
            const int total = n * TC;
            for (int e = tid; e < total; e += kThreads) {
                const int i = e / TC, k = e - i * TC;
                const int64_t c = c0 + k;
                if (c < d) {
                    const int sw = (k >> 2) ^ ((i / RPL) & (CPR - 1));
                    cp_async4(sbase + (uint32_t)(i * TC + sw * 4 + (k & 3)) * 4u,
                              copies + (int64_t)rows[i] * ld + c);
                }
            }
        }
        cp_async_commit();
    };

    if (tid < TC) {
        s_lo[tid] = 0xffffffffu;
        s_hi[tid] = 0u;
    }
    int64_t t = blockIdx.x;
    int buf = 0;
    if (t < ntiles) issue(t, tiles[0]);
    for (; t < ntiles; t += gridDim.x) {
        const int64_t tn = t + gridDim.x;
        if (tn < ntiles) issue(tn, tiles[buf ^ 1]);
        else cp_async_commit();
        cp_async_wait<1>();
        __syncthreads();
        uint32_t *tile = tiles[buf];
        const int64_t c0 = t * TC;
        const bool live = c0 + cc < d;

        if constexpr (MODE == 1) {
            // ---- mean: compensated sums per lane, combined per coordinate
            float s = 0.f, e = 0.f;
            if (live) {
                const uint32_t *p = tile + off0;
                for (int j = 0; j < nmine; ++j, p += stride) {
                    float ns, ne;
                    two_sum(s, __uint_as_float(*p), ns, ne);
                    s = ns;
                    e += ne;
                }
            }
            float2 *pp = reinterpret_cast<float2 *>(part);
            pp[gf * TC + cc] = make_float2(s, e);
            group_sync<WS>(cw);
            if (gf == 0 && live) {
                float S = 0.f, E = 0.f;
                for (int q = 0; q < G; ++q) {
                    const float2 v = pp[q * TC + cc];
                    float ns, ne;
                    two_sum(S, v.x, ns, ne);
                    S = ns;
                    E += ne + v.y;
                }
                out[c0 + cc] = (float)(((double)S + (double)E) / (double)n);
            }
        } else {
            // ---- pass A: keys in place, min / max
            uint32_t mn = 0xffffffffu, mx = 0u;
            {
                uint32_t *p = tile + off0;
                for (int j = 0; j < nmine; ++j, p += stride) {
                    const uint32_t k = to_key(*p);
                    *p = k;
                    mn = min(mn, k);
                    mx = max(mx, k);
                }
            }
            mn = min(mn, __shfl_xor_sync(0xffffffffu, mn, 4));
            mx = max(mx, __shfl_xor_sync(0xffffffffu, mx, 4));
            mn = min(mn, __shfl_xor_sync(0xffffffffu, mn, 8));
            mx = max(mx, __shfl_xor_sync(0xffffffffu, mx, 8));
            mn = min(mn, __shfl_xor_sync(0xffffffffu, mn, 16));
            mx = max(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
            if (g8 == 0) {
                if constexpr (WS == 1) {
                    s_lo[cc] = mn;
                    s_hi[cc] = mx;
                } else {
                    atomicMin(&s_lo[cc], mn);
                    atomicMax(&s_hi[cc], mx);
                }
            }
            group_sync<WS>(cw);
            if (gf == 0) {
                s_krem[cc] = krank;
                s_cnt[cc] = (uint32_t)n;
                const bool single = s_lo[cc] == s_hi[cc];
                s_done[cc] = (!live || single) ? 1u : 0u;
                s_res[cc] = s_lo[cc];
            }
            group_sync<WS>(cw);

            for (;;) {
                const bool dn = s_done[cc] != 0u;
                const uint32_t lo = s_lo[cc], hi = s_hi[cc], cnt = s_cnt[cc];
                const bool compact = !dn && cnt <= (uint32_t)kCap;
                const bool hmode = !dn && !compact;
                const uint32_t W = hi - lo;
                const int bits = 32 - __clz(W);
                const int shift = hmode && bits > kLogNB ? bits - kLogNB : 0;
                if (hmode)
                    for (int b = gf; b < kNB; b += G) hist[b * TC + cc] = 0u;
                if (compact && gf == 0) s_ccount[cc] = 0u;
                group_sync<WS>(cw);
                if (!dn) {
                    const uint32_t *p = tile + off0;
                    if (compact) {
                        for (int j = 0; j < nmine; ++j, p += stride) {
                            const uint32_t k = *p;
                            if (k - lo <= W) cand[cc * kCap + atomicAdd(&s_ccount[cc], 1u)] = k;
                        }
                    } else {
                        for (int j = 0; j < nmine; ++j, p += stride) {
                            const uint32_t dk = *p - lo;
                            if (dk <= W) atomicAdd(&hist[(dk >> shift) * TC + cc], 1u);
                        }
                    }
                }
                group_sync<WS>(cw);
                if (hmode) {
                    constexpr int BPG = kNB / G;            // bins summed by each lane
                    uint32_t s = 0;
#pragma unroll
                    for (int b = 0; b < BPG; ++b) s += hist[(gf * BPG + b) * TC + cc];
                    part[gf * TC + cc] = s;
                } else if (compact) {
                    const uint32_t krem = s_krem[cc];
                    for (uint32_t m = gf; m < cnt; m += G) {
                        const uint32_t x = cand[cc * kCap + m];
                        uint32_t lt = 0, le = 0;
                        for (uint32_t q = 0; q < cnt; ++q) {
                            const uint32_t y = cand[cc * kCap + q];
                            lt += y < x;
                            le += y <= x;
                        }
                        if (lt <= krem && krem < le) s_res[cc] = x;
                    }
                }
                group_sync<WS>(cw);
                if (gf == 0) {
                    if (hmode) {
                        constexpr int BPG = kNB / G;
                        uint32_t krem = s_krem[cc];
                        int g = 0;
                        for (; g < G - 1; ++g) {
                            const uint32_t v = part[g * TC + cc];
                            if (krem < v) break;
                            krem -= v;
                        }
                        int b = g * BPG;
                        for (; b < g * BPG + BPG - 1; ++b) {
                            const uint32_t v = hist[b * TC + cc];
                            if (krem < v) break;
                            krem -= v;
                        }
                        const uint32_t nlo = lo + ((uint32_t)b << shift);
                        const uint64_t top = (uint64_t)nlo + ((1ull << shift) - 1ull);
                        const uint32_t nhi = top < (uint64_t)hi ? (uint32_t)top : hi;
                        s_lo[cc] = nlo;
                        s_hi[cc] = nhi;
                        s_krem[cc] = krem;
                        s_cnt[cc] = hist[b * TC + cc];
                        if (nlo == nhi) {
                            s_done[cc] = 1u;
                            s_res[cc] = nlo;
                        }
                    } else if (compact) {
                        s_done[cc] = 1u;
                    }
                }
                group_sync<WS>(cw);
                const int base = cw * 4;
                if (s_done[base] & s_done[base + 1] & s_done[base + 2] & s_done[base + 3]) break;
            }
            if (gf == 0 && live) out[c0 + cc] = __uint_as_float(from_key(s_res[cc]));
            if (gf == 0) {
                s_lo[cc] = 0xffffffffu;
                s_hi[cc] = 0u;
            }
        }
        __syncthreads();
        buf ^= 1;
    }
    cp_async_wait<0>();
}

template <int TC, bool VEC, int MODE>
cudaError_t launch_tc(const float *copies, int64_t f, int r, int64_t d, int64_t ld,
                      const int8_t *sel, aspis_detection *det, float *out, cudaStream_t stream)
{
    const Layout L = make_layout<TC>(f);
    auto kern = aggregate_kernel<TC, VEC, MODE>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)L.total);
    if (e != cudaSuccess) return e;
    const int64_t ntiles = (d + TC - 1) / TC;
    int64_t grid = sm_count();
    if (grid > ntiles) grid = ntiles;
    kern<<<(unsigned)grid, kThreads, L.total, stream>>>(copies, f, r, d, ld, sel, det, out);
    return cudaGetLastError();
}

template <bool VEC, int MODE>
cudaError_t launch_mode(int tc, const float *copies, int64_t f, int r, int64_t d, int64_t ld,
                        const int8_t *sel, aspis_detection *det, float *out, cudaStream_t stream)
{
    switch (tc) {
    case 32: return launch_tc<32, VEC, MODE>(copies, f, r, d, ld, sel, det, out, stream);
    case 16: return launch_tc<16, VEC, MODE>(copies, f, r, d, ld, sel, det, out, stream);
    case 8: return launch_tc<8, VEC, MODE>(copies, f, r, d, ld, sel, det, out, stream);
    default: return launch_tc<4, VEC, MODE>(copies, f, r, d, ld, sel, det, out, stream);
    }
}

// Largest tile width whose double-buffered tile fits in shared memory.
int pick_tc(int64_t f, size_t smem_cap)
{
    if (make_layout<32>(f).total <= smem_cap) return 32;
    if (make_layout<16>(f).total <= smem_cap) return 16;
    if (make_layout<8>(f).total <= smem_cap) return 8;
    if (make_layout<4>(f).total <= smem_cap) return 4;
    return 0;
}

}  // namespace

size_t aggregate_smem_bytes(int64_t f, int *tc_out)
{
    int dev = 0, cap = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&cap, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    const int tc = pick_tc(f, (size_t)cap - 1024);
    if (tc_out) *tc_out = tc;
    if (!tc) return 0;
    switch (tc) {
    case 32: return make_layout<32>(f).total;
    case 16: return make_layout<16>(f).total;
    case 8: return make_layout<8>(f).total;
    default: return make_layout<4>(f).total;
    }
}

cudaError_t launch_aggregate(const float *copies, int64_t f, int r, int64_t d, int64_t ld,
                             const int8_t *sel, aspis_detection *det, int mode, float *out,
                             cudaStream_t stream)
{
    int tc = 0;
    if (!aggregate_smem_bytes(f, &tc) || !tc) return cudaErrorInvalidValue;
    const bool vec = ((uintptr_t)copies % 16 == 0) && (ld % 4 == 0);
    if (vec)
        return mode == 0 ? launch_mode<true, 0>(tc, copies, f, r, d, ld, sel, det, out, stream)
                         : launch_mode<true, 1>(tc, copies, f, r, d, ld, sel, det, out, stream);
    return mode == 0 ? launch_mode<false, 0>(tc, copies, f, r, d, ld, sel, det, out, stream)
                     : launch_mode<false, 1>(tc, copies, f, r, d, ld, sel, det, out, stream);
}

}  // namespace aspis
