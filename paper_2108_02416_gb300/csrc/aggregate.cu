// Step 5 of the PS round: coordinate-wise aggregation of the chosen copies
// (Algorithm 1: median of the majority gradients; mean in Case 1).
//
// Data path.  Persistent CTAs of 8 warps.  A tile is TC consecutive
// coordinates of all n kept rows.  It is staged in shared memory by 16-byte
// cp.async copies in which consecutive lanes fetch one row's 16*TC/4 bytes,
// so every memory request carries whole lines (a gather of 16-byte pieces of
// many rows runs ~10x below the streaming rate).  Either two CTAs share an SM
// with one tile each (their load and reduce phases overlap), or one CTA
// keeps STAGES tiles in flight.  Rows of a tile are TC floats; the 16-byte
// chunks of row i are XOR-swizzled by (i / (32/TC)) so that the reads below
// are conflict-free.
//
// Compute.  Warp w takes the 4 coordinates of chunk column cw = w % (TC/4);
// the WS = 8/(TC/4) warps of a column split the rows.  Lane = (cq = lane & 3,
// g8 = lane >> 2): coordinate cq of the column, rows i = gf, gf + G, ...
// with gf = 8*(w / (TC/4)) + g8 and G = 8*WS.  The G lanes of one
// coordinate hold identical copies of its search state.  Every barrier and
// warp collective below is reached by all lanes; per-coordinate decisions
// only predicate the state updates.
//
// Lower median, exact (IEEE totalOrder through a monotone uint32 key; the
// key map is a bijection, so the output has the chosen element's bits).  Per
// coordinate, a small state machine:
//   VH  value-space histogram: 128 bins, bins 1..126 evenly over the range of
//       a sample (two values per lane), 0 / 127 catching everything below /
//       above.  The bin map x -> bits(fma(x, s, c)) - bits(2^23), clamped,
//       is monotone in totalOrder, so bins are contiguous value ranges; each
//       value's bin is also kept as a byte.  A scan over the coordinate's
//       lanes finds the bin holding the target rank.  (Key-space bins cannot
//       do this in one pass: values of both signs near zero span ~2^31 keys.)
//   VC  each lane compares its bytes with that bin (branch-free, 32 rows at
//       a time into a bit mask; rows past n hold a byte no bin has), the
//       members' keys are stored at a prefix over the coordinate's lanes and
//       the <= 32 of them are ranked directly.
//   VM  a bin with more than 32 members: their exact key range [lo, hi];
//   VR  value-space bins over that range for the members only (every other
//       tag becomes 0xFF), then VC or VM again.  At most two such levels,
//       each at least 4x smaller; otherwise key-space passes on [lo, hi].
// Exact key-space fallback, taken when the sample range is degenerate or not
// finite, a NaN is seen or refinement stalls:
//   KA  min / max of the keys -> range [lo, hi]
//   KH  128 equal-width key-space bins over [lo, hi]; the bin holding the
//       rank becomes [lo, hi] (each pass shrinks the range by at least 2^6)
//   KC  the keys left in [lo, hi] are gathered with warp ballots and ranked.
// One pass body serves every mode; it is instantiated three times: a VH-only
// pass and a VC-only pass that every tile runs first (the common case ends
// there), and the general pass, looped only while a coordinate is left.  The
// pass cap only guards against an inconsistent state.
#include <climits>
#include <type_traits>

#include "aspis_internal.cuh"
#include "median_common.cuh"

namespace aspis {
namespace {

constexpr int kThreads = 256;     // 8 warps
constexpr int kWarps = kThreads / 32;
constexpr int kHistStride = kNB + 4;   // words per coordinate row (rows start 4 banks apart)
constexpr int kListStride = kCap + 1;

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

// Sync of the WS warps of one chunk column (barrier ids 1..8; 0 is __syncthreads).
template <int WS>
__device__ __forceinline__ void col_sync(int cw)
{
    if constexpr (WS == 1) {
        __syncwarp();
    } else {
        asm volatile("bar.sync %0, %1;\n" ::"r"(cw + 1), "r"(WS * 32) : "memory");
    }
}

struct Layout {
    size_t tiles, bins, rows, hist, list, lcnt, red, state, total, tile_bytes;
};

template <int TC>
__host__ __device__ inline int bin_row(int64_t f)
{
    // tag bytes per lane: its rows' tags are contiguous, four per word; an odd
    // word count puts the 32 lanes of a warp in 32 different banks
    constexpr int G = 8 * (kWarps / (TC / 4));
    const int rows = (int)((f + G - 1) / G);
    int words = (rows + 3) / 4;
    if ((words & 1) == 0) ++words;
    return words * 4;
}

template <int TC, int STAGES>
__host__ __device__ inline Layout make_layout(int64_t f)
{
    constexpr int WS = kWarps / (TC / 4);
    Layout L{};
    size_t o = 0;
    L.tile_bytes = ((size_t)f * TC * 4 + 127) / 128 * 128;
    L.tiles = o; o += STAGES * L.tile_bytes;
    L.bins = o; o += ((size_t)TC * 8 * WS * bin_row<TC>(f) + 15) / 16 * 16;
    L.rows = o; o += ((size_t)f * 4 + 15) / 16 * 16;
    L.hist = o; o += (size_t)TC * kHistStride * 4;
    L.list = o; o += (size_t)TC * WS * kListStride * 4;
    L.lcnt = o; o += (size_t)TC * WS * 4;
    L.red = o; o += (size_t)TC * WS * 8;
    L.state = o; o += (size_t)TC * 8 * 4;
    L.total = o;
    return L;
}

template <int TC, int STAGES, int MINB, bool VEC, int MODE>
__global__ void __launch_bounds__(kThreads, MINB)
aggregate_kernel(const float *__restrict__ copies, int64_t f, int r, int64_t d, int64_t ld,
                 const int8_t *__restrict__ sel, aspis_detection *det, float *__restrict__ out)
{
    constexpr int CPR = TC / 4;            // 16-byte chunks (= chunk columns) per tile row
    constexpr int WS = kWarps / CPR;       // warps per chunk column
    constexpr int G = 8 * WS;              // lanes per coordinate
    constexpr int RPL = 32 / TC;           // tile rows per 128-byte line
    constexpr int BPL = kNB / G;           // histogram bins summed per lane (16, 8, 4, 2)
    constexpr int RPI = kThreads / CPR;    // tile rows covered by one copy round
    extern __shared__ __align__(128) unsigned char smem[];
    const Layout L = make_layout<TC, STAGES>(f);
    unsigned char *tiles = smem + L.tiles;
    uint8_t *bins = smem + L.bins;                                    // [WS][TC][8][JP] tags
    int32_t *rows = reinterpret_cast<int32_t *>(smem + L.rows);
    uint32_t *hist = reinterpret_cast<uint32_t *>(smem + L.hist);     // [TC][kHistStride]
    uint32_t *list = reinterpret_cast<uint32_t *>(smem + L.list);     // [TC][WS][kListStride]
    uint32_t *lcnt = reinterpret_cast<uint32_t *>(smem + L.lcnt);     // [TC][WS]
    uint32_t *red = reinterpret_cast<uint32_t *>(smem + L.red);       // [TC][WS][2]
    uint32_t *st = reinterpret_cast<uint32_t *>(smem + L.state);      // [8][TC]
    __shared__ int warp_tot[kWarps];

    const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
    const int cq = lane & 3, g8 = lane >> 2;
    const int cw = w % CPR, ws = w / CPR;
    const int cc = cw * 4 + cq;            // coordinate within the tile
    const int gf = ws * 8 + g8;            // file group of this lane
    const unsigned full = 0xffffffffu;
    const unsigned seg = 0x11111111u << cq;                  // lanes of this coordinate
    const unsigned below = (1u << lane) - 1u;

    // ---- kept files: rows[k] = i*r + sel[i] for the k-th file with sel >= 0
    int n = 0;
    for (int64_t b0 = 0; b0 < f; b0 += kThreads) {
        const int64_t i = b0 + tid;
        const int s = i < f ? (int)sel[i] : -1;
        const unsigned m = __ballot_sync(full, s >= 0);
        if (lane == 0) warp_tot[w] = __popc(m);
        __syncthreads();
        int off = n, tot = 0;
        for (int q = 0; q < kWarps; ++q) {
            off += q < w ? warp_tot[q] : 0;
            tot += warp_tot[q];
        }
        if (s >= 0) rows[off + __popc(m & below)] = (int32_t)(i * r + s);
        n += tot;
        __syncthreads();
    }
    if (n == 0) {
        if (blockIdx.x == 0 && tid == 0) det->status = ASPIS_E_EMPTY;
        return;
    }
    const uint32_t krank = (uint32_t)((n - 1) / 2);
    const int64_t ntiles = (d + TC - 1) / TC;

    // lane's first element (in words) and the stride between its rows
    const int fl = (gf / RPL) & (CPR - 1);
    const int off0 = gf * TC + ((cw ^ fl) << 2) + cq;
    constexpr int kStride = G * TC;
    const int JP = bin_row<TC>(f);
    const int nmine = n > gf ? (n - gf + G - 1) / G : 0;

    // copy role (vector path): this thread always moves chunk ch_me of rows
    // i0_me + RPI*k; its swizzled chunk is the same for all of them
    const int ch_me = tid % CPR, i0_me = tid / CPR;
    const int sw_me = ch_me ^ ((i0_me / RPL) & (CPR - 1));

    auto issue = [&](int64_t t, int stage) {
        if (t < ntiles) {
            const int64_t c0 = t * TC;
            const uint32_t sbase = (uint32_t)__cvta_generic_to_shared(tiles + stage * L.tile_bytes);
            if constexpr (VEC) {
                const int64_t c = c0 + ch_me * 4;
                if (c < d) {
                    const float *src = copies + c;
                    uint32_t dst = sbase + (uint32_t)(i0_me * TC + sw_me * 4) * 4u;
                    int i = i0_me;
                    for (; i + 3 * RPI < n; i += 4 * RPI, dst += 4 * RPI * TC * 4) {
                        const int32_t r0 = rows[i], r1 = rows[i + RPI];
                        const int32_t r2 = rows[i + 2 * RPI], r3 = rows[i + 3 * RPI];
                        cp_async16(dst, src + (int64_t)r0 * ld);
                        cp_async16(dst + RPI * TC * 4, src + (int64_t)r1 * ld);
                        cp_async16(dst + 2 * RPI * TC * 4, src + (int64_t)r2 * ld);
                        cp_async16(dst + 3 * RPI * TC * 4, src + (int64_t)r3 * ld);
                    }
                    for (; i < n; i += RPI, dst += RPI * TC * 4)
                        cp_async16(dst, src + (int64_t)rows[i] * ld);
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
        }
        cp_async_commit();
    };

    const int64_t t0 = blockIdx.x;
    // One stage: the next tile is fetched into the same buffer as soon as this
    // one is no longer read (after the list pass, when no coordinate needs
    // the general passes), else at the end of the tile.  More stages: tile
    // t + (STAGES-1) grids is fetched when tile t starts.
    if constexpr (STAGES == 1) {
        issue(t0, 0);
    } else {
#pragma unroll
        for (int s = 0; s < STAGES - 1; ++s) issue(t0 + (int64_t)s * gridDim.x, s);
    }

    int stage = 0;
    for (int64_t t = t0; t < ntiles; t += gridDim.x) {
        if constexpr (STAGES > 1)
            issue(t + (int64_t)(STAGES - 1) * gridDim.x, (stage + STAGES - 1) % STAGES);
        bool fetched = false;             // the next tile is on its way (one stage)
        cp_async_wait<STAGES - 1>();
        __syncthreads();
        uint32_t *tile = reinterpret_cast<uint32_t *>(tiles + stage * L.tile_bytes);
        const int64_t c0 = t * TC;
        const bool live = c0 + cc < d;

        if constexpr (MODE == 1) {
            // ---- mean: compensated per-lane sums, combined in a fixed order
            float s = 0.f, e = 0.f;
            const uint32_t *p = tile + off0;
            for (int j = 0; j < nmine; ++j, p += kStride) {
                float ns, ne;
                two_sum(s, __uint_as_float(*p), ns, ne);
                s = ns;
                e += ne;
            }
#pragma unroll
            for (int o = 4; o < 32; o <<= 1) {
                const float os = __shfl_xor_sync(full, s, o);
                const float oe = __shfl_xor_sync(full, e, o);
                float ns, ne;
                two_sum(s, os, ns, ne);
                s = ns;
                e += ne + oe;
            }
            if constexpr (WS > 1) {
                if (g8 == 0) {
                    red[(cc * WS + ws) * 2] = __float_as_uint(s);
                    red[(cc * WS + ws) * 2 + 1] = __float_as_uint(e);
                }
                col_sync<WS>(cw);
                s = 0.f;
                e = 0.f;
                for (int u = 0; u < WS; ++u) {
                    float ns, ne;
                    two_sum(s, __uint_as_float(red[(cc * WS + u) * 2]), ns, ne);
                    s = ns;
                    e += ne + __uint_as_float(red[(cc * WS + u) * 2 + 1]);
                }
            }
            if (gf == 0 && live) out[c0 + cc] = (float)(((double)s + (double)e) / (double)n);
        } else {
            // ---- sample range: the first two values of each lane of the
            // coordinate; bins 1..kNB-2 split [min, max] of the sample evenly
            uint32_t slo = 0xffffffffu, shi = 0u;
            if (nmine > 0) {
                const uint32_t k = to_key(tile[off0]);
                slo = min(slo, k);
                shi = max(shi, k);
            }
            if (nmine > 1) {
                const uint32_t k = to_key(tile[off0 + kStride]);
                slo = min(slo, k);
                shi = max(shi, k);
            }
#pragma unroll
            for (int o = 4; o < 32; o <<= 1) {
                slo = min(slo, __shfl_xor_sync(full, slo, o));
                shi = max(shi, __shfl_xor_sync(full, shi, o));
            }
            if constexpr (WS > 1) {
                if (g8 == 0) {
                    red[(cc * WS + ws) * 2] = slo;
                    red[(cc * WS + ws) * 2 + 1] = shi;
                }
                if (gf == 0) st[4 * TC + cc] = 0u;     // NaN flag of this tile
                col_sync<WS>(cw);
                for (int u = 0; u < WS; ++u) {
                    slo = min(slo, red[(cc * WS + u) * 2]);
                    shi = max(shi, red[(cc * WS + u) * 2 + 1]);
                }
                col_sync<WS>(cw);
            }
            const float xs_lo = __uint_as_float(from_key(slo));
            const float xs_hi = __uint_as_float(from_key(shi));
            const float vs = (float)(kNB - 2) / (xs_hi - xs_lo);
            const float vc = 8388609.0f - xs_lo * vs;    // xs_lo -> about 2^23 + 1
            float rs = 0.f, rc = 0.f;                    // bin map of the refinement passes
            const bool vspace = isfinite(xs_lo) && isfinite(xs_hi) && xs_hi > xs_lo &&
                                isfinite(vs) && isfinite(vc);

            int mode = !live ? M_DONE : (vspace ? M_VH : M_KA);
            uint32_t lo = 0u, hi = 0u, krem = krank, cnt = (uint32_t)n, res = 0u, vb = 0u;
            int vr_levels = 0;
            // this lane's tags, one byte per row, contiguous
            uint8_t *bmine = bins + ((ws * TC + cc) * 8 + g8) * JP;

            auto pass = [&](auto kind) {

                constexpr int K = decltype(kind)::value;   // 0 all modes, 1 VH only, 2 VC only
                const int m0 = mode;
                const bool cmode = m0 == M_VC || m0 == M_KC;
                const uint32_t W = hi - lo;
                const int bits = 32 - __clz(W);
                const int sh = bits > kLogNB ? bits - kLogNB : 0;
                uint32_t *h = hist + cc * kHistStride;
                if (K != 2 && (m0 == M_VH || m0 == M_KH || m0 == M_VR))
                    for (int b = gf * 4; b < kNB; b += G * 4)
                        *reinterpret_cast<uint4 *>(h + b) = make_uint4(0u, 0u, 0u, 0u);
                col_sync<WS>(cw);

                // ---- sweep over the lane's values
                const uint32_t *p = tile + off0;
                uint32_t amin = 0xffffffffu, amax = 0u;
                bool nanf = false;
                if (K != 2 && m0 == M_VH) {
                    uint32_t *pb = reinterpret_cast<uint32_t *>(bmine);
                    int j = 0;
                    for (; j + 4 <= nmine; j += 4, p += 4 * kStride, ++pb) {
                        const float y0 = fmaf(__uint_as_float(p[0]), vs, vc);
                        const float y1 = fmaf(__uint_as_float(p[kStride]), vs, vc);
                        const float y2 = fmaf(__uint_as_float(p[2 * kStride]), vs, vc);
                        const float y3 = fmaf(__uint_as_float(p[3 * kStride]), vs, vc);
                        nanf |= (y0 != y0) | (y1 != y1) | (y2 != y2) | (y3 != y3);
                        const uint32_t b0 = vbin(y0), b1 = vbin(y1), b2 = vbin(y2), b3 = vbin(y3);
                        atomicAdd(h + b0, 1u);
                        atomicAdd(h + b1, 1u);
                        atomicAdd(h + b2, 1u);
                        atomicAdd(h + b3, 1u);
                        *pb = b0 | (b1 << 8) | (b2 << 16) | (b3 << 24);
                    }
                    if (j < nmine) {
                        // last, partial word: missing rows get tag 0xFF, which no bin has
                        uint32_t word = 0xFFFFFFFFu;
                        for (int q = 0; j < nmine; ++j, ++q, p += kStride) {
                            const float y = fmaf(__uint_as_float(*p), vs, vc);
                            nanf |= y != y;
                            const uint32_t b = vbin(y);
                            atomicAdd(h + b, 1u);
                            word = (word & ~(0xFFu << (8 * q))) | (b << (8 * q));
                        }
                        *pb = word;
                    }
                }
                if constexpr (K == 0) {
                if (m0 == M_KA) {
                    for (int j = 0; j < nmine; ++j, p += kStride) {
                        const uint32_t k = to_key(*p);
                        amin = min(amin, k);
                        amax = max(amax, k);
                    }
                } else if (m0 == M_KH) {
                    for (int j = 0; j < nmine; ++j, p += kStride) {
                        const uint32_t dk = to_key(*p) - lo;
                        if (dk <= W) atomicAdd(h + (dk >> sh), 1u);
                    }
                }
                }
                // VC: one 32-bit load tests four of the lane's rows against the
                // bin; members are counted, stored at a prefix over the
                // coordinate's lanes, and only the words holding one are revisited
                if constexpr (K != 1) {
                if (__any_sync(full, m0 == M_VC)) {
                    uint32_t *lst = list + (cc * WS + ws) * kListStride;
                    const uint32_t *pw = reinterpret_cast<const uint32_t *>(bmine);
                    const uint32_t vbx = vb * 0x01010101u;
                    const int nw = m0 == M_VC ? (nmine + 3) >> 2 : 0;
                    uint32_t nm = 0u, wm = 0u;
#pragma unroll 4
                    for (int q = 0; q < nw; ++q) {
                        const uint32_t z = tag_match(pw[q], vbx);
                        nm += __popc(z);
                        wm |= (q < 32 && z != 0u) ? 1u << q : 0u;
                    }
                    uint32_t incl = nm;
#pragma unroll
                    for (int o = 1; o < 8; o <<= 1) {
                        const uint32_t tv = __shfl_up_sync(full, incl, 4 * o);
                        if (g8 >= o) incl += tv;
                    }
                    const uint32_t tot = __shfl_sync(full, incl, 28 + cq);
                    uint32_t pos = incl - nm;
                    for (; wm; wm &= wm - 1) {
                        const int q = __ffs(wm) - 1;
                        for (uint32_t z = tag_match(pw[q], vbx); z; z &= z - 1)
                            lst[pos++] = to_key(tile[off0 + (q * 4 + ((__ffs(z) - 1) >> 3)) * kStride]);
                    }
                    for (int q = 32; q < nw; ++q)            // rows past 128 of a lane
                        for (uint32_t z = tag_match(pw[q], vbx); z; z &= z - 1)
                            lst[pos++] = to_key(tile[off0 + (q * 4 + ((__ffs(z) - 1) >> 3)) * kStride]);
                    if (m0 == M_VC && g8 == 0) lcnt[cc * WS + ws] = tot;
                }
                }
                if constexpr (K == 2 && STAGES == 1) {
                    // every warp is past the tile unless a coordinate still
                    // needs the general passes (which read it)
                    if (!__syncthreads_or(m0 != M_VC && m0 != M_DONE)) {
                        issue(t + gridDim.x, 0);
                        fetched = true;
                    }
                }
                if constexpr (K == 0) {
                // VM: key range of the members of bin vb (too many to list)
                if (__any_sync(full, m0 == M_VM)) {
                    uint32_t kmin = 0xffffffffu, kmax = 0u;
                    if (m0 == M_VM)
                        for (int j = 0; j < nmine; ++j)
                            if (bmine[j] == vb) {
                                const uint32_t k = to_key(tile[off0 + j * kStride]);
                                kmin = min(kmin, k);
                                kmax = max(kmax, k);
                            }
#pragma unroll
                    for (int o = 4; o < 32; o <<= 1) {
                        kmin = min(kmin, __shfl_xor_sync(full, kmin, o));
                        kmax = max(kmax, __shfl_xor_sync(full, kmax, o));
                    }
                    if constexpr (WS > 1) {
                        if (g8 == 0 && m0 == M_VM) {
                            red[(cc * WS + ws) * 2] = kmin;
                            red[(cc * WS + ws) * 2 + 1] = kmax;
                        }
                        col_sync<WS>(cw);
                        if (m0 == M_VM)
                            for (int u = 0; u < WS; ++u) {
                                kmin = min(kmin, red[(cc * WS + u) * 2]);
                                kmax = max(kmax, red[(cc * WS + u) * 2 + 1]);
                            }
                        col_sync<WS>(cw);
                    }
                    if (m0 == M_VM) {
                        // members are the values with keys in [kmin, kmax]: bins are
                        // contiguous value ranges at every level
                        lo = kmin;
                        hi = kmax;
                        if (lo == hi) {
                            res = lo;
                            mode = M_DONE;
                        } else {
                            const float xlo = __uint_as_float(from_key(kmin));
                            const float xhi = __uint_as_float(from_key(kmax));
                            rs = (float)(kNB - 2) / (xhi - xlo);
                            rc = 8388609.0f - xlo * rs;
                            mode = isfinite(rs) && isfinite(rc) && rs > 0.f ? M_VR : M_KH;
                        }
                    }
                }
                // VR: value-space bins over [kmin, kmax] for the members only;
                // every other tag becomes 0xFF, which no bin has
                if (m0 == M_VR) {
                    uint8_t *pbr = bmine;
                    for (int j = 0; j < nmine; ++j, ++pbr) {
                        uint32_t b = 0xFFu;
                        if (*pbr == vb) {
                            b = vbin(fmaf(__uint_as_float(tile[off0 + j * kStride]), rs, rc));
                            atomicAdd(h + b, 1u);
                        }
                        *pbr = (uint8_t)b;
                    }
                }
                // KC (fallback): ballot-gathered list of the keys in [lo, hi]
                if (__any_sync(full, m0 == M_KC)) {
                    uint32_t *lst = list + (cc * WS + ws) * kListStride;
                    const int iters = (int)__reduce_max_sync(full, m0 == M_KC ? (unsigned)nmine : 0u);
                    const uint32_t *pc = tile + off0;
                    uint32_t nlist = 0u;
                    for (int j = 0; j < iters; ++j, pc += kStride) {
                        const bool pk = m0 == M_KC && j < nmine && to_key(*pc) - lo <= W;
                        const unsigned m = __ballot_sync(full, pk);
                        if (m) {
                            if (pk) lst[nlist + __popc(m & seg & below)] = to_key(*pc);
                            nlist += __popc(m & seg);
                        }
                    }
                    if (m0 == M_KC && g8 == 0) lcnt[cc * WS + ws] = nlist;
                }
                }
                bool nan_any = false;
                if constexpr (WS == 1) {
                    nan_any = (__ballot_sync(full, nanf) & seg) != 0u;
                } else {
                    if (nanf) atomicOr(&st[4 * TC + cc], 1u);
                }
                col_sync<WS>(cw);
                if constexpr (WS > 1) nan_any = st[4 * TC + cc] != 0u;

                if constexpr (K == 0) {
                // ---- key range of the fallback path (pass KA)
                if (__any_sync(full, m0 == M_KA)) {
#pragma unroll
                    for (int o = 4; o < 32; o <<= 1) {
                        amin = min(amin, __shfl_xor_sync(full, amin, o));
                        amax = max(amax, __shfl_xor_sync(full, amax, o));
                    }
                    if constexpr (WS > 1) {
                        if (g8 == 0) {
                            red[(cc * WS + ws) * 2] = amin;
                            red[(cc * WS + ws) * 2 + 1] = amax;
                        }
                        col_sync<WS>(cw);
                        for (int u = 0; u < WS; ++u) {
                            amin = min(amin, red[(cc * WS + u) * 2]);
                            amax = max(amax, red[(cc * WS + u) * 2 + 1]);
                        }
                        col_sync<WS>(cw);
                    }
                    if (m0 == M_KA) {
                        lo = amin;
                        hi = amax;
                        krem = krank;
                        cnt = (uint32_t)n;
                        if (lo == hi) {
                            res = lo;
                            mode = M_DONE;
                        } else {
                            mode = cnt <= (uint32_t)kCap ? M_KC : M_KH;
                        }
                    }
                }

                }
                // ---- bin search (value-space or key-space histogram)
                const bool hm = m0 == M_VH || m0 == M_KH || m0 == M_VR;
                uint32_t nbin = 0, nrr = 0, ncb = 0;
                if constexpr (K != 2) {
                if constexpr (WS == 1) {
                    if (__any_sync(full, hm)) {
                        // level 1: lane g8 sums bins [16*g8, 16*g8 + 16); scan over g8
                        uint32_t sum = 0;
#pragma unroll
                        for (int b = 0; b < BPL; b += 4) {
                            const uint4 v = *reinterpret_cast<const uint4 *>(h + g8 * BPL + b);
                            sum += (v.x + v.y) + (v.z + v.w);
                        }
                        uint32_t incl = sum;
#pragma unroll
                        for (int o = 1; o < 8; o <<= 1) {
                            const uint32_t tv = __shfl_up_sync(full, incl, 4 * o);
                            if (g8 >= o) incl += tv;
                        }
                        const unsigned m1 = __ballot_sync(full, incl > krem) & seg;
                        const int owner = m1 ? __ffs(m1) - 1 : cq;
                        const uint32_t before = __shfl_sync(full, incl - sum, owner);
                        const int og = owner >> 2;
                        // level 2: lane g8 takes 2 bins of the owner's 16
                        const uint2 c = *reinterpret_cast<const uint2 *>(h + og * BPL + g8 * 2);
                        const uint32_t s2 = c.x + c.y;
                        uint32_t incl2 = s2;
#pragma unroll
                        for (int o = 1; o < 8; o <<= 1) {
                            const uint32_t tv = __shfl_up_sync(full, incl2, 4 * o);
                            if (g8 >= o) incl2 += tv;
                        }
                        const uint32_t r2 = krem - before;
                        const unsigned m2 = __ballot_sync(full, incl2 > r2) & seg;
                        const int owner2 = m2 ? __ffs(m2) - 1 : cq;
                        uint32_t rr = r2 - (incl2 - s2), cb = c.y;
                        int b = 1;
                        if (rr < c.x) {
                            b = 0;
                            cb = c.x;
                        } else {
                            rr -= c.x;
                        }
                        const uint32_t bin = (uint32_t)(og * BPL + g8 * 2 + b);
                        nbin = __shfl_sync(full, bin, owner2);
                        nrr = __shfl_sync(full, rr, owner2);
                        ncb = __shfl_sync(full, cb, owner2);
                    }
                } else {
                    // WS warps per coordinate: per-lane partial sums through shared
                    // memory (the coordinate's list area is free here), then the
                    // lane with gf == 0 finishes the search
                    uint32_t *part = list + cc * WS * kListStride;    // G <= WS * kListStride
                    if (hm) {
                        uint32_t sum = 0;
#pragma unroll
                        for (int b = 0; b < BPL; ++b) sum += h[gf * BPL + b];
                        part[gf] = sum;
                    }
                    col_sync<WS>(cw);
                    if (hm && gf == 0) {
                        uint32_t rr = krem;
                        int g = 0;
                        for (; g < G - 1; ++g) {
                            if (rr < part[g]) break;
                            rr -= part[g];
                        }
                        int b = g * BPL;
                        for (; b < g * BPL + BPL - 1; ++b) {
                            if (rr < h[b]) break;
                            rr -= h[b];
                        }
                        st[0 * TC + cc] = (uint32_t)b;
                        st[1 * TC + cc] = rr;
                        st[2 * TC + cc] = h[b];
                    }
                    col_sync<WS>(cw);
                    nbin = st[0 * TC + cc];
                    nrr = st[1 * TC + cc];
                    ncb = st[2 * TC + cc];
                }
                }
                if (K != 2 && (m0 == M_VH || m0 == M_VR)) {
                    if (nan_any) {
                        mode = M_KA;             // exact key-space passes instead
                    } else if (m0 == M_VR && ncb > (uint32_t)kCap &&
                               (4u * ncb > cnt || ++vr_levels >= 2)) {
                        // little progress (values spread over many scales, say):
                        // key-space bins on the members' range [lo, hi] instead
                        mode = M_KH;
                    } else {
                        vb = nbin;
                        krem = nrr;
                        cnt = ncb;
                        mode = ncb <= (uint32_t)kCap ? M_VC : M_VM;
                    }
                } else if (K == 0 && m0 == M_KH) {
                    const uint32_t nlo = lo + (nbin << sh);
                    const uint64_t top = (uint64_t)nlo + ((1ull << sh) - 1ull);
                    hi = top < (uint64_t)hi ? (uint32_t)top : hi;
                    lo = nlo;
                    krem = nrr;
                    cnt = ncb;
                    if (lo == hi) {
                        res = lo;
                        mode = M_DONE;
                    } else {
                        mode = cnt <= (uint32_t)kCap ? M_KC : M_KH;
                    }
                }

                // ---- rank the listed keys: lane gf takes entries gf, gf+G, ...
                bool any = false;
                uint32_t hit = 0u;
                if constexpr (WS == 1) {
                    if (K != 1 && __any_sync(full, cmode)) {
                        const uint32_t cmax = __reduce_max_sync(full, cmode ? cnt : 0u);
                        const uint32_t *cl = list + cc * kListStride;
                        for (uint32_t e0 = (uint32_t)g8; e0 < cmax; e0 += 8) {
                            const bool mine = cmode && e0 < cnt;
                            const uint32_t x = mine ? cl[e0] : 0u;
                            uint32_t lt = 0, le = 0;
                            for (uint32_t t2 = 0; t2 < cmax; ++t2) {
                                const uint32_t y = t2 < cnt ? cl[t2] : 0xffffffffu;
                                lt += (t2 < cnt) & (y < x);
                                le += (t2 < cnt) & (y <= x);
                            }
                            if (mine && lt <= krem && krem < le) {
                                hit = x;
                                any = true;
                            }
                        }
                    }
                } else if (K != 1 && cmode) {
                    for (uint32_t e0 = (uint32_t)gf; e0 < cnt; e0 += G) {
                        // entry e0 of the concatenated per-warp lists
                        uint32_t m = e0;
                        int u = 0;
                        for (; u < WS - 1 && m >= lcnt[cc * WS + u]; ++u) m -= lcnt[cc * WS + u];
                        const uint32_t x = list[(cc * WS + u) * kListStride + m];
                        uint32_t lt = 0, le = 0;
                        for (int u2 = 0; u2 < WS; ++u2) {
                            const uint32_t cu = lcnt[cc * WS + u2];
                            const uint32_t *cl = list + (cc * WS + u2) * kListStride;
                            for (uint32_t t2 = 0; t2 < cu; ++t2) {
                                const uint32_t y = cl[t2];
                                lt += y < x;
                                le += y <= x;
                            }
                        }
                        if (lt <= krem && krem < le) {
                            hit = x;
                            any = true;
                        }
                    }
                }
                if constexpr (WS == 1) {
                    if constexpr (K != 1) {
                        const unsigned mh = __ballot_sync(full, any) & seg;
                        const uint32_t v = __shfl_sync(full, hit, mh ? __ffs(mh) - 1 : lane);
                        if (cmode) res = v;
                    }
                } else {
                    if (any) st[3 * TC + cc] = hit;
                    col_sync<WS>(cw);
                    if (cmode) res = st[3 * TC + cc];
                    if (gf == 0) st[4 * TC + cc] = 0u;   // NaN flag, next pass
                    col_sync<WS>(cw);
                }
                if (K != 1 && cmode) mode = M_DONE;
                        };
            // two lean passes (histogram, list) while every coordinate of the
            // column is in VH, VC or done; then the general passes, if any
            pass(std::integral_constant<int, 1>{});
            pass(std::integral_constant<int, 2>{});
            if (__builtin_expect((__ballot_sync(full, mode == M_DONE) & 0xfu) != 0xfu, 0)) {
                for (int k2 = 0; k2 < 20; ++k2) {
                    // the column's warps hold identical states: the exit is uniform
                    if ((__ballot_sync(full, mode == M_DONE) & 0xfu) == 0xfu) break;
                    pass(std::integral_constant<int, 0>{});
                }
            }
            if (gf == 0 && live) out[c0 + cc] = __uint_as_float(from_key(res));
        }
        if (!fetched) {
            __syncthreads();
            if constexpr (STAGES == 1) issue(t + gridDim.x, 0);
        }
        stage = (stage + 1) % STAGES;
    }
    cp_async_wait<0>();
}

size_t smem_cap()
{
    int dev = 0, cap = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&cap, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    return (size_t)cap - 1024;        // static shared memory and reserve
}

template <int TC, int STAGES, int MINB, bool VEC, int MODE>
cudaError_t try_launch(bool &launched, const float *copies, int64_t f, int r, int64_t d,
                       int64_t ld, const int8_t *sel, aspis_detection *det, float *out,
                       cudaStream_t stream)
{
    launched = false;
    const Layout L = make_layout<TC, STAGES>(f);
    if (L.total > smem_cap()) return cudaSuccess;
    auto kern = aggregate_kernel<TC, STAGES, MINB, VEC, MODE>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)L.total);
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kThreads, L.total);
    if (e != cudaSuccess) return e;
    if (per_sm < MINB) return cudaSuccess;        // the next configuration is tried
    const int64_t ntiles = (d + TC - 1) / TC;
    int64_t grid = (int64_t)sm_count() * per_sm;
    if (grid > ntiles) grid = ntiles;
    kern<<<(unsigned)grid, kThreads, L.total, stream>>>(copies, f, r, d, ld, sel, det, out);
    launched = true;
    return cudaGetLastError();
}

template <bool VEC, int MODE>
cudaError_t launch_mode(const float *copies, int64_t f, int r, int64_t d, int64_t ld,
                        const int8_t *sel, aspis_detection *det, float *out, cudaStream_t stream)
{
    bool ok = false;
    cudaError_t e = cudaSuccess;
#define ASPIS_TRY(TC, ST, MB)                                                                  \
    e = try_launch<TC, ST, MB, VEC, MODE>(ok, copies, f, r, d, ld, sel, det, out, stream);     \
    if (e != cudaSuccess || ok) return e;
    if constexpr (VEC) {
        ASPIS_TRY(32, 1, 2)
        ASPIS_TRY(32, 3, 1)
        ASPIS_TRY(32, 2, 1)
        ASPIS_TRY(16, 3, 1)
        ASPIS_TRY(16, 2, 1)
        ASPIS_TRY(8, 3, 1)
        ASPIS_TRY(8, 2, 1)
        ASPIS_TRY(8, 1, 1)
        ASPIS_TRY(4, 2, 1)
    }
    ASPIS_TRY(4, 1, 1)
#undef ASPIS_TRY
    return cudaErrorInvalidValue;
}

}  // namespace

cudaError_t launch_aggregate(const float *copies, int64_t f, int r, int64_t d, int64_t ld,
                             const int8_t *sel, aspis_detection *det, int mode, float *out,
                             cudaStream_t stream)
{
    if (f > ASPIS_MAX_AGG_FILES) return cudaErrorInvalidValue;
    const bool vec = ((uintptr_t)copies % 16 == 0) && (ld % 4 == 0);
    if (vec)
        return mode == 0 ? launch_mode<true, 0>(copies, f, r, d, ld, sel, det, out, stream)
                         : launch_mode<true, 1>(copies, f, r, d, ld, sel, det, out, stream);
    return mode == 0 ? launch_mode<false, 0>(copies, f, r, d, ld, sel, det, out, stream)
                     : launch_mode<false, 1>(copies, f, r, d, ld, sel, det, out, stream);
}

}  // namespace aspis
