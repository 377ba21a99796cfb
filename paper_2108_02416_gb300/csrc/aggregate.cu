// Step 5 of the PS round: coordinate-wise aggregation of the chosen copies
// (Algorithm 1: median of the majority gradients; mean in Case 1).
//
// Data path.  Persistent CTAs of 8 warps.  A tile is TC consecutive
// coordinates of all n kept rows.  It is staged in shared memory by 16-byte
// cp.async copies in which 8 consecutive lanes fetch one row's 128 bytes, so
// every memory request carries a whole line (a gather of 16-byte pieces of
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
//   VH  value-space histogram: 256 bins, bins 1..254 evenly over the range of
//       a sample (each lane's first value), 0 / 255 catching everything below
//       / above.  The bin map x -> bits(fma(x, s, c)) - bits(2^23), clamped,
//       is monotone in totalOrder, so bins are contiguous value ranges; a
//       scan over the coordinate's lanes finds the bin holding the target
//       rank.  (Key-space bins cannot do this in one pass: values of both
//       signs near zero span ~2^31 keys.)
//   VC  each lane copies the keys of that bin (at most kSlots per lane) and
//       the <= 32 of them are ranked directly.
// Exact fallback, taken when the sample range is degenerate or not finite,
// a NaN is seen, the bin holds more than 32 values or a lane runs out of
// slots:
//   KA  min / max of the keys -> range [lo, hi]
//   KH  256 equal-width key-space bins over [lo, hi]; the bin holding the
//       rank becomes [lo, hi] (each pass shrinks the range by at least 2^7)
//   KC  as VC for the keys left in [lo, hi].
// The pass cap only guards against an inconsistent state.
#include <climits>

#include "aspis_internal.cuh"

namespace aspis {
namespace {

constexpr int kThreads = 256;     // 8 warps
constexpr int kWarps = kThreads / 32;
constexpr int kNB = 256;          // histogram bins per pass
constexpr int kLogNB = 8;
constexpr int kHistStride = kNB + 4;   // words per coordinate row (rows start 4 banks apart)
constexpr int kCap = 32;          // keys ranked directly
constexpr int kSlots = 8;         // candidate slots per lane
constexpr int kSlotStride = kSlots + 1;

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

// Value-space bin of y = fma(x, s, c): the integer part of y read from its
// bits (y is near 2^23, where one unit is one ulp), clamped to [0, 255].
// Rounding is monotone and the clamp sends negative y, -inf and -NaN-free
// underflow to 0 and +inf / large y to 255, so the map is monotone in the
// IEEE totalOrder of x for every non-NaN x (NaNs are detected separately:
// fma returns a canonical NaN whatever the sign of x).
__device__ __forceinline__ int vraw(float y) { return (int)__float_as_uint(y) - 0x4B000000; }

__device__ __forceinline__ uint32_t vbin(float y)
{
    return (uint32_t)min(max(vraw(y), 0), kNB - 1);
}

enum { M_DONE = 0, M_VH, M_VC, M_KA, M_KH, M_KC };

// Two-sum: s + e == a + b exactly (Knuth); no products, so nothing to fuse.
__device__ __forceinline__ void two_sum(float a, float b, float &s, float &e)
{
    s = a + b;
    const float bp = s - a;
    e = (a - (s - bp)) + (b - bp);
}

struct Layout {
    size_t tiles, rows, hist, cand, ccnt, red, state, total, tile_bytes;
};

template <int TC, int STAGES>
__host__ __device__ inline Layout make_layout(int64_t f)
{
    constexpr int G = 8 * (kWarps / (TC / 4));
    Layout L{};
    size_t o = 0;
    L.tile_bytes = ((size_t)f * TC * 4 + 127) / 128 * 128;
    L.tiles = o; o += STAGES * L.tile_bytes;
    L.rows = o; o += ((size_t)f * 4 + 15) / 16 * 16;
    L.hist = o; o += (size_t)TC * kHistStride * 4;
    L.cand = o; o += (size_t)TC * G * kSlotStride * 4;
    L.ccnt = o; o += (size_t)TC * G * 4;
    L.red = o; o += (size_t)TC * G * 8;
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
    constexpr int BPL = kNB / G;           // histogram bins summed per lane
    constexpr int RPI = kThreads / CPR;    // tile rows covered by one copy round
    extern __shared__ __align__(128) unsigned char smem[];
    const Layout L = make_layout<TC, STAGES>(f);
    unsigned char *tiles = smem + L.tiles;
    int32_t *rows = reinterpret_cast<int32_t *>(smem + L.rows);
    uint32_t *hist = reinterpret_cast<uint32_t *>(smem + L.hist);     // [TC][kHistStride]
    uint32_t *cand = reinterpret_cast<uint32_t *>(smem + L.cand);     // [TC][G][kSlotStride]
    uint32_t *ccnt = reinterpret_cast<uint32_t *>(smem + L.ccnt);     // [TC][G]
    uint32_t *red = reinterpret_cast<uint32_t *>(smem + L.red);       // [TC][G][2]
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
                    for (int i = i0_me; i < n; i += RPI, dst += RPI * TC * 4)
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
#pragma unroll
    for (int s = 0; s < STAGES - 1; ++s) issue(t0 + (int64_t)s * gridDim.x, s);

    int stage = 0;
    for (int64_t t = t0; t < ntiles; t += gridDim.x) {
        issue(t + (int64_t)(STAGES - 1) * gridDim.x, (stage + STAGES - 1) % STAGES);
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
                    red[(cc * G + ws) * 2] = __float_as_uint(s);
                    red[(cc * G + ws) * 2 + 1] = __float_as_uint(e);
                }
                col_sync<WS>(cw);
                s = 0.f;
                e = 0.f;
                for (int u = 0; u < WS; ++u) {
                    float ns, ne;
                    two_sum(s, __uint_as_float(red[(cc * G + u) * 2]), ns, ne);
                    s = ns;
                    e += ne + __uint_as_float(red[(cc * G + u) * 2 + 1]);
                }
            }
            if (gf == 0 && live) out[c0 + cc] = (float)(((double)s + (double)e) / (double)n);
        } else {
            // ---- sample range: the first value of each lane of the coordinate.
            // Value-space bins 1..254 split [sample min, sample max] evenly;
            // bins 0 and 255 catch everything below / above (see vbin below).
            uint32_t slo = nmine > 0 ? to_key(tile[off0]) : 0xffffffffu;
            uint32_t shi = nmine > 0 ? slo : 0u;
#pragma unroll
            for (int o = 4; o < 32; o <<= 1) {
                slo = min(slo, __shfl_xor_sync(full, slo, o));
                shi = max(shi, __shfl_xor_sync(full, shi, o));
            }
            if constexpr (WS > 1) {
                if (g8 == 0) {
                    red[(cc * G + ws) * 2] = slo;
                    red[(cc * G + ws) * 2 + 1] = shi;
                }
                if (gf == 0) st[4 * TC + cc] = 0u;     // NaN flag of this tile
                col_sync<WS>(cw);
                for (int u = 0; u < WS; ++u) {
                    slo = min(slo, red[(cc * G + u) * 2]);
                    shi = max(shi, red[(cc * G + u) * 2 + 1]);
                }
                col_sync<WS>(cw);
            }
            const float xs_lo = __uint_as_float(from_key(slo));
            const float xs_hi = __uint_as_float(from_key(shi));
            const float vs = 254.0f / (xs_hi - xs_lo);
            const float vc = 8388609.0f - xs_lo * vs;    // xs_lo -> about 2^23 + 1
            const bool vspace = isfinite(xs_lo) && isfinite(xs_hi) && xs_hi > xs_lo &&
                                isfinite(vs) && isfinite(vc);

            int mode = !live ? M_DONE : (vspace ? M_VH : M_KA);
            uint32_t lo = 0u, hi = 0u, krem = krank, cnt = (uint32_t)n, res = 0u;
            int vlo = 0, vhi = 0;           // raw value-space bin bounds of the chosen bin

            for (int pass = 0; pass < 20; ++pass) {
                // the column's warps hold identical states: the exit is uniform
                if ((__ballot_sync(full, mode == M_DONE) & 0xfu) == 0xfu) break;
                const int m0 = mode;
                const uint32_t W = hi - lo;
                const int bits = 32 - __clz(W);
                const int sh = bits > kLogNB ? bits - kLogNB : 0;
                uint32_t *h = hist + cc * kHistStride;
                if (m0 == M_VH || m0 == M_KH)
                    for (int b = gf * 4; b < kNB; b += G * 4)
                        *reinterpret_cast<uint4 *>(h + b) = make_uint4(0u, 0u, 0u, 0u);
                col_sync<WS>(cw);

                // ---- sweep over the lane's values
                const uint32_t *p = tile + off0;
                uint32_t mycnt = 0, amin = 0xffffffffu, amax = 0u;
                bool nanf = false;
                uint32_t *slots = cand + (cc * G + gf) * kSlotStride;
                if (m0 == M_VH) {
                    int j = 0;
                    for (; j + 4 <= nmine; j += 4, p += 4 * kStride) {
                        const float y0 = fmaf(__uint_as_float(p[0]), vs, vc);
                        const float y1 = fmaf(__uint_as_float(p[kStride]), vs, vc);
                        const float y2 = fmaf(__uint_as_float(p[2 * kStride]), vs, vc);
                        const float y3 = fmaf(__uint_as_float(p[3 * kStride]), vs, vc);
                        nanf |= (y0 != y0) | (y1 != y1) | (y2 != y2) | (y3 != y3);
                        atomicAdd(h + vbin(y0), 1u);
                        atomicAdd(h + vbin(y1), 1u);
                        atomicAdd(h + vbin(y2), 1u);
                        atomicAdd(h + vbin(y3), 1u);
                    }
                    for (; j < nmine; ++j, p += kStride) {
                        const float y = fmaf(__uint_as_float(*p), vs, vc);
                        nanf |= y != y;
                        atomicAdd(h + vbin(y), 1u);
                    }
                } else if (m0 == M_VC) {
                    for (int j = 0; j < nmine; ++j, p += kStride) {
                        const uint32_t u = *p;
                        const int raw = vraw(fmaf(__uint_as_float(u), vs, vc));
                        if (raw >= vlo && raw <= vhi) {
                            if (mycnt < (uint32_t)kSlots) slots[mycnt] = to_key(u);
                            ++mycnt;
                        }
                    }
                    ccnt[cc * G + gf] = mycnt;
                } else if (m0 == M_KA) {
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
                } else if (m0 == M_KC) {
                    for (int j = 0; j < nmine; ++j, p += kStride) {
                        const uint32_t k = to_key(*p);
                        if (k - lo <= W) {
                            if (mycnt < (uint32_t)kSlots) slots[mycnt] = k;
                            ++mycnt;
                        }
                    }
                    ccnt[cc * G + gf] = mycnt;
                }
                bool nan_any = false;
                if constexpr (WS == 1) {
                    nan_any = (__ballot_sync(full, nanf) & seg) != 0u;
                } else {
                    if (nanf) atomicOr(&st[4 * TC + cc], 1u);
                }
                col_sync<WS>(cw);
                if constexpr (WS > 1) nan_any = st[4 * TC + cc] != 0u;

                // ---- key range of the fallback path (pass A)
                if (__any_sync(full, m0 == M_KA)) {
#pragma unroll
                    for (int o = 4; o < 32; o <<= 1) {
                        amin = min(amin, __shfl_xor_sync(full, amin, o));
                        amax = max(amax, __shfl_xor_sync(full, amax, o));
                    }
                    if constexpr (WS > 1) {
                        if (g8 == 0) {
                            red[(cc * G + ws) * 2] = amin;
                            red[(cc * G + ws) * 2 + 1] = amax;
                        }
                        col_sync<WS>(cw);
                        for (int u = 0; u < WS; ++u) {
                            amin = min(amin, red[(cc * G + u) * 2]);
                            amax = max(amax, red[(cc * G + u) * 2 + 1]);
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

                // ---- bin search (value-space or key-space histogram)
                const bool hm = m0 == M_VH || m0 == M_KH;
                uint32_t nbin = 0, nrr = 0, ncb = 0;
                if constexpr (WS == 1) {
                    if (__any_sync(full, hm)) {
                        // level 1: lane g8 sums bins [32*g8, 32*g8 + 32); scan over g8
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
                        // level 2: lane g8 takes 4 bins of the owner's 32
                        const uint4 c = *reinterpret_cast<const uint4 *>(h + og * BPL + g8 * 4);
                        const uint32_t s2 = (c.x + c.y) + (c.z + c.w);
                        uint32_t incl2 = s2;
#pragma unroll
                        for (int o = 1; o < 8; o <<= 1) {
                            const uint32_t tv = __shfl_up_sync(full, incl2, 4 * o);
                            if (g8 >= o) incl2 += tv;
                        }
                        const uint32_t r2 = krem - before;
                        const unsigned m2 = __ballot_sync(full, incl2 > r2) & seg;
                        const int owner2 = m2 ? __ffs(m2) - 1 : cq;
                        uint32_t rr = r2 - (incl2 - s2), cb = c.w;
                        int b = 3;
                        if (rr < c.x) {
                            b = 0;
                            cb = c.x;
                        } else if ((rr -= c.x) < c.y) {
                            b = 1;
                            cb = c.y;
                        } else if ((rr -= c.y) < c.z) {
                            b = 2;
                            cb = c.z;
                        } else {
                            rr -= c.z;
                        }
                        const uint32_t bin = (uint32_t)(og * BPL + g8 * 4 + b);
                        nbin = __shfl_sync(full, bin, owner2);
                        nrr = __shfl_sync(full, rr, owner2);
                        ncb = __shfl_sync(full, cb, owner2);
                    }
                } else {
                    // WS warps per coordinate: per-lane partial sums through shared
                    // memory (the coordinate's candidate slots are free here),
                    // then the lane with gf == 0 finishes the search
                    uint32_t *part = cand + cc * G * kSlotStride;
                    if (hm) {
                        uint32_t sum = 0;
#pragma unroll
                        for (int b = 0; b < BPL; b += 4) {
                            const uint4 v = *reinterpret_cast<const uint4 *>(h + gf * BPL + b);
                            sum += (v.x + v.y) + (v.z + v.w);
                        }
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
                if (m0 == M_VH) {
                    if (nan_any || ncb > (uint32_t)kCap) {
                        mode = M_KA;             // exact key-space passes instead
                    } else {
                        vlo = nbin == 0 ? INT_MIN : (int)nbin;
                        vhi = nbin == kNB - 1 ? INT_MAX : (int)nbin;
                        krem = nrr;
                        cnt = ncb;
                        mode = M_VC;
                    }
                } else if (m0 == M_KH) {
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

                // ---- ranking of the collected keys: every lane ranks its own
                // candidates (two at a time) against all of the coordinate's
                const bool cm = m0 == M_VC || m0 == M_KC;
                bool ovf = false, any = false;
                uint32_t hit = 0u;
                if (cm) {
                    for (int u = 0; u < G; ++u) ovf |= ccnt[cc * G + u] > (uint32_t)kSlots;
                    if (!ovf) {
                        const uint32_t mine = mycnt;
                        for (uint32_t k0 = 0; k0 < mine; k0 += 2) {
                            const uint32_t x0 = slots[k0];
                            const bool two = k0 + 1 < mine;
                            const uint32_t x1 = two ? slots[k0 + 1] : 0u;
                            uint32_t lt0 = 0, le0 = 0, lt1 = 0, le1 = 0;
                            for (int u = 0; u < G; ++u) {
                                const uint32_t cu = ccnt[cc * G + u];
                                const uint32_t *cl = cand + (cc * G + u) * kSlotStride;
                                for (uint32_t t2 = 0; t2 < cu; ++t2) {
                                    const uint32_t y = cl[t2];
                                    lt0 += y < x0;
                                    le0 += y <= x0;
                                    lt1 += y < x1;
                                    le1 += y <= x1;
                                }
                            }
                            if (lt0 <= krem && krem < le0) {
                                hit = x0;
                                any = true;
                            }
                            if (two && lt1 <= krem && krem < le1) {
                                hit = x1;
                                any = true;
                            }
                        }
                    }
                }
                if constexpr (WS == 1) {
                    const unsigned mh = __ballot_sync(full, any) & seg;
                    const uint32_t v = __shfl_sync(full, hit, mh ? __ffs(mh) - 1 : lane);
                    if (cm && !ovf) res = v;
                } else {
                    if (any) st[3 * TC + cc] = hit;
                    col_sync<WS>(cw);
                    if (cm && !ovf) res = st[3 * TC + cc];
                    if (gf == 0) st[4 * TC + cc] = 0u;   // NaN flag, next pass
                    col_sync<WS>(cw);
                }
                if (cm) {
                    if (!ovf) mode = M_DONE;
                    else mode = m0 == M_VC ? M_KA : M_KH;   // a lane ran out of slots
                }
            }
            if (gf == 0 && live) out[c0 + cc] = __uint_as_float(from_key(res));
        }
        __syncthreads();
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
    }
    ASPIS_TRY(4, 2, 1)
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
