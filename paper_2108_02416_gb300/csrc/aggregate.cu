// Step 5 of the PS round: coordinate-wise aggregation of the chosen copies
// (Algorithm 1: median of the majority gradients; mean in Case 1).
//
// Layout.  A tile is TC consecutive coordinates (TC = 32, 16, 8 or 4) of all
// n kept rows, staged row-major in shared memory ([row][TC] floats) by
// 16-byte cp.async copies, TC/4 consecutive threads per row, so every
// request carries the row's whole TC*4-byte segment.  Lane l of a warp works
// on coordinate c = l % TC of the tile; the SUB = 32/TC lanes of a warp that
// share a coordinate and the 8 warps split its rows: thread (w, s) owns slot
// w*SUB + s and rows slot, slot + NS, slot + 2*NS, ... (NS = 8*SUB slots).
// With this assignment every shared access of the per-value loops is free of
// bank conflicts by construction: the 32 lanes of a load read 32 consecutive
// words of the tile; each lane counts into its own histogram column (bank =
// lane); tag words are laid out [word][slot][TC].  Two CTAs share an SM, or
// one CTA keeps STAGES tiles in flight.
//
// Lower median, exact (IEEE totalOrder through a monotone uint32 key; the
// key map is a bijection, so the output has the chosen element's bits).  Per
// tile:
//   S   sample: the key range [min, max] of the first two values of every
//       slot (16 values per coordinate for TC = 32).
//   VH  value-space histogram of all values: 128 bins, bins 1..126 evenly
//       over the sample range, 0 / 127 catching everything below / above.
//       The bin map x -> bits(fma(x, s, c)) - bits(2^23), clamped, is
//       monotone in totalOrder, so bins are contiguous value ranges.  Every
//       value's bin is kept as a tag byte.  NaNs are detected on the way.
//   B   bin search: per-slot partial sums over the bins, then the slot whose
//       bins hold the target rank finds the bin, the rank inside it and its
//       count (bins of one slot stay in its registers).
//   VC  the bin's members (found by comparing four tag bytes per word) are
//       written to a per-coordinate list of at most 32 keys; each candidate
//       is ranked against the list directly.
// Exact fallback, for the coordinates that need it (NaN seen, degenerate or
// non-finite sample range, more than 32 members in the target bin):
//   VM  the exact key range [lo, hi] of the crowded bin's members
//   KA  the key range [lo, hi] of all values
//   KH  128 equal-width key-space bins over [lo, hi]; the bin holding the
//       rank becomes [lo, hi] (each pass shrinks the range by 2^7)
//   KC  the at most 32 keys left in [lo, hi] are listed and ranked.
// The fallback loop is bounded (kMaxPasses); every wait is a block barrier.
#include <climits>

#include "aspis_internal.cuh"
#include "median_common.cuh"

namespace aspis {
namespace {

constexpr int kThreads = 256;     // 8 warps
constexpr int kWarps = kThreads / 32;
constexpr int kMaxPasses = 12;    // fallback passes: KA/VM, at most 5 KH, KC

// per-coordinate state words (arrays of TC words in shared memory)
enum { S_SMIN, S_SMAX, S_NAN, S_LCNT, S_BIN, S_REM, S_CNT, S_KMIN, S_KMAX, kStateWords };

template <int TC>
struct Geo {
    static constexpr int SUB = 32 / TC;          // lanes of a warp on one coordinate
    static constexpr int NS = kWarps * SUB;      // row slots of a CTA
    static constexpr int CPR = TC / 4;           // 16-byte chunks per tile row
    static constexpr int RPI = kThreads / CPR;   // tile rows per copy round
    static constexpr int BPT = kNB / NS;         // bins per slot in the bin search
    static constexpr int VS = NS * TC;           // words between a lane's consecutive rows
};

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

// max that propagates NaN: a NaN anywhere in the chain survives
__device__ __forceinline__ float max_nan(float a, float b)
{
    float r;
    asm("max.NaN.f32 %0, %1, %2;" : "=f"(r) : "f"(a), "f"(b));
    return r;
}

// the low bytes of four words, packed into one word
__device__ __forceinline__ uint32_t pack4(uint32_t b0, uint32_t b1, uint32_t b2, uint32_t b3)
{
    return __byte_perm(__byte_perm(b0, b1, 0x0040), __byte_perm(b2, b3, 0x0040), 0x5410);
}

struct Layout {
    size_t tiles, tile_bytes, tags, hist, part, list, state, rows, total;
    int jw;                       // tag words per slot
};

template <int TC, int STAGES>
__host__ __device__ inline Layout make_layout(int64_t f)
{
    using G = Geo<TC>;
    Layout L{};
    const int64_t per_slot = (f + G::NS - 1) / G::NS;
    L.jw = (int)((per_slot + 3) / 4);
    size_t o = 0;
    L.tile_bytes = ((size_t)f * TC * 4 + 127) / 128 * 128;
    L.tiles = o; o += STAGES * L.tile_bytes;
    L.tags = o; o += (size_t)L.jw * G::VS * 4;
    L.hist = o; o += (size_t)kNB * 32 * 4;
    L.part = o; o += (size_t)2 * G::NS * TC * 4;
    L.list = o; o += (size_t)kCap * TC * 4;
    L.state = o; o += (size_t)kStateWords * TC * 4;
    L.rows = o; o += ((size_t)f * 4 + 15) / 16 * 16;
    L.total = o;
    return L;
}

template <int TC, int STAGES, int MINB, bool VEC, int MODE>
__global__ void __launch_bounds__(kThreads, MINB)
aggregate_kernel(const float *__restrict__ copies, int64_t f, int r, int64_t d, int64_t ld,
                 const int8_t *__restrict__ sel, aspis_detection *det, float *__restrict__ out)
{
    using G = Geo<TC>;
    constexpr int SUB = G::SUB, NS = G::NS, CPR = G::CPR, RPI = G::RPI, BPT = G::BPT;
    constexpr int VS = G::VS;
    extern __shared__ __align__(128) unsigned char smem[];
    const Layout L = make_layout<TC, STAGES>(f);
    unsigned char *tiles = smem + L.tiles;
    uint32_t *tags = reinterpret_cast<uint32_t *>(smem + L.tags);    // [jw][NS][TC]
    uint32_t *hist = reinterpret_cast<uint32_t *>(smem + L.hist);    // [kNB][32]
    uint32_t *part = reinterpret_cast<uint32_t *>(smem + L.part);    // [2][NS][TC]
    uint32_t *list = reinterpret_cast<uint32_t *>(smem + L.list);    // [kCap][TC]
    uint32_t *st = reinterpret_cast<uint32_t *>(smem + L.state);     // [kStateWords][TC]
    int32_t *rows = reinterpret_cast<int32_t *>(smem + L.rows);
    __shared__ int warp_tot[kWarps];

    const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
    const int c = lane % TC, s = lane / TC;
    const int slot = w * SUB + s;
    const unsigned full = 0xffffffffu;
    auto S = [&](int k) -> uint32_t & { return st[k * TC + c]; };

    // ---- kept files: rows[k] = i*r + sel[i] for the k-th file with sel >= 0
    int n = 0;
    for (int64_t b0 = 0; b0 < f; b0 += kThreads) {
        const int64_t i = b0 + tid;
        const int sv = i < f ? (int)sel[i] : -1;
        const unsigned m = __ballot_sync(full, sv >= 0);
        if (lane == 0) warp_tot[w] = __popc(m);
        __syncthreads();
        int off = n, tot = 0;
        for (int q = 0; q < kWarps; ++q) {
            off += q < w ? warp_tot[q] : 0;
            tot += warp_tot[q];
        }
        if (sv >= 0) rows[off + __popc(m & ((1u << lane) - 1u))] = (int32_t)(i * r + sv);
        n += tot;
        __syncthreads();
    }
    if (n == 0) {
        if (blockIdx.x == 0 && tid == 0) det->status = ASPIS_E_EMPTY;
        return;
    }
    const uint32_t krank = (uint32_t)((n - 1) / 2);
    const int64_t ntiles = (d + TC - 1) / TC;
    const int nmine = n > slot ? (n - slot + NS - 1) / NS : 0;   // rows of this slot

    if constexpr (MODE == 0) {
        for (int i = tid * 4; i < kNB * 32; i += kThreads * 4)
            *reinterpret_cast<uint4 *>(hist + i) = make_uint4(0u, 0u, 0u, 0u);
        if (tid < TC) {
            st[S_SMIN * TC + tid] = 0xffffffffu;
            st[S_SMAX * TC + tid] = 0u;
            st[S_NAN * TC + tid] = 0u;
            st[S_LCNT * TC + tid] = 0u;
            st[S_KMIN * TC + tid] = 0xffffffffu;
            st[S_KMAX * TC + tid] = 0u;
        }
    }

    // copy role (vector path): this thread moves chunk ch_me of rows i0_me + RPI*k
    const int ch_me = tid % CPR, i0_me = tid / CPR;

    auto issue = [&](int64_t t, int stage) {
        if (t < ntiles) {
            const int64_t c0 = t * TC;
            const uint32_t sbase = (uint32_t)__cvta_generic_to_shared(tiles + stage * L.tile_bytes);
            if constexpr (VEC) {
                const int64_t cg = c0 + ch_me * 4;
                if (cg < d) {
                    const float *src = copies + cg;
                    uint32_t dst = sbase + (uint32_t)(i0_me * TC + ch_me * 4) * 4u;
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
                    if (c0 + k < d)
                        cp_async4(sbase + (uint32_t)e * 4u, copies + (int64_t)rows[i] * ld + c0 + k);
                }
            }
        }
        cp_async_commit();
    };

    const int64_t t0 = blockIdx.x;
    if constexpr (STAGES == 1) {
        issue(t0, 0);
    } else {
#pragma unroll
        for (int q = 0; q < STAGES - 1; ++q) issue(t0 + (int64_t)q * gridDim.x, q);
    }

    // Bin search over the 128 bins of the coordinates whose threads pass hm:
    // slot u sums bins [u*BPT, u*BPT + BPT) over the coordinate's SUB
    // columns; the slot holding rank `rank` resolves the bin and writes
    // S_BIN, S_REM (rank inside the bin) and S_CNT.  Leaves the histogram
    // zeroed.  Called by every thread (two block barriers).
    auto bin_search = [&](bool hm, uint32_t rank) {
        uint32_t cb[BPT];
        uint32_t sum = 0u;
#pragma unroll
        for (int j = 0; j < BPT; ++j) {
            uint32_t v = 0u;
            if (hm) {
                const int b = slot * BPT + j;
#pragma unroll
                for (int s2 = 0; s2 < SUB; ++s2) v += hist[b * 32 + s2 * TC + c];
            }
            cb[j] = v;
            sum += v;
        }
        if (hm) part[slot * TC + c] = sum;
        __syncthreads();
        for (int i = tid * 4; i < kNB * 32; i += kThreads * 4)
            *reinterpret_cast<uint4 *>(hist + i) = make_uint4(0u, 0u, 0u, 0u);
        if (hm) {
            uint32_t rem = rank;
            int owner = NS - 1;
            bool fd = false;
            for (int u = 0; u < NS; ++u) {
                const uint32_t pu = part[u * TC + c];
                const bool hit = !fd && rem < pu;
                if (hit) owner = u;
                if (!fd && !hit) rem -= pu;
                fd |= hit;
            }
            if (owner == slot) {
                uint32_t bsel = BPT - 1, csel = cb[BPT - 1];
                bool f2 = false;
#pragma unroll
                for (int j = 0; j < BPT; ++j) {
                    const bool hit = !f2 && rem < cb[j];
                    if (hit) {
                        bsel = (uint32_t)j;
                        csel = cb[j];
                    }
                    if (!f2 && !hit) rem -= cb[j];
                    f2 |= hit;
                }
                S(S_BIN) = (uint32_t)(slot * BPT) + bsel;
                S(S_REM) = rem;
                S(S_CNT) = csel;
            }
        }
        __syncthreads();
    };

    // rank the cnt keys of the coordinate's list; the candidate(s) of rank
    // `rank` write the output
    auto rank_list = [&](bool act, uint32_t cnt, uint32_t rank, int64_t oc) {
        if (!act) return;
        for (uint32_t e = (uint32_t)slot; e < cnt; e += NS) {
            const uint32_t x = list[e * TC + c];
            uint32_t lt = 0u, le = 0u;
            for (uint32_t t2 = 0; t2 < cnt; ++t2) {
                const uint32_t y = list[t2 * TC + c];
                lt += y < x;
                le += y <= x;
            }
            if (lt <= rank && rank < le) out[oc] = __uint_as_float(from_key(x));
        }
    };

    int stage = 0;
    for (int64_t t = t0; t < ntiles; t += gridDim.x) {
        if constexpr (STAGES > 1)
            issue(t + (int64_t)(STAGES - 1) * gridDim.x, (stage + STAGES - 1) % STAGES);
        bool fetched = false;
        cp_async_wait<STAGES - 1>();
        __syncthreads();
        const uint32_t *tile = reinterpret_cast<const uint32_t *>(tiles + stage * L.tile_bytes);
        const int64_t c0 = t * TC;
        const int64_t oc = c0 + c;
        const bool live = oc < d;
        const uint32_t *pv = tile + slot * TC + c;       // value j of this slot: pv[j * VS]

        if constexpr (MODE == 1) {
            // ---- mean: compensated per-slot sums, combined in slot order
            float sm = 0.f, e = 0.f;
            for (int j = 0; j < nmine; ++j) {
                float ns, ne;
                two_sum(sm, __uint_as_float(pv[j * VS]), ns, ne);
                sm = ns;
                e += ne;
            }
            part[slot * TC + c] = __float_as_uint(sm);
            part[(NS + slot) * TC + c] = __float_as_uint(e);
            __syncthreads();
            if (slot == 0 && live) {
                float a = 0.f, ae = 0.f;
                for (int u = 0; u < NS; ++u) {
                    float ns, ne;
                    two_sum(a, __uint_as_float(part[u * TC + c]), ns, ne);
                    a = ns;
                    ae += ne + __uint_as_float(part[(NS + u) * TC + c]);
                }
                out[oc] = (float)(((double)a + (double)ae) / (double)n);
            }
        } else {
            uint32_t *tw = tags + slot * TC + c;         // tag word q of this slot: tw[q * VS]

            // ---- S: sample key range
            uint32_t klo = 0xffffffffu, khi = 0u;
            if (live && nmine > 0) {
                const uint32_t k = to_key(pv[0]);
                klo = min(klo, k);
                khi = max(khi, k);
            }
            if (live && nmine > 1) {
                const uint32_t k = to_key(pv[VS]);
                klo = min(klo, k);
                khi = max(khi, k);
            }
#pragma unroll
            for (int o = TC; o < 32; o <<= 1) {
                klo = min(klo, __shfl_xor_sync(full, klo, o));
                khi = max(khi, __shfl_xor_sync(full, khi, o));
            }
            if (s == 0 && live) {
                atomicMin(&S(S_SMIN), klo);
                atomicMax(&S(S_SMAX), khi);
            }
            __syncthreads();
            const float xs_lo = __uint_as_float(from_key(S(S_SMIN)));
            const float xs_hi = __uint_as_float(from_key(S(S_SMAX)));
            const float vs = (float)(kNB - 2) / (xs_hi - xs_lo);
            const float vc = 8388609.0f - xs_lo * vs;    // xs_lo -> about 2^23 + 1
            const bool vspace = isfinite(xs_lo) && isfinite(xs_hi) && xs_hi > xs_lo &&
                                isfinite(vs) && isfinite(vc);
            int mode = !live ? M_DONE : (vspace ? M_VH : M_KA);

            // ---- VH: histogram of every value, tags, NaN check
            if (mode == M_VH) {
                uint32_t *hl = hist + lane;
                float nacc = 0.f;
                const uint32_t *p = pv;
                uint32_t *q4 = tw;
                int j = 0;
#pragma unroll 2
                for (; j + 4 <= nmine; j += 4, p += 4 * VS, q4 += VS) {
                    const float y0 = fmaf(__uint_as_float(p[0]), vs, vc);
                    const float y1 = fmaf(__uint_as_float(p[VS]), vs, vc);
                    const float y2 = fmaf(__uint_as_float(p[2 * VS]), vs, vc);
                    const float y3 = fmaf(__uint_as_float(p[3 * VS]), vs, vc);
                    nacc = max_nan(max_nan(nacc, max_nan(y0, y1)), max_nan(y2, y3));
                    const uint32_t b0 = vbin(y0), b1 = vbin(y1), b2 = vbin(y2), b3 = vbin(y3);
                    atomicAdd(hl + b0 * 32, 1u);
                    atomicAdd(hl + b1 * 32, 1u);
                    atomicAdd(hl + b2 * 32, 1u);
                    atomicAdd(hl + b3 * 32, 1u);
                    *q4 = pack4(b0, b1, b2, b3);
                }
                if (j < nmine) {
                    // last, partial word: missing rows get tag 0xFF, which no bin has
                    uint32_t word = 0xFFFFFFFFu;
                    for (int k = 0; j < nmine; ++j, ++k, p += VS) {
                        const float y = fmaf(__uint_as_float(*p), vs, vc);
                        nacc = max_nan(nacc, y);
                        const uint32_t b = vbin(y);
                        atomicAdd(hl + b * 32, 1u);
                        word = (word & ~(0xFFu << (8 * k))) | (b << (8 * k));
                    }
                    *q4 = word;
                }
                if (nacc != nacc) atomicOr(&S(S_NAN), 1u);
            }
            __syncthreads();
            if (mode == M_VH && S(S_NAN) != 0u) mode = M_KA;     // exact key-space passes
            if (slot == 0) {
                S(S_SMIN) = 0xffffffffu;
                S(S_SMAX) = 0u;
            }

            // ---- B: the bin holding the median
            bin_search(mode == M_VH, krank);
            uint32_t vb = 0u, krem = krank, cnt = (uint32_t)n;
            if (mode == M_VH) {
                vb = S(S_BIN);
                krem = S(S_REM);
                cnt = S(S_CNT);
                mode = cnt <= (uint32_t)kCap ? M_VC : M_VM;
            }
            if (slot == 0) S(S_NAN) = 0u;

            // ---- VC: list the members of bin vb
            if (mode == M_VC) {
                const uint32_t vbx = vb * 0x01010101u;
                const int nw = (nmine + 3) >> 2;
                uint32_t wm = 0u;                     // words holding a member (first 32)
                for (int q = 0; q < nw && q < 32; ++q)
                    wm |= (tag_match(tw[q * VS], vbx) != 0u ? 1u : 0u) << q;
                for (; wm; wm &= wm - 1u) {
                    const int q = __ffs(wm) - 1;
                    uint32_t z = tag_match(tw[q * VS], vbx);
                    uint32_t pos = atomicAdd(&S(S_LCNT), (uint32_t)__popc(z));
                    for (; z && pos < (uint32_t)kCap; z &= z - 1u)
                        list[(pos++) * TC + c] = to_key(pv[(q * 4 + ((__ffs(z) - 1) >> 3)) * VS]);
                }
                for (int q = 32; q < nw; ++q) {       // slots with more than 128 rows
                    uint32_t z = tag_match(tw[q * VS], vbx);
                    if (z) {
                        uint32_t pos = atomicAdd(&S(S_LCNT), (uint32_t)__popc(z));
                        for (; z && pos < (uint32_t)kCap; z &= z - 1u)
                            list[(pos++) * TC + c] = to_key(pv[(q * 4 + ((__ffs(z) - 1) >> 3)) * VS]);
                    }
                }
            }
            const bool general = __syncthreads_or(mode != M_DONE && mode != M_VC);
            if (slot == 0) S(S_LCNT) = 0u;
            if constexpr (STAGES == 1) {
                if (!general) {
                    issue(t + gridDim.x, 0);          // the tile is no longer read
                    fetched = true;
                }
            }
            rank_list(mode == M_VC, cnt, krem, oc);
            if (mode == M_VC) mode = M_DONE;

            if (general) {
                // ---- exact fallback passes (rare)
                uint32_t lo = 0u, hi = 0u;
                for (int it = 0; it < kMaxPasses; ++it) {
                    const int m0 = mode;
                    const uint32_t W = hi - lo;
                    const int bits = 32 - __clz(W);
                    const int sh = bits > kLogNB ? bits - kLogNB : 0;
                    if (m0 == M_VM || m0 == M_KA) {
                        uint32_t a = 0xffffffffu, b = 0u;
                        const uint8_t *tb = reinterpret_cast<const uint8_t *>(tw);
                        for (int j = 0; j < nmine; ++j) {
                            const bool take = m0 == M_KA || tb[(j >> 2) * VS * 4 + (j & 3)] == vb;
                            if (take) {
                                const uint32_t k = to_key(pv[j * VS]);
                                a = min(a, k);
                                b = max(b, k);
                            }
                        }
                        if (a <= b) {
                            atomicMin(&S(S_KMIN), a);
                            atomicMax(&S(S_KMAX), b);
                        }
                    } else if (m0 == M_KH) {
                        for (int j = 0; j < nmine; ++j) {
                            const uint32_t dk = to_key(pv[j * VS]) - lo;
                            if (dk <= W) atomicAdd(hist + (dk >> sh) * 32 + lane, 1u);
                        }
                    } else if (m0 == M_KC) {
                        for (int j = 0; j < nmine; ++j) {
                            const uint32_t k = to_key(pv[j * VS]);
                            if (k - lo <= W) {
                                const uint32_t pos = atomicAdd(&S(S_LCNT), 1u);
                                if (pos < (uint32_t)kCap) list[pos * TC + c] = k;
                            }
                        }
                    }
                    __syncthreads();
                    if (m0 == M_VM || m0 == M_KA) {
                        lo = S(S_KMIN);
                        hi = S(S_KMAX);
                        if (m0 == M_KA) {
                            krem = krank;
                            cnt = (uint32_t)n;
                        }
                        if (lo == hi) {
                            if (slot == 0) out[oc] = __uint_as_float(from_key(lo));
                            mode = M_DONE;
                        } else {
                            mode = cnt <= (uint32_t)kCap ? M_KC : M_KH;
                        }
                    }
                    rank_list(m0 == M_KC, cnt, krem, oc);
                    if (m0 == M_KC) mode = M_DONE;
                    if (__syncthreads_or(m0 == M_KH)) {
                        bin_search(m0 == M_KH, krem);
                        if (m0 == M_KH) {
                            const uint32_t nb = S(S_BIN);
                            krem = S(S_REM);
                            cnt = S(S_CNT);
                            const uint32_t nlo = lo + (nb << sh);
                            const uint64_t top = (uint64_t)nlo + ((1ull << sh) - 1ull);
                            hi = top < (uint64_t)hi ? (uint32_t)top : hi;
                            lo = nlo;
                            if (lo == hi) {
                                if (slot == 0) out[oc] = __uint_as_float(from_key(lo));
                                mode = M_DONE;
                            } else {
                                mode = cnt <= (uint32_t)kCap ? M_KC : M_KH;
                            }
                        }
                    }
                    if (slot == 0) {
                        S(S_KMIN) = 0xffffffffu;
                        S(S_KMAX) = 0u;
                        S(S_LCNT) = 0u;
                    }
                    if (!__syncthreads_or(mode != M_DONE)) break;
                }
            }
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
        ASPIS_TRY(32, 2, 1)
        ASPIS_TRY(16, 1, 2)
        ASPIS_TRY(16, 2, 1)
        ASPIS_TRY(8, 1, 2)
        ASPIS_TRY(8, 2, 1)
        ASPIS_TRY(8, 1, 1)
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
