// Step 5 of the PS round: coordinate-wise aggregation of the chosen copies
// (Algorithm 1: median of the majority gradients; mean in Case 1).
//
// Data path.  A tile is TC = 32*V consecutive coordinates (V = 4, 2 or 1) of
// all n kept rows.  Lane l of every warp holds coordinates [l*V, l*V + V) of
// the tile and the 8 warps split the rows: warp w reads rows w, w + 8, ...
// straight from global memory with one V-wide load per row, so a warp-wide
// load is one contiguous 128*V-byte segment of a row.  (Gathering 128-byte
// segments of 455 rows that lie 45 MB apart runs at about 4.9 TB/s on GB300,
// 512-byte segments at 7.0; staging whole tiles in shared memory would limit
// the segments to 128 bytes.)  Each value is used once, from registers: rows
// come in batches of kU (8, or 24 for V <= 2 with one CTA per SM) per thread, every
// register refilled with the next batch's row as soon as it is read, and the
// last batch of a tile refills with the first rows of the CTA's next tile,
// whose loads then overlap this tile's remaining phases.  Shared memory holds one tag byte per value, the
// histograms, the member lists and small per-coordinate state; two CTAs of
// 12 warps share an SM.
//
// Lower median, exact (IEEE totalOrder through a monotone uint32 key; the key
// map is a bijection, so the output has the chosen element's bits).  Per
// tile:
//   S   sample: key range of the first two rows of every warp (24 values per
//       coordinate).
//   VH  value-space histogram of every value: bins 1..125 evenly over the
//       sample range, 0 and 126 catch everything below / above (vbin_bits);
//       each value's bin is kept as a tag byte; NaNs are detected.  Counters
//       are the 16-bit halves of words in per-lane columns, so the 32 shared
//       atomics of a warp instruction hit 32 different banks.
//   B   bin search: per-warp partial sums over kBPW bins, then one thread per
//       coordinate finds the bin that holds the target rank, the rank inside
//       it and its count.
//   VC  right after the bin search, four tag bytes are compared per word; the
//       bin's members (about n/80) are copied from global memory (the tile is
//       still in L2) into a list of at most CAP values per coordinate (4096 / TC) by
//       4-byte cp.async; they land during the next tile's sweep, after which
//       one thread per coordinate sorts its keys in registers.
// Exact fallback for the coordinates that need it (NaN seen, degenerate or
// non-finite sample range, more than CAP members in the bin), values
// re-read from global memory:
//   VM  exact key range [lo, hi] of the crowded bin's members
//   KA  key range [lo, hi] of all values
//   KH  128 equal-width key-space bins over [lo, hi]; the bin holding the
//       rank becomes [lo, hi] (each pass shrinks the range by 2^7)
//   KC  the at most CAP keys left in [lo, hi] are listed and ranked.
// The fallback loop is bounded (kMaxPasses); every wait is a block barrier.
#include <type_traits>

#include "aspis_internal.cuh"
#include "median_common.cuh"

namespace aspis {
namespace {

constexpr int kMaxPasses = 12;            // fallback: VM/KA, at most 5 KH, KC
constexpr int kListWords = 4096;          // member lists: 32, 64 or 128 per coordinate
constexpr int kListWords2 = 16384;        // two-pass median: 128 per coordinate

// per-coordinate state, arrays of TC words
enum { S_MIN, S_MAX, S_NAN, S_LCNT, S_MODE, S_BIN, S_REM, S_CNT, S_LO, S_HI, S_PCNT, S_PREM,
       S_FILT, kStateWords };
// S_PCNT / S_PREM: count and rank of the listed bin of the pending tile
// (S_PCNT = 0: nothing to rank for that coordinate).  S_FILT: the exact
// passes of this coordinate search inside its value bin, whose members are
// the values whose tag byte is the bin (only they are re-read).

template <int V> struct Vec;
template <> struct Vec<4> { using T = uint4; };
template <> struct Vec<2> { using T = uint2; };
template <> struct Vec<1> { using T = uint32_t; };

template <int V>
__device__ __forceinline__ uint32_t elem(const typename Vec<V>::T &x, int k)
{
    if constexpr (V == 4) return k == 0 ? x.x : k == 1 ? x.y : k == 2 ? x.z : x.w;
    else if constexpr (V == 2) return k == 0 ? x.x : x.y;
    else return x;
}

template <int V>
__device__ __forceinline__ typename Vec<V>::T load_row(const float *p)
{
    if constexpr (V == 4) return __ldcg(reinterpret_cast<const uint4 *>(p));
    else if constexpr (V == 2) return __ldcg(reinterpret_cast<const uint2 *>(p));
    else return __ldcg(reinterpret_cast<const unsigned int *>(p));
}

// Histogram increment.  No memory clobber: the counters are read only after a
// block barrier, so ordinary loads and stores may move across these.
template <uint32_t INC>
__device__ __forceinline__ void red_shared(uint32_t saddr)
{
    asm volatile("red.shared.add.u32 [%0], %1;\n" ::"r"(saddr), "n"(INC));
}

__device__ __forceinline__ void cp_async4(uint32_t saddr, const void *g)
{
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;\n" ::"r"(saddr), "l"(g) : "memory");
}

__device__ __forceinline__ void prefetch_l2(const void *p)
{
    asm volatile("prefetch.global.L2 [%0];\n" ::"l"(p));
}

__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }

__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;\n" ::: "memory"); }

// ascending bitonic sorting network over N registers (N a power of two)
template <int N>
__device__ __forceinline__ void sort_net(uint32_t (&y)[N])
{
#pragma unroll
    for (int k = 2; k <= N; k <<= 1)
#pragma unroll
        for (int j = k >> 1; j > 0; j >>= 1)
#pragma unroll
            for (int i = 0; i < N; ++i) {
                const int l = i ^ j;
                if (l > i) {
                    const uint32_t a = y[i], b = y[l];
                    const bool up = (i & k) == 0;
                    y[i] = up ? min(a, b) : max(a, b);
                    y[l] = up ? max(a, b) : min(a, b);
                }
            }
}

// the 32 values of a warp (one per lane) sorted ascending across the lanes
// (bitonic: lane i meets lane i ^ j; the lower lane of an ascending block
// keeps the minimum)
__device__ __forceinline__ uint32_t warp_sort32(uint32_t x, int lane)
{
#pragma unroll
    for (int k = 2; k <= 32; k <<= 1)
#pragma unroll
        for (int j = k >> 1; j > 0; j >>= 1) {
            const uint32_t y = __shfl_xor_sync(0xffffffffu, x, j);
            const bool up = (lane & k) == 0, lower = (lane & j) == 0;
            x = lower == up ? min(x, y) : max(x, y);
        }
    return x;
}

// flag |= 1 if any of a, b, c, e is NaN (one compare per pair)
__device__ __forceinline__ void nan_check(uint32_t &flag, float a, float b, float c, float e)
{
    asm("{\n .reg .pred p;\n setp.nan.f32 p, %1, %2;\n setp.nan.or.f32 p, %3, %4, p;\n"
        " @p mov.b32 %0, 1;\n}\n" : "+r"(flag) : "f"(a), "f"(b), "f"(c), "f"(e));
}

// the low bytes of four words, packed into one word
__device__ __forceinline__ uint32_t pack4(uint32_t b0, uint32_t b1, uint32_t b2, uint32_t b3)
{
    return __byte_perm(__byte_perm(b0, b1, 0x0040), __byte_perm(b2, b3, 0x0040), 0x5410);
}

template <int V>
struct Geo {
    static constexpr int TC = 32 * V;                 // coordinates per tile
    static constexpr int NP = V >= 2 ? V / 2 : 1;     // key-space histogram words per (bin, lane)
    static constexpr int SHB = NP == 2 ? 8 : 7;       // log2 of the bytes per key-space row
    // value-space histogram: one word per (bin, lane) holding the lane's V
    // counters, 8-bit for V = 4 (an overflow is detected by the bin search),
    // 16-bit otherwise
    static constexpr int HW = kVB * 32 > kNB * NP * 32 ? kVB * 32 : kNB * NP * 32;   // histogram words
    static constexpr int RPW = 4 / V;                 // rows per tag word
    static constexpr int CAP = kListWords / TC;       // list entries per coordinate
};

struct Layout {
    size_t tags, hist, list, state, rows, total;
};

template <int V, int NT, int MODE>
__host__ __device__ inline Layout make_layout(int64_t f)
{
    using G = Geo<V>;
    constexpr int kWarps = NT / 32;
    Layout L{};
    const int64_t per_slot = (f + kWarps - 1) / kWarps;
    const int64_t jw = (per_slot + G::RPW - 1) / G::RPW;     // tag words per thread
    size_t o = 0;
    // the mean and the two-pass median keep no tags
    L.tags = o; o += MODE == 0 ? (size_t)jw * kWarps * 32 * 4 : 0;
    L.hist = o; o += (size_t)G::HW * 4;
    L.list = o; o += (size_t)(MODE == 2 ? kListWords2 : kListWords) * 4;   // also the partial sums
    L.state = o; o += (size_t)kStateWords * G::TC * 4;
    L.rows = o; o += ((size_t)f * 2 + 15) / 16 * 16;
    L.total = o;
    return L;
}

template <int V, int MINB, bool W32, int MODE, int NT>
__global__ void __launch_bounds__(NT, MINB)
aggregate_kernel(const float *__restrict__ copies, int64_t f, int r, int64_t d, int64_t ld,
                 const int8_t *__restrict__ sel, aspis_detection *det, float *__restrict__ out)
{
    using G = Geo<V>;
    using T = typename Vec<V>::T;
    constexpr int TC = G::TC, NP = G::NP, SHB = G::SHB, RPW = G::RPW;
    constexpr int CAP = (MODE == 2 ? kListWords2 : kListWords) / TC;   // list entries per coordinate
    constexpr int kThreads = NT, kWarps = NT / 32;           // warps = row slots of a CTA
    constexpr int kBPW = (kVB + kWarps - 1) / kWarps;        // bins per warp in the bin search
    constexpr int kShort = MINB >= 2 ? 8 : 16;                // longest list one thread sorts
    constexpr int HW = G::HW;
    // rows per load batch and thread: deeper for narrow rows when one CTA
    // has the SM's registers
    constexpr int kU = (MINB >= 2 || V == 4) ? 8 : 24;
    extern __shared__ __align__(16) unsigned char smem[];
    const Layout L = make_layout<V, NT, MODE>(f);
    uint32_t *tags = reinterpret_cast<uint32_t *>(smem + L.tags);     // [word][kWarps][32]
    uint32_t *hist = reinterpret_cast<uint32_t *>(smem + L.hist);     // [kVB][32] or [kNB][NP][32]
    uint32_t *list = reinterpret_cast<uint32_t *>(smem + L.list);     // [CAP][TC]
    uint32_t *st = reinterpret_cast<uint32_t *>(smem + L.state);      // [kStateWords][TC]
    uint16_t *rows = reinterpret_cast<uint16_t *>(smem + L.rows);
    __shared__ int warp_tot[kWarps];
    __shared__ int n_long;              // listed bins of the pending tile with more than kShort members
    __shared__ int any_exact;           // some coordinate of this tile takes the exact passes
    __shared__ uint8_t long_c[G::TC];   // their coordinates

    const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
    const unsigned full = 0xffffffffu;
    const uint32_t hist_s = (uint32_t)__cvta_generic_to_shared(hist);
    const uint32_t list_s = (uint32_t)__cvta_generic_to_shared(list);
    auto S = [&](int k, int c) -> uint32_t & { return st[k * TC + c]; };

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
        if (sv >= 0) rows[off + __popc(m & ((1u << lane) - 1u))] = (uint16_t)(i * r + sv);
        n += tot;
        __syncthreads();
    }
    if (n == 0) {
        if (blockIdx.x == 0 && tid == 0) det->status = ASPIS_E_EMPTY;
        return;
    }
    const uint32_t krank = (uint32_t)((n - 1) / 2);
    // With 8-bit counters the bins span more than the sample range as n
    // grows, so that the two outer bins (the values outside it) stay well
    // below 256; a wider span also puts more values in the median's bin.
    const float wf = (V != 4 || n <= 640) ? 1.0f : n <= 1024 ? 1.25f : n <= 1536 ? 1.5f : 2.0f;
    const int nmine = n > w ? (n - w + kWarps - 1) / kWarps : 0;     // rows of this warp
    const int nwords = (nmine + RPW - 1) / RPW;
    const int64_t ntiles = (d + TC - 1) / TC;
    const uint64_t ldb = (uint64_t)ld * 4u;                          // row pitch in bytes

    if (tid == 0) {
        n_long = 0;
        any_exact = 0;
    }
    for (int i = tid; i < TC; i += kThreads) {
        S(S_MIN, i) = 0xffffffffu;
        S(S_MAX, i) = 0u;
        S(S_NAN, i) = 0u;
        S(S_LCNT, i) = 0u;
        S(S_PCNT, i) = 0u;
    }
    for (int i = tid * 4; i < HW; i += kThreads * 4)
        *reinterpret_cast<uint4 *>(hist + i) = make_uint4(0u, 0u, 0u, 0u);

    // address of row j of this warp at the lane's chunk of a tile
    auto row_ptr = [&](const char *lb, int j) -> const float * {
        const uint32_t row = rows[w + j * kWarps];
        if constexpr (W32) return reinterpret_cast<const float *>(lb + (uint64_t)row * (uint32_t)ldb);
        else return reinterpret_cast<const float *>(lb + (uint64_t)row * ldb);
    };
    auto lane_base = [&](int64_t t) -> const char * {
        return reinterpret_cast<const char *>(copies + t * TC + lane * V);
    };

    T xa[kU];                            // the batch being processed (then the next one)
    {
        const int64_t t = blockIdx.x;
        const bool lv = t < ntiles && t * TC + lane * V < d;
#pragma unroll
        for (int u = 0; u < kU; ++u) {
            xa[u] = T{};
            if (lv && u < nmine) xa[u] = load_row<V>(row_ptr(lane_base(t), u));
        }
    }
    __syncthreads();

    uint32_t exact_cnt = 0u;        // coordinates resolved by the exact passes (thread 0)

    // The previous tile ("pending"): its median bins are known, its members
    // are listed during the next sweep and ranked after it.
    bool have_p = false;
    const char *lb_p = nullptr;
    int64_t c0_p = 0;
    uint32_t vbx_p = 0xFFFFFFFFu, vcm_p = 0u;

    // The members of the pending tile's bins: its tag words are compared with
    // the target bins eight at a time (one mask bit per byte), and each
    // member's value is copied (4-byte cp.async) into its coordinate's list
    // column while the tile's rows are still in L2; the copies complete
    // during the next sweep.
    auto capture_members = [&]() {
        if (!vcm_p) return;
        // bytes of the lane's coordinates that search a value bin
        uint32_t vmask = 0u;
#pragma unroll
        for (int q = 0; q < 4; ++q) vmask |= ((vcm_p >> (q % V)) & 1u) ? 0xFFu << (8 * q) : 0u;
        for (int g = 0; g < nwords; g += 8) {
            uint32_t m = 0u;
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                if (g + i < nwords) {
                    const uint32_t z = tag_match(tags[((g + i) * kWarps + w) * 32 + lane], vbx_p);
                    m |= z >> (7 - i);
                }
            }
            for (m &= vmask; m; m &= m - 1u) {
                const int b = __ffs(m) - 1;
                const int pos = b >> 3, q = g + (b & 7);
                const int j = q * RPW + pos / V, k = pos % V;
                const int c = lane * V + k;
                const uint32_t at = atomicAdd(&S(S_LCNT, c), 1u);
                if (at < (uint32_t)CAP)
                    cp_async4(list_s + (at * TC + c) * 4u, row_ptr(lb_p, j) + k);
            }
        }
        cp_async_commit();
    };

    // Rank the pending tile's listed bins.  Lists of at most kShort keys (the
    // common case): one thread per coordinate sorts them in registers (16
    // keys where one block has the SM's registers, else 8).
    // Longer lists (queued by the bin search): one warp per coordinate, a
    // warp-wide sort for up to 32 keys, else every lane counting, for its
    // candidates, the listed keys below and at them.
    auto rank_pending = [&]() {
        for (int c = tid; c < TC; c += kThreads) {
            const uint32_t cnt = S(S_PCNT, c);
            if (cnt == 0u || cnt > (uint32_t)kShort) continue;
            const uint32_t rk = S(S_PREM, c);
            uint32_t y[kShort];
#pragma unroll
            for (int e = 0; e < kShort; ++e) y[e] = (uint32_t)e < cnt ? to_key(list[e * TC + c]) : 0xffffffffu;
            sort_net<kShort>(y);
            uint32_t res = y[0];
#pragma unroll
            for (int e = 1; e < kShort; ++e) res = (uint32_t)e == rk ? y[e] : res;
            out[c0_p + c] = __uint_as_float(from_key(res));
        }
        // dealt first to the warps without a coordinate of their own above
        constexpr int kSW = TC / 32 < kWarps ? TC / 32 : 0;
        for (int q = (w - kSW + kWarps) % kWarps; q < n_long; q += kWarps) {
            const int c = long_c[q];
            const uint32_t cnt = S(S_PCNT, c);               // the same in every lane
            const uint32_t rk = S(S_PREM, c);
            if (cnt <= 32u) {
                const uint32_t x = warp_sort32((uint32_t)lane < cnt ? to_key(list[lane * TC + c])
                                                                     : 0xffffffffu, lane);
                const uint32_t res = __shfl_sync(full, x, (int)rk);
                if (lane == 0) out[c0_p + c] = __uint_as_float(from_key(res));
                continue;
            }
            for (uint32_t e = (uint32_t)lane; e < cnt; e += 32u) {
                const uint32_t x = to_key(list[e * TC + c]);
                uint32_t lt = 0u, le = 0u;
                for (uint32_t t2 = 0; t2 < cnt; ++t2) {
                    const uint32_t y = to_key(list[t2 * TC + c]);
                    lt += y < x;
                    le += y <= x;
                }
                if (lt <= rk && rk < le) out[c0_p + c] = __uint_as_float(from_key(x));
            }
        }
    };

    for (int64_t t = blockIdx.x; t < ntiles; t += gridDim.x) {
        const int64_t c0 = t * TC;
        const bool lv = c0 + lane * V < d;                 // some coordinate of the lane is live
        const char *lb = lane_base(t);
        const int64_t tn = t + gridDim.x;
        const bool lvn = tn < ntiles && tn * TC + lane * V < d;
        const char *lbn = lvn ? lane_base(tn) : lb;

        // One pass over this warp's rows, batch by batch: pre(j0) at the start
        // of a batch, fn(x, j, u) for every row; each register is refilled
        // right after it is used, the last batch with the first rows of the
        // next tile (or of this tile again when a second pass follows).
        auto sweep = [&](auto pre, auto fn, auto againc) {
            constexpr bool AGAIN = decltype(againc)::value;
            const char *lr = AGAIN ? lb : lbn;
            const bool lvr = AGAIN ? lv : lvn;
            auto batch = [&](auto lastc, int j0) {
                constexpr bool LAST = decltype(lastc)::value;
                pre(j0);
                if constexpr (!LAST) {
                    // the rows of the batch after next into L2, one 128-byte
                    // line (32 coordinates) per lane: line q % V of row
                    // j0 + 2 kU + q / V for q = lane, lane + 32, ...
#pragma unroll
                    for (int q0 = 0; q0 < kU * V; q0 += 32) {
                        const int q = q0 + lane, jp = j0 + 2 * kU + q / V, ln = q % V;
                        if (q < kU * V && jp < nmine && c0 + ln * 32 < d)
                            prefetch_l2(reinterpret_cast<const char *>(copies + c0 + ln * 32) +
                                        (uint64_t)rows[w + jp * kWarps] * ldb);
                    }
                }
#pragma unroll
                for (int u = 0; u < kU; ++u) {
                    if constexpr (LAST) {
                        if (j0 + u < nmine) fn(xa[u], j0 + u, u);
                        if (lvr && u < nmine) xa[u] = load_row<V>(row_ptr(lr, u));
                    } else {
                        fn(xa[u], j0 + u, u);
                        const int jn = j0 + kU + u;
                        if (lv && jn < nmine) xa[u] = load_row<V>(row_ptr(lb, jn));
                    }
                }
            };
            int j0 = 0;
            for (; j0 + kU < nmine; j0 += kU) batch(std::false_type{}, j0);
            batch(std::true_type{}, j0);
        };

        if constexpr (MODE == 1) {
            // ---- mean: compensated per-thread sums, combined in warp order
            float sm[V], se[V];
#pragma unroll
            for (int k = 0; k < V; ++k) sm[k] = se[k] = 0.f;
            sweep([](int) {}, [&](const T &x, int, int) {
#pragma unroll
                for (int k = 0; k < V; ++k) {
                    float ns, ne;
                    two_sum(sm[k], __uint_as_float(elem<V>(x, k)), ns, ne);
                    sm[k] = ns;
                    se[k] += ne;
                }
            }, std::false_type{});
#pragma unroll
            for (int k = 0; k < V; ++k) {
                list[(2 * w) * TC + lane * V + k] = __float_as_uint(sm[k]);
                list[(2 * w + 1) * TC + lane * V + k] = __float_as_uint(se[k]);
            }
            __syncthreads();
            for (int c = tid; c < TC; c += kThreads) {
                if (c0 + c >= d) continue;
                float a = 0.f, ae = 0.f;
                for (int u = 0; u < kWarps; ++u) {
                    float ns, ne;
                    two_sum(a, __uint_as_float(list[(2 * u) * TC + c]), ns, ne);
                    a = ns;
                    ae += ne + __uint_as_float(list[(2 * u + 1) * TC + c]);
                }
                out[c0 + c] = (float)(((double)a + (double)ae) / (double)n);
            }
            __syncthreads();
        } else {
            // ---- S: key range of the sample (rows 0 and 1 of every warp)
            if (lv) {
#pragma unroll
                for (int k = 0; k < V; ++k) {
                    if (c0 + lane * V + k >= d) continue;
                    uint32_t lo = 0xffffffffu, hi = 0u;
                    if (nmine > 0) {
                        const uint32_t q = to_key(elem<V>(xa[0], k));
                        lo = min(lo, q);
                        hi = max(hi, q);
                    }
                    if (nmine > 1) {
                        const uint32_t q = to_key(elem<V>(xa[1], k));
                        lo = min(lo, q);
                        hi = max(hi, q);
                    }
                    if (lo <= hi) {
                        atomicMin(&S(S_MIN, lane * V + k), lo);
                        atomicMax(&S(S_MAX, lane * V + k), hi);
                    }
                }
            }
            __syncthreads();                                        // (B)
            float vs[V], vc[V];
#pragma unroll
            for (int k = 0; k < V; ++k) {
                const float xlo = __uint_as_float(from_key(S(S_MIN, lane * V + k)));
                const float xhi = __uint_as_float(from_key(S(S_MAX, lane * V + k)));
                // the sample range, widened by wf around its centre -> y in
                // [1/254, 253/254]: bins 1..253; values outside go to 0 and 254
                const float wd = wf * (xhi - xlo);
                const float x0 = xlo - 0.5f * (wf - 1.0f) * (xhi - xlo);
                const float sc = (252.0f / 254.0f) / wd;
                const float cc = fmaf(-x0, sc, 1.0f / 254.0f);
                const bool ok = isfinite(xlo) && isfinite(xhi) && xhi > xlo && isfinite(sc) &&
                                sc > 0.f && isfinite(cc);
                vs[k] = ok ? sc : 0.f;
                vc[k] = ok ? cc : 0.f;
                if (w == 0) {
                    const bool live = c0 + lane * V + k < d;
                    S(S_MODE, lane * V + k) = !live ? M_DONE : (ok ? M_VH : M_KA);
                }
            }
            const uint32_t hb = hist_s + (uint32_t)lane * 4u - (0x4B000000u << 7);

            // ---- sweep: the pending tile's members (old tag words), then
            // VH for this tile (histogram, new tag words, NaN check)
            uint32_t nanf = 0u, tacc = 0u;
            sweep([](int) {}, [&](const T &x, int j, int u) {
                uint32_t bb[V];
#pragma unroll
                for (int k = 0; k < V; ++k) {
                    bb[k] = vbin_bits(__uint_as_float(elem<V>(x, k)), vs[k], vc[k]);
                    const uint32_t a = (bb[k] << 7) + hb;
                    if constexpr (V == 4) {
                        if (k == 0) red_shared<1u>(a);
                        else if (k == 1) red_shared<0x100u>(a);
                        else if (k == 2) red_shared<0x10000u>(a);
                        else red_shared<0x1000000u>(a);
                    } else {
                        if (k & 1) red_shared<0x10000u>(a);
                        else red_shared<1u>(a);
                    }
                }
                if constexpr (V == 4) {
                    nan_check(nanf, __uint_as_float(x.x), __uint_as_float(x.y),
                              __uint_as_float(x.z), __uint_as_float(x.w));
                    if constexpr (MODE == 0)
                        tags[(j * kWarps + w) * 32 + lane] = pack4(bb[0], bb[1], bb[2], bb[3]);
                } else if constexpr (V == 2) {
                    nan_check(nanf, __uint_as_float(x.x), __uint_as_float(x.y),
                              __uint_as_float(x.x), __uint_as_float(x.y));
                    const uint32_t h = __byte_perm(bb[0], bb[1], 0x0040) & 0xFFFFu;
                    if ((u & 1) == 0) {
                        tacc = h | (kPadTag * 0x01010000u);
                        if (j + 1 >= nmine) tags[((j >> 1) * kWarps + w) * 32 + lane] = tacc;
                    } else {
                        tags[((j >> 1) * kWarps + w) * 32 + lane] = (tacc & 0xFFFFu) | (h << 16);
                    }
                } else {
                    nan_check(nanf, __uint_as_float(x), __uint_as_float(x),
                              __uint_as_float(x), __uint_as_float(x));
                    const int sh = 8 * (u & 3);
                    tacc = ((u & 3) == 0 ? kPadTag * 0x01010101u : tacc);
                    tacc = (tacc & ~(0xFFu << sh)) | ((bb[0] & 0xFFu) << sh);
                    if ((u & 3) == 3 || j + 1 >= nmine) tags[((j >> 2) * kWarps + w) * 32 + lane] = tacc;
                }
            }, std::integral_constant<bool, MODE == 2>{});
            if (nanf) {
#pragma unroll
                for (int k = 0; k < V; ++k) atomicOr(&S(S_NAN, lane * V + k), 1u);
            }
            cp_async_wait_all();
            __syncthreads();                                        // (C)
            if (have_p) rank_pending();
            if (w == 0) {
#pragma unroll
                for (int k = 0; k < V; ++k) {
                    const int c = lane * V + k;
                    if (S(S_MODE, c) == M_VH && S(S_NAN, c)) S(S_MODE, c) = M_KA;
                    S(S_NAN, c) = 0u;
                    S(S_MIN, c) = 0xffffffffu;
                    S(S_MAX, c) = 0u;
                }
            }
            __syncthreads();                                        // (R)
            if (tid == 0) {                        // both read by every thread before (R)
                n_long = 0;
                any_exact = 0;
            }
            for (int c = tid; c < TC; c += kThreads) S(S_LCNT, c) = 0u;

            // ---- B1: per-warp partial sums over bins [kBPW*w, kBPW*w + kBPW);
            // 8-bit counters are summed as two pairs of 16-bit fields
            {
                uint32_t ps0 = 0u, ps1 = 0u;
#pragma unroll
                for (int b = 0; b < kBPW; ++b)
                    if (w * kBPW + b < kVB) {
                        const uint32_t x = hist[(w * kBPW + b) * 32 + lane];
                        if constexpr (V == 4) {
                            ps0 += x & 0x00FF00FFu;
                            ps1 += (x >> 8) & 0x00FF00FFu;
                        } else {
                            ps0 += x;
                        }
                    }
                if constexpr (V == 4) {
                    // one 16-byte store per lane: its four coordinates' sums
                    *reinterpret_cast<uint4 *>(list + w * TC + lane * 4) =
                        make_uint4(ps0 & 0xFFFFu, ps1 & 0xFFFFu, ps0 >> 16, ps1 >> 16);
                } else {
#pragma unroll
                    for (int k = 0; k < V; ++k) list[w * TC + lane * V + k] = (ps0 >> (16 * (k & 1))) & 0xFFFFu;
                }
            }
            __syncthreads();                                        // (D)
            // ---- B2: one thread per coordinate resolves its bin
            for (int c = tid; c < TC; c += kThreads) {
                uint32_t pc = 0u;
                if (S(S_MODE, c) == M_VH) {
                    uint32_t rem = krank, tot = 0u;
                    int owner = kWarps - 1;
                    bool fd = false;
                    for (int u = 0; u < kWarps; ++u) {
                        const uint32_t pu = list[u * TC + c];
                        const bool hit = !fd && rem < pu;
                        if (hit) owner = u;
                        if (!fd && !hit) rem -= pu;
                        fd |= hit;
                        tot += pu;
                    }
                    const int lc = c / V, k = c % V;
                    const uint32_t *h = hist + lc;
                    const int shf = V == 4 ? 8 * k : 16 * (k & 1);
                    const uint32_t msk = V == 4 ? 0xFFu : 0xFFFFu;
                    int bin = min(owner * kBPW + kBPW, kVB) - 1;
                    uint32_t cnt = 0u;
                    bool f2 = false;
                    uint32_t cbs[kBPW];                        // the owner's bins, loaded at once
#pragma unroll
                    for (int i = 0; i < kBPW; ++i) {
                        const int b = owner * kBPW + i;
                        cbs[i] = b < kVB ? (h[b * 32] >> shf) & msk : 0u;
                    }
#pragma unroll
                    for (int i = 0; i < kBPW; ++i) {
                        const uint32_t cb = cbs[i];
                        const bool hit = !f2 && rem < cb;
                        if (hit) {
                            bin = owner * kBPW + i;
                            cnt = cb;
                        }
                        if (!f2 && !hit) rem -= cb;
                        f2 |= hit;
                    }
                    S(S_BIN, c) = (uint32_t)bin;
                    S(S_REM, c) = rem;
                    S(S_CNT, c) = cnt;
                    S(S_PREM, c) = rem;
                    // an 8-bit counter that overflowed changes its coordinate's total
                    const bool exact = tot == (uint32_t)n;
                    const bool vcm = exact && cnt <= (uint32_t)CAP;
                    // (without tags the exact passes cannot read a bin's members
                    // alone: a crowded bin starts them over all values)
                    S(S_MODE, c) = !exact ? M_KA : (vcm ? M_VC : (MODE == 2 ? M_KA : M_VM));
                    pc = vcm ? cnt : 0u;
                }
                S(S_PCNT, c) = pc;
                if (pc > (uint32_t)kShort) long_c[atomicAdd(&n_long, 1)] = (uint8_t)c;
                const uint32_t mdn = S(S_MODE, c);
                if (mdn == M_VM || mdn == M_KA) any_exact = 1;
            }
            __syncthreads();                                        // (E)
            // the same in every thread: no barrier decides the exact passes
            const bool exact_pass = any_exact != 0;
            for (int i = tid * 4; i < HW; i += kThreads * 4)
                *reinterpret_cast<uint4 *>(hist + i) = make_uint4(0u, 0u, 0u, 0u);

            // this tile becomes the pending one: target bins of its coordinates
            uint32_t vbx = 0u, vcm = 0u;
#pragma unroll
            for (int k = 0; k < V; ++k) {
                const uint32_t md = S(S_MODE, lane * V + k);
                const uint32_t vb = md == M_VC ? S(S_BIN, lane * V + k) : 0xFFu;
                vcm |= (md == M_VC ? 1u : 0u) << k;
#pragma unroll
                for (int q = k; q < 4; q += V) vbx |= vb << (8 * q);
            }
            if constexpr (MODE == 0) {
                // two blocks per SM: the next tile's second batch into L2 while
                // this tile's tail runs (with one block per SM and its larger
                // tiles the extra lines cost more than they save)
                if constexpr (MINB >= 2) {
                    if (tn < ntiles) {
#pragma unroll
                        for (int q0 = 0; q0 < kU * V; q0 += 32) {
                            const int q = q0 + lane, jp = kU + q / V, ln = q % V;
                            if (jp < nmine && tn * TC + ln * 32 < d)
                                prefetch_l2(reinterpret_cast<const char *>(copies + tn * TC + ln * 32) +
                                            (uint64_t)rows[w + jp * kWarps] * ldb);
                        }
                    }
                }
                have_p = true;
                lb_p = lb;
                c0_p = c0;
                vbx_p = vbx;
                vcm_p = vcm;
                capture_members();
            } else {
                // ---- second pass over the tile's rows (two-pass median): the
                // values whose bin is their coordinate's target go straight
                // from the registers into the list; then they are ranked
                uint32_t tgt[V];
#pragma unroll
                for (int k = 0; k < V; ++k)
                    tgt[k] = ((vcm >> k) & 1u) ? 0x4B000000u | S(S_BIN, lane * V + k) : 0xFFFFFFFFu;
                sweep([](int) {}, [&](const T &x, int, int) {
                    uint32_t bb[V];
                    bool hit = false;
#pragma unroll
                    for (int k = 0; k < V; ++k) {
                        bb[k] = vbin_bits(__uint_as_float(elem<V>(x, k)), vs[k], vc[k]);
                        hit |= bb[k] == tgt[k];
                    }
                    if (hit) {
#pragma unroll
                        for (int k = 0; k < V; ++k) {
                            if (bb[k] != tgt[k]) continue;
                            const int c = lane * V + k;
                            const uint32_t at = atomicAdd(&S(S_LCNT, c), 1u);
                            if (at < (uint32_t)CAP) list[at * TC + c] = elem<V>(x, k);
                        }
                    }
                }, std::false_type{});
                __syncthreads();
                c0_p = c0;
                rank_pending();
            }

            if (exact_pass) {
                // ---- exact fallback passes (rare), values re-read from global memory
                {
                    const uint32_t md0 = tid < TC ? S(S_MODE, tid) : (uint32_t)M_DONE;
                    if (tid < TC) S(S_FILT, tid) = 0u;
                    const int ne = __syncthreads_count(md0 == M_VM || md0 == M_KA);
                    if (tid == 0) exact_cnt += (uint32_t)ne;
                }
                auto reread = [&](int j, int k) -> uint32_t {
                    return __ldcg(reinterpret_cast<const unsigned int *>(row_ptr(lb, j)) + k);
                };
                for (int it = 0; it < kMaxPasses; ++it) {
                    // pass over the values of the coordinates still searching
                    if (lv) {
                        for (int k = 0; k < V; ++k) {
                            const int c = lane * V + k;
                            const uint32_t md = S(S_MODE, c);
                            if (md == M_DONE || md == M_VC) continue;
                            const uint32_t lo = S(S_LO, c), hi = S(S_HI, c);
                            const uint32_t W = hi - lo;
                            const int bits = 32 - __clz(W);
                            const int sh = bits > kLogNB ? bits - kLogNB : 0;
                            const uint32_t vb = S(S_BIN, c);
                            const uint8_t *tb = reinterpret_cast<const uint8_t *>(tags);
                            // inside a value bin only its members (tag == bin) are read
                            const bool filt = MODE == 0 && (md == M_VM || S(S_FILT, c) != 0u);
                            uint32_t a = 0xffffffffu, bmax = 0u;
                            if (filt) {
                                // the members' rows from the tag bytes first, then
                                // their loads, four at a time
                                for (int j0 = 0; j0 < nmine; j0 += 32) {
                                    uint32_t m = 0u;
                                    for (int u = 0; u < 32 && j0 + u < nmine; ++u) {
                                        const int j = j0 + u, q = j / RPW, p = (j % RPW) * V + k;
                                        if (tb[((q * kWarps + w) * 32 + lane) * 4 + p] == vb) m |= 1u << u;
                                    }
                                    while (m) {
                                        uint32_t vals[4], ok = 0u;
#pragma unroll
                                        for (int u = 0; u < 4; ++u) {
                                            vals[u] = 0u;
                                            if (m) {
                                                vals[u] = reread(j0 + __ffs(m) - 1, k);
                                                m &= m - 1u;
                                                ok |= 1u << u;
                                            }
                                        }
#pragma unroll
                                        for (int u = 0; u < 4; ++u) {
                                            if (!((ok >> u) & 1u)) continue;
                                            const uint32_t key = to_key(vals[u]);
                                            if (md == M_VM) {
                                                a = min(a, key);
                                                bmax = max(bmax, key);
                                            } else if (key - lo <= W) {
                                                if (md == M_KH) {
                                                    atomicAdd(hist + (((key - lo) >> sh) * NP + k / 2) * 32 + lane,
                                                              (k & 1) ? 0x10000u : 1u);
                                                } else {
                                                    const uint32_t at = atomicAdd(&S(S_LCNT, c), 1u);
                                                    if (at < (uint32_t)CAP) list[at * TC + c] = key;
                                                }
                                            }
                                        }
                                    }
                                }
                            } else {
                                for (int j0 = 0; j0 < nmine; j0 += 8) {
                                    uint32_t vals[8];
#pragma unroll
                                    for (int u = 0; u < 8; ++u)    // eight loads in flight
                                        if (j0 + u < nmine) vals[u] = reread(j0 + u, k);
#pragma unroll
                                    for (int u = 0; u < 8; ++u) {
                                        const int j = j0 + u;
                                        if (j >= nmine) break;
                                        const uint32_t key = to_key(vals[u]);
                                        if (md == M_KA) {
                                            a = min(a, key);
                                            bmax = max(bmax, key);
                                        } else if (key - lo <= W) {
                                            if (md == M_KH) {
                                                atomicAdd(hist + (((key - lo) >> sh) * NP + k / 2) * 32 + lane,
                                                          (k & 1) ? 0x10000u : 1u);
                                            } else {
                                                const uint32_t at = atomicAdd(&S(S_LCNT, c), 1u);
                                                if (at < (uint32_t)CAP) list[at * TC + c] = key;
                                            }
                                        }
                                    }
                                }
                            }
                            if ((md == M_VM || md == M_KA) && a <= bmax) {
                                atomicMin(&S(S_MIN, c), a);
                                atomicMax(&S(S_MAX, c), bmax);
                            }
                        }
                    }
                    __syncthreads();
                    // resolution, one thread per coordinate
                    for (int c = tid; c < TC; c += kThreads) {
                        const uint32_t md = S(S_MODE, c);
                        if (md == M_DONE || md == M_VC) continue;
                        uint32_t lo = S(S_LO, c), hi = S(S_HI, c);
                        uint32_t rk = S(S_REM, c), cnt = S(S_CNT, c);
                        uint32_t nm = md;
                        if (md == M_VM || md == M_KA) {
                            lo = S(S_MIN, c);
                            hi = S(S_MAX, c);
                            if (md == M_KA) {
                                rk = krank;
                                cnt = (uint32_t)n;
                            } else {
                                S(S_FILT, c) = 1u;             // [lo, hi] lies inside the value bin
                            }
                            nm = lo == hi ? M_DONE : (cnt <= (uint32_t)CAP ? M_KC : M_KH);
                        } else if (md == M_KH) {
                            const uint32_t W = hi - lo;
                            const int bits = 32 - __clz(W);
                            const int sh = bits > kLogNB ? bits - kLogNB : 0;
                            const int lc = c / V, k = c % V;
                            const uint32_t *h = hist + (k / 2) * 32 + lc;
                            const int shf = 16 * (k & 1);
                            uint32_t b = 0;
                            for (; b < (uint32_t)kNB - 1; ++b) {
                                const uint32_t cb = (h[b * NP * 32] >> shf) & 0xFFFFu;
                                if (rk < cb) break;
                                rk -= cb;
                            }
                            cnt = (h[b * NP * 32] >> shf) & 0xFFFFu;
                            const uint32_t nlo = lo + (b << sh);
                            const uint64_t top = (uint64_t)nlo + ((1ull << sh) - 1ull);
                            hi = top < (uint64_t)hi ? (uint32_t)top : hi;
                            lo = nlo;
                            nm = lo == hi ? M_DONE : (cnt <= (uint32_t)CAP ? M_KC : M_KH);
                        } else if (md == M_KC) {
                            const uint32_t m = min(cnt, (uint32_t)CAP);
                            for (uint32_t e = 0; e < m; ++e) {
                                const uint32_t x = list[e * TC + c];
                                uint32_t lt = 0u, le = 0u;
                                for (uint32_t t2 = 0; t2 < m; ++t2) {
                                    const uint32_t y = list[t2 * TC + c];
                                    lt += y < x;
                                    le += y <= x;
                                }
                                if (lt <= rk && rk < le) {
                                    lo = x;
                                    break;
                                }
                            }
                            hi = lo;
                            nm = M_DONE;
                        }
                        if (nm == M_DONE) out[c0 + c] = __uint_as_float(from_key(lo));
                        S(S_LO, c) = lo;
                        S(S_HI, c) = hi;
                        S(S_REM, c) = rk;
                        S(S_CNT, c) = cnt;
                        S(S_MODE, c) = nm;
                        S(S_MIN, c) = 0xffffffffu;
                        S(S_MAX, c) = 0u;
                        S(S_LCNT, c) = 0u;
                    }
                    __syncthreads();
                    for (int i = tid * 4; i < HW; i += kThreads * 4)
                        *reinterpret_cast<uint4 *>(hist + i) = make_uint4(0u, 0u, 0u, 0u);
                    bool more = false;
                    for (int c = tid; c < TC; c += kThreads) {
                        const uint32_t md = S(S_MODE, c);
                        more |= md != M_DONE && md != M_VC;
                    }
                    if (!__syncthreads_or(more)) break;
                }
            }
        }
    }
    if constexpr (MODE != 1) {
        // the last tile's listed members are ranked once their copies land
        if (MODE == 0 && have_p) {
            cp_async_wait_all();
            __syncthreads();
            rank_pending();
        }
        if (tid == 0 && exact_cnt) atomicAdd(&det->median_exact, exact_cnt);
    }
}

// Lower median for rows that are not 16-byte aligned (no two-pass 128-
// coordinate tiles) and more kept files than the tag bytes of even a
// 32-coordinate tile can hold in shared memory (about 5,800): an exact 8-bit radix select
// on the totalOrder keys, four passes per tile, each re-reading the tile's
// kept values.  A tile is 32 coordinates (lane l of every warp holds
// coordinate l; the warps split the rows); the histogram has one 32-bit
// counter per (digit, coordinate).  Four times the reads of the tagged
// kernel, no per-value state.
constexpr int kRadixThreads = 256;

__global__ void __launch_bounds__(kRadixThreads)
median_radix_kernel(const float *__restrict__ copies, int64_t f, int r, int64_t d, int64_t ld,
                    const int8_t *__restrict__ sel, aspis_detection *det, float *__restrict__ out)
{
    constexpr int kW = kRadixThreads / 32;
    extern __shared__ __align__(16) unsigned char smem[];
    uint32_t *hist = reinterpret_cast<uint32_t *>(smem);              // [256 digits][32 coordinates]
    uint32_t *pre = hist + 256 * 32;                                  // per coordinate: key prefix
    uint32_t *rnk = pre + 32;                                         // per coordinate: rank left
    uint16_t *rows = reinterpret_cast<uint16_t *>(rnk + 32);         // kept rows
    __shared__ int warp_tot[kW];
    const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
    const unsigned full = 0xffffffffu;
    int n = 0;
    for (int64_t b0 = 0; b0 < f; b0 += kRadixThreads) {
        const int64_t i = b0 + tid;
        const int sv = i < f ? (int)sel[i] : -1;
        const unsigned m = __ballot_sync(full, sv >= 0);
        if (lane == 0) warp_tot[w] = __popc(m);
        __syncthreads();
        int off = n, tot = 0;
        for (int u = 0; u < kW; ++u) {
            off += u < w ? warp_tot[u] : 0;
            tot += warp_tot[u];
        }
        if (sv >= 0) rows[off + __popc(m & ((1u << lane) - 1u))] = (uint16_t)(i * r + sv);
        n += tot;
        __syncthreads();
    }
    if (n == 0) {
        if (blockIdx.x == 0 && tid == 0) det->status = ASPIS_E_EMPTY;
        return;
    }
    const uint32_t krank = (uint32_t)((n - 1) / 2);
    const int64_t ntiles = (d + 31) / 32;
    for (int64_t t = blockIdx.x; t < ntiles; t += gridDim.x) {
        const int64_t col = t * 32 + lane;
        const bool live = col < d;
        if (tid < 32) {
            pre[tid] = 0u;
            rnk[tid] = krank;
        }
        for (int p = 0; p < 4; ++p) {
            const int sh = 24 - 8 * p;
            const uint32_t pmask = p == 0 ? 0u : 0xFFFFFFFFu << (32 - 8 * p);
            for (int i = tid; i < 256 * 32; i += kRadixThreads) hist[i] = 0u;
            __syncthreads();
            const uint32_t want = pre[lane];
            for (int j0 = w; j0 < n; j0 += kW * 8) {
                uint32_t v[8];
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const int j = j0 + u * kW;
                    v[u] = live && j < n ? __ldcg(reinterpret_cast<const unsigned int *>(
                                               copies + (int64_t)rows[j] * ld + col))
                                         : 0u;
                }
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const int j = j0 + u * kW;
                    const uint32_t key = to_key(v[u]);
                    if (live && j < n && (key & pmask) == want)
                        atomicAdd(&hist[((key >> sh) & 0xFFu) * 32 + lane], 1u);
                }
            }
            __syncthreads();
            // warp w settles coordinates 4w..4w+3: a warp scan over the 256 digits
            for (int q = 0; q < 4; ++q) {
                const int cc = 4 * w + q;
                uint32_t cb[8], sum = 0u;
#pragma unroll
                for (int b = 0; b < 8; ++b) {
                    cb[b] = hist[(lane * 8 + b) * 32 + cc];
                    sum += cb[b];
                }
                uint32_t inc = sum;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const uint32_t y = __shfl_up_sync(full, inc, o);
                    if (lane >= o) inc += y;
                }
                const uint32_t rk = rnk[cc], exc = inc - sum;
                const bool mine = exc <= rk && rk < inc;
                uint32_t dig = 0u, r2 = rk - exc;
                if (mine) {
                    bool hit = false;
#pragma unroll
                    for (int b = 0; b < 8; ++b) {
                        if (!hit && r2 < cb[b]) {
                            dig = (uint32_t)(lane * 8 + b);
                            hit = true;
                        }
                        if (!hit) r2 -= cb[b];
                    }
                }
                const unsigned bal = __ballot_sync(full, mine);
                const int src = bal ? __ffs(bal) - 1 : 0;
                dig = __shfl_sync(full, dig, src);
                r2 = __shfl_sync(full, r2, src);
                if (lane == 0 && bal) {
                    pre[cc] |= dig << sh;
                    rnk[cc] = r2;
                }
            }
            __syncthreads();
        }
        if (w == 0 && live) out[col] = __uint_as_float(from_key(pre[lane]));
        __syncthreads();
    }
    // every coordinate of this path is resolved exactly
    if (tid == 0) {
        uint32_t cnt = 0u;
        for (int64_t t = blockIdx.x; t < ntiles; t += gridDim.x) cnt += (uint32_t)min((int64_t)32, d - t * 32);
        atomicAdd(&det->median_exact, cnt);
    }
}

size_t smem_cap()
{
    int dev = 0, cap = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&cap, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    return (size_t)cap - 1024;        // static shared memory and reserve
}

template <int V, int MINB, bool W32, int MODE, int NT>
cudaError_t try_launch(bool &launched, const float *copies, int64_t f, int r, int64_t d,
                       int64_t ld, const int8_t *sel, aspis_detection *det, float *out,
                       cudaStream_t stream)
{
    launched = false;
    const Layout L = make_layout<V, NT, MODE>(f);
    if (L.total > smem_cap()) return cudaSuccess;
    auto kern = aggregate_kernel<V, MINB, W32, MODE, NT>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)L.total);
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, NT, L.total);
    if (e != cudaSuccess) return e;
    if (per_sm < MINB) return cudaSuccess;        // the next configuration is tried
    const int64_t ntiles = (d + Geo<V>::TC - 1) / Geo<V>::TC;
    int64_t grid = (int64_t)sm_count() * per_sm;
    if (grid > ntiles) grid = ntiles;
    kern<<<(unsigned)grid, NT, L.total, stream>>>(copies, f, r, d, ld, sel, det, out);
    launched = true;
    return cudaGetLastError();
}

cudaError_t launch_radix(const float *copies, int64_t f, int r, int64_t d, int64_t ld,
                         const int8_t *sel, aspis_detection *det, float *out, cudaStream_t stream)
{
    const size_t smem = (size_t)(256 * 32 + 64) * 4 + ((size_t)f * 2 + 15) / 16 * 16;
    if (smem > smem_cap()) return cudaErrorInvalidValue;
    cudaError_t e = cudaFuncSetAttribute(median_radix_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, median_radix_kernel, kRadixThreads, smem);
    if (e != cudaSuccess) return e;
    const int64_t ntiles = (d + 31) / 32;
    int64_t grid = (int64_t)sm_count() * (per_sm > 0 ? per_sm : 1);
    if (grid > ntiles) grid = ntiles;
    median_radix_kernel<<<(unsigned)grid, kRadixThreads, smem, stream>>>(copies, f, r, d, ld, sel, det, out);
    return cudaGetLastError();
}

template <int MODE, bool W32>
cudaError_t launch_mode(int align, const float *copies, int64_t f, int r, int64_t d, int64_t ld,
                        const int8_t *sel, aspis_detection *det, float *out, cudaStream_t stream)
{
    bool ok = false;
    cudaError_t e = cudaSuccess;
#define ASPIS_TRY(V, MB, NT)                                                                    \
    e = try_launch<V, MB, W32, MODE, NT>(ok, copies, f, r, d, ld, sel, det, out, stream);       \
    if (e != cudaSuccess || ok) return e;
    if (align >= 4) {
        ASPIS_TRY(4, 2, 384)
    }
    if (align >= 2) {
        ASPIS_TRY(2, 2, 384)
    }
    if (align >= 4) {
        ASPIS_TRY(4, 1, 384)
    }
    if (align >= 2) {
        ASPIS_TRY(2, 1, 384)
    }
    if constexpr (MODE == 0) {
        // more files than the tag bytes of 64-coordinate tiles hold: two
        // passes over 128-coordinate tiles (twice the reads, 512-byte row
        // segments) before the narrow one-pass tiles
        if (align >= 4) {
            e = try_launch<4, 2, W32, 2, 384>(ok, copies, f, r, d, ld, sel, det, out, stream);
            if (e != cudaSuccess || ok) return e;
            e = try_launch<4, 1, W32, 2, 384>(ok, copies, f, r, d, ld, sel, det, out, stream);
            if (e != cudaSuccess || ok) return e;
        }
    }
    ASPIS_TRY(1, 2, 384)
    ASPIS_TRY(1, 1, 384)
#undef ASPIS_TRY
    if constexpr (MODE == 0) return launch_radix(copies, f, r, d, ld, sel, det, out, stream);
    return cudaErrorInvalidValue;
}

}  // namespace

cudaError_t launch_aggregate(const float *copies, int64_t f, int r, int64_t d, int64_t ld,
                             const int8_t *sel, aspis_detection *det, int mode, float *out,
                             cudaStream_t stream)
{
    if (f > ASPIS_MAX_AGG_FILES || f * r > 65535) return cudaErrorInvalidValue;
    // widest load every row start allows: 16 bytes (V = 4), 8 (V = 2), else 4
    const uintptr_t p = (uintptr_t)copies;
    const int align = (p % 16 == 0 && ld % 4 == 0) ? 4 : (p % 8 == 0 && ld % 2 == 0) ? 2 : 1;
    const bool w32 = (uint64_t)ld * 4u < (1ull << 32);     // row pitch fits a 32-bit multiplier
    if (mode == 0)
        return w32 ? launch_mode<0, true>(align, copies, f, r, d, ld, sel, det, out, stream)
                   : launch_mode<0, false>(align, copies, f, r, d, ld, sel, det, out, stream);
    return w32 ? launch_mode<1, true>(align, copies, f, r, d, ld, sel, det, out, stream)
               : launch_mode<1, false>(align, copies, f, r, d, ld, sel, det, out, stream);
}

}  // namespace aspis
