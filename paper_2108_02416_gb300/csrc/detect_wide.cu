// Algorithm 3 beyond 32 workers: all maximum cliques of an agreement graph
// of up to 128 workers, with vertex sets as four 32-bit words.
//
// Bron-Kerbosch with Tomita pivoting (pivot = the vertex of P u X with most
// neighbours in P), spread over the warps of a thread-block cluster (CB
// blocks of four warps) in two levels.  Level 1: the k-th candidate c_k of
// the root starts from R = {c_k}, P = (V minus c_0..c_{k-1}) n N(c_k),
// X = {c_0..c_{k-1}} n N(c_k), exactly the branch sequential Bron-Kerbosch
// takes; every block settles all of these frames into a table in its shared
// memory.  Level 2: the children of those frames, numbered in sequential
// order, are dealt one at a time from a counter in block 0's shared memory
// (a distributed-shared-memory atomic), so a few large subtrees of the first
// branches no longer leave the other warps idle.  A warp that finds a larger
// clique writes its size into every block's bound with a distributed-shared-
// memory max (rare), so the pruning test reads only local shared memory;
// block 0 combines the blocks' results at the end through distributed shared
// memory.  Each warp walks its items cooperatively: the current frame
// (R, P, X, candidates) is the same in all lanes, lane l holds the adjacency
// rows of workers l, l + 32, l + 64, l + 96 in registers, so the pivot is one
// row-count per lane and a warp max, and parent frames wait on a stack in
// shared memory (at most K deep: every push adds one worker to R).  Workers of
// P adjacent to all the rest of P are in every maximal clique of their branch
// and move to R without branching, so the long chains of nearly complete
// agreement graphs take one step.  Detection mode prunes a frame whose
// |R| + |P| cannot reach the largest clique any warp has found (level-1
// frames are settled without pruning, so that every block's table is the
// same); enumeration mode (ASPIS_WIDE_ALL_MAXIMAL) prunes nothing and counts
// every maximal clique.  A node budget per warp bounds the search.
#include "aspis_internal.cuh"

namespace {

constexpr int kMaxK = ASPIS_WIDE_MAX_K;
constexpr uint32_t kDefaultBudget = 1u << 20;   // nodes per warp

struct VS {
    uint32_t w[4];
};

__device__ __forceinline__ VS vs_and(const VS &a, const uint32_t *b)
{
    return VS{{a.w[0] & b[0], a.w[1] & b[1], a.w[2] & b[2], a.w[3] & b[3]}};
}

__device__ __forceinline__ VS vs_andnot(const VS &a, const uint32_t *b)
{
    return VS{{a.w[0] & ~b[0], a.w[1] & ~b[1], a.w[2] & ~b[2], a.w[3] & ~b[3]}};
}

__device__ __forceinline__ int vs_count(const VS &a)
{
    return __popc(a.w[0]) + __popc(a.w[1]) + __popc(a.w[2]) + __popc(a.w[3]);
}

__device__ __forceinline__ int vs_count_and(const VS &a, const VS &b)
{
    return __popc(a.w[0] & b.w[0]) + __popc(a.w[1] & b.w[1]) + __popc(a.w[2] & b.w[2]) +
           __popc(a.w[3] & b.w[3]);
}

__device__ __forceinline__ bool vs_empty(const VS &a)
{
    return (a.w[0] | a.w[1] | a.w[2] | a.w[3]) == 0u;
}

// index of the lowest member, -1 if empty
__device__ __forceinline__ int vs_lowest(const VS &a)
{
#pragma unroll
    for (int i = 0; i < 4; ++i)
        if (a.w[i]) return 32 * i + __ffs(a.w[i]) - 1;
    return -1;
}

// (word selected by comparison, not by index, so sets stay in registers)
__device__ __forceinline__ void vs_set(VS &a, int k)
{
#pragma unroll
    for (int i = 0; i < 4; ++i) a.w[i] |= (k >> 5) == i ? 1u << (k & 31) : 0u;
}

__device__ __forceinline__ void vs_clear(VS &a, int k)
{
#pragma unroll
    for (int i = 0; i < 4; ++i) a.w[i] &= (k >> 5) == i ? ~(1u << (k & 31)) : 0xffffffffu;
}

// a < b as 128-bit numbers, word 3 most significant
__device__ __forceinline__ bool vs_less(const VS &a, const VS &b)
{
#pragma unroll
    for (int i = 3; i >= 0; --i)
        if (a.w[i] != b.w[i]) return a.w[i] < b.w[i];
    return false;
}

constexpr int kWarps = 4;

__device__ __forceinline__ uint32_t cta_rank()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
__device__ __forceinline__ uint32_t cta_count()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(r));
    return r;
}
// shared::cluster address of a shared variable of this block in block `rank`
__device__ __forceinline__ uint32_t peer(const void *p, uint32_t rank)
{
    uint32_t a = (uint32_t)__cvta_generic_to_shared(p), r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(rank));
    return r;
}
__device__ __forceinline__ uint32_t ld_peer32(const void *p, uint32_t rank)
{
    uint32_t v;
    asm volatile("ld.shared::cluster.u32 %0, [%1];" : "=r"(v) : "r"(peer(p, rank)) : "memory");
    return v;
}
__device__ __forceinline__ uint64_t ld_peer64(const void *p, uint32_t rank)
{
    uint64_t v;
    asm volatile("ld.shared::cluster.u64 %0, [%1];" : "=l"(v) : "r"(peer(p, rank)) : "memory");
    return v;
}
__device__ __forceinline__ void max_peer(const int *p, uint32_t rank, int v)
{
    asm volatile("red.shared::cluster.max.s32 [%0], %1;" ::"r"(peer(p, rank)), "r"(v) : "memory");
}
__device__ __forceinline__ void cluster_sync_all()
{
    asm volatile("barrier.cluster.arrive.release.aligned;\n"
                 "barrier.cluster.wait.acquire.aligned;\n" ::: "memory");
}

__global__ void __launch_bounds__(kWarps * 32)
detect_wide_kernel(const uint32_t *__restrict__ adj_g, int K, aspis_detection_wide *det)
{
    __shared__ uint32_t raw[kMaxK][4];
    __shared__ uint32_t adj[kMaxK][4];
    __shared__ uint32_t stack[kWarps][kMaxK][16];      // R, P, X, C of waiting parents
    __shared__ uint32_t tab[kMaxK][16];                 // R, P, X, C of the root's branches
    __shared__ int pre[kMaxK + 1];                      // their child counts, then prefix sums
    __shared__ uint32_t ticket;                         // next level-2 item (read in block 0)
    __shared__ int shared_best;
    __shared__ int w_best[kWarps], w_over[kWarps];
    __shared__ unsigned long long w_count[kWarps], w_maximal[kWarps], w_nodes[kWarps];
    __shared__ uint32_t w_first[kWarps][4];
    const int tid = threadIdx.x, lane = tid & 31, wp = tid >> 5;
    const unsigned full = 0xffffffffu;
    const uint32_t rank = cta_rank(), nblocks = cta_count();
    const int gw = (int)rank * kWarps + wp, nwarps = (int)nblocks * kWarps;
    for (int i = tid; i < kMaxK * 4; i += kWarps * 32) raw[i >> 2][i & 3] = (i >> 2) < K ? adj_g[i] : 0u;
    if (tid == 0) {
        shared_best = 0;
        ticket = 0u;
    }
    __syncthreads();
    cluster_sync_all();             // bounds and the counter are initialised before any access
    // symmetric part: bit k of row j iff both rows list the edge; no self
    // loops, nothing at or beyond K
    for (int j = tid; j < kMaxK; j += kWarps * 32) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            uint32_t m = 0u;
            uint32_t x = j < K ? raw[j][i] : 0u;
            while (x) {
                const int b = __ffs(x) - 1;
                x &= x - 1u;
                const int k = 32 * i + b;
                if (k < K && k != j && ((raw[k][j >> 5] >> (j & 31)) & 1u)) m |= 1u << b;
            }
            adj[j][i] = m;
        }
    }
    __syncthreads();

    const uint32_t budget = det->node_budget ? det->node_budget : kDefaultBudget;
    const bool all = (det->flags & ASPIS_WIDE_ALL_MAXIMAL) != 0u;
    // this lane's rows: workers lane + 32 j
    const VS own0{{adj[lane][0], adj[lane][1], adj[lane][2], adj[lane][3]}};
    const VS own1{{adj[lane + 32][0], adj[lane + 32][1], adj[lane + 32][2], adj[lane + 32][3]}};
    const VS own2{{adj[lane + 64][0], adj[lane + 64][1], adj[lane + 64][2], adj[lane + 64][3]}};
    const VS own3{{adj[lane + 96][0], adj[lane + 96][1], adj[lane + 96][2], adj[lane + 96][3]}};

    int best = 0;
    uint64_t count = 0, maximal = 0, nodes = 0;
    VS first{{0xffffffffu, 0xffffffffu, 0xffffffffu, 0xffffffffu}};
    bool over = false;
    bool live = true;           // false while every warp settles the same root frame
    auto report = [&](const VS R) {
        if (!live) return;
        const int sz = vs_count(R);
        ++maximal;
        if (sz > best) {
            best = sz;
            count = 1;
            first = R;
            if (lane == 0 && sz > *(volatile int *)&shared_best)
                for (uint32_t b = 0; b < nblocks; ++b) max_peer(&shared_best, b, sz);
        } else if (sz == best) {
            ++count;
            if (vs_less(R, first)) first = R;
        }
    };

    // Settles a new frame (R, P, X).  Workers of P adjacent to all the rest
    // of P lie in every maximal clique of the branch, so they move to R at
    // once (X keeps only their common neighbours); when P is a clique that
    // leaves P empty, and R is maximal iff X is empty.  Returns true with
    // the candidates C = P minus the pivot's neighbours when the frame must
    // be branched, false when it is finished (reported or pruned).  Every
    // pass of the loop moves at least one worker out of P.
    auto settle = [&](VS &R, VS &P, VS &X, VS &C, bool prune) -> bool {
        while (true) {
            if (vs_empty(P)) {
                if (vs_empty(X)) report(R);
                return false;
            }
            if (prune) {
                const int bound = max(best, *(volatile int *)&shared_best);
                if (vs_count(R) + vs_count(P) < bound) return false;
            }
            const uint32_t np1 = (uint32_t)vs_count(P);          // |P|; a universal worker has |P| - 1
            uint32_t key = 0u;
            VS U{{0u, 0u, 0u, 0u}};
            VS common{{0xffffffffu, 0xffffffffu, 0xffffffffu, 0xffffffffu}};
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int u = lane + 32 * j;
                const bool inP = (P.w[j] >> lane) & 1u, inX = (X.w[j] >> lane) & 1u;
                const VS &oj = j == 0 ? own0 : j == 1 ? own1 : j == 2 ? own2 : own3;
                uint32_t c = 0u;
                if (inP || inX) {
                    c = (uint32_t)vs_count_and(P, oj);
                    key = max(key, ((c + 1u) << 8) | (uint32_t)(255 - u));
                }
                const bool uni = inP && c + 1u == np1;
                U.w[j] = __ballot_sync(full, uni);
                if (uni) {
#pragma unroll
                    for (int i = 0; i < 4; ++i) common.w[i] &= oj.w[i];
                }
            }
            if (!vs_empty(U)) {
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    common.w[i] = __reduce_and_sync(full, common.w[i]);
                    R.w[i] |= U.w[i];
                    P.w[i] &= ~U.w[i];
                    X.w[i] &= common.w[i];
                }
                continue;
            }
            // pivot: the worker of P u X with most neighbours in P, lowest
            // index on ties (any pivot enumerates the same cliques)
            key = __reduce_max_sync(full, key);
            const int piv = 255 - (int)(key & 255u);      // P is not empty, so key != 0
            C = vs_andnot(P, adj[piv]);
            return true;
        }
    };

    // Depth-first walk below a settled frame (R, P, X, C): children in
    // increasing worker order, parents waiting on this warp's stack.
    auto dfs = [&](VS R, VS P, VS X, VS C) {
        int sp = 0;
        while (true) {
            const int u = vs_lowest(C);
            if (u < 0) {
                if (sp == 0) return;
                --sp;                                   // back to the parent
                __syncwarp();
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    R.w[i] = stack[wp][sp][i];
                    P.w[i] = stack[wp][sp][4 + i];
                    X.w[i] = stack[wp][sp][8 + i];
                    C.w[i] = stack[wp][sp][12 + i];
                }
                __syncwarp();
                continue;
            }
            if (++nodes > budget) {
                over = true;
                return;
            }
            vs_clear(C, u);
            VS Ru = R, Cu;
            vs_set(Ru, u);
            VS Pu = vs_and(P, adj[u]);
            VS Xu = vs_and(X, adj[u]);
            vs_clear(P, u);
            vs_set(X, u);
            if (!settle(Ru, Pu, Xu, Cu, !all)) continue;
            if (sp >= kMaxK) {                          // unreachable: |R| grows by one per frame
                over = true;
                return;
            }
            // the parent waits on the stack; the child becomes the frame
            if (lane < 16) {
                uint32_t val = 0u;
#pragma unroll
                for (int i = 0; i < 4; ++i)
                    if ((lane & 3) == i) val = lane < 4 ? R.w[i] : lane < 8 ? P.w[i] : lane < 12 ? X.w[i] : C.w[i];
                stack[wp][sp][lane] = val;
            }
            __syncwarp();
            ++sp;
            R = Ru;
            P = Pu;
            X = Xu;
            C = Cu;
        }
    };

    // the root frame, settled by every warp alike (reports counted once)
    VS R0{{0u, 0u, 0u, 0u}}, P0{{0u, 0u, 0u, 0u}}, X0{{0u, 0u, 0u, 0u}}, C0{{0u, 0u, 0u, 0u}};
    for (int v = 0; v < K; ++v) vs_set(P0, v);
    live = gw == 0;
    const bool branch0 = settle(R0, P0, X0, C0, !all);
    live = true;
    if (!branch0) C0 = VS{{0u, 0u, 0u, 0u}};

    // Level 1: the root's branches c_0 < c_1 < ... (the members of C0), each
    // with R, P and X as sequential Bron-Kerbosch leaves them.  Every block
    // settles all of them, without pruning, so that every block holds the
    // same table of frames; warp wp of a block takes k = wp, wp + 4, ...,
    // and only the owner of k in the cluster (warp k mod nwarps) reports and
    // counts.  cnt[k] = the number of children of frame k (0 if it was
    // finished by its settling).
    const int nb = vs_count(C0);
    {
        VS Cr = C0, Pr = P0, Xr = X0;
        for (int k = 0; k < nb; ++k) {
            const int ck = vs_lowest(Cr);
            vs_clear(Cr, ck);
            if ((k & (kWarps - 1)) == wp) {
                VS R = R0, P = vs_and(Pr, adj[ck]), X = vs_and(Xr, adj[ck]), C{{0u, 0u, 0u, 0u}};
                vs_set(R, ck);
                const bool own = (k % nwarps) == gw;
                live = own;
                if (own) ++nodes;
                const bool br = settle(R, P, X, C, false);
                live = true;
                if (lane < 16) {
                    uint32_t val = 0u;
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        if ((lane & 3) == i) val = lane < 4 ? R.w[i] : lane < 8 ? P.w[i] : lane < 12 ? X.w[i] : C.w[i];
                    tab[k][lane] = val;
                }
                if (lane == 0) pre[k] = br ? vs_count(C) : 0;
            }
            vs_clear(Pr, ck);
            vs_set(Xr, ck);
        }
    }
    __syncthreads();
    if (tid == 0) {                     // exclusive prefix sums of the child counts
        int acc = 0;
        for (int k = 0; k < nb; ++k) {
            const int c = pre[k];
            pre[k] = acc;
            acc += c;
        }
        pre[nb] = acc;
    }
    __syncthreads();

    // Level 2: item t = child j of frame k with pre[k] <= t < pre[k + 1],
    // dealt from a cluster-wide counter in block 0's shared memory (the next
    // ticket is fetched before the item is walked).  Child j is the j-th
    // member u of C_k: R = R_k + u, P = (P_k minus the members of C_k below
    // u) n N(u), X = (X_k plus those members) n N(u).
    const uint32_t total = (uint32_t)pre[nb];
    const uint32_t tk_addr = peer(&ticket, 0);
    auto take = [&]() -> uint32_t {
        uint32_t t = 0u;
        if (lane == 0) asm volatile("atom.shared::cluster.add.u32 %0, [%1], 1;" : "=r"(t) : "r"(tk_addr) : "memory");
        return __shfl_sync(full, t, 0);
    };
    uint32_t t = total ? take() : 0u;
    while (!over && t < total) {
        const uint32_t tn = take();
        int k = 0;
        for (int base = 0; base < nb; base += 32) {
            const unsigned m = __ballot_sync(full, base + lane < nb && (uint32_t)pre[base + lane] <= t);
            if (m) k = base + 31 - __clz(m);
        }
        VS R, P, X, C;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            R.w[i] = tab[k][i];
            P.w[i] = tab[k][4 + i];
            X.w[i] = tab[k][8 + i];
            C.w[i] = tab[k][12 + i];
        }
        // u = the j-th lowest member of C_k; below = its members under u
        uint32_t j = t - (uint32_t)pre[k];
        int u = -1;
        VS below{{0u, 0u, 0u, 0u}};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const uint32_t c = (uint32_t)__popc(C.w[i]);
            if (u < 0) {
                if (j < c) {
                    uint32_t x = C.w[i];
                    for (uint32_t q = 0; q < j; ++q) x &= x - 1u;
                    const int b = __ffs(x) - 1;
                    u = 32 * i + b;
                    below.w[i] = C.w[i] & ((1u << b) - 1u);
                } else {
                    below.w[i] = C.w[i];
                    j -= c;
                }
            }
        }
        if (++nodes > budget) {
            over = true;
            break;
        }
        vs_set(R, u);
        VS Pu = vs_and(vs_andnot(P, below.w), adj[u]);
        VS Xu{{(X.w[0] | below.w[0]) & adj[u][0], (X.w[1] | below.w[1]) & adj[u][1],
               (X.w[2] | below.w[2]) & adj[u][2], (X.w[3] | below.w[3]) & adj[u][3]}};
        VS Cu;
        if (settle(R, Pu, Xu, Cu, !all)) dfs(R, Pu, Xu, Cu);
        t = tn;
    }

    // reduction: first over the warps of this block, then block 0's first
    // warp gathers the blocks' summaries (lane b reads block b) and combines
    // them; omega, the maximum cliques of that size, the smallest of them
    if (lane == 0) {
        w_best[wp] = best;
        w_over[wp] = over ? 1 : 0;
        w_count[wp] = count;
        w_maximal[wp] = maximal;
        w_nodes[wp] = nodes;
#pragma unroll
        for (int i = 0; i < 4; ++i) w_first[wp][i] = count ? first.w[i] : 0xffffffffu;
    }
    __syncthreads();
    __shared__ int b_best, b_over;
    __shared__ unsigned long long b_count, b_maximal, b_nodes;
    __shared__ uint32_t b_first[4];
    if (tid == 0) {
        int om = 0;
        for (int q = 0; q < kWarps; ++q) om = max(om, w_best[q]);
        unsigned long long n = 0, nmx = 0, nds = 0;
        int ov = 0;
        VS c{{0xffffffffu, 0xffffffffu, 0xffffffffu, 0xffffffffu}};
        for (int q = 0; q < kWarps; ++q) {
            nmx += w_maximal[q];
            nds += w_nodes[q];
            ov |= w_over[q];
            if (w_best[q] == om && w_count[q]) {
                n += w_count[q];
                const VS f{{w_first[q][0], w_first[q][1], w_first[q][2], w_first[q][3]}};
                if (vs_less(f, c)) c = f;
            }
        }
        b_best = om;
        b_over = ov;
        b_count = n;
        b_maximal = nmx;
        b_nodes = nds;
#pragma unroll
        for (int i = 0; i < 4; ++i) b_first[i] = c.w[i];
    }
    cluster_sync_all();             // every block's summary is complete
    if (rank == 0 && wp == 0) {
        const bool has = (uint32_t)lane < nblocks;
        const int bb = has ? (int)ld_peer32(&b_best, lane) : 0;
        const uint64_t bc = has ? ld_peer64(&b_count, lane) : 0ull;
        uint64_t nmx = has ? ld_peer64(&b_maximal, lane) : 0ull;
        uint64_t nds = has ? ld_peer64(&b_nodes, lane) : 0ull;
        const uint32_t bo = has ? ld_peer32(&b_over, lane) : 0u;
        VS f{{0xffffffffu, 0xffffffffu, 0xffffffffu, 0xffffffffu}};
        if (has)
#pragma unroll
            for (int i = 0; i < 4; ++i) f.w[i] = ld_peer32(&b_first[i], lane);
        const int omega = __reduce_max_sync(full, bb);
        const bool at = has && bb == omega && bc != 0ull;
        uint64_t n = at ? bc : 0ull;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            n += __shfl_xor_sync(full, n, o);
            nmx += __shfl_xor_sync(full, nmx, o);
            nds += __shfl_xor_sync(full, nds, o);
        }
        const bool any_over = __any_sync(full, bo != 0u);
        // the smallest first clique among the blocks at omega: compare
        // 128-bit values from the most significant word down
        VS c = at ? f : VS{{0xffffffffu, 0xffffffffu, 0xffffffffu, 0xffffffffu}};
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            VS y;
#pragma unroll
            for (int i = 0; i < 4; ++i) y.w[i] = __shfl_xor_sync(full, c.w[i], o);
            if (vs_less(y, c)) c = y;
        }
        if (lane == 0) {
#pragma unroll
            for (int i = 0; i < 4; ++i) det->clique_mask[i] = c.w[i];
            det->n_max_cliques = n;
            det->n_maximal = nmx;
            det->search_nodes = nds;
            det->omega = omega;
            det->success = (n == 1u && !any_over) ? 1 : 0;
            det->status = any_over ? ASPIS_E_LIMIT : ASPIS_OK;
        }
    }
    cluster_sync_all();             // block 0 has read every block's records
}

// Blocks per cluster: 16 where the device allows clusters of that size
// (non-portable), else 8; decided once per device.
int cluster_blocks()
{
    static int cached[64] = {0};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev < 0 || dev >= 64) dev = 0;
    if (cached[dev]) return cached[dev];
    int best = 8;
    if (cudaFuncSetAttribute(detect_wide_kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) ==
        cudaSuccess) {
        cudaLaunchConfig_t cfg = {};
        cudaLaunchAttribute at[1];
        at[0].id = cudaLaunchAttributeClusterDimension;
        at[0].val.clusterDim.x = 16;
        at[0].val.clusterDim.y = 1;
        at[0].val.clusterDim.z = 1;
        cfg.gridDim = dim3(16);
        cfg.blockDim = dim3(kWarps * 32);
        cfg.attrs = at;
        cfg.numAttrs = 1;
        int n = 0;
        if (cudaOccupancyMaxActiveClusters(&n, detect_wide_kernel, &cfg) == cudaSuccess && n > 0) best = 16;
    }
    cudaGetLastError();
    cached[dev] = best;
    return best;
}

}  // namespace

extern "C" aspis_status aspis_detect_wide(const uint32_t *adj, int K, aspis_detection_wide *det,
                                          void *stream)
{
    if (!adj || !det || K < 1) return ASPIS_E_INVAL;
    if (K > ASPIS_WIDE_MAX_K) return ASPIS_E_RANGE;
    const int cb = cluster_blocks();
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = (unsigned)cb;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.gridDim = dim3((unsigned)cb);
    cfg.blockDim = dim3(kWarps * 32);
    cfg.stream = (cudaStream_t)stream;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    if (cudaLaunchKernelEx(&cfg, detect_wide_kernel, adj, K, det) != cudaSuccess) return ASPIS_E_CUDA;
    return cudaGetLastError() == cudaSuccess ? ASPIS_OK : ASPIS_E_CUDA;
}
