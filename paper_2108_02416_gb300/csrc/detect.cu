// Steps 3-4 of the PS round.
//
// detect: all maximum cliques of G (Algorithm 3).  One warp; lane v explores
// the cliques whose smallest vertex is v (R = {v}, P = later neighbours,
// X = earlier neighbours), so every maximal clique is reported by exactly one
// lane.  Inside a branch: Bron-Kerbosch with Tomita pivoting over 32-bit
// vertex masks, an explicit stack in shared memory, and pruning of branches
// that cannot reach the best clique size found so far by any lane.  Each lane
// has a node budget; running out sets ASPIS_E_LIMIT and success = 0, so a
// pathological graph ends the search instead of stalling the stream.
//
// select: one copy per file (Algorithm 1): Case 1 honest copy / Case 2
// majority class of bitwise-equal copies, read from the mismatch word.
#include "aspis_internal.cuh"

namespace aspis {
namespace {

constexpr uint32_t kDefaultNodeBudget = 1u << 20;   // per lane

struct Frame {
    uint32_t R, P, X, cand;
};

__device__ __forceinline__ int pick_pivot(uint32_t P, uint32_t X, const uint32_t *adj)
{
    uint32_t PX = P | X;
    int piv = __ffs(PX) - 1, best = -1;
    while (PX) {
        const int u = __ffs(PX) - 1;
        PX &= PX - 1;
        const int c = __popc(P & adj[u]);
        if (c > best) {
            best = c;
            piv = u;
        }
    }
    return piv;
}

__global__ void __launch_bounds__(32)
detect_kernel(const uint32_t *__restrict__ adj_g, int K, aspis_detection *det)
{
    __shared__ uint32_t adj[32];
    __shared__ Frame stack[32][32];          // [depth][lane]
    __shared__ int shared_best;
    const int v = threadIdx.x;
    adj[v] = v < K ? adj_g[v] : 0u;
    if (v == 0) shared_best = 0;
    const uint32_t budget = det->node_budget ? det->node_budget : kDefaultNodeBudget;
    __syncwarp();

    int best = 0;
    uint32_t count = 0, first = 0xffffffffu, nodes = 0;
    bool over = false;

    if (v < K) {
        int sp = 0;
        auto report = [&](uint32_t R) {
            const int sz = __popc(R);
            if (sz > best) {
                best = sz;
                count = 1;
                first = R;
                atomicMax(&shared_best, sz);
            } else if (sz == best) {
                ++count;
                if (R < first) first = R;
            }
        };
        // a child node: report it if maximal, else push it unless it cannot
        // reach the best size known to any lane
        auto visit = [&](uint32_t R, uint32_t P, uint32_t X) {
            if (P == 0u) {
                if (X == 0u) report(R);
                return;
            }
            const int bound = max(best, *(volatile int *)&shared_best);
            if (__popc(R) + __popc(P) < bound) return;
            stack[sp][v] = Frame{R, P, X, P & ~adj[pick_pivot(P, X, adj)]};
            ++sp;
        };
        const uint32_t bit = 1u << v;
        visit(bit, adj[v] & ~(bit | (bit - 1u)), adj[v] & (bit - 1u));
        while (sp > 0) {
            Frame &fr = stack[sp - 1][v];
            if (fr.cand == 0u) {
                --sp;
                continue;
            }
            if (++nodes > budget) {
                over = true;
                break;
            }
            const int u = __ffs(fr.cand) - 1;
            const uint32_t ub = 1u << u;
            fr.cand &= ~ub;
            const uint32_t R = fr.R | ub, P = fr.P & adj[u], X = fr.X & adj[u];
            fr.P &= ~ub;
            fr.X |= ub;
            visit(R, P, X);
        }
    }
    const unsigned full = 0xffffffffu;
    const int omega = __reduce_max_sync(full, best);
    const uint32_t n = __reduce_add_sync(full, best == omega ? count : 0u);
    const uint32_t canon = __reduce_min_sync(full, (best == omega && count) ? first : 0xffffffffu);
    const uint32_t total = __reduce_add_sync(full, nodes);
    const bool any_over = __any_sync(full, over);
    if (v == 0) {
        det->clique_mask = canon;
        det->omega = omega;
        det->n_max_cliques = n;
        det->success = (n == 1u && !any_over) ? 1 : 0;
        det->n_sel = 0;
        det->median_exact = 0u;
        det->status = any_over ? ASPIS_E_LIMIT : ASPIS_OK;
        det->search_nodes = total;
    }
}

template <int R>
__device__ __forceinline__ int majority_slot(uint32_t w)
{
    // size of the class of slot s = 1 + number of slots equal to it
    int pick = 0, best = 0;
#pragma unroll
    for (int s = 0; s < R; ++s) {
        int size = 1, p = 0;
#pragma unroll
        for (int a = 0; a < R; ++a)
#pragma unroll
            for (int b = a + 1; b < R; ++b, ++p)
                if ((a == s || b == s) && !((w >> p) & 1u)) ++size;
        if (size > best) {
            best = size;
            pick = s;
        }
    }
    return pick;
}

template <int R>
__global__ void __launch_bounds__(256)
select_kernel(const uint32_t *__restrict__ file_neq, aspis_detection *det,
              const uint8_t *__restrict__ fw, int64_t f, int8_t *__restrict__ sel)
{
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int success = det->success;
    const uint32_t clique = det->clique_mask;
    int pick = -1;
    if (i < f) {
        if (success) {
#pragma unroll
            for (int s = R - 1; s >= 0; --s)
                if ((clique >> fw[i * R + s]) & 1u) pick = s;
        } else {
            pick = majority_slot<R>(file_neq[i]);
        }
        sel[i] = (int8_t)pick;
    }
    const int kept = __syncthreads_count(pick >= 0);
    if (threadIdx.x == 0 && kept) atomicAdd(&det->n_sel, kept);
}

}  // namespace

cudaError_t launch_detect(const uint32_t *adj, int K, aspis_detection *det, cudaStream_t stream)
{
    detect_kernel<<<1, 32, 0, stream>>>(adj, K, det);
    return cudaGetLastError();
}

cudaError_t launch_select(const uint32_t *file_neq, aspis_detection *det,
                          const uint8_t *dev_file_workers, int64_t f, int r, int8_t *sel,
                          cudaStream_t stream)
{
    const unsigned grid = (unsigned)((f + 255) / 256);
    switch (r) {
    case 2: select_kernel<2><<<grid, 256, 0, stream>>>(file_neq, det, dev_file_workers, f, sel); break;
    case 3: select_kernel<3><<<grid, 256, 0, stream>>>(file_neq, det, dev_file_workers, f, sel); break;
    case 4: select_kernel<4><<<grid, 256, 0, stream>>>(file_neq, det, dev_file_workers, f, sel); break;
    case 5: select_kernel<5><<<grid, 256, 0, stream>>>(file_neq, det, dev_file_workers, f, sel); break;
    case 6: select_kernel<6><<<grid, 256, 0, stream>>>(file_neq, det, dev_file_workers, f, sel); break;
    case 7: select_kernel<7><<<grid, 256, 0, stream>>>(file_neq, det, dev_file_workers, f, sel); break;
    case 8: select_kernel<8><<<grid, 256, 0, stream>>>(file_neq, det, dev_file_workers, f, sel); break;
    default: return cudaErrorInvalidValue;
    }
    return cudaGetLastError();
}

}  // namespace aspis
