// Steps 1-2 of the PS round: per-file agreement of the r copies (Section 4,
// definition of alpha_i^{(j1,j2)}) and the agreement graph G (an edge iff the
// pair agrees on all C(K-2,r-2) shared files, Algorithm 3).
//
// compare: HBM-streaming kernel.  Work item = (file, chunk of kChunkVec float4
// per row).  Each thread keeps U*R 128-bit loads in flight, XORs every slot
// pair, ORs the pair's "differs" bit into a register word, and each warp
// issues one atomicOr per item into file_neq[file] (only if a bit is set).
// graph: one block folds the per-file words into per-worker disagreement
// masks in shared memory and writes adj = complement.
#include "aspis_internal.cuh"

namespace aspis {
namespace {

constexpr int kCmpThreads = 256;
constexpr int64_t kChunkVec = 4096;   // 64 KiB of each row per work item

__device__ __forceinline__ uint32_t vdiff(const uint4 &a, const uint4 &b)
{
    return (a.x ^ b.x) | (a.y ^ b.y) | (a.z ^ b.z) | (a.w ^ b.w);
}

template <int R, int U>
__global__ void __launch_bounds__(kCmpThreads)
compare_vec_kernel(const float *__restrict__ copies, int64_t f, int64_t d, int64_t ld,
                   int64_t nvec, int64_t nchunks, uint32_t *__restrict__ file_neq)
{
    const int64_t ldv = ld >> 2;
    const uint4 *base = reinterpret_cast<const uint4 *>(copies);
    const int64_t items = f * nchunks;
    const int tail = (int)(d - nvec * 4);                 // 0..3 scalars after the vectors
    for (int64_t item = blockIdx.x; item < items; item += gridDim.x) {
        const int64_t i = item / nchunks;
        const int64_t ch = item - i * nchunks;
        const uint4 *row = base + i * R * ldv;
        const int64_t v0 = ch * kChunkVec;
        const int64_t v1 = v0 + kChunkVec < nvec ? v0 + kChunkVec : nvec;
        uint32_t neq = 0;
        for (int64_t v = v0 + threadIdx.x; v < v1; v += (int64_t)kCmpThreads * U) {
            uint4 x[U][R];
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int64_t vv = v + (int64_t)u * kCmpThreads;
#pragma unroll
                for (int s = 0; s < R; ++s)
                    x[u][s] = vv < v1 ? __ldcs(row + s * ldv + vv) : make_uint4(0, 0, 0, 0);
            }
#pragma unroll
            for (int u = 0; u < U; ++u) {
                int p = 0;
#pragma unroll
                for (int s = 0; s < R; ++s)
#pragma unroll
                    for (int t = s + 1; t < R; ++t, ++p)
                        neq |= (vdiff(x[u][s], x[u][t]) != 0u ? 1u : 0u) << p;
            }
        }
        if (tail && ch == nchunks - 1 && threadIdx.x < (unsigned)tail) {
            const uint32_t *rw = reinterpret_cast<const uint32_t *>(copies) + i * R * ld;
            const int64_t c = nvec * 4 + threadIdx.x;
            uint32_t y[R];
#pragma unroll
            for (int s = 0; s < R; ++s) y[s] = rw[s * ld + c];
            int p = 0;
#pragma unroll
            for (int s = 0; s < R; ++s)
#pragma unroll
                for (int t = s + 1; t < R; ++t, ++p)
                    neq |= (y[s] != y[t] ? 1u : 0u) << p;
        }
        neq = __reduce_or_sync(0xffffffffu, neq);
        if ((threadIdx.x & 31) == 0 && neq) atomicOr(&file_neq[i], neq);
    }
}

// 4-byte path for buffers that are not 16-byte aligned or have ld % 4 != 0.
template <int R>
__global__ void __launch_bounds__(kCmpThreads)
compare_scalar_kernel(const float *__restrict__ copies, int64_t f, int64_t d, int64_t ld,
                      int64_t nchunks, uint32_t *__restrict__ file_neq)
{
    const uint32_t *base = reinterpret_cast<const uint32_t *>(copies);
    const int64_t chunk = kChunkVec * 4;
    const int64_t items = f * nchunks;
    for (int64_t item = blockIdx.x; item < items; item += gridDim.x) {
        const int64_t i = item / nchunks;
        const int64_t ch = item - i * nchunks;
        const uint32_t *row = base + i * R * ld;
        const int64_t c0 = ch * chunk;
        const int64_t c1 = c0 + chunk < d ? c0 + chunk : d;
        uint32_t neq = 0;
        for (int64_t c = c0 + threadIdx.x; c < c1; c += kCmpThreads) {
            uint32_t y[R];
#pragma unroll
            for (int s = 0; s < R; ++s) y[s] = __ldcs(row + s * ld + c);
            int p = 0;
#pragma unroll
            for (int s = 0; s < R; ++s)
#pragma unroll
                for (int t = s + 1; t < R; ++t, ++p)
                    neq |= (y[s] != y[t] ? 1u : 0u) << p;
        }
        neq = __reduce_or_sync(0xffffffffu, neq);
        if ((threadIdx.x & 31) == 0 && neq) atomicOr(&file_neq[i], neq);
    }
}

// One block: per-worker disagreement masks from the per-file words, then
// adj[j] = workers j agrees with on every shared file.
__global__ void __launch_bounds__(1024)
graph_kernel(const uint32_t *__restrict__ file_neq, const uint8_t *__restrict__ fw,
             int64_t f, int r, int K, uint32_t *__restrict__ adj)
{
    __shared__ uint32_t dis[32];
    if (threadIdx.x < 32) dis[threadIdx.x] = 0;
    __syncthreads();
    for (int64_t i = threadIdx.x; i < f; i += blockDim.x) {
        uint32_t w = file_neq[i];
        while (w) {
            int rem = __ffs(w) - 1;
            w &= w - 1;
            int s = 0;
            while (rem >= r - 1 - s) {
                rem -= r - 1 - s;
                ++s;
            }
            const int t = s + 1 + rem;
            const int a = fw[i * r + s], b = fw[i * r + t];
            atomicOr(&dis[a], 1u << b);
            atomicOr(&dis[b], 1u << a);
        }
    }
    __syncthreads();
    if (threadIdx.x < (unsigned)K) {
        const uint32_t all = (1u << K) - 1u;                 // K <= 31
        adj[threadIdx.x] = ~dis[threadIdx.x] & all & ~(1u << threadIdx.x);
    }
}

template <int R, int U>
cudaError_t launch_vec(const float *copies, int64_t f, int64_t d, int64_t ld,
                       uint32_t *file_neq, cudaStream_t stream)
{
    const int64_t nvec = d >> 2;
    int64_t nchunks = (nvec + kChunkVec - 1) / kChunkVec;
    if (nchunks < 1) nchunks = 1;
    int per_sm = 0;
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, compare_vec_kernel<R, U>,
                                                  kCmpThreads, 0);
    if (per_sm < 1) per_sm = 1;
    int64_t grid = (int64_t)sm_count() * per_sm;
    if (grid > f * nchunks) grid = f * nchunks;
    compare_vec_kernel<R, U><<<(unsigned)grid, kCmpThreads, 0, stream>>>(
        copies, f, d, ld, nvec, nchunks, file_neq);
    return cudaGetLastError();
}

template <int R>
cudaError_t launch_scalar(const float *copies, int64_t f, int64_t d, int64_t ld,
                          uint32_t *file_neq, cudaStream_t stream)
{
    const int64_t chunk = kChunkVec * 4;
    int64_t nchunks = (d + chunk - 1) / chunk;
    if (nchunks < 1) nchunks = 1;
    int64_t grid = (int64_t)sm_count() * 8;
    if (grid > f * nchunks) grid = f * nchunks;
    compare_scalar_kernel<R><<<(unsigned)grid, kCmpThreads, 0, stream>>>(
        copies, f, d, ld, nchunks, file_neq);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_compare(const float *copies, int64_t f, int r, int64_t d, int64_t ld,
                           uint32_t *file_neq, cudaStream_t stream)
{
    const bool vec = ((uintptr_t)copies % 16 == 0) && (ld % 4 == 0);
    if (vec) {
        switch (r) {
        case 2: return launch_vec<2, 8>(copies, f, d, ld, file_neq, stream);
        case 3: return launch_vec<3, 4>(copies, f, d, ld, file_neq, stream);
        case 4: return launch_vec<4, 4>(copies, f, d, ld, file_neq, stream);
        case 5: return launch_vec<5, 3>(copies, f, d, ld, file_neq, stream);
        case 6: return launch_vec<6, 2>(copies, f, d, ld, file_neq, stream);
        case 7: return launch_vec<7, 2>(copies, f, d, ld, file_neq, stream);
        case 8: return launch_vec<8, 2>(copies, f, d, ld, file_neq, stream);
        default: return cudaErrorInvalidValue;
        }
    }
    switch (r) {
    case 2: return launch_scalar<2>(copies, f, d, ld, file_neq, stream);
    case 3: return launch_scalar<3>(copies, f, d, ld, file_neq, stream);
    case 4: return launch_scalar<4>(copies, f, d, ld, file_neq, stream);
    case 5: return launch_scalar<5>(copies, f, d, ld, file_neq, stream);
    case 6: return launch_scalar<6>(copies, f, d, ld, file_neq, stream);
    case 7: return launch_scalar<7>(copies, f, d, ld, file_neq, stream);
    case 8: return launch_scalar<8>(copies, f, d, ld, file_neq, stream);
    default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_graph(const uint32_t *file_neq, const uint8_t *dev_file_workers, int64_t f,
                         int r, int K, uint32_t *adj, cudaStream_t stream)
{
    graph_kernel<<<1, 1024, 0, stream>>>(file_neq, dev_file_workers, f, r, K, adj);
    return cudaGetLastError();
}

}  // namespace aspis
