// aspis_round_static: the whole PS round for callers that cannot allocate
// device memory.  Some hosts of this library hand it device buffers they own
// (an embedding runtime with its own memory pool, a process whose allocator
// is locked or budgeted, code running where a cudaMalloc would synchronize
// or fail) but cannot let it call cudaMalloc or cudaFree.  aspis_round needs
// three per-round intermediates from its caller (the per-file mismatch
// words, the graph and the selection) and a device copy of the assignment
// table; here all four live in one fixed file-scope device array instead.
//
// The array is ASPIS_STATIC_SCRATCH_BYTES bytes and is held by every GPU
// that loads the library until the process exits.  Every call shares it, so
// calls that overlap on the GPU (different streams without ordering, or
// several host threads) race on it; calls on one stream are ordered.  Its
// contents carry over from the previous call: the mismatch words, the only
// part that must start at zero, are cleared on the stream by every call.
#include <mutex>

#include "aspis_internal.cuh"

namespace {

constexpr size_t kFwBytes = (size_t)ASPIS_STATIC_MAX_FILES * ASPIS_MAX_R;   // file -> workers
constexpr size_t kNeqOff = kFwBytes;
constexpr size_t kAdjOff = kNeqOff + (size_t)ASPIS_STATIC_MAX_FILES * 4;     // mismatch words
constexpr size_t kSelOff = kAdjOff + 32 * 4;                                 // graph
constexpr size_t kEnd = kSelOff + (size_t)ASPIS_STATIC_MAX_FILES;            // selection
static_assert(kEnd <= ASPIS_STATIC_SCRATCH_BYTES, "static scratch layout exceeds its size");
static_assert(kNeqOff % 256 == 0 && kAdjOff % 4 == 0, "scratch sections must stay aligned");

__device__ __align__(256) unsigned char g_round_scratch[ASPIS_STATIC_SCRATCH_BYTES];

// Host code cannot use g_round_scratch as an address: on the host the name
// refers to a host-side shadow.  The device address is looked up once per
// device, with that device current, and kept here for the life of the
// process (a cudaDeviceReset of the device makes it stale; the header says
// so).
constexpr int kMaxDevices = 64;
std::mutex g_mu;
unsigned char *g_dev_ptr[kMaxDevices] = {nullptr};

aspis_status scratch_for_current_device(unsigned char **out)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return ASPIS_E_CUDA;
    if (dev < 0 || dev >= kMaxDevices) return ASPIS_E_RANGE;
    std::lock_guard<std::mutex> g(g_mu);
    if (!g_dev_ptr[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_round_scratch) != cudaSuccess || !p) return ASPIS_E_CUDA;
        g_dev_ptr[dev] = static_cast<unsigned char *>(p);
    }
    *out = g_dev_ptr[dev];
    return ASPIS_OK;
}

}  // namespace

extern "C" aspis_status aspis_round_static(const float *copies, int64_t d, int64_t ld,
                                           const aspis_assignment *a, aspis_detection *det,
                                           int mode, float *out, void *stream)
{
    using namespace aspis;
    if (!a || !a->file_workers || !copies || !det || !out) return ASPIS_E_INVAL;
    if (a->r < 2 || a->K < a->r || a->f < 1 || d < 1 || ld < d) return ASPIS_E_INVAL;
    if (mode != 0 && mode != 1) return ASPIS_E_INVAL;
    if (a->K > ASPIS_MAX_K || a->r > ASPIS_MAX_R) return ASPIS_E_RANGE;
    if (a->f > ASPIS_STATIC_MAX_FILES) return ASPIS_E_RANGE;
    if (ld > (int64_t)(INT64_MAX / 8) / (a->f * a->r)) return ASPIS_E_RANGE;

    unsigned char *base = nullptr;
    aspis_status s = scratch_for_current_device(&base);
    if (s != ASPIS_OK) return s;
    uint8_t *fw = base;
    uint32_t *file_neq = reinterpret_cast<uint32_t *>(base + kNeqOff);
    uint32_t *adj = reinterpret_cast<uint32_t *>(base + kAdjOff);
    int8_t *sel = reinterpret_cast<int8_t *>(base + kSelOff);

    cudaStream_t st = (cudaStream_t)stream;
    const int64_t f = a->f;
    const int r = a->r;
    if (cudaMemcpyAsync(fw, a->file_workers, (size_t)(f * r), cudaMemcpyHostToDevice, st) !=
        cudaSuccess)
        return ASPIS_E_CUDA;
    if (cudaMemsetAsync(file_neq, 0, sizeof(uint32_t) * (size_t)f, st) != cudaSuccess)
        return ASPIS_E_CUDA;
    if (launch_compare(copies, f, r, d, ld, file_neq, st) != cudaSuccess) return ASPIS_E_CUDA;
    if (launch_graph(file_neq, fw, f, r, a->K, adj, st) != cudaSuccess) return ASPIS_E_CUDA;
    if (launch_detect(adj, a->K, det, st) != cudaSuccess) return ASPIS_E_CUDA;
    if (launch_select(file_neq, det, fw, f, r, sel, st) != cudaSuccess) return ASPIS_E_CUDA;
    if (launch_aggregate(copies, f, r, d, ld, sel, det, mode, out, st) != cudaSuccess)
        return ASPIS_E_CUDA;
    return ASPIS_OK;
}
