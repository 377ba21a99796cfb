// C-ABI entry points of libaspis: argument checks, then the kernel launches
// of check.cu, detect.cu and aggregate.cu on the caller's stream.
#include <cstdlib>
#include <cstring>
#include <mutex>

#include "aspis_internal.cuh"

namespace aspis {


int sm_count()
{
    static std::mutex mu;
    static int cached[64] = {0};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev < 0 || dev >= 64) dev = 0;
    std::lock_guard<std::mutex> g(mu);
    if (!cached[dev]) {
        int n = 0;
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
        cached[dev] = n > 0 ? n : 1;
    }
    return cached[dev];
}

}  // namespace aspis

using namespace aspis;

namespace {

// Pinned host memory is mapped into the device's address space, and over the
// Grace-Blackwell host link SM loads of it stream at the link's rate (about
// 205 GB/s for a 61 GB buffer, steady from run to run) where the copy engines
// moved the same buffer at 135-210 GB/s.  So a large copy from a
// device-mapped host buffer is a grid-stride kernel of 16-byte loads and
// stores; returns false (nothing enqueued) when the buffer is not
// device-mapped or not 16-byte aligned, and the copy engines take it.
__global__ void __launch_bounds__(256)
h2d_copy_kernel(const uint4 *__restrict__ src, uint4 *__restrict__ dst, int64_t n16)
{
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n16;
         i += (int64_t)gridDim.x * blockDim.x)
        dst[i] = __ldcs(src + i);
}

bool h2d_sm(void *dst, const void *src, size_t bytes, cudaStream_t st, cudaError_t &err)
{
    cudaPointerAttributes at{};
    if (cudaPointerGetAttributes(&at, src) != cudaSuccess) {
        cudaGetLastError();                          // not a pointer CUDA knows: clear the error
        return false;
    }
    if (at.type != cudaMemoryTypeHost || !at.devicePointer) return false;
    if (((uintptr_t)at.devicePointer | (uintptr_t)dst | (uintptr_t)bytes) % 16 != 0) return false;
    const int64_t n16 = (int64_t)(bytes / 16);
    int64_t grid = (int64_t)sm_count() * 8;
    if (grid > (n16 + 255) / 256) grid = (n16 + 255) / 256;
    h2d_copy_kernel<<<(unsigned)grid, 256, 0, st>>>(static_cast<const uint4 *>(at.devicePointer),
                                                    static_cast<uint4 *>(dst), n16);
    err = cudaGetLastError();
    return true;
}

// The copy and the compare of aspis_round_host overlap for pinned inputs: the
// copy kernel moves file-aligned chunks over the host link on the caller's
// stream with two CTAs per SM (the link saturates well below that), and each
// chunk's compare runs on a library-owned stream as soon as the chunk has
// landed, on the SMs the copy leaves free.  Only the last chunk's compare,
// the graph and the rest of the round follow the last byte.  Events are
// recorded and waited on under one lock, so concurrent callers cannot mix
// them up (their compares then share the side stream).
constexpr int kPipeChunks = 8;
struct PipeLanes {
    bool ready = false;
    cudaStream_t side;
    cudaEvent_t landed[kPipeChunks], compared;
};
std::mutex g_pipe_mu;
PipeLanes g_pipe[64];

bool copy_and_compare(const float *host, float *dev, int64_t d, int64_t ld,
                      const aspis_assignment *a, uint32_t *file_neq, cudaStream_t st,
                      cudaError_t &err)
{
    cudaPointerAttributes at{};
    if (cudaPointerGetAttributes(&at, host) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    if (at.type != cudaMemoryTypeHost || !at.devicePointer) return false;
    // every chunk starts at a file boundary: 16-byte aligned when ld % 4 == 0
    if (((uintptr_t)at.devicePointer | (uintptr_t)dev) % 16 != 0 || ld % 4 != 0) return false;
    int devno = 0;
    if ((err = cudaGetDevice(&devno)) != cudaSuccess) return true;
    if (devno < 0 || devno >= 64) return false;
    std::lock_guard<std::mutex> g(g_pipe_mu);
    PipeLanes &L = g_pipe[devno];
    if (!L.ready) {
        if ((err = cudaStreamCreateWithFlags(&L.side, cudaStreamNonBlocking)) != cudaSuccess) return true;
        for (int k = 0; k < kPipeChunks; ++k)
            if ((err = cudaEventCreateWithFlags(&L.landed[k], cudaEventDisableTiming)) != cudaSuccess)
                return true;
        if ((err = cudaEventCreateWithFlags(&L.compared, cudaEventDisableTiming)) != cudaSuccess)
            return true;
        L.ready = true;
    }
    const int64_t f = a->f, r = a->r, row = r * ld;               // floats per file
    if ((err = cudaMemsetAsync(file_neq, 0, sizeof(uint32_t) * (size_t)f, st)) != cudaSuccess)
        return true;
    const int64_t per = (f + kPipeChunks - 1) / kPipeChunks;
    const float *src = static_cast<const float *>(at.devicePointer);
    for (int k = 0; k < kPipeChunks; ++k) {
        const int64_t i0 = k * per, i1 = i0 + per < f ? i0 + per : f;
        if (i0 >= i1) break;
        const int64_t n16 = (i1 - i0) * row / 4;
        int64_t grid = (int64_t)sm_count() * 2;
        if (grid > (n16 + 255) / 256) grid = (n16 + 255) / 256;
        h2d_copy_kernel<<<(unsigned)grid, 256, 0, st>>>(reinterpret_cast<const uint4 *>(src + i0 * row),
                                                        reinterpret_cast<uint4 *>(dev + i0 * row), n16);
        if ((err = cudaGetLastError()) != cudaSuccess) return true;
        if ((err = cudaEventRecord(L.landed[k], st)) != cudaSuccess) return true;
        if ((err = cudaStreamWaitEvent(L.side, L.landed[k], 0)) != cudaSuccess) return true;
        if ((err = launch_compare(dev + i0 * row, i1 - i0, (int)r, d, ld, file_neq + i0, L.side)) !=
            cudaSuccess)
            return true;
    }
    if ((err = cudaEventRecord(L.compared, L.side)) != cudaSuccess) return true;
    err = cudaStreamWaitEvent(st, L.compared, 0);
    return true;
}

// Other host-to-device copies of the round's inputs are split over kLanes streams
// so that several copy engines move them at once; the caller's stream waits
// for all of them.  Streams and events are created once per device.
constexpr int kLanes = 4;
struct CopyLanes {
    bool ready = false;
    cudaStream_t s[kLanes];
    cudaEvent_t start, done[kLanes];
};
std::mutex g_lanes_mu;
CopyLanes g_lanes[64];

cudaError_t h2d_split(void *dst, const void *src, size_t bytes, cudaStream_t st)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64 || bytes < ((size_t)64 << 20))
        return cudaMemcpyAsync(dst, src, bytes, cudaMemcpyHostToDevice, st);
    std::lock_guard<std::mutex> g(g_lanes_mu);
    CopyLanes &L = g_lanes[dev];
    if (!L.ready) {
        for (int i = 0; i < kLanes; ++i) {
            if ((e = cudaStreamCreateWithFlags(&L.s[i], cudaStreamNonBlocking)) != cudaSuccess) return e;
            if ((e = cudaEventCreateWithFlags(&L.done[i], cudaEventDisableTiming)) != cudaSuccess) return e;
        }
        if ((e = cudaEventCreateWithFlags(&L.start, cudaEventDisableTiming)) != cudaSuccess) return e;
        L.ready = true;
    }
    if ((e = cudaEventRecord(L.start, st)) != cudaSuccess) return e;
    const size_t chunk = (bytes / kLanes + 4095) / 4096 * 4096;
    for (int i = 0; i < kLanes; ++i) {
        const size_t off = (size_t)i * chunk;
        if (off >= bytes) break;
        const size_t len = bytes - off < chunk ? bytes - off : chunk;
        if ((e = cudaStreamWaitEvent(L.s[i], L.start, 0)) != cudaSuccess) return e;
        e = cudaMemcpyAsync(static_cast<char *>(dst) + off, static_cast<const char *>(src) + off, len,
                            cudaMemcpyHostToDevice, L.s[i]);
        if (e != cudaSuccess) return e;
        if ((e = cudaEventRecord(L.done[i], L.s[i])) != cudaSuccess) return e;
        if ((e = cudaStreamWaitEvent(st, L.done[i], 0)) != cudaSuccess) return e;
    }
    return cudaSuccess;
}

}  // namespace

namespace {

inline aspis_status cuda_status(cudaError_t e) { return e == cudaSuccess ? ASPIS_OK : ASPIS_E_CUDA; }

aspis_status check_assignment(const aspis_assignment *a)
{
    if (!a || !a->dev_file_workers) return ASPIS_E_INVAL;
    if (a->r < 2 || a->K < a->r || a->f < 1) return ASPIS_E_INVAL;
    if (a->K > ASPIS_MAX_K || a->r > ASPIS_MAX_R) return ASPIS_E_RANGE;
    return ASPIS_OK;
}

aspis_status check_copies(const float *copies, int64_t d, int64_t ld, const aspis_assignment *a)
{
    if (!copies || d < 1 || ld < d) return ASPIS_E_INVAL;
    // every element index i*r*ld + s*ld + c must fit in int64
    const int64_t rows = a->f * a->r;
    if (ld > (int64_t)(INT64_MAX / 8) / rows) return ASPIS_E_RANGE;
    return ASPIS_OK;
}

}  // namespace

extern "C" aspis_status aspis_assignment_to_device(aspis_assignment *a)
{
    if (!a || !a->file_workers || a->f < 1 || a->r < 2) return ASPIS_E_INVAL;
    if (a->dev_file_workers) return ASPIS_OK;
    uint8_t *p = nullptr;
    const size_t bytes = (size_t)(a->f * a->r);
    if (cudaMalloc(&p, bytes) != cudaSuccess) return ASPIS_E_CUDA;
    if (cudaMemcpy(p, a->file_workers, bytes, cudaMemcpyHostToDevice) != cudaSuccess) {
        cudaFree(p);
        return ASPIS_E_CUDA;
    }
    a->dev_file_workers = p;
    return ASPIS_OK;
}

extern "C" void aspis_assignment_free(aspis_assignment *a)
{
    if (!a) return;
    std::free(a->file_workers);
    std::free(a->worker_files);
    std::free(a->slot_of);
    if (a->dev_file_workers) cudaFree(a->dev_file_workers);
    std::memset(a, 0, sizeof(*a));
}

extern "C" aspis_status aspis_check(const float *copies, int64_t d, int64_t ld,
                                    const aspis_assignment *a, uint32_t *file_neq,
                                    uint32_t *adj, void *stream)
{
    aspis_status s = check_assignment(a);
    if (s != ASPIS_OK) return s;
    if ((s = check_copies(copies, d, ld, a)) != ASPIS_OK) return s;
    if (!file_neq || !adj) return ASPIS_E_INVAL;
    cudaStream_t st = (cudaStream_t)stream;
    if (cudaMemsetAsync(file_neq, 0, sizeof(uint32_t) * (size_t)a->f, st) != cudaSuccess)
        return ASPIS_E_CUDA;
    if ((s = cuda_status(launch_compare(copies, a->f, a->r, d, ld, file_neq, st))) != ASPIS_OK)
        return s;
    return cuda_status(launch_graph(file_neq, a->dev_file_workers, a->f, a->r, a->K, adj, st));
}

extern "C" aspis_status aspis_graph(const uint32_t *file_neq, const aspis_assignment *a,
                                    uint32_t *adj, void *stream)
{
    aspis_status s = check_assignment(a);
    if (s != ASPIS_OK) return s;
    if (!file_neq || !adj) return ASPIS_E_INVAL;
    return cuda_status(launch_graph(file_neq, a->dev_file_workers, a->f, a->r, a->K, adj,
                                    (cudaStream_t)stream));
}

extern "C" aspis_status aspis_detect(const uint32_t *adj, int K, aspis_detection *det,
                                     void *stream)
{
    if (!adj || !det) return ASPIS_E_INVAL;
    if (K < 2) return ASPIS_E_INVAL;
    if (K > ASPIS_MAX_K) return ASPIS_E_RANGE;
    return cuda_status(launch_detect(adj, K, det, (cudaStream_t)stream));
}

extern "C" aspis_status aspis_select(const uint32_t *file_neq, aspis_detection *det,
                                     const aspis_assignment *a, int8_t *sel, void *stream)
{
    aspis_status s = check_assignment(a);
    if (s != ASPIS_OK) return s;
    if (!file_neq || !det || !sel) return ASPIS_E_INVAL;
    return cuda_status(launch_select(file_neq, det, a->dev_file_workers, a->f, a->r, sel,
                                     (cudaStream_t)stream));
}

extern "C" aspis_status aspis_aggregate(const float *copies, int64_t d, int64_t ld,
                                        const aspis_assignment *a, const int8_t *sel,
                                        aspis_detection *det, int mode, float *out,
                                        void *stream)
{
    aspis_status s = check_assignment(a);
    if (s != ASPIS_OK) return s;
    if ((s = check_copies(copies, d, ld, a)) != ASPIS_OK) return s;
    if (!sel || !det || !out || (mode != 0 && mode != 1)) return ASPIS_E_INVAL;
    if (a->f > ASPIS_MAX_AGG_FILES) return ASPIS_E_RANGE;
    return cuda_status(launch_aggregate(copies, a->f, a->r, d, ld, sel, det, mode, out,
                                        (cudaStream_t)stream));
}

extern "C" aspis_status aspis_round(const float *copies, int64_t d, int64_t ld,
                                    const aspis_assignment *a, uint32_t *file_neq,
                                    uint32_t *adj, aspis_detection *det, int8_t *sel,
                                    int mode, float *out, void *stream)
{
    aspis_status s = check_assignment(a);
    if (s != ASPIS_OK) return s;
    if ((s = check_copies(copies, d, ld, a)) != ASPIS_OK) return s;
    if (!file_neq || !adj || !det || !sel || !out || (mode != 0 && mode != 1))
        return ASPIS_E_INVAL;
    if (a->f > ASPIS_MAX_AGG_FILES) return ASPIS_E_RANGE;
    if ((s = aspis_check(copies, d, ld, a, file_neq, adj, stream)) != ASPIS_OK) return s;
    if ((s = aspis_detect(adj, a->K, det, stream)) != ASPIS_OK) return s;
    if ((s = aspis_select(file_neq, det, a, sel, stream)) != ASPIS_OK) return s;
    return aspis_aggregate(copies, d, ld, a, sel, det, mode, out, stream);
}

extern "C" aspis_status aspis_round_host(const float *host_copies, float *dev_copies,
                                         int64_t d, int64_t ld, const aspis_assignment *a,
                                         uint32_t *file_neq, uint32_t *adj,
                                         aspis_detection *det, int8_t *sel, int mode,
                                         float *dev_out, float *host_out,
                                         aspis_detection *host_det, void *stream)
{
    aspis_status s = check_assignment(a);
    if (s != ASPIS_OK) return s;
    if (!host_copies || !host_out || !host_det) return ASPIS_E_INVAL;
    if ((s = check_copies(dev_copies, d, ld, a)) != ASPIS_OK) return s;
    cudaStream_t st = (cudaStream_t)stream;
    const size_t bytes = sizeof(float) * (size_t)(a->f * a->r) * (size_t)ld;
    if (!file_neq || !adj || !det || !sel || !dev_out || (mode != 0 && mode != 1))
        return ASPIS_E_INVAL;
    if (a->f > ASPIS_MAX_AGG_FILES) return ASPIS_E_RANGE;
    cudaError_t e = cudaSuccess;
    const bool piped = bytes >= ((size_t)64 << 20) &&
                       copy_and_compare(host_copies, dev_copies, d, ld, a, file_neq, st, e);
    if (e != cudaSuccess) return ASPIS_E_CUDA;
    if (piped) {
        // the copies are on the device and compared: the rest of the round
        if ((s = aspis_graph(file_neq, a, adj, stream)) != ASPIS_OK) return s;
        if ((s = aspis_detect(adj, a->K, det, stream)) != ASPIS_OK) return s;
        if ((s = aspis_select(file_neq, det, a, sel, stream)) != ASPIS_OK) return s;
        if ((s = aspis_aggregate(dev_copies, d, ld, a, sel, det, mode, dev_out, stream)) != ASPIS_OK)
            return s;
    } else {
        const bool by_sm =
            bytes >= ((size_t)64 << 20) && h2d_sm(dev_copies, host_copies, bytes, st, e);
        if (!by_sm) e = h2d_split(dev_copies, host_copies, bytes, st);
        if (e != cudaSuccess) return ASPIS_E_CUDA;
        s = aspis_round(dev_copies, d, ld, a, file_neq, adj, det, sel, mode, dev_out, stream);
        if (s != ASPIS_OK) return s;
    }
    if (cudaMemcpyAsync(host_out, dev_out, sizeof(float) * (size_t)d, cudaMemcpyDeviceToHost,
                        st) != cudaSuccess)
        return ASPIS_E_CUDA;
    if (cudaMemcpyAsync(host_det, det, sizeof(aspis_detection), cudaMemcpyDeviceToHost, st) !=
        cudaSuccess)
        return ASPIS_E_CUDA;
    return ASPIS_OK;
}
