// Internal declarations shared by the libaspis translation units.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "aspis.h"

namespace aspis {

// Launch helpers: enqueue on `stream`, return cudaGetLastError().
cudaError_t launch_compare(const float *copies, int64_t f, int r, int64_t d,
                           int64_t ld, uint32_t *file_neq, cudaStream_t stream);
cudaError_t launch_graph(const uint32_t *file_neq, const uint8_t *dev_file_workers,
                         int64_t f, int r, int K, uint32_t *adj, cudaStream_t stream);
cudaError_t launch_detect(const uint32_t *adj, int K, aspis_detection *det,
                          cudaStream_t stream);
cudaError_t launch_select(const uint32_t *file_neq, aspis_detection *det,
                          const uint8_t *dev_file_workers, int64_t f, int r,
                          int8_t *sel, cudaStream_t stream);
cudaError_t launch_aggregate(const float *copies, int64_t f, int r, int64_t d,
                             int64_t ld, const int8_t *sel, aspis_detection *det,
                             int mode, float *out, cudaStream_t stream);

// Number of SMs of the current device (cached per device).
int sm_count();

__host__ __device__ inline int pair_count(int r) { return r * (r - 1) / 2; }

}  // namespace aspis
