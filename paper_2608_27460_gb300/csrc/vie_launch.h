// vie_launch.h - host-side entry points of the kernel instantiations, one
// translation unit per query-group width so they compile in parallel.
#pragma once

#include <cuda_runtime.h>

#include "vie_stream_topk.cuh"

namespace vie {

// Launches stream_topk_kernel<nb, mm, r> on `grid` CTAs; nb in {1,2,4,8},
// mm in {2,8,32}, r in {1,2,4}.  Returns the launch error
// (cudaErrorInvalidValue for an unsupported combination).
cudaError_t launch_stream_topk(int nb, int mm, int r, const StreamTopkParams &p, int grid,
                               uint32_t smem, cudaStream_t stream);

cudaError_t launch_stream_topk_nb1(int mm, int r, const StreamTopkParams &p, int grid,
                                   uint32_t smem, cudaStream_t stream);
cudaError_t launch_stream_topk_nb2(int mm, int r, const StreamTopkParams &p, int grid,
                                   uint32_t smem, cudaStream_t stream);
cudaError_t launch_stream_topk_nb4(int mm, int r, const StreamTopkParams &p, int grid,
                                   uint32_t smem, cudaStream_t stream);
cudaError_t launch_stream_topk_nb8(int mm, int r, const StreamTopkParams &p, int grid,
                                   uint32_t smem, cudaStream_t stream);

}  // namespace vie
