// vie_stream_topk_inst.cuh - body shared by the per-width instantiation
// units: sets the shared-memory opt-in once per device and launches.
#pragma once

#include "vie_launch.h"

namespace vie {

template <int NB, int MM, int kR, bool Q8>
cudaError_t launch_one(const StreamTopkParams &p, int grid, uint32_t smem, cudaStream_t stream) {
    static bool configured[64] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    if (!configured[dev]) {
        e = cudaFuncSetAttribute(stream_topk_kernel<NB, MM, kR, Q8>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, 232448);
        if (e != cudaSuccess) return e;
        configured[dev] = true;
    }
    stream_topk_kernel<NB, MM, kR, Q8><<<grid, threads_for<NB>(), smem, stream>>>(p);
    return cudaGetLastError();
}

template <int NB, int R, bool Q8>
cudaError_t launch_rows(int mm, const StreamTopkParams &p, int grid, uint32_t smem,
                        cudaStream_t stream) {
    // 2: register lists (k <= 64); 0: shared-memory candidate buffers
    switch (mm) {
        case 2: return launch_one<NB, 2, R, Q8>(p, grid, smem, stream);
        case 0: return launch_one<NB, 0, R, Q8>(p, grid, smem, stream);
        default: return cudaErrorInvalidValue;
    }
}

template <int NB, bool Q8>
cudaError_t launch_width(int mm, int r, const StreamTopkParams &p, int grid, uint32_t smem,
                         cudaStream_t stream) {
    switch (r) {
        case 1: return launch_rows<NB, 1, Q8>(mm, p, grid, smem, stream);
        case 2: return launch_rows<NB, 2, Q8>(mm, p, grid, smem, stream);
        case 4: return launch_rows<NB, 4, Q8>(mm, p, grid, smem, stream);
        case 8:  // narrow rows, one query: 64-row stages
            if constexpr (NB == 1) return launch_rows<NB, 8, Q8>(mm, p, grid, smem, stream);
            return cudaErrorInvalidValue;
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace vie
