// vie_tc_launch.cuh - launch helpers of the tensor-core head, shared by the
// translation units that instantiate its kernel (bf16 and e4m3 rows).
#pragma once

#include <cuda_runtime.h>

#include <utility>

#include "vie_tc_topk.cuh"

namespace vie {

// Launch with programmatic stream serialisation (the kernel calls
// griddep_wait before it touches what the previous kernel wrote).
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, uint32_t smem,
                       cudaStream_t stream, Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...);
}

template <int NQ, bool Q8>
cudaError_t launch_tc_one(const CUtensorMap &mapW, const CUtensorMap &mapH, const TcParams &p,
                          int grid, uint32_t smem, cudaStream_t stream) {
    static bool configured[64] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    if (!configured[dev]) {
        e = cudaFuncSetAttribute(tc_topk_kernel<NQ, Q8>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 232448);
        if (e != cudaSuccess) return e;
        configured[dev] = true;
    }
    return launch_pdl(tc_topk_kernel<NQ, Q8>, dim3(grid), dim3(TcShape<NQ, Q8>::kThreads), smem, stream,
                      mapW, mapH, p);
}

}  // namespace vie
