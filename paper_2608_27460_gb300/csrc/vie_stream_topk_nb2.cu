// Instantiations of the streaming top-k kernel for query groups of 2.
#include "vie_stream_topk_inst.cuh"

namespace vie {
cudaError_t launch_stream_topk_nb2(int mm, int r, const StreamTopkParams &p, int grid,
                                   uint32_t smem, cudaStream_t stream) {
    return launch_width<2, false>(mm, r, p, grid, smem, stream);
}
}  // namespace vie
