// Instantiations of the streaming top-k kernel on e4m3 rows for query groups of 4.
#include "vie_stream_topk_inst.cuh"

namespace vie {
cudaError_t launch_stream_topk_e4m3_nb4(int mm, int r, const StreamTopkParams &p, int grid,
                                        uint32_t smem, cudaStream_t stream) {
    return launch_width<4, true>(mm, r, p, grid, smem, stream);
}
}  // namespace vie
