// vie_tc_topk.cu - launchers of the tensor-core head: hi/lo query prep, and
// the tcgen05 projection with per-CTA top-k and the merge in its last CTA.
#include <cuda_bf16.h>

#include <utility>

#include "vie_launch.h"
#include "vie_tc_topk.cuh"

namespace vie {

// hB[n_rows][d_pad] bf16: row 2q = rn(h_q), row 2q+1 = rn(h_q - rn(h_q)),
// rows of absent queries and columns >= d are zero.
__global__ void prep_queries_kernel(const float *__restrict__ h, int nq, int d, int d_pad,
                                    int n_rows, __nv_bfloat16 *__restrict__ hB) {
    griddep_launch_dependents();  // the projection kernel may start its prologue now
    const int64_t n = static_cast<int64_t>(n_rows) * d_pad;
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int r = static_cast<int>(i / d_pad), j = static_cast<int>(i - static_cast<int64_t>(r) * d_pad);
        const int q = r >> 1;
        const float x = (q < nq && j < d) ? h[static_cast<int64_t>(q) * d + j] : 0.0f;
        const __nv_bfloat16 hi = __float2bfloat16_rn(x);
        hB[i] = (r & 1) ? __float2bfloat16_rn(x - __bfloat162float(hi)) : hi;
    }
}

namespace {

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

template <int NQ>
cudaError_t launch_tc_one(const CUtensorMap &mapW, const CUtensorMap &mapH, const TcParams &p,
                          int grid, uint32_t smem, cudaStream_t stream) {
    static bool configured[64] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    if (!configured[dev]) {
        e = cudaFuncSetAttribute(tc_topk_kernel<NQ>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 232448);
        if (e != cudaSuccess) return e;
        configured[dev] = true;
    }
    return launch_pdl(tc_topk_kernel<NQ>, dim3(grid), dim3(TcShape<NQ>::kThreads), smem, stream, mapW,
                      mapH, p);
}

template <int NQ>
int tc_stage_bytes() {
    return TcShape<NQ>::kStageBytes;
}

}  // namespace

bool tc_shape(int nq_tmpl, int kps, int *stages, uint32_t *smem) {
    int score_bytes = 0, buf_bytes = 0, stage_bytes = 0;
    switch (nq_tmpl) {
        case 8: score_bytes = TcShape<8>::kScoreBytes; buf_bytes = TcShape<8>::kBufBytes;
                stage_bytes = TcShape<8>::kStageBytes; break;
        case 16: score_bytes = TcShape<16>::kScoreBytes; buf_bytes = TcShape<16>::kBufBytes;
                 stage_bytes = TcShape<16>::kStageBytes; break;
        case 32: score_bytes = TcShape<32>::kScoreBytes; buf_bytes = TcShape<32>::kBufBytes;
                 stage_bytes = TcShape<32>::kStageBytes; break;
        case 64: score_bytes = TcShape<64>::kScoreBytes; buf_bytes = TcShape<64>::kBufBytes;
                 stage_bytes = TcShape<64>::kStageBytes; break;
        default: return false;
    }
    for (int s = kTcMaxStages; s >= 2; --s) {
        const TcSmemLayout L(score_bytes, buf_bytes, s, kps * stage_bytes);
        if (L.total <= 232448u) {
            *stages = s;
            *smem = L.total;
            return true;
        }
    }
    return false;
}

int tc_max_k(int nq_tmpl) {
    switch (nq_tmpl) {
        case 8: return TcShape<8>::kMaxK;
        case 16: return TcShape<16>::kMaxK;
        case 32: return TcShape<32>::kMaxK;
        case 64: return TcShape<64>::kMaxK;
        default: return 0;
    }
}

cudaError_t launch_tc_topk(int nq_tmpl, const CUtensorMap &mapW, const CUtensorMap &mapH,
                           const TcParams &p, int grid, uint32_t smem, cudaStream_t stream) {
    switch (nq_tmpl) {
        case 8: return launch_tc_one<8>(mapW, mapH, p, grid, smem, stream);
        case 16: return launch_tc_one<16>(mapW, mapH, p, grid, smem, stream);
        case 32: return launch_tc_one<32>(mapW, mapH, p, grid, smem, stream);
        case 64: return launch_tc_one<64>(mapW, mapH, p, grid, smem, stream);
        default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_prep_queries(const float *h, int nq, int d, int d_pad, int n_rows, void *hB,
                                int sms, cudaStream_t stream) {
    const int64_t n = static_cast<int64_t>(n_rows) * d_pad;
    int64_t blocks = (n + 255) / 256;
    if (blocks > 4LL * sms) blocks = 4LL * sms;
    prep_queries_kernel<<<static_cast<unsigned>(blocks), 256, 0, stream>>>(
        h, nq, d, d_pad, n_rows, static_cast<__nv_bfloat16 *>(hB));
    return cudaGetLastError();
}

}  // namespace vie
