// vie_tc_topk_e4m3.cu - the tensor-core head on e4m3 rows (tcgen05
// kind::f8f6f4): the query prep that splits each fp32 query into e4m3 pieces,
// and the kernel instances for 4, 8, 16 and 32 query slots.
#include <cuda_fp16.h>
#include <cuda_fp8.h>

#include "vie_launch.h"
#include "vie_tc_launch.cuh"

namespace vie {

namespace {

__device__ float block_max(float v, float *red) {
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xFFFFFFFFu, v, o));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    __syncthreads();  // red is reused from the previous call
    if (lane == 0) red[warp] = v;
    __syncthreads();
    v = lane < static_cast<int>(blockDim.x >> 5) ? red[lane] : 0.0f;
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xFFFFFFFFu, v, o));
    return v;
}

}  // namespace

// Query q of the group, columns [1024 x, 1024 x + 1024) per CTA (grid
// (ceil(d_pad / 1024), NQ)).  With M = max_j |h_qj| and s_0 = the least power
// of two >= M / 448, piece p has the scale s_p = s_0 2^-4p and the codes
//   c_pj = e4m3(r_pj / s_p)  (round to nearest even; the quotient is exact),
//   r_0j = h_qj,  r_(p+1)j = r_pj - s_p e4m3(c_pj)  (exact).
// A residual is at most half an e4m3 step of its code: |r_1 / s_0| <= 16, so
// |r_1 / s_1| <= 256, then 128, then 64 - no piece saturates, and each takes
// 4 more significand bits, leaving |r_4j| <= 2^-16 |h_qj| (plus at most
// s_0 2^-22 for entries far below M).  One reduction per CTA (M, over the whole
// query) and no other synchronisation.
//   hQ[4q + p][j] = c_pj  (uint8 [4 NQ][d_pad]),   qscale[4q + p] = s_p.
constexpr int kPrepCols = 1024;
__global__ void __launch_bounds__(256) prep_queries_e4m3_kernel(const float *__restrict__ h, int nq, int d,
                                                                int d_pad, uint8_t *__restrict__ hQ,
                                                                float *__restrict__ qscale) {
    griddep_launch_dependents();  // the projection kernel may start its prologue now
    __shared__ float red[32];
    const int q = blockIdx.y;
    const bool real = q < nq;
    const float *hq = h + static_cast<int64_t>(q) * d;
    float mx = 0.0f;
    if (real)
        for (int j = threadIdx.x; j < d; j += blockDim.x) mx = fmaxf(mx, fabsf(hq[j]));
    mx = block_max(mx, red);
    const float s0 = pow2_at_least(mx / 448.0f);
    const int j0 = blockIdx.x * kPrepCols;
    for (int j = j0 + threadIdx.x; j < j0 + kPrepCols && j < d_pad; j += blockDim.x) {
        float r = (real && j < d) ? hq[j] : 0.0f;
        float s = s0;
#pragma unroll
        for (int pc = 0; pc < kQ8Pieces; ++pc) {
            const uint8_t c = e4m3_code(r / s);
            hQ[static_cast<int64_t>(kQ8Pieces * q + pc) * d_pad + j] = c;
            r -= s * e4m3_value(c);
            s *= 0x1p-4f;
        }
    }
    if (blockIdx.x == 0 && threadIdx.x < kQ8Pieces)
        qscale[kQ8Pieces * q + threadIdx.x] = s0 * __uint_as_float((127u - 4u * threadIdx.x) << 23);
}

cudaError_t launch_prep_queries_e4m3(const float *h, int nq, int nq_tmpl, int d, int d_pad, void *hQ,
                                     float *qscale, cudaStream_t stream) {
    const dim3 grid(static_cast<unsigned>((d_pad + kPrepCols - 1) / kPrepCols), static_cast<unsigned>(nq_tmpl));
    prep_queries_e4m3_kernel<<<grid, 256, 0, stream>>>(h, nq, d, d_pad, static_cast<uint8_t *>(hQ), qscale);
    return cudaGetLastError();
}

cudaError_t launch_tc_topk_e4m3(int nq_tmpl, const CUtensorMap &mapW, const CUtensorMap &mapH,
                                const TcParams &p, int grid, uint32_t smem, cudaStream_t stream) {
    switch (nq_tmpl) {
        case 4: return launch_tc_one<4, true>(mapW, mapH, p, grid, smem, stream);
        case 8: return launch_tc_one<8, true>(mapW, mapH, p, grid, smem, stream);
        case 16: return launch_tc_one<16, true>(mapW, mapH, p, grid, smem, stream);
        case 32: return launch_tc_one<32, true>(mapW, mapH, p, grid, smem, stream);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace vie
