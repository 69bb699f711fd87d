// vie_launch.h - host-side entry points of the kernel instantiations, one
// translation unit per query-group width so they compile in parallel.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>

#include "vie_stream_topk.cuh"

namespace vie {

// Launches stream_topk_kernel<nb, mm, r> on `grid` CTAs; nb in {1,2,4,8},
// mm in {2 (register lists), 0 (candidate buffers)}, r in {1,2,4,8}.  Returns the launch error
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
// The same on rows of e4m3 codes with per-row scales (p.row_scale).
cudaError_t launch_stream_topk_e4m3_nb1(int mm, int r, const StreamTopkParams &p, int grid,
                                        uint32_t smem, cudaStream_t stream);
cudaError_t launch_stream_topk_e4m3_nb2(int mm, int r, const StreamTopkParams &p, int grid,
                                        uint32_t smem, cudaStream_t stream);
cudaError_t launch_stream_topk_e4m3_nb4(int mm, int r, const StreamTopkParams &p, int grid,
                                        uint32_t smem, cudaStream_t stream);
cudaError_t launch_stream_topk_e4m3_nb8(int mm, int r, const StreamTopkParams &p, int grid,
                                        uint32_t smem, cudaStream_t stream);


// ---- tensor-core head (vie_tc_topk.cu) ----
struct TcParams;

// Recall@k: per query, how many exact top-k indices the candidates contain.
cudaError_t launch_recall_hits(const int32_t *exact, int k, const int32_t *approx, int m, int64_t n,
                               int32_t *hits, cudaStream_t stream);
// Top-k sampling: one draw per query from its k sorted candidates.
cudaError_t launch_sample_topk(const int32_t *idx, const float *logits, int batch, int k, float T,
                               float top_p, float min_p, uint64_t seed, uint64_t step,
                               int32_t *out_token, float *out_prob, cudaStream_t stream);

// Largest k the tensor-core kernel with nq_tmpl query slots handles (q8: on
// e4m3 rows).
int tc_max_k(int nq_tmpl, bool q8 = false);
// Rows of W per tile of that kernel (128, or 256 for the 64-query bf16 tile).
int tc_tile_rows(int nq_tmpl, bool q8 = false);
// Ring depth, score-ring depth and dynamic shared memory for query groups of
// nq_tmpl (8, 16, 32 or 64; 4, 8, 16 or 32 on e4m3 rows), kps K-blocks per
// stage and hres_bytes of query operand built in shared memory; false if
// unsupported.
bool tc_shape(int nq_tmpl, bool q8, int kps, int hres_bytes, int *stages, int *slots, uint32_t *smem);
// Bytes of the query operand each CTA builds in shared memory itself for this
// group shape and n_kb K-blocks (0: a prep kernel writes it and its boxes
// travel with every ring stage).
int tc_hres_bytes(int nq_tmpl, bool q8, int n_kb);

// Launches tc_topk_kernel<nq_tmpl, q8>.
cudaError_t launch_tc_topk(int nq_tmpl, bool q8, const CUtensorMap &mapW, const CUtensorMap &mapH,
                           const TcParams &p, int grid, uint32_t smem, cudaStream_t stream);
cudaError_t launch_tc_topk_e4m3(int nq_tmpl, const CUtensorMap &mapW, const CUtensorMap &mapH,
                                const TcParams &p, int grid, uint32_t smem, cudaStream_t stream);

// e4m3 query pieces hQ [4 nq_tmpl][d_pad] and their scales [4 nq_tmpl] for
// the tensor-core kernel on e4m3 rows (d_pad <= 24576).
cudaError_t launch_prep_queries_e4m3(const float *h, int nq, int nq_tmpl, int d, int d_pad, void *hQ,
                                     float *qscale, cudaStream_t stream);

// hi/lo bf16 query matrix [n_rows][d_pad] for the tensor-core kernel.
cudaError_t launch_prep_queries(const float *h, int nq, int d, int d_pad, int n_rows, void *hB,
                                int sms, cudaStream_t stream);

}  // namespace vie
