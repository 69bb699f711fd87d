// vie_recall.cu - Recall@k bookkeeping on the device (paper, Section 4.3:
// recall is the share of the exact head's top-k tokens that an approximate
// search also retrieves, over many hidden states).
//
// Per query q, one warp: hits[q] = #{ j < k : exact[q, j] >= 0 and
// exact[q, j] is among approx[q, 0..m-1] }.  The candidates act as a set (a
// repeated candidate is found once per exact entry) and negative entries are
// empty slots.  Each lane holds KPL exact entries (lane, lane + 32, ...) and a
// bit per entry; the candidates stream past in coalesced blocks of 32, each
// broadcast to the warp by a shuffle and compared with every held entry.
// Integer work only: the result is exact.
#include <cuda_runtime.h>

#include <cstdint>

#include "vie_device.cuh"
#include "vie_launch.h"

namespace vie {

constexpr int kRecallWarps = 8;

template <int KPL>
__global__ void __launch_bounds__(kRecallWarps * 32) recall_hits_kernel(const int32_t *__restrict__ exact,
                                                                       int k,
                                                                       const int32_t *__restrict__ approx,
                                                                       int m, int64_t n,
                                                                       int32_t *__restrict__ hits) {
    griddep_wait();  // the lists may come from the kernels before this one
    const int lane = threadIdx.x & 31;
    const int64_t q = static_cast<int64_t>(blockIdx.x) * kRecallWarps + (threadIdx.x >> 5);
    if (q >= n) return;
    int32_t e[KPL];
#pragma unroll
    for (int t = 0; t < KPL; ++t) {
        const int j = lane + 32 * t;
        e[t] = j < k ? exact[q * k + j] : -1;
    }
    uint32_t found = 0;
    const int32_t *aq = approx + q * m;
    for (int i0 = 0; i0 < m; i0 += 32) {
        const int32_t mine = i0 + lane < m ? aq[i0 + lane] : -1;
        const int cnt = min(32, m - i0);
        for (int s = 0; s < cnt; ++s) {
            const int32_t a = __shfl_sync(0xFFFFFFFFu, mine, s);
            if (a < 0) continue;  // the same a in every lane: a uniform branch
#pragma unroll
            for (int t = 0; t < KPL; ++t) found |= static_cast<uint32_t>(e[t] == a) << t;
        }
    }
    const int cnt = static_cast<int>(__reduce_add_sync(0xFFFFFFFFu, static_cast<unsigned>(__popc(found))));
    if (lane == 0) hits[q] = cnt;
}

cudaError_t launch_recall_hits(const int32_t *exact, int k, const int32_t *approx, int m, int64_t n,
                               int32_t *hits, cudaStream_t stream) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>((n + kRecallWarps - 1) / kRecallWarps));
    cfg.blockDim = dim3(kRecallWarps * 32);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (k <= 32) return cudaLaunchKernelEx(&cfg, recall_hits_kernel<1>, exact, k, approx, m, n, hits);
    if (k <= 128) return cudaLaunchKernelEx(&cfg, recall_hits_kernel<4>, exact, k, approx, m, n, hits);
    return cudaLaunchKernelEx(&cfg, recall_hits_kernel<32>, exact, k, approx, m, n, hits);
}

}  // namespace vie
