// vie_sample.cu - top-k sampling on the k candidates of each query (paper,
// Section 2: top-k sampling draws the next token from the k most probable
// tokens; Section 3: top-p and min-p act as a second stage on the retrieved
// logits; Section 4 samples with k = 50).
//
// Per query, one warp, in fp32:
//   s_j = z_j / T;  e_j = exp(s_j - max s);  C_j = e_0 + ... + e_j
//   top-p keeps the shortest prefix with C_{n-1} >= top_p * C_{k-1} (>= 1),
//   min-p keeps the j with e_j >= min_p * e_0; the kept set is the shorter
//   prefix (both filters keep prefixes of the sorted candidates);
//   the draw is the first kept j with C_j > u * C_{n-1}.
// u is the top 24 bits of the first word of Philox4x32-10 (Salmon, Moraes,
// Dror, Shaw, SC 2011) at counter (step lo, step hi, query, 0) and key
// (seed lo, seed hi), times 2^-24.
#include <cuda_runtime.h>

#include <cstdint>

#include "vie_device.cuh"
#include "vie_launch.h"

namespace vie {

// Philox4x32 with 10 rounds, from the published round function: the two
// 32x32 -> 64-bit products of words 0 and 2 with the round multipliers, their
// halves crossed with words 1 and 3 and the key, the key advanced by the two
// Weyl constants between rounds.
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint2 key) {
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        if (r > 0) {
            key.x += 0x9E3779B9u;
            key.y += 0xBB67AE85u;
        }
        const uint32_t lo0 = 0xD2511F53u * c.x, hi0 = __umulhi(0xD2511F53u, c.x);
        const uint32_t lo1 = 0xCD9E8D57u * c.z, hi1 = __umulhi(0xCD9E8D57u, c.z);
        c = make_uint4(hi1 ^ c.y ^ key.x, lo1, hi0 ^ c.w ^ key.y, lo0);
    }
    return c;
}

// Candidates per lane: PER contiguous positions lane*PER .. lane*PER+PER-1.
template <int PER>
__global__ void __launch_bounds__(128) sample_topk_kernel(const int32_t *__restrict__ idx,
                                                         const float *__restrict__ logits,
                                                         int batch, int k, float T, float top_p,
                                                         float min_p, uint64_t seed, uint64_t step,
                                                         int32_t *__restrict__ out_token,
                                                         float *__restrict__ out_prob) {
    griddep_wait();  // the candidates may come from the kernel before this one
    const int lane = threadIdx.x & 31;
    const int q = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (q >= batch) return;
    const float *zq = logits + static_cast<int64_t>(q) * k;
    const int j0 = lane * PER;

    float e[PER];
    float mx = -INFINITY;
#pragma unroll
    for (int t = 0; t < PER; ++t) {
        const int j = j0 + t;
        e[t] = j < k ? zq[j] / T : -INFINITY;
        mx = fmaxf(mx, e[t]);
    }
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xFFFFFFFFu, mx, o));
    // weights and this lane's running sums
    float run = 0.0f;
#pragma unroll
    for (int t = 0; t < PER; ++t) {
        e[t] = j0 + t < k ? expf(e[t] - mx) : 0.0f;
        run += e[t];
    }
    // exclusive prefix over lanes: the cumulative weight before this lane's block
    float incl = run;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const float v = __shfl_up_sync(0xFFFFFFFFu, incl, o);
        if (lane >= o) incl += v;
    }
    const float before = incl - run;
    const float total = __shfl_sync(0xFFFFFFFFu, incl, 31);
    const float e0 = __shfl_sync(0xFFFFFFFFu, e[0], 0);

    // top-p: the first j with C_j >= top_p * total gives n_p = j + 1
    // min-p: the number of j with e_j >= min_p * e_0
    const float tp = top_p * total, tm = min_p * e0;
    int first_p = k;
    int n_m = 0;
    float c = before;
#pragma unroll
    for (int t = 0; t < PER; ++t) {
        const int j = j0 + t;
        if (j < k) {
            c += e[t];
            if (c >= tp && first_p == k) first_p = j;
            n_m += e[t] >= tm ? 1 : 0;
        }
    }
    first_p = __reduce_min_sync(0xFFFFFFFFu, first_p);
    n_m = static_cast<int>(__reduce_add_sync(0xFFFFFFFFu, static_cast<unsigned>(n_m)));
    const int n_p = first_p < k ? first_p + 1 : k;
    const int n = max(1, min(n_p, n_m));

    // kept mass M = C_{n-1}, then the inverse CDF at u * M
    float cn = 0.0f;
    c = before;
#pragma unroll
    for (int t = 0; t < PER; ++t) {
        c += e[t];
        if (j0 + t == n - 1) cn = c;
    }
    const float M = __shfl_sync(0xFFFFFFFFu, cn, (n - 1) / PER);
    const uint4 r = philox4x32_10(make_uint4(static_cast<uint32_t>(step), static_cast<uint32_t>(step >> 32),
                                             static_cast<uint32_t>(q), 0u),
                                  make_uint2(static_cast<uint32_t>(seed), static_cast<uint32_t>(seed >> 32)));
    const float u = static_cast<float>(r.x >> 8) * (1.0f / 16777216.0f);
    const float target = u * M;
    int pick = n - 1;
    c = before;
#pragma unroll
    for (int t = 0; t < PER; ++t) {
        const int j = j0 + t;
        c += e[t];
        if (j < n && c > target && pick == n - 1 && j < n - 1) pick = j;
    }
    pick = __reduce_min_sync(0xFFFFFFFFu, pick);
    if (lane == pick / PER) {
        float ep = 0.0f;
#pragma unroll
        for (int t = 0; t < PER; ++t)
            if (j0 + t == pick) ep = e[t];
        out_token[q] = idx[static_cast<int64_t>(q) * k + pick];
        out_prob[q] = ep / M;
    }
}

cudaError_t launch_sample_topk(const int32_t *idx, const float *logits, int batch, int k, float T,
                               float top_p, float min_p, uint64_t seed, uint64_t step,
                               int32_t *out_token, float *out_prob, cudaStream_t stream) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>((batch + 3) / 4));
    cfg.blockDim = dim3(128);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (k <= 64)
        return cudaLaunchKernelEx(&cfg, sample_topk_kernel<2>, idx, logits, batch, k, T, top_p, min_p,
                                  seed, step, out_token, out_prob);
    if (k <= 256)
        return cudaLaunchKernelEx(&cfg, sample_topk_kernel<8>, idx, logits, batch, k, T, top_p, min_p,
                                  seed, step, out_token, out_prob);
    return cudaLaunchKernelEx(&cfg, sample_topk_kernel<32>, idx, logits, batch, k, T, top_p, min_p, seed,
                              step, out_token, out_prob);
}

}  // namespace vie
