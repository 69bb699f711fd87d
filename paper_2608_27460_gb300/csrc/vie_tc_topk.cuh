// vie_tc_topk.cuh - the batched output head on the 5th-generation tensor
// cores: Z[V, b] = W[V, d] * H[d, b] (paper, Section 3, z = W_out h for b
// queries at once) with the exact per-CTA top-k fused into the epilogue.
//
// h is fp32; tcgen05 kind::f16 needs both operands in bf16, so each query
// enters as two bf16 columns hi = rn(h), lo = rn(h - hi) and its logit is the
// sum of the two accumulator columns (residual error <= 2^-16 |h| per term).
// N = 2 * NQ accumulator columns per tile.
//
// One persistent CTA per SM walks 128-row tiles of W (round robin, then an
// atomic pool).  Per tile, d/64 K-blocks flow through a shared-memory ring;
// a stage is one 2-D TMA box of W (128 rows x 64 bf16, 128-byte swizzle)
// plus the matching box of the hi/lo query matrix (N rows x 64).
//   warp 0       TMA producer;
//   warp 1       TMEM allocator and the single MMA-issuing thread:
//                4 x tcgen05.mma (M=128, N, K=16) per stage into one of two
//                TMEM accumulators, tcgen05.commit frees the stage;
//   warps 2-5    epilogue: tcgen05.ld of the 128 x N accumulator (warp w
//                owns TMEM lanes 32*(w%4)..), hi + lo per query, logits into
//                a score ring laid out [query][row];
//   warps 6..    selectors, one query each (two when NQ = 32, four when
//                NQ = 64): per query a sorted list of the best keys so far,
//                spread over the warp's registers (the streaming kernel's
//                WarpList); a row enters only when its key beats the list's
//                k-th, so the lists are final when the stream ends.
// Each CTA writes its per-query lists and takes a completion ticket; the
// last CTAs to finish merge them, one query each.  All waits are bounded.
//
// Q8 (e4m3 rows with one fp32 scale each, tcgen05 kind::f8f6f4): a K-block
// is 128 codes (the same 128-byte swizzle row), and each query enters as four
// e4m3 columns c_0..c_3 with power-of-two scales s_0..s_3 such that
// h ~ sum_p s_p c_p (each piece takes 4 more significand bits of what the
// previous left, so the residual is below 2^-16 |h| per term, as with the bf16
// hi/lo split); the logit of row i is scale_i * sum_p s_p acc_p.
//
// Small e4m3 groups (h_resident): every CTA builds the whole query operand
// (the four e4m3 pieces of each query) itself, straight into shared memory in
// the 128-byte-swizzled K-major layout the MMA reads, so the call needs no
// separate query-prep kernel and the ring carries weights only.  (For the
// 8-query bf16 tile the same build measured slower than the prep kernel.)
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_fp8.h>
#include <cstdint>

#include "vie_stream_topk.cuh"
#include "vie_tcgen05.cuh"

namespace vie {

constexpr int kTcTile = 128;       // rows per tile (MMA M)
constexpr int kTcKBlock = 64;      // bf16 columns per K-block (one 128-byte swizzle row)
constexpr int kTcScoreSlots = 8;   // score ring depth, at most (chosen per launch)
constexpr int kTcMaxStages = 16;
constexpr int kTcHRows = 128;      // rows of the hi/lo query matrix (N <= 128)
constexpr int kTcMaxK = 128;       // largest k of this path
constexpr int kTcListKeys = 4096;  // keys of the per-CTA lists per CTA: NQ * k <= this
constexpr int kTcMaxKPS = 4;       // K-blocks per stage, at most
constexpr int kTcMergeE = 8;       // merge: keys per list in the heads area
constexpr int kQ8Pieces = 4;       // e4m3 columns per query on the Q8 path
constexpr int kTcMaxMergers = 64;  // CTAs that merge, at most (one per query)

struct TcParams {
    int64_t V;
    int32_t d_pad;
    int32_t k;
    int32_t nq;              // queries of this launch (<= NQ)
    int32_t stages;          // ring depth
    int32_t static_tiles;    // tiles each CTA owns before drawing from the pool
    int32_t kb_per_stage;    // K-blocks per ring stage (1..kTcMaxKPS)
    int32_t score_slots;     // score ring depth (TcShape::kMinSlots..kTcScoreSlots)
    uint64_t *cand;          // [NQ][G][k] keys
    uint64_t *heads;         // [NQ][G][kTcMergeE]: the first keys of each list
    uint32_t *ticket;        // CTA completion counter (self-resetting)
    uint32_t *next_tile;     // pool counter (self-resetting)
    uint32_t *epoch;         // launch counter word (advanced by the last CTA to finish)
    uint32_t *flags;         // [G] publication words: flags[c] = epoch + 1 once CTA c's lists are written
    uint32_t *err;           // device flag word
    int32_t *out_idx;        // [nq, k]
    float *out_logits;       // [nq, k]
    float *sparse;           // [nq, V] fp32 or nullptr: slices filled with -inf here
    const float *row_scale;  // Q8: fp32 scale per row [V]
    const float *qscale;     // Q8: [NQ][kQ8Pieces] power-of-two piece scales (from the prep kernel)
    int32_t h_resident;      // 1: each CTA builds the whole query operand in shared memory itself
    const float *h;          // h_resident: the queries [nq, d] fp32
    int32_t d;               // h_resident: their length
};

template <int NQ, bool Q8 = false>
struct TcShape {
    static constexpr int kCols = Q8 ? kQ8Pieces : 2;  // accumulator columns per query
    static constexpr int N = kCols * NQ;
    static constexpr int kKB = Q8 ? 2 * kTcKBlock : kTcKBlock;  // elements per 128-byte K-block
    static constexpr int kQPW = NQ >= 64 ? 4 : (NQ >= 32 ? 2 : 1);  // queries per selector warp
    static constexpr int kSelWarps = NQ / kQPW;
    static constexpr int kWarps = 6 + kSelWarps;
    static constexpr int kThreads = 32 * kWarps;
    // 128-row halves per tile (two M = 128 MMAs into two accumulators per
    // K-block: a query box rides with twice the weight bytes).  Measured: at
    // 256 rows the 64-query tile finishes later, its coarser tiles leaving the
    // CTAs up to a tile apart at the end (~30 us at d = 3072), so every tile
    // is 128 rows.
    static constexpr int kMH = 1;
    static constexpr int kTileRows = kTcTile * kMH;
    static constexpr int kHalfA = kTcTile * 128;   // 16 KB: one 128-row box of a K-block of W
    static constexpr int kStageA = kMH * kHalfA;   // W bytes per K-block (128 B per row)
    static constexpr int kStageB = N * 128;        // N x 128 B per K-block of H
    static constexpr int kStageBytes = kStageA + kStageB;    // per K-block; a multiple of 1024
    static constexpr int kAccCols = kMH * N;  // accumulator columns of one tile
    static constexpr int kTmemCols = (2 * kAccCols <= 32) ? 32 : (2 * kAccCols <= 64 ? 64 :
                                     (2 * kAccCols <= 128 ? 128 : (2 * kAccCols <= 256 ? 256 : 512)));
    // score ring depth (e4m3 tiles: 2, leaving shared memory to the weight ring)
    static constexpr int kMinSlots = NQ >= 64 ? 1 : 2;     // score ring depth, at least
    static constexpr int kSlotBytes = NQ * kTcTile * 4;    // one tile's logits, [query][row]
    // A selector keeps each query's best keys either in a register list of
    // 32 * kMM positions (2 at 64 queries, where k <= 64; else 4), one
    // insertion per key above the list's k-th, or - for the 4-query e4m3
    // tile, whose weight stream is short beside a burst of insertions - in a
    // shared buffer of kCap candidates above a bound, compacted to the best k
    // by bisection when it fills and sorted once at the end.
    static constexpr bool kBufSel = Q8 && NQ == 4;
    static constexpr int kMM = NQ >= 64 ? 2 : 4;
    static constexpr int kCap = 256;
    static constexpr int kMaxK0 = kBufSel ? kTcMaxK : (32 * kMM < kTcMaxK ? 32 * kMM : kTcMaxK);
    static constexpr int kMaxK = kMaxK0 < kTcListKeys / NQ ? kMaxK0 : kTcListKeys / NQ;  // largest k
    // shared memory next to the scores: the Q8 piece scales [NQ][4] fp32, then
    // (buffer selectors) the counts [NQ], bounds [NQ] and buffers [NQ][kCap]
    static constexpr int kQsBytes = Q8 ? NQ * kQ8Pieces * 4 : 0;
    static constexpr int kCntOff = kQsBytes, kTauOff = (kCntOff + NQ * 4 + 7) & ~7;
    static constexpr int kBufOff = (kTauOff + NQ * 8 + 15) & ~15;
    static constexpr int kBufBytes = 16 + (kBufSel ? kBufOff + NQ * kCap * 8 : kQsBytes);
};

struct TcMisc {
    uint32_t tmem_base;
    int abort;
    int stage_tile[kTcMaxStages];  // tile of a stage that starts a tile (-1: end)
    int buf_tile[2];               // tile held by each TMEM accumulator
    int slot_tile[kTcScoreSlots];  // 128-row block (row / 128) of each score slot (-1: end)
    int merger;                    // m >= 0: this CTA merges queries m, m + X, ...
    uint32_t epoch;                // the launch counter, read after the previous kernel finished
};

// The ring (1024-byte aligned at run time) starts with the resident query
// boxes when there are any (hres_bytes, a multiple of 1024), then the stages.
struct TcSmemLayout {
    uint32_t bars, misc, scores, bufs, ring, total;
    __host__ __device__ TcSmemLayout(int score_bytes, int buf_bytes, int stages, int stage_bytes,
                                     int hres_bytes = 0) {
        bars = 0;
        misc = 512;
        scores = 1024;
        bufs = scores + score_bytes;
        ring = (bufs + buf_bytes + 1023u) & ~1023u;
        total = ring + hres_bytes + stages * stage_bytes + 1024;  // +1024: room to align the ring
    }
};

// The least power of two >= v for v >= 0, at least 2^-100 (so that the
// piece scales s_0 2^-4p and their reciprocals stay normal fp32 numbers):
// exact bit arithmetic on the fp32 encoding.
__device__ __forceinline__ float pow2_at_least(float v) {
    const uint32_t b = __float_as_uint(v);
    if (b <= 0x0D800000u) return 0x1p-100f;  // zero, or at most 2^-100
    if ((b & 0x007FFFFFu) == 0) return v;   // already a power of two
    return __uint_as_float((b & 0x7F800000u) + 0x00800000u);
}

// x rounded to the nearest e4m3 value (ties to even, saturated at +-448),
// and an e4m3 code's exact value.
__device__ __forceinline__ uint8_t e4m3_code(float x) {
    return static_cast<uint8_t>(__nv_cvt_float_to_fp8(x, __NV_SATFINITE, __NV_E4M3));
}
__device__ __forceinline__ float e4m3_value(uint8_t c) {
    return __half2float(__half(__nv_cvt_fp8_to_halfraw(static_cast<__nv_fp8_storage_t>(c), __NV_E4M3)));
}

// Keeps the k largest of the cnt (k < cnt <= 32 * PER) nonzero keys in buf, unsorted at
// buf[0..k), and returns k; *tau becomes a bound T <= the k-th key such that
// exactly k keys are >= T.  T is found by bisection: first on the high words
// (the logit order), then, only if several keys tie on the k-th high word,
// on the low words (the row order) among the tied keys.  Out of line and
// loop-based: a few hundred instructions, and little code next to the
// latency-critical producer and MMA loops.
template <int PER>
static __device__ __noinline__ int keep_best(uint64_t *buf, int cnt, int k, uint64_t *tau, int lane) {
    uint64_t v[PER];
#pragma unroll
    for (int j = 0; j < PER; ++j) {
        const int e = j * 32 + lane;
        v[j] = e < cnt ? buf[e] : 0ull;  // 0 is below every key
    }
    // two bits per step: the counts at the three candidate digits are
    // independent reductions, so the chain of dependent ones halves
    uint32_t th = 0;
#pragma unroll 1
    for (int bit = 30; bit >= 0; bit -= 2) {
        const uint32_t c1 = th | (1u << bit), c2 = th | (2u << bit), c3 = th | (3u << bit);
        int n1 = 0, n2 = 0, n3 = 0;
#pragma unroll
        for (int j = 0; j < PER; ++j) {
            const uint32_t hi = static_cast<uint32_t>(v[j] >> 32);
            n1 += hi >= c1 ? 1 : 0;
            n2 += hi >= c2 ? 1 : 0;
            n3 += hi >= c3 ? 1 : 0;
        }
        n1 = static_cast<int>(__reduce_add_sync(0xFFFFFFFFu, n1));
        n2 = static_cast<int>(__reduce_add_sync(0xFFFFFFFFu, n2));
        n3 = static_cast<int>(__reduce_add_sync(0xFFFFFFFFu, n3));
        th = n3 >= k ? c3 : (n2 >= k ? c2 : (n1 >= k ? c1 : th));
    }
    int n_gt = 0, n_ge = 0;
#pragma unroll
    for (int j = 0; j < PER; ++j) {
        const uint32_t hi = static_cast<uint32_t>(v[j] >> 32);
        n_gt += hi > th ? 1 : 0;
        n_ge += hi >= th ? 1 : 0;
    }
    n_gt = static_cast<int>(__reduce_add_sync(0xFFFFFFFFu, n_gt));
    n_ge = static_cast<int>(__reduce_add_sync(0xFFFFFFFFu, n_ge));
    uint32_t tl = 0;
    if (n_ge > k) {
        // ties on the k-th logit: the (k - n_gt) largest low words among them
        const int need = k - n_gt;
#pragma unroll 1
        for (int bit = 31; bit >= 0; --bit) {
            const uint32_t c = tl | (1u << bit);
            int n = 0;
#pragma unroll
            for (int j = 0; j < PER; ++j)
                n += (static_cast<uint32_t>(v[j] >> 32) == th && static_cast<uint32_t>(v[j]) >= c) ? 1 : 0;
            if (static_cast<int>(__reduce_add_sync(0xFFFFFFFFu, n)) >= need) tl = c;
        }
    }
    const uint64_t T = (static_cast<uint64_t>(th) << 32) | tl;
    __syncwarp();
    const unsigned lt_mask = (1u << lane) - 1u;
    int base = 0;
#pragma unroll
    for (int j = 0; j < PER; ++j) {
        const bool in = v[j] >= T;
        const unsigned m = __ballot_sync(0xFFFFFFFFu, in);
        if (in) buf[base + __popc(m & lt_mask)] = v[j];
        base += __popc(m);
    }
    if (lane == 0) *tau = T;
    __syncwarp();
    return k;
}

// The final list of one query: the best min(k, cnt) keys of buf (cnt <=
// 32 * CAP_PER), sorted descending, written to dst[0..k) (zeros after them),
// and its first kTcMergeE keys also to head[0..kTcMergeE).  The sort network
// spans 32 * PER keys, the least that holds k (k <= 32 * PER): its dependent
// shuffles are the tail of the launch.
template <int CAP_PER, int PER>
static __device__ __noinline__ void write_sorted_list(uint64_t *buf, int cnt, int k, uint64_t *tau,
                                                      uint64_t *dst, uint64_t *head, int lane) {
    // (up to 32 * PER keys are sorted as they are; the first k are kept)
    if (cnt > 32 * PER) cnt = keep_best<CAP_PER>(buf, cnt, k, tau, lane);
    uint64_t v[PER];
#pragma unroll
    for (int j = 0; j < PER; ++j) {
        const int e = lane * PER + j;
        v[j] = e < cnt ? buf[e] : 0ull;
    }
    warp_sort_desc<PER>(v, lane);
#pragma unroll
    for (int j = 0; j < PER; ++j) {
        const int e = lane * PER + j;
        if (e < k) dst[e] = v[j];
        if (e < kTcMergeE) head[e] = v[j];
    }
}

template <int NQ, bool Q8>
__global__ void __launch_bounds__(TcShape<NQ, Q8>::kThreads, 1)
    tc_topk_kernel(const __grid_constant__ CUtensorMap mapW, const __grid_constant__ CUtensorMap mapH,
                   const TcParams p) {
    using Sh = TcShape<NQ, Q8>;
    constexpr int N = Sh::N;
    constexpr int KB = Sh::kKB;
    extern __shared__ __align__(1024) unsigned char tc_smem[];
    unsigned char *smem = tc_smem;
    const int S = p.stages;
    const int KPS = p.kb_per_stage;
    const bool hres = p.h_resident != 0;
    const int n_kb = (p.d_pad + KB - 1) / KB;
    // a stage: [KPS boxes of W][KPS boxes of H], or W only when H is resident
    const int kb_bytes = hres ? Sh::kStageA : Sh::kStageBytes;
    const int stage_bytes = KPS * kb_bytes;
    const int hres_bytes = hres ? n_kb * Sh::kStageB : 0;
    const int SL = p.score_slots;
    const TcSmemLayout L(SL * Sh::kSlotBytes, Sh::kBufBytes, S, stage_bytes, hres_bytes);
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + L.bars);
    uint64_t *empty = full + kTcMaxStages;
    uint64_t *tfull = empty + kTcMaxStages;
    uint64_t *tempty = tfull + 2;
    uint64_t *sfull = tempty + 2;
    uint64_t *sempty = sfull + kTcScoreSlots;
    uint64_t *final_bar = sempty + kTcScoreSlots;
    TcMisc *mc = reinterpret_cast<TcMisc *>(smem + L.misc);
    float *scores = reinterpret_cast<float *>(smem + L.scores);
    uint64_t *bufs = reinterpret_cast<uint64_t *>(smem + L.bufs);
    // the 128-byte swizzle needs 1024-byte aligned tiles in the shared window
    unsigned char *ring = smem + L.ring;
    ring += (1024u - (smem_addr(ring) & 1023u)) & 1023u;
    unsigned char *hq_res = ring;  // [n_kb][N rows x 128 B] when H is resident
    ring += hres_bytes;
    volatile int *abort_flag = &mc->abort;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int G = gridDim.x, cta = blockIdx.x;
    const int n_st = (n_kb + KPS - 1) / KPS;  // stages per tile
    constexpr int MH = Sh::kMH;
    constexpr int TR = Sh::kTileRows;
    const int n_tiles = static_cast<int>((p.V + TR - 1) / TR);

    if (tid == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&tfull[b], 2);
            mbar_init(&tempty[b], 4);
        }
        for (int s = 0; s < SL; ++s) {
            mbar_init(&sfull[s], 4);
            mbar_init(&sempty[s], Sh::kSelWarps);
        }
        mbar_init(final_bar, 1);
        mc->abort = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(&mc->tmem_base, Sh::kTmemCols);
        tmem_relinquish();
        tc_fence_before_sync();
    }
    __syncthreads();
    tc_fence_after_sync();
    const uint32_t tmem = mc->tmem_base;
    if (tid == 0) griddep_launch_dependents();  // a kernel launched after this one may be scheduled
    // Q8: the piece scales of the queries, next to the selectors' counts
    float *qs = reinterpret_cast<float *>(bufs);

    if (Q8 && hres && warp > 0) {
        // ---------------- the query operand, built in shared memory ----------------
        // Row r of a K-block is 128 bytes; 8-row groups are 1024 bytes apart;
        // the 16-byte chunk c of row r sits at chunk c ^ (r % 8) (the 128-byte
        // swizzle TMA would apply).  Columns past d are zero.
        griddep_wait();  // h comes from the kernel before this one
        const int T = Sh::kThreads - 32, t = tid - 32;
        const int width = n_kb * KB;  // columns of the operand, K-block padded
        auto at = [&](int r, int byte_in_row, int kb) -> unsigned char * {
            const int c = byte_in_row >> 4;
            return hq_res + kb * Sh::kStageB + (r >> 3) * 1024 + (r & 7) * 128 +
                   (((c ^ (r & 7)) << 4) | (byte_in_row & 15));
        };
        // rows of absent queries: zero, 16 bytes at a time (a row is 128 B in
        // every K-block; the swizzle only permutes chunks within a row)
        const int r_real = Sh::kCols * p.nq;
        for (int e = t; e < n_kb * (N - r_real) * 8; e += T) {
            const int kb = e / ((N - r_real) * 8), rem = e - kb * (N - r_real) * 8;
            const int r = r_real + (rem >> 3);
            *reinterpret_cast<uint4 *>(hq_res + kb * Sh::kStageB + (r >> 3) * 1024 + (r & 7) * 128 +
                                       ((rem & 7) << 4)) = make_uint4(0u, 0u, 0u, 0u);
        }
        constexpr int U = 8;  // independent loads of h in flight per thread
        {
            // s_0 = the least power of two >= max_j |h_qj| / 448, s_p = s_0 2^-4p:
            // every residual then stays within the pieces' range (448, 256, 128,
            // 64) and each piece takes 4 more significand bits
            const int q = warp - 1;
            if (q < p.nq) {
                float m = 0.0f;
                for (int j = lane; j < p.d; j += 32) m = fmaxf(m, fabsf(p.h[static_cast<int64_t>(q) * p.d + j]));
#pragma unroll
                for (int o = 16; o >= 1; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
                const float s0 = pow2_at_least(m / 448.0f);
                if (lane < kQ8Pieces) qs[kQ8Pieces * q + lane] = s0 * __uint_as_float((127u - 4u * lane) << 23);
            } else if (q < NQ && lane < kQ8Pieces) {
                qs[kQ8Pieces * q + lane] = 0.0f;
            }
            named_barrier_sync(3, T);
            for (int q = 0; q < p.nq; ++q) {
                const float *hq = p.h + static_cast<int64_t>(q) * p.d;
                // 1 / s_p is exact: s_p is a power of two within fp32's normal range
                const float inv0 = 1.0f / qs[kQ8Pieces * q], s0 = qs[kQ8Pieces * q];
                for (int j0 = t; j0 < width; j0 += U * T) {
                    float x[U];
#pragma unroll
                    for (int u = 0; u < U; ++u) {
                        const int j = j0 + u * T;
                        x[u] = j < p.d ? hq[j] : 0.0f;
                    }
#pragma unroll
                    for (int u = 0; u < U; ++u) {
                        const int j = j0 + u * T;
                        if (j < width) {
                            float r = x[u], sp = s0, inv = inv0;
#pragma unroll
                            for (int pc = 0; pc < kQ8Pieces; ++pc) {
                                const uint8_t c = e4m3_code(r * inv);
                                *at(kQ8Pieces * q + pc, j & (KB - 1), j / KB) = c;
                                r -= sp * e4m3_value(c);
                                sp *= 0x1p-4f;
                                inv *= 16.0f;
                            }
                        }
                    }
                }
            }
        }
        fence_proxy_async_smem();  // the MMAs read these bytes through the async proxy
        named_barrier_sync(3, T);
    }

    if (warp == 0) {
        // ---------------- TMA producer ----------------
        if (lane == 0) {
            tma_prefetch_map(&mapW);
            tma_prefetch_map(&mapH);
            const uint64_t pol = l2_evict_first_policy();
            const int Ns = p.static_tiles;
            const int pool0 = G * Ns;
            // The pool counter is re-armed by the previous launch's last
            // merging CTA, and this launch may start before that one ends
            // (programmatic dependent launch): the first draw waits for it.
            // With static tiles to issue first, the wait has long been over.
            if (Ns == 0) griddep_wait();
            uint32_t draw = (Ns == 0) ? atomic_add_relaxed_gpu(p.next_tile, 1u) : 0u;
            int it = 0, issued = 0;
            bool ok = true;
            for (int ti = 0; ok; ++ti) {
                int tile;
                if (ti < Ns) {
                    tile = ti * G + cta;
                } else {
                    tile = pool0 + static_cast<int>(draw);
                    if (tile >= n_tiles) tile = -1;
                }
                if (tile >= 0 && ti + 1 >= Ns) {
                    if (ti + 1 == Ns) griddep_wait();
                    draw = atomic_add_relaxed_gpu(p.next_tile, 1u);
                }
                const int nst = tile < 0 ? 1 : n_st;
                for (int st_i = 0; st_i < nst; ++st_i, ++it) {
                    const int s = it % S, u = it / S;
                    if (it >= S && !mbar_wait(&empty[s], (u - 1) & 1, abort_flag)) {
                        ok = false;
                        break;
                    }
                    if (st_i == 0) mc->stage_tile[s] = tile;
                    if (tile < 0) {
                        mbar_arrive(&full[s]);  // closes the stream: no bytes
                        break;
                    }
                    const int kb0 = st_i * KPS, nin = min(KPS, n_kb - kb0);
                    mbar_arrive_expect_tx(&full[s], nin * kb_bytes);
                    unsigned char *st = ring + s * stage_bytes;
                    for (int i = 0; i < nin; ++i)
#pragma unroll
                        for (int h = 0; h < MH; ++h)
                            tma_load_2d(st + i * Sh::kStageA + h * Sh::kHalfA, &mapW, (kb0 + i) * KB,
                                        tile * TR + h * kTcTile, &full[s], pol);
                    if (!hres) {
                        if (it == 0) griddep_wait();  // the query matrix comes from the prep kernel
                        for (int i = 0; i < nin; ++i)
                            tma_load_2d(st + KPS * Sh::kStageA + i * Sh::kStageB, &mapH,
                                        (kb0 + i) * KB, 0, &full[s], pol);
                    }
                    issued = it + 1;
                }
                if (tile < 0) break;
            }
            if (!ok) {
                atomicOr(p.err, kErrWaitTimeout);
                mc->abort = 1;
                const int never = 0;
                for (int t2 = max(0, issued - S); t2 < issued; ++t2)
                    mbar_wait(&full[t2 % S], (t2 / S) & 1, const_cast<volatile int *>(&never));
            }
        }
        // the other lanes wait for the producer lane here, so the whole warp
        // reaches the CTA barrier below together (bar.sync counts warps)
        __syncwarp();
    } else if (warp == 1) {
        // ---------------- MMA issuer ----------------
        if (lane == 0) {
            constexpr uint32_t idesc = Q8 ? umma_idesc_e4m3_f32(kTcTile, N) : umma_idesc_bf16_f32(kTcTile, N);
            int it = 0;
            bool ok = true;
            for (int ti = 0; ok; ++ti) {
                const int b = ti & 1, ub = ti >> 1;
                const int s0 = it % S, u0 = it / S;
                if (!mbar_wait(&full[s0], u0 & 1, abort_flag)) {
                    ok = false;
                    break;
                }
                const int tile = mc->stage_tile[s0];
                if (ti >= 2 && !mbar_wait(&tempty[b], (ub - 1) & 1, abort_flag)) {
                    ok = false;
                    break;
                }
                tc_fence_after_sync();
                if (tile < 0) {
                    mc->buf_tile[b] = -1;
                    mbar_arrive(&tfull[b]);
                    mbar_arrive(&tfull[b]);
                    break;
                }
                mc->buf_tile[b] = tile;
                const uint32_t d = tmem + static_cast<uint32_t>(b * Sh::kAccCols);
                for (int st_i = 0; st_i < n_st; ++st_i, ++it) {
                    const int s = it % S, u = it / S;
                    if (st_i > 0 && !mbar_wait(&full[s], u & 1, abort_flag)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after_sync();
                    unsigned char *st = ring + s * stage_bytes;
                    const int kb0 = st_i * KPS, nin = min(KPS, n_kb - kb0);
                    for (int i = 0; i < nin; ++i) {
                        const uint64_t ad = umma_desc_k_sw128(st + i * Sh::kStageA);
                        const uint64_t bd = umma_desc_k_sw128(
                            hres ? hq_res + (kb0 + i) * Sh::kStageB : st + KPS * Sh::kStageA + i * Sh::kStageB);
#pragma unroll
                        for (int k4 = 0; k4 < 4; ++k4) {  // +32 bytes per MMA (K = 16 bf16 or 32 e4m3)
#pragma unroll
                            for (int h = 0; h < MH; ++h) {  // rows h*128.. of the tile: accumulator h
                                const uint64_t adh = ad + static_cast<uint64_t>(h * (Sh::kHalfA >> 4));
                                const uint32_t acc = ((kb0 + i) | k4) != 0 ? 1u : 0u;
                                if constexpr (Q8)
                                    umma_e4m3(d + h * N, adh + 2 * k4, bd + 2 * k4, idesc, acc);
                                else
                                    umma_bf16(d + h * N, adh + 2 * k4, bd + 2 * k4, idesc, acc);
                            }
                        }
                    }
                    umma_commit(&empty[s]);
                }
                if (!ok) break;
                umma_commit(&tfull[b]);
                mbar_arrive(&tfull[b]);  // publishes buf_tile[b]
            }
            if (!ok) {
                atomicOr(p.err, kErrWaitTimeout);
                mc->abort = 1;
            }
            // every MMA this thread issued has finished before TMEM is freed
            umma_commit(final_bar);
            const int never = 0;
            mbar_wait(final_bar, 0, const_cast<volatile int *>(&never));
        }
        __syncwarp();  // the whole warp reaches the CTA barrier together
    } else if (warp < 6) {
        // ---------------- epilogue: TMEM -> logits ----------------
        const int qw = warp & 3;  // TMEM lane quarter this warp may access
        const int row = 32 * qw + lane;
        if (Q8 && !hres) {
            griddep_wait();  // the prep kernel wrote them
            const int e = (warp - 2) * 32 + lane;
            if (e < NQ * kQ8Pieces) qs[e] = p.qscale[e];
            named_barrier_sync(2, 128);  // the four epilogue warps
        }
        for (int ti = 0;; ++ti) {
            const int b = ti & 1, ub = ti >> 1;
            if (!mbar_wait(&tfull[b], ub & 1, abort_flag)) {
                if (lane == 0) {
                    atomicOr(p.err, kErrWaitTimeout);
                    mc->abort = 1;
                }
                break;
            }
            tc_fence_after_sync();
            const int tile = mc->buf_tile[b];
            const int ss = ti % SL, su = ti / SL;
            // Q8: this row's scale, loaded under the accumulator reads
            float rsc = 1.0f;
            if constexpr (Q8) {
                const int64_t gr = static_cast<int64_t>(tile) * TR + row;  // MH == 1 on e4m3 rows
                if (tile >= 0 && gr < p.V) rsc = __ldg(p.row_scale + gr);
            }
            if constexpr (N > 64) {
                // wide tiles: per 128-row half, wait for a score slot first,
                // then drain that half's accumulator 32 columns (16 queries)
                // at a time; the TMEM buffer is handed back after the last half
                bool failed = false;
#pragma unroll 1
                for (int h = 0; h < MH; ++h) {
                    const int si = ti * MH + h, ssh = si % SL, suh = si / SL;
                    if (si >= SL && !mbar_wait(&sempty[ssh], (suh - 1) & 1, abort_flag)) {
                        if (lane == 0) {
                            atomicOr(p.err, kErrWaitTimeout);
                            mc->abort = 1;
                        }
                        failed = true;
                        break;
                    }
                    if (tile >= 0) {
                        const uint32_t tb = tmem + (static_cast<uint32_t>(32 * qw) << 16) + b * Sh::kAccCols + h * N;
                        float *sc = scores + ssh * NQ * kTcTile;
                        constexpr int QC = 32 / Sh::kCols;  // queries per 32 accumulator columns
#pragma unroll
                        for (int c = 0; c < N / 16; c += 2) {
                            uint32_t r[2][16];
                            tmem_ld_32x32b_x16(tb + 16 * c, r[0]);
                            tmem_ld_32x32b_x16(tb + 16 * (c + 1), r[1]);
                            tmem_wait_ld();
#pragma unroll
                            for (int qq = 0; qq < QC; ++qq) {
                                const int q = QC * (c / 2) + qq, c0 = Sh::kCols * qq;
                                float z;
                                if constexpr (Q8) {
                                    z = 0.0f;
#pragma unroll
                                    for (int pc = 0; pc < kQ8Pieces; ++pc)
                                        z = fmaf(qs[kQ8Pieces * q + pc],
                                                 __uint_as_float(r[(c0 + pc) / 16][(c0 + pc) % 16]), z);
                                    z *= rsc;
                                } else {
                                    z = __uint_as_float(r[c0 / 16][c0 % 16]) +
                                        __uint_as_float(r[c0 / 16][c0 % 16 + 1]);
                                }
                                sc[q * kTcTile + row] = z;
                            }
                        }
                    }
                    if (h == MH - 1 || tile < 0) {
                        tc_fence_before_sync();
                        __syncwarp();
                        if (lane == 0) mbar_arrive(&tempty[b]);
                    }
                    if (warp == 2 && lane == 0) mc->slot_tile[ssh] = tile >= 0 ? tile * MH + h : -1;
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&sfull[ssh]);
                    if (tile < 0) break;
                }
                if (failed || tile < 0) break;
                continue;
            }
            float lg[NQ];
            if (tile >= 0) {
                const uint32_t tb = tmem + (static_cast<uint32_t>(32 * qw) << 16) + b * N;
                uint32_t r[N / 16][16];
#pragma unroll
                for (int c = 0; c < N / 16; ++c) tmem_ld_32x32b_x16(tb + 16 * c, r[c]);
                tmem_wait_ld();
#pragma unroll
                for (int q = 0; q < NQ; ++q) {
                    const int c0 = Sh::kCols * q;
                    if constexpr (Q8) {
                        float z = 0.0f;
#pragma unroll
                        for (int pc = 0; pc < kQ8Pieces; ++pc)
                            z = fmaf(qs[kQ8Pieces * q + pc], __uint_as_float(r[(c0 + pc) / 16][(c0 + pc) % 16]), z);
                        lg[q] = z * rsc;
                    } else {
                        lg[q] = __uint_as_float(r[c0 / 16][c0 % 16]) + __uint_as_float(r[c0 / 16][c0 % 16 + 1]);
                    }
                }
            }
            tc_fence_before_sync();
            __syncwarp();
            if (lane == 0) mbar_arrive(&tempty[b]);
            if (ti >= SL && !mbar_wait(&sempty[ss], (su - 1) & 1, abort_flag)) {
                if (lane == 0) {
                    atomicOr(p.err, kErrWaitTimeout);
                    mc->abort = 1;
                }
                break;
            }
            if (tile >= 0) {
                float *sc = scores + ss * NQ * kTcTile;
#pragma unroll
                for (int q = 0; q < NQ; ++q) sc[q * kTcTile + row] = lg[q];
            }
            if (warp == 2 && lane == 0) mc->slot_tile[ss] = tile;  // MH == 1: the tile is the row block
            __syncwarp();
            if (lane == 0) mbar_arrive(&sfull[ss]);
            if (tile < 0) break;
        }
    } else {
        // ---------------- selectors ----------------
        const int sel = warp - 6;
        griddep_wait();  // writes below must follow the previous kernel on the stream
        // the launch counter, now that the kernel before this one has finished
        // (it may have advanced it)
        if (sel == 0 && lane == 0) mc->epoch = *reinterpret_cast<volatile uint32_t *>(p.epoch);
        if (p.sparse != nullptr) {
            // this CTA's fixed slice of every sparse row = -inf (values come later)
            const float ninf = __uint_as_float(0xFF800000u);
            const int64_t base = p.V / G, rem = p.V % G;
            const int64_t f0 = cta * base + (cta < rem ? cta : rem);
            const int64_t fn = base + (cta < rem ? 1 : 0);
            for (int q = 0; q < p.nq; ++q) {
                float *rw = p.sparse + static_cast<int64_t>(q) * p.V + f0;
                for (int64_t i = sel * 32 + lane; i < fn; i += Sh::kSelWarps * 32) rw[i] = ninf;
            }
        }
        constexpr int QPW = Sh::kQPW;
        if constexpr (Sh::kBufSel) {
            // per query of this warp: candidates above the bound tau in a shared
            // buffer, their count and tau next to it (only this warp touches them)
            constexpr int CAP = Sh::kCap, CAP_PER = CAP / 32;
            unsigned char *bb = reinterpret_cast<unsigned char *>(bufs);
            int *cnt_s = reinterpret_cast<int *>(bb + Sh::kCntOff) + QPW * sel;
            uint64_t *tau_s = reinterpret_cast<uint64_t *>(bb + Sh::kTauOff) + QPW * sel;
            uint64_t *buf0 = reinterpret_cast<uint64_t *>(bb + Sh::kBufOff);
            if (lane < QPW) {
                cnt_s[lane] = 0;
                tau_s[lane] = 0;
            }
            __syncwarp();
            const unsigned lt_mask = (1u << lane) - 1u;
            for (int ti = 0;; ++ti) {
                const int ss = ti % SL, su = ti / SL;
                if (!mbar_wait(&sfull[ss], su & 1, abort_flag)) {
                    if (lane == 0) {
                        atomicOr(p.err, kErrWaitTimeout);
                        mc->abort = 1;
                    }
                    break;
                }
                const int rblk = mc->slot_tile[ss];
                if (rblk < 0) break;
                const int64_t row0 = static_cast<int64_t>(rblk) * kTcTile;
                const int rows = static_cast<int>(min(static_cast<int64_t>(kTcTile), p.V - row0));
                const float *sc = scores + ss * NQ * kTcTile;
#pragma unroll 1
                for (int j = 0; j < QPW; ++j) {
                    const int q = QPW * sel + j;
                    if (q >= p.nq) break;
                    uint64_t *buf = buf0 + q * CAP;
                    int cnt = cnt_s[j];
                    uint64_t tau = tau_s[j];
                    for (int rb = 0; rb < rows; rb += 32) {
                        if (cnt > CAP - 32) {  // room for one more row block
                            cnt = keep_best<CAP_PER>(buf, cnt, p.k, &tau_s[j], lane);
                            tau = tau_s[j];
                        }
                        const int r = rb + lane;
                        const uint64_t key =
                            (r < rows) ? make_key(sc[q * kTcTile + r], static_cast<uint32_t>(row0 + r)) : 0;
                        const bool in = key > tau;
                        const unsigned m = __ballot_sync(0xFFFFFFFFu, in);
                        if (in) buf[cnt + __popc(m & lt_mask)] = key;
                        cnt += __popc(m);
                    }
                    __syncwarp();
                    if (lane == 0) cnt_s[j] = cnt;
                    __syncwarp();
                }
                if (lane == 0) mbar_arrive(&sempty[ss]);
            }
            // this CTA's sorted top-k per query and its first keys -> scratch
            // (written even after a wait gave up: the merge then stays in bounds)
#pragma unroll 1
            for (int j = 0; j < QPW; ++j) {
                const int q = QPW * sel + j;
                if (q >= p.nq) break;
                uint64_t *dst = p.cand + (static_cast<size_t>(q) * G + cta) * p.k;
                uint64_t *head = p.heads + (static_cast<size_t>(q) * G + cta) * kTcMergeE;
                uint64_t *buf = buf0 + q * CAP;
                if (p.k <= 32)
                    write_sorted_list<CAP_PER, 1>(buf, cnt_s[j], p.k, &tau_s[j], dst, head, lane);
                else if (p.k <= 64)
                    write_sorted_list<CAP_PER, 2>(buf, cnt_s[j], p.k, &tau_s[j], dst, head, lane);
                else
                    write_sorted_list<CAP_PER, kTcMaxK / 32>(buf, cnt_s[j], p.k, &tau_s[j], dst, head, lane);
            }
        } else {
            // per query of this warp: its best keys so far as a sorted list spread
            // over the warp's registers, and the k-th of them as the entry bound
            constexpr int MM = Sh::kMM;
            WarpList<MM> list[QPW];
            uint64_t tau[QPW];
#pragma unroll
            for (int j = 0; j < QPW; ++j) {
                list[j].clear();
                tau[j] = 0;
            }
            for (int ti = 0;; ++ti) {
                const int ss = ti % SL, su = ti / SL;
                if (!mbar_wait(&sfull[ss], su & 1, abort_flag)) {
                    if (lane == 0) {
                        atomicOr(p.err, kErrWaitTimeout);
                        mc->abort = 1;
                    }
                    break;
                }
                const int rblk = mc->slot_tile[ss];
                if (rblk < 0) break;
                const int64_t row0 = static_cast<int64_t>(rblk) * kTcTile;
                const int rows = static_cast<int>(min(static_cast<int64_t>(kTcTile), p.V - row0));
                const float *sc = scores + ss * NQ * kTcTile;
#pragma unroll
                for (int j = 0; j < QPW; ++j) {
                    const int q = QPW * sel + j;
                    if (q < p.nq) {
                        for (int rb = 0; rb < rows; rb += 32) {
                            const int r = rb + lane;
                            const uint64_t key =
                                (r < rows) ? make_key(sc[q * kTcTile + r], static_cast<uint32_t>(row0 + r)) : 0;
                            // every key above the block's entry bound goes in (one that
                            // an earlier key of the block pushed below the k-th lands
                            // past position k, harmlessly); the bound is refreshed once
                            // per block
                            unsigned m = __ballot_sync(0xFFFFFFFFu, key > tau[j]);
                            if (m) {
                                do {
                                    const int src = __ffs(m) - 1;
                                    m &= m - 1;
                                    list[j].insert(shfl_u64(key, src), lane);
                                } while (m);
                                tau[j] = list[j].at(p.k - 1);
                            }
                        }
                    }
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(&sempty[ss]);
            }
            // this CTA's sorted top-k per query and its first keys -> scratch
            // (written even after a wait gave up: the merge then stays in bounds)
#pragma unroll
            for (int j = 0; j < QPW; ++j) {
                const int q = QPW * sel + j;
                if (q < p.nq) {
                    uint64_t *dst = p.cand + (static_cast<size_t>(q) * G + cta) * p.k;
                    uint64_t *head = p.heads + (static_cast<size_t>(q) * G + cta) * kTcMergeE;
#pragma unroll
                    for (int s2 = 0; s2 < MM; ++s2) {
                        const int pos = lane * MM + s2;
                        if (pos < p.k) dst[pos] = list[j].v[s2];
                        if (pos < kTcMergeE) head[pos] = list[j].v[s2];
                    }
                }
            }
        }
    }

    __syncthreads();
    if (warp == 1) {
        tc_fence_after_sync();
        tmem_dealloc(tmem, Sh::kTmemCols);
    }

    // ---------------- publication, then the merge (first X CTAs) ----------------
    // bar.sync orders every thread's writes (lists, heads, sparse fill) before
    // thread 0's release store of epoch + 1 into this CTA's publication word.
    // A relaxed ticket then ranks the CTAs by finishing order: the first X
    // merge (queries m, m + X, ...), taking each CTA's lists as they are
    // published, while the others still stream; the last re-arms the tile
    // pool and the ticket and advances the epoch (every CTA has drawn its
    // last tile and taken its ticket by then).
    const int X = min(p.nq, min(G, kTcMaxMergers));
    const uint32_t target = mc->epoch + 1u;
    if (tid == 0) {
        st_release_gpu(p.flags + cta, target);
        const uint32_t ticket = atomic_add_relaxed_gpu(p.ticket, 1u);
        if (ticket == static_cast<uint32_t>(G - 1)) {
            *p.next_tile = 0;
            *p.ticket = 0;
            *reinterpret_cast<volatile uint32_t *>(p.epoch) = target;
        }
        mc->merger = ticket < static_cast<uint32_t>(X) ? static_cast<int>(ticket) : -1;
    }
    __syncthreads();
    const int m = mc->merger;
    if (m < 0) return;

    // ---------------- merge ----------------
    // Scores, buffers and ring are free now.  Per query: the first kFastE keys
    // of every list (the heads area) go to shared memory as the lists are
    // published, the fast merge settles the query from them, or the full
    // merge reads the lists.  (Every CTA wrote full lists and heads, valid
    // keys or zeros, even if it gave up on a wait: the merge stays in bounds,
    // the flag reports the call.)
    {
        static_assert(kTcMergeE == kFastE, "the heads area feeds the fast merge");
        unsigned char *ws = smem + L.scores;
        const uint32_t ms_off = (SmemLayout::merge_fixed_bytes() + 15u) & ~15u;
        MiscSmem *ms = reinterpret_cast<MiscSmem *>(ws + ms_off);
        uint64_t *fe = reinterpret_cast<uint64_t *>(ws + ms_off + ((sizeof(MiscSmem) + 15u) & ~15u));
        for (int q = m; q < p.nq; q += X) {
            int32_t *oi = p.out_idx + static_cast<size_t>(q) * p.k;
            float *ol = p.out_logits + static_cast<size_t>(q) * p.k;
            float *sp = p.sparse != nullptr ? p.sparse + static_cast<int64_t>(q) * p.V : nullptr;
            merge_published(p.flags, target, p.heads + static_cast<size_t>(q) * G * kFastE,
                            p.cand + static_cast<size_t>(q) * G * p.k, G, p.k, ws, fe, ms, p.err, oi, ol, sp);
            __syncthreads();
        }
    }
}

}  // namespace vie
