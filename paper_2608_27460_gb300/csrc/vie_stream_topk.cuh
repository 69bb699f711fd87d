// vie_stream_topk.cuh - the small-batch output head in one launch:
// streaming projection z = W_out h (paper, Section 3) fused with the exact
// top-k selection (exhaustive MIPS, Sections 2-3).
//
// One persistent CTA per SM owns a contiguous slice of the vocabulary rows.
//   warp 0     producer: 1-D bulk copies (TMA) of whole row groups into a
//              ring of shared-memory stages, L2 evict-first, mbarrier
//              transaction counts;
//   warps 2-9  projection: each warp takes rows of a stage, every lane a
//              strided set of 16-byte column chunks; bf16 -> fp32 widening,
//              fp32 FMA against h (staged in shared memory, one load per
//              chunk reused for R rows), then a warp-shuffle butterfly sum;
//   warp 1     selector: keeps the best keys seen so far as a sorted list
//              spread over the warp's registers; a row enters only if it
//              beats the current k-th key.
// The full logit vector never leaves the chip.  After the stream, each CTA
// writes its sorted top-k list to scratch and takes a ticket; the CTA that
// draws the last ticket merges the G lists into the final top-k:
//   1. tau* = k-th largest key among the first J = ceil(k/G) entries of all
//      lists (a lower bound of the true k-th key: k keys are >= it);
//   2. every list contributes its prefix of keys >= tau*;
//   3. exact top-k of those candidates (rank counting, or radix select when
//      there are many), written best first.
#pragma once

#include <cstdint>

#include "vie_device.cuh"

namespace vie {

constexpr int kDotWarps = 8;
constexpr int kThreads = 32 * (2 + kDotWarps);
constexpr int kMaxStages = 16;
constexpr int kMergePrefixCap = 2048;  // keys: first-J prefixes of all lists
constexpr int kMergeCandCap = 2048;    // keys: gathered candidates
constexpr int kRankCountMax = 640;     // rank counting below this many keys
constexpr int kMaxLists = 1024;        // G <= 1024 CTAs

struct StreamTopkParams {
    const uint16_t *W;   // padded [V, d_pad] bf16 bits
    const float *h;      // [nq, d] fp32
    int32_t nq;          // queries in this launch (<= NB)
    int64_t V;
    int32_t d, d_pad;
    int32_t k;
    int32_t rows_per_stage;  // RS
    int32_t stages;          // S
    uint64_t *cand;          // [NB][G][k] keys
    uint32_t *ticket;        // CTA completion counter (self-resetting)
    uint32_t *err;           // device flag word
    int32_t *out_idx;        // [nq, k]
    float *out_logits;       // [nq, k]
};

// Shared-memory carve-up; all offsets are multiples of 128 bytes.
struct SmemLayout {
    uint32_t bars, misc, h, scores, ring, merge, total;
    __host__ __device__ static uint32_t align128(uint32_t x) { return (x + 127u) & ~127u; }
    __host__ __device__ SmemLayout(int nb, int d_pad, int rs, int stages, int row_bytes) {
        bars = 0;
        misc = align128(bars + 3u * kMaxStages * 8u);
        h = align128(misc + 128u);
        scores = align128(h + 4u * nb * d_pad);
        ring = align128(scores + 4u * stages * rs * nb);
        merge = ring;  // the merge reuses the ring once the stream is drained
        uint32_t ring_end = ring + static_cast<uint32_t>(stages) * rs * row_bytes;
        uint32_t merge_end = merge + 8u * (kMergePrefixCap + kMergeCandCap + 1024) +
                             4u * (2 * kMaxLists + 256 + 32);
        total = ring_end > merge_end ? ring_end : merge_end;
    }
};

struct MiscSmem {
    int abort;
    int is_last;
    int remaining;
    int bin_count;
    int n_cand;
    int n_win;
    unsigned long long tau;
    unsigned long long prefix;
};

// --------------------------------------------------------------------------
// Warp-distributed sorted list of the best keys (descending).  Lane L holds
// positions L*MM .. L*MM+MM-1.  Unused positions hold 0.
template <int MM>
struct WarpList {
    uint64_t v[MM];

    __device__ __forceinline__ void clear() {
#pragma unroll
        for (int s = 0; s < MM; ++s) v[s] = 0;
    }

    // Inserts key x (the same on every lane), dropping the last position.
    __device__ __forceinline__ void insert(uint64_t x, int lane) {
        int c = 0;
#pragma unroll
        for (int s = 0; s < MM; ++s) c += (v[s] > x) ? 1 : 0;
        const int pos = __reduce_add_sync(0xFFFFFFFFu, c);
        const uint64_t up = shfl_up_u64(v[MM - 1], 1);
#pragma unroll
        for (int s = MM - 1; s >= 0; --s) {
            const int e = lane * MM + s;
            const uint64_t prev = (s > 0) ? v[s > 0 ? s - 1 : 0] : up;
            v[s] = (e > pos) ? prev : ((e == pos) ? x : v[s]);
        }
    }

    // Key at position p (same p on every lane).
    __device__ __forceinline__ uint64_t at(int p) const {
        const int slot = p % MM;
        uint64_t x = 0;
#pragma unroll
        for (int s = 0; s < MM; ++s)
            if (s == slot) x = v[s];
        return shfl_u64(x, p / MM);
    }
};

// --------------------------------------------------------------------------
// Block-wide helpers for the merge (all kThreads threads call them).

struct SmemKeys {
    const uint64_t *p;
    __device__ __forceinline__ uint64_t operator[](int i) const { return p[i]; }
};
struct GlobalKeys {
    const uint64_t *p;
    __device__ __forceinline__ uint64_t operator[](int i) const {
        return __ldcg(reinterpret_cast<const unsigned long long *>(p) + i);
    }
};

// Threshold T such that exactly k of the keys with key >= lo (lo >= 1) are
// >= T (keys are unique apart from 0, which is never counted).  MSB-first
// radix select over 8-bit digits, stopping early once the selected bin
// holds exactly the keys still needed.
template <class Keys>
__device__ uint64_t block_radix_threshold(Keys keys, int n, int k, uint64_t lo, uint32_t *hist,
                                          MiscSmem *ms) {
    const int tid = threadIdx.x;
    uint64_t prefix = 0, mask = 0;
    int remaining = k;
    for (int shift = 56; shift >= 0; shift -= 8) {
        for (int i = tid; i < 256; i += kThreads) hist[i] = 0;
        __syncthreads();
        for (int i = tid; i < n; i += kThreads) {
            const uint64_t x = keys[i];
            if (x >= lo && x != 0 && (x & mask) == prefix)
                atomicAdd(&hist[(x >> shift) & 255u], 1u);
        }
        __syncthreads();
        if (tid < 32) {
            const int lane = tid;
            int cnt[8];
            int local = 0;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                cnt[j] = static_cast<int>(hist[255 - 8 * lane - j]);
                local += cnt[j];
            }
            int incl = local;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int t = __shfl_up_sync(0xFFFFFFFFu, incl, o);
                if (lane >= o) incl += t;
            }
            const int excl = incl - local;
            if (excl < remaining && remaining <= incl) {
                int run = excl;
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    if (run < remaining && remaining <= run + cnt[j]) {
                        const uint64_t dgt = static_cast<uint64_t>(255 - 8 * lane - j);
                        ms->prefix = prefix | (dgt << shift);
                        ms->remaining = remaining - run;
                        ms->bin_count = cnt[j];
                    }
                    run += cnt[j];
                }
            }
        }
        __syncthreads();
        prefix = ms->prefix;
        mask |= static_cast<uint64_t>(255) << shift;
        remaining = ms->remaining;
        const bool done = (ms->bin_count == remaining);
        __syncthreads();
        if (done) break;
    }
    return prefix;
}

// Exact top-k of n unique nonzero keys in shared memory, written best first
// to out_idx / out_logits.  Uses rank counting for small n, otherwise a
// radix-select threshold followed by rank counting of the k winners.
__device__ inline void block_topk_to_output(const uint64_t *keys, int n, int k, uint64_t *win,
                                     uint32_t *hist, MiscSmem *ms, int32_t *out_idx,
                                     float *out_logits) {
    const int tid = threadIdx.x;
    const uint64_t *src = keys;
    int m = n;
    if (n > kRankCountMax && n > k) {
        const uint64_t T = block_radix_threshold(SmemKeys{keys}, n, k, 1, hist, ms);
        if (tid == 0) ms->n_win = 0;
        __syncthreads();
        for (int i = tid; i < n; i += kThreads) {
            const uint64_t x = keys[i];
            if (x >= T) win[atomicAdd(&ms->n_win, 1)] = x;
        }
        __syncthreads();
        src = win;
        m = k;
    }
    for (int i = tid; i < m; i += kThreads) {
        const uint64_t x = src[i];
        int rank = 0;
        for (int j = 0; j < m; ++j) rank += (src[j] > x) ? 1 : 0;
        if (rank < k) {
            out_idx[rank] = key_index(x);
            out_logits[rank] = key_value(x);
        }
    }
    __syncthreads();
}

// --------------------------------------------------------------------------
template <int NB, int MM, int R>
__global__ void __launch_bounds__(kThreads, 1) stream_topk_kernel(const StreamTopkParams p) {
    extern __shared__ __align__(128) unsigned char smem[];
    const int RS = p.rows_per_stage;
    const int S = p.stages;
    const int row_bytes = p.d_pad * 2;
    const SmemLayout L(NB, p.d_pad, RS, S, row_bytes);
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + L.bars);
    uint64_t *empty = full + kMaxStages;
    uint64_t *sfull = empty + kMaxStages;
    MiscSmem *ms = reinterpret_cast<MiscSmem *>(smem + L.misc);
    float *h_s = reinterpret_cast<float *>(smem + L.h);
    float *scores = reinterpret_cast<float *>(smem + L.scores);
    unsigned char *ring = smem + L.ring;
    volatile int *abort_flag = &ms->abort;

    const int tid = threadIdx.x;
    const int warp = tid >> 5;
    const int lane = tid & 31;
    const int G = gridDim.x;
    const int cta = blockIdx.x;
    const int64_t base = p.V / G, rem = p.V % G;
    const int64_t r0 = cta * base + (cta < rem ? cta : rem);
    const int n_rows = static_cast<int>(base + (cta < rem ? 1 : 0));
    const int n_st = (n_rows + RS - 1) / RS;
    const int C = p.d_pad >> 3;  // 16-byte chunks per row
    const int stage_bytes = RS * row_bytes;

    if (tid == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], kDotWarps + 1);
            mbar_init(&sfull[s], kDotWarps);
        }
        ms->abort = 0;
        ms->is_last = 0;
        fence_mbar_init();
    }
    // h -> shared memory as [nb][half][chunk][4] so a lane's two float4 loads
    // of one chunk fall in distinct bank groups; zero pad, zero unused queries.
    for (int i = tid; i < NB * p.d_pad; i += kThreads) {
        const int nb = i / p.d_pad, j = i - nb * p.d_pad;
        const float v = (nb < p.nq && j < p.d) ? p.h[static_cast<int64_t>(nb) * p.d + j] : 0.0f;
        const int c = j >> 3, e = j & 7;
        h_s[(nb * 2 + (e >> 2)) * (C * 4) + c * 4 + (e & 3)] = v;
    }
    __syncthreads();

    if (warp == 0) {
        // ---------------- producer ----------------
        if (lane == 0) {
            const uint64_t pol = l2_evict_first_policy();
            const unsigned char *src = reinterpret_cast<const unsigned char *>(p.W) +
                                       static_cast<size_t>(r0) * row_bytes;
            int issued = 0;
            bool ok = true;
            for (int t = 0; t < n_st; ++t) {
                const int s = t % S, u = t / S;
                if (t >= S && !mbar_wait(&empty[s], (u - 1) & 1, abort_flag)) {
                    ok = false;
                    break;
                }
                const int rows = min(RS, n_rows - t * RS);
                const uint32_t bytes = static_cast<uint32_t>(rows * row_bytes);
                mbar_arrive_expect_tx(&full[s], bytes);
                bulk_g2s(ring + s * stage_bytes, src + static_cast<size_t>(t) * stage_bytes, bytes,
                         &full[s], pol);
                issued = t + 1;
            }
            if (!ok) {
                atomicOr(p.err, kErrWaitTimeout);
                ms->abort = 1;
                // drain: copies still in flight must land before the CTA exits
                const int never = 0;
                for (int t = max(0, issued - S); t < issued; ++t)
                    mbar_wait(&full[t % S], (t / S) & 1, const_cast<volatile int *>(&never));
            }
        }
    } else if (warp == 1) {
        // ---------------- selector ----------------
        WarpList<MM> list[NB];
        uint64_t tau[NB];
#pragma unroll
        for (int nb = 0; nb < NB; ++nb) {
            list[nb].clear();
            tau[nb] = 0;
        }
        for (int t = 0; t < n_st; ++t) {
            const int s = t % S, u = t / S;
            if (!mbar_wait(&sfull[s], u & 1, abort_flag)) {
                if (lane == 0) {
                    atomicOr(p.err, kErrWaitTimeout);
                    ms->abort = 1;
                }
                break;
            }
            const int rows = min(RS, n_rows - t * RS);
            const uint32_t row_base = static_cast<uint32_t>(r0 + static_cast<int64_t>(t) * RS);
            const float *sc = scores + s * RS * NB;
#pragma unroll
            for (int nb = 0; nb < NB; ++nb) {
                if (nb >= p.nq) break;
                for (int rb = 0; rb < rows; rb += 32) {
                    const int r = rb + lane;
                    const uint64_t key = (r < rows) ? make_key(sc[r * NB + nb], row_base + r) : 0;
                    unsigned m = __ballot_sync(0xFFFFFFFFu, key > tau[nb]);
                    while (m) {
                        const int src = __ffs(m) - 1;
                        m &= m - 1;
                        const uint64_t x = shfl_u64(key, src);
                        if (x > tau[nb]) {
                            list[nb].insert(x, lane);
                            tau[nb] = list[nb].at(p.k - 1);
                        }
                    }
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty[s]);
        }
        // this CTA's sorted top-k per query -> scratch
#pragma unroll
        for (int nb = 0; nb < NB; ++nb) {
            uint64_t *dst = p.cand + (static_cast<size_t>(nb) * G + cta) * p.k;
#pragma unroll
            for (int s = 0; s < MM; ++s) {
                const int pos = lane * MM + s;
                if (pos < p.k) dst[pos] = list[nb].v[s];
            }
        }
        __threadfence();
    } else {
        // ---------------- projection ----------------
        const int w = warp - 2;
        for (int t = 0; t < n_st; ++t) {
            const int s = t % S, u = t / S;
            if (!mbar_wait(&full[s], u & 1, abort_flag)) {
                if (lane == 0) {
                    atomicOr(p.err, kErrWaitTimeout);
                    ms->abort = 1;
                }
                break;
            }
            const int rows = min(RS, n_rows - t * RS);
            const unsigned char *stage = ring + s * stage_bytes;
            float *sc = scores + s * RS * NB;
            // rows of this stage owned by warp w: global row index = w mod 8
            const int first = (w - ((t * RS) & (kDotWarps - 1)) + kDotWarps) & (kDotWarps - 1);
            for (int rg = first; rg < rows; rg += kDotWarps * R) {
                int rr[R];
#pragma unroll
                for (int i = 0; i < R; ++i) rr[i] = min(rg + i * kDotWarps, rows - 1);
                float acc[R][NB];
#pragma unroll
                for (int i = 0; i < R; ++i)
#pragma unroll
                    for (int nb = 0; nb < NB; ++nb) acc[i][nb] = 0.0f;
                for (int c = lane; c < C; c += 32) {
                    uint4 wv[R];
#pragma unroll
                    for (int i = 0; i < R; ++i)
                        wv[i] = *reinterpret_cast<const uint4 *>(stage + rr[i] * row_bytes + c * 16);
#pragma unroll
                    for (int nb = 0; nb < NB; ++nb) {
                        const float4 ha =
                            *reinterpret_cast<const float4 *>(h_s + (nb * 2 + 0) * (C * 4) + c * 4);
                        const float4 hb =
                            *reinterpret_cast<const float4 *>(h_s + (nb * 2 + 1) * (C * 4) + c * 4);
#pragma unroll
                        for (int i = 0; i < R; ++i) {
                            float a = acc[i][nb];
                            a = fmaf(bf16_lo(wv[i].x), ha.x, a);
                            a = fmaf(bf16_hi(wv[i].x), ha.y, a);
                            a = fmaf(bf16_lo(wv[i].y), ha.z, a);
                            a = fmaf(bf16_hi(wv[i].y), ha.w, a);
                            a = fmaf(bf16_lo(wv[i].z), hb.x, a);
                            a = fmaf(bf16_hi(wv[i].z), hb.y, a);
                            a = fmaf(bf16_lo(wv[i].w), hb.z, a);
                            a = fmaf(bf16_hi(wv[i].w), hb.w, a);
                            acc[i][nb] = a;
                        }
                    }
                }
#pragma unroll
                for (int i = 0; i < R; ++i)
#pragma unroll
                    for (int nb = 0; nb < NB; ++nb) {
                        float a = acc[i][nb];
#pragma unroll
                        for (int o = 16; o >= 1; o >>= 1) a += __shfl_xor_sync(0xFFFFFFFFu, a, o);
                        acc[i][nb] = a;
                    }
                if (lane == 0) {
#pragma unroll
                    for (int i = 0; i < R; ++i) {
                        const int r = rg + i * kDotWarps;
                        if (r < rows) {
#pragma unroll
                            for (int nb = 0; nb < NB; ++nb) sc[r * NB + nb] = acc[i][nb];
                        }
                    }
                }
            }
            __syncwarp();
            if (lane == 0) {
                mbar_arrive(&empty[s]);
                mbar_arrive(&sfull[s]);
            }
        }
    }

    // ---------------- completion ticket ----------------
    __syncthreads();
    if (tid == 0) {
        __threadfence();
        const uint32_t ticket = atomicAdd(p.ticket, 1u);
        ms->is_last = (ticket == static_cast<uint32_t>(G - 1)) ? 1 : 0;
    }
    __syncthreads();
    if (!ms->is_last) return;
    __threadfence();

    // ---------------- global merge (last CTA) ----------------
    uint64_t *pref = reinterpret_cast<uint64_t *>(smem + L.merge);
    uint64_t *cands = pref + kMergePrefixCap;
    uint64_t *win = cands + kMergeCandCap;
    int *counts = reinterpret_cast<int *>(win + 1024);
    int *offsets = counts + kMaxLists;
    uint32_t *hist = reinterpret_cast<uint32_t *>(offsets + kMaxLists);
    const int k = p.k;
    const int J = (k + G - 1) / G;
    const int P = G * J;
    const bool aborted = (*reinterpret_cast<volatile uint32_t *>(p.err) & kErrWaitTimeout) != 0;

    for (int nb = 0; nb < p.nq && !aborted; ++nb) {
        const uint64_t *lists = p.cand + static_cast<size_t>(nb) * G * k;
        int32_t *oi = p.out_idx + static_cast<size_t>(nb) * k;
        float *ol = p.out_logits + static_cast<size_t>(nb) * k;

        // 1. tau*: k-th largest among the first J entries of every list
        uint64_t tau = 0;
        if (P <= kMergePrefixCap) {
            for (int i = tid; i < P; i += kThreads) {
                const int c = i / J, j = i - c * J;
                pref[i] = __ldcg(reinterpret_cast<const unsigned long long *>(lists) +
                                 static_cast<size_t>(c) * k + j);
            }
            if (tid == 0) ms->tau = 0;
            __syncthreads();
            if (P <= kRankCountMax) {
                for (int i = tid; i < P; i += kThreads) {
                    const uint64_t x = pref[i];
                    if (x == 0) continue;
                    int rank = 0;
                    for (int j = 0; j < P; ++j) rank += (pref[j] > x) ? 1 : 0;
                    if (rank == k - 1) ms->tau = x;
                }
                __syncthreads();
                tau = ms->tau;
            } else {
                int nz = 0;  // nonzero keys among the prefixes
                for (int i = 0; i < P; ++i) nz += pref[i] != 0;
                tau = (nz >= k) ? block_radix_threshold(SmemKeys{pref}, P, k, 1, hist, ms) : 0;
            }
        }
        // 2. per-list count of keys >= tau* (lists are sorted descending); the
        //    first J entries are already in shared memory, deeper entries are
        //    fetched eight at a time with independent loads.
        const uint64_t lo = tau > 0 ? tau : 1;
        const bool have_pref = P <= kMergePrefixCap;
        for (int c = tid; c < G; c += kThreads) {
            const unsigned long long *lc =
                reinterpret_cast<const unsigned long long *>(lists) + static_cast<size_t>(c) * k;
            int n = 0;
            if (have_pref)
                while (n < J && pref[c * J + n] >= lo) ++n;
            if (!have_pref || n == J) {
                for (int b = n; b < k && n == b; b += 8) {
                    uint64_t e[8];
#pragma unroll
                    for (int q = 0; q < 8; ++q) e[q] = (b + q < k) ? __ldcg(lc + b + q) : 0;
#pragma unroll
                    for (int q = 0; q < 8; ++q)
                        if (n == b + q && b + q < k && e[q] >= lo) ++n;
                }
            }
            counts[c] = n;
        }
        __syncthreads();
        if (tid < 32) {
            // exclusive scan of counts[0..G) by one warp, chunk per lane
            const int per = (G + 31) / 32;
            const int b0 = tid * per;
            int local = 0;
            for (int c = b0; c < min(G, b0 + per); ++c) local += counts[c];
            int incl = local;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int t2 = __shfl_up_sync(0xFFFFFFFFu, incl, o);
                if (tid >= o) incl += t2;
            }
            int run = incl - local;
            for (int c = b0; c < min(G, b0 + per); ++c) {
                offsets[c] = run;
                run += counts[c];
            }
            if (tid == 31) ms->n_cand = incl;
        }
        __syncthreads();
        const int M = ms->n_cand;
        if (M <= kMergeCandCap) {
            // 3a. gather the candidates, exact top-k among them
            for (int c = tid; c < G; c += kThreads) {
                const unsigned long long *lc =
                    reinterpret_cast<const unsigned long long *>(lists) + static_cast<size_t>(c) * k;
                for (int j = 0; j < counts[c]; ++j)
                    cands[offsets[c] + j] = (have_pref && j < J) ? pref[c * J + j] : __ldcg(lc + j);
            }
            __syncthreads();
            block_topk_to_output(cands, M, k, win, hist, ms, oi, ol);
        } else {
            // 3b. too many candidates: radix-select the threshold over all lists
            const uint64_t T = block_radix_threshold(GlobalKeys{lists}, G * k, k, lo, hist, ms);
            if (tid == 0) ms->n_win = 0;
            __syncthreads();
            for (int i = tid; i < G * k; i += kThreads) {
                const uint64_t x = __ldcg(reinterpret_cast<const unsigned long long *>(lists) + i);
                if (x >= T && x >= lo) win[atomicAdd(&ms->n_win, 1)] = x;
            }
            __syncthreads();
            block_topk_to_output(win, k, k, win, hist, ms, oi, ol);
        }
    }
    if (tid == 0) *p.ticket = 0;  // re-arm for the next launch
}

}  // namespace vie
