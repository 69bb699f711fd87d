// vie_stream_topk.cuh - the small-batch output head in one launch:
// streaming projection z = W_out h (paper, Section 3) fused with the exact
// top-k selection (exhaustive MIPS, Sections 2-3) and, optionally, the
// sparse -inf logit tensor (Section 3).
//
// One persistent CTA per SM.  The vocabulary is cut into chunks of RS rows
// (one weight stage each).  The first G * Ns chunks are dealt round robin
// (chunk c to CTA c mod G, so the CTAs sweep W together and keep every HBM
// channel busy); the rest form a pool that CTAs draw from in order with an
// atomic counter once their own chunks are done, so all CTAs finish together.
//   warp 0     producer: 1-D bulk copies (TMA) of chunks into a ring of
//              shared-memory stages (mbarrier transaction counts, L2
//              evict-first); the chunk id travels with the stage; an id of
//              -1 closes the stream;
//   warps 1..NS  selectors, NS = one per query up to four (selector s takes
//              query slots s, s + NS, ..): per query, the best keys seen so
//              far as a sorted list spread over the warp's registers; a row
//              enters only if it beats the current k-th key.  They never
//              hold a weight stage.  Wide lists (k > 64): every key above
//              the bound tau goes into a shared-memory buffer of the query
//              (ballot and append); a full buffer is cut back to a set
//              holding its best k by a bisection on the keys, which raises
//              tau.  After the stream the whole CTA turns each buffer into
//              the sorted list (radix select of the best k, then a bitonic
//              sort: runs of 128 keys in registers, merged through shared
//              memory);
//   the next 8 warps  projection: warp w owns rows w, w+8, .. (at most R) of
//              each stage and every lane a strided set of 16-byte column
//              chunks; bf16 -> fp32 widening, fp32 FMA against h (staged in
//              shared memory, one load per chunk reused for the warp's
//              rows).  The stage is released as soon as its last
//              shared-memory read retires; the warp-shuffle sums then go to
//              a separate, deeper score ring.
// The full logit vector never leaves the chip.  Afterwards each CTA writes
// its sorted top-k list to scratch and takes a ticket (an acq_rel atomic, no
// full fences); the CTA that draws the last ticket copies every list into
// shared memory in one pass (when they fit) and merges them:
//   1. tau* = k-th largest key among the first J = ceil(k/G) entries of all
//      lists (a lower bound of the true k-th key: k keys are >= it);
//   2. every list contributes its prefix of keys >= tau*;
//   3. exact top-k of those candidates (rank counting, or radix select when
//      there are many), written best first.
// Single-query launches with k <= 64 merge early instead: CTA 0 streams only
// its round-robin chunks (never the pool), so it finishes first, and then
// merges the CTAs' lists as they are published (merge_published: a release
// store of the launch's epoch per CTA, polled with acquire loads, the lists'
// first keys gathered in shared memory as they come); after the last list
// only one poll, one load and the fast merge over those keys remain.
// Launches of several queries publish their lists the same way; the first
// CTAs to finish (one per query, round robin) merge them as they arrive.
// With a sparse output, every CTA first fills a fixed slice of each output
// row with -inf; the merging CTA writes the k logits after every CTA has
// finished (the last ticket, or the last published list), so each fill
// happens before the value at the same position.
#pragma once

#include <cuda_fp16.h>
#include <cuda_fp8.h>

#include <cstdint>
#include <type_traits>

#include "vie_device.cuh"

namespace vie {

constexpr int kDotWarps = 8;
constexpr int kThreads = 32 * (2 + kDotWarps);  // single-query launches (the fewest threads)

// Selector warps of a launch with NB query slots, one per query up to four
// (selector s takes slots s, s + NS, ...), and the launch's thread count.
template <int NB>
__host__ __device__ constexpr int sel_warps() { return NB < 4 ? NB : 4; }
template <int NB>
__host__ __device__ constexpr int threads_for() { return 32 * (1 + sel_warps<NB>() + kDotWarps); }
constexpr int kMaxStages = 16;         // weight ring depth limit
constexpr int kScoreStages = 16;       // score ring depth
constexpr int kMergePrefixCap = 2048;  // keys: first-J prefixes of all lists
constexpr int kMergeCandCap = 2048;    // keys: gathered candidates
constexpr int kRankCountMax = 640;     // rank counting below this many keys
constexpr int kMaxLists = 1024;        // G <= 1024 CTAs
constexpr int kFastE = 8;              // fast merge: entries read per list (even)
constexpr int kFastMaxK = 64;          // fast merge: largest k
constexpr int kSelRun = 128;           // keys of one sorted run (a warp's registers)
constexpr int kRankRunsMin = kRankCountMax;  // merge output: a bitonic sort above this many keys

// Keys per query of the shared-memory candidate buffer of the wide lists
// (k > kFastMaxK): room for k keys and as many again, so a cut-back keeps k
// and frees at least k; 0 for the register lists.
__host__ __device__ inline int sel_cap_for(int k) {
    if (k <= kFastMaxK) return 0;
    const int c = (2 * k + 63) & ~63;
    return c < 256 ? 256 : c;
}

struct StreamTopkParams {
    const uint16_t *W;   // padded [V, d_pad] bf16 bits, or [V, d_pad] e4m3 codes (bytes)
    const float *row_scale;  // e4m3 rows: fp32 scale per row [V]; nullptr for bf16 rows
    const float *h;      // [nq, d] fp32
    int32_t nq;          // queries in this launch (<= NB)
    int64_t V;
    int32_t d, d_pad;
    int32_t k;
    int32_t rows_per_stage;  // RS <= 8 * R: rows of one chunk / weight stage
    int32_t stages;          // S, weight ring depth
    int32_t static_chunks;   // chunks each CTA owns before drawing from the pool
    int32_t pool_rows;       // rows of a pool piece (<= rows_per_stage)
    int32_t half_rows;       // 1: each half-warp projects its own row (R >= 2)
    int32_t sel_cap;         // wide lists: buffer keys per query (sel_cap_for(k)); else 0
    uint64_t *cand;          // [NB][G][k] keys
    uint64_t *heads;         // [NB][G][kFastE]: the first keys of each list
    uint32_t *ticket;        // CTA completion counter (self-resetting)
    uint32_t *next_chunk;    // pool counter (self-resetting)
    uint32_t *err;           // device flag word
    int32_t early;           // 1: CTA 0 merges the lists as they are published (nq == 1)
    int32_t pmerge;          // 1: the first min(nq, G) CTAs to finish merge the queries,
                             //    each taking the lists as they are published (nq > 1)
    uint32_t *epoch;         // launch counter word (early merge or pmerge)
    uint32_t *flags;         // [G] publication words (early merge or pmerge)
    int32_t *out_idx;        // [nq, k]
    float *out_logits;       // [nq, k]
    float *sparse;           // [nq, V] fp32 or nullptr
};

// Shared-memory carve-up; all offsets are multiples of 128 bytes.
struct SmemLayout {
    uint32_t bars, misc, h, scores, sel, ring, merge, total;
    __host__ __device__ static uint32_t align128(uint32_t x) { return (x + 127u) & ~127u; }
    __host__ __device__ SmemLayout(int nb, int d_pad, int rs, int stages, int row_bytes, int sel_cap) {
        bars = 0;
        misc = align128(bars + 8u * (2 * kMaxStages + 2 * kScoreStages));
        h = align128(misc + 256u);
        scores = align128(h + 4u * nb * d_pad);
        sel = align128(scores + 4u * kScoreStages * rs * nb);  // wide lists: [nb][sel_cap] keys
        ring = align128(sel + 8u * nb * sel_cap);
        merge = ring;  // the merge reuses the ring once the stream is drained
        uint32_t ring_end = ring + static_cast<uint32_t>(stages) * rs * row_bytes;
        uint32_t merge_end = merge + merge_fixed_bytes();
        total = ring_end > merge_end ? ring_end : merge_end;
    }
    __host__ __device__ static uint32_t merge_fixed_bytes() {
        return 8u * (kMergePrefixCap + kMergeCandCap + 1024) + 4u * (2 * kMaxLists + 256 + 32);
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
    unsigned int tau_v;
    int overflow;
    uint32_t epoch;
    int merger;                  // pmerge: m >= 0 merges queries m, m + X, ...
    int sel_cnt[8];              // wide lists: keys in each query's buffer
    int chunk_w[kMaxStages];     // first row of each weight stage (-1: end)
    int chunk_s[kScoreStages];   // first row of each score stage (-1: end)
};
static_assert(sizeof(MiscSmem) <= 256, "MiscSmem fits its 256-byte slot");

__device__ __forceinline__ uint32_t atomic_add_acq_rel_gpu(uint32_t *p, uint32_t v) {
    uint32_t old;
    asm volatile("atom.add.acq_rel.gpu.u32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
    return old;
}

__device__ __forceinline__ uint32_t atomic_add_relaxed_gpu(uint32_t *p, uint32_t v) {
    uint32_t old;
    asm volatile("atom.add.relaxed.gpu.u32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
    return old;
}

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

// Bitonic sort, descending, of the 32 * PER keys a warp holds (lane l holds
// elements l*PER .. l*PER + PER - 1).  Steps with a stride below PER swap
// registers; wider steps exchange with lane ^ (stride / PER).
template <int PER>
__device__ __forceinline__ void warp_sort_desc(uint64_t (&v)[PER], int lane) {
#pragma unroll
    for (int size = 2; size <= 32 * PER; size <<= 1) {
#pragma unroll
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            if (stride < PER) {
#pragma unroll
                for (int j = 0; j < PER; ++j) {
                    const int pj = j ^ stride;
                    if (pj > j) {
                        const bool desc = ((lane * PER + j) & size) == 0;
                        const uint64_t a = v[j], b = v[pj];
                        if (desc ? (a < b) : (a > b)) {
                            v[j] = b;
                            v[pj] = a;
                        }
                    }
                }
            } else {
                const int ls = stride / PER;
                const bool lower = (lane & ls) == 0;
#pragma unroll
                for (int j = 0; j < PER; ++j) {
                    const uint64_t o = shfl_xor_u64(v[j], ls);
                    const bool desc = ((lane * PER + j) & size) == 0;
                    const bool keep_max = lower == desc;
                    v[j] = keep_max ? (v[j] > o ? v[j] : o) : (v[j] < o ? v[j] : o);
                }
            }
        }
    }
}

// --------------------------------------------------------------------------
// Block-wide helpers for the merge: every thread of the CTA calls them, for
// any block size of at least 32 threads (merge_queries: at least kThreads).

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
// holds exactly the keys still needed.  The lanes of a warp that hit the
// same bin add their count with one atomic (the keys of a top-k share their
// leading digits, so a bin can draw most of the block's increments).  The
// block size is a multiple of 32.
template <class Keys>
__device__ uint64_t block_radix_threshold(Keys keys, int n, int k, uint64_t lo, uint32_t *hist,
                                          MiscSmem *ms) {
    const int tid = threadIdx.x, lane = tid & 31;
    uint64_t prefix = 0, mask = 0;
    int remaining = k;
    for (int shift = 56; shift >= 0; shift -= 8) {
        for (int i = tid; i < 256; i += static_cast<int>(blockDim.x)) hist[i] = 0;
        __syncthreads();
        for (int i0 = tid - lane; i0 < n; i0 += static_cast<int>(blockDim.x)) {
            const int i = i0 + lane;
            const uint64_t x = i < n ? keys[i] : 0ull;
            const bool in = x >= lo && x != 0 && (x & mask) == prefix;
            const unsigned bin = in ? static_cast<unsigned>((x >> shift) & 255u) : 256u;
            const unsigned peers = __match_any_sync(0xFFFFFFFFu, bin);
            if (in && (__ffs(peers) - 1) == lane) atomicAdd(&hist[bin], static_cast<unsigned>(__popc(peers)));
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

// Number of keys in keys[0..n) (shared memory, 16-byte aligned) above x.
// Every thread of a warp reads the same address, so each load is a broadcast;
// two keys per load and an unrolled loop keep many loads in flight.
__device__ __forceinline__ int rank_among(const uint64_t *keys, int n, uint64_t x) {
    const ulonglong2 *k2 = reinterpret_cast<const ulonglong2 *>(keys);
    const int n2 = n >> 1;
    int r0 = 0, r1 = 0;
#pragma unroll 8
    for (int j = 0; j < n2; ++j) {
        const ulonglong2 v = k2[j];
        r0 += (v.x > x) ? 1 : 0;
        r1 += (v.y > x) ? 1 : 0;
    }
    if (n & 1) r0 += (keys[n - 1] > x) ? 1 : 0;
    return r0 + r1;
}

// The last merge of a warp's sort network: the 32 * PER keys it holds
// (bitonic) sorted descending by half-cleaners of strides 16 * PER .. 1.
template <int PER>
__device__ __forceinline__ void warp_merge_desc(uint64_t (&v)[PER], int lane) {
#pragma unroll
    for (int stride = 16 * PER; stride > 0; stride >>= 1) {
        if (stride < PER) {
#pragma unroll
            for (int j = 0; j < PER; ++j) {
                const int pj = j ^ stride;
                if (pj > j && v[j] < v[pj]) {
                    const uint64_t a = v[j];
                    v[j] = v[pj];
                    v[pj] = a;
                }
            }
        } else {
            const int ls = stride / PER;
            const bool lower = (lane & ls) == 0;
#pragma unroll
            for (int j = 0; j < PER; ++j) {
                const uint64_t o = shfl_xor_u64(v[j], ls);
                v[j] = lower ? (v[j] > o ? v[j] : o) : (v[j] < o ? v[j] : o);
            }
        }
    }
}

// Sorts the m unique nonzero keys a[0..m) (shared memory) descending in
// place.  a must have room for P keys, P the power of two >= max(m,
// kSelRun); a[m..P) is zero-filled (zeros sort last).  Bitonic: runs of
// kSelRun keys sorted in registers (a warp each), then per doubling of the
// sorted length a mirror compare-exchange between the two runs of each pair
// and half-cleaners of strides >= kSelRun in shared memory, and the strides
// below kSelRun in registers.  Every thread of the CTA calls it; it ends
// with a barrier.
__device__ inline void block_sort_desc(uint64_t *a, int m) {
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int nthr = static_cast<int>(blockDim.x), nw = nthr >> 5;
    constexpr int PER = kSelRun / 32;
    int P = kSelRun;
    while (P < m) P <<= 1;
    for (int i = m + tid; i < P; i += nthr) a[i] = 0ull;
    __syncthreads();
    const int nruns = P / kSelRun;
    for (int r = warp; r < nruns; r += nw) {
        uint64_t v[PER];
#pragma unroll
        for (int j = 0; j < PER; ++j) v[j] = a[r * kSelRun + lane * PER + j];
        warp_sort_desc<PER>(v, lane);
#pragma unroll
        for (int j = 0; j < PER; ++j) a[r * kSelRun + lane * PER + j] = v[j];
    }
    for (int size = 2 * kSelRun; size <= P; size <<= 1) {
        const int half = size >> 1;
        __syncthreads();
        for (int i = tid; i < (P >> 1); i += nthr) {
            const int blk = i / half, j = i - blk * half;
            const int lo = blk * size + j, hi = blk * size + size - 1 - j;
            const uint64_t x = a[lo], y = a[hi];
            if (x < y) {
                a[lo] = y;
                a[hi] = x;
            }
        }
        for (int stride = half >> 1; stride >= kSelRun; stride >>= 1) {
            __syncthreads();
            for (int i = tid; i < (P >> 1); i += nthr) {
                const int lo = (i / stride) * 2 * stride + (i % stride), hi = lo + stride;
                const uint64_t x = a[lo], y = a[hi];
                if (x < y) {
                    a[lo] = y;
                    a[hi] = x;
                }
            }
        }
        __syncthreads();
        for (int r = warp; r < nruns; r += nw) {
            uint64_t v[PER];
#pragma unroll
            for (int j = 0; j < PER; ++j) v[j] = a[r * kSelRun + lane * PER + j];
            warp_merge_desc<PER>(v, lane);
#pragma unroll
            for (int j = 0; j < PER; ++j) a[r * kSelRun + lane * PER + j] = v[j];
        }
    }
    __syncthreads();
}

// Exact top-k of n unique nonzero keys in shared memory, written best first
// to out_idx / out_logits (and into the sparse row, if any).  Rank counting
// for small n, otherwise a radix-select threshold and rank counting of the
// k winners.
__device__ inline void block_topk_to_output(uint64_t *keys, int n, int k, uint64_t *win,
                                            uint32_t *hist, MiscSmem *ms, int32_t *out_idx,
                                            float *out_logits, float *sparse_row) {
    const int tid = threadIdx.x;
    uint64_t *src = keys;
    int m = n;
    if (n > kRankCountMax && n > k) {
        const uint64_t T = block_radix_threshold(SmemKeys{keys}, n, k, 1, hist, ms);
        if (tid == 0) ms->n_win = 0;
        __syncthreads();
        for (int i = tid; i < n; i += static_cast<int>(blockDim.x)) {
            const uint64_t x = keys[i];
            if (x >= T) win[atomicAdd(&ms->n_win, 1)] = x;
        }
        __syncthreads();
        src = win;
        m = k;
    }
    if (m > kRankRunsMin) {
        // many keys: a bitonic sort (rank counting is m^2); src has room for
        // the sort's power of two (at most 1024 keys here)
        block_sort_desc(src, m);
        for (int i = tid; i < min(m, k); i += static_cast<int>(blockDim.x)) {
            const uint64_t x = src[i];
            out_idx[i] = key_index(x);
            out_logits[i] = key_value(x);
            if (sparse_row != nullptr) sparse_row[key_index(x)] = key_value(x);
        }
        __syncthreads();
        return;
    }
    for (int i = tid; i < m; i += static_cast<int>(blockDim.x)) {
        const uint64_t x = src[i];
        const int rank = rank_among(src, m, x);
        if (rank < k) {
            out_idx[rank] = key_index(x);
            out_logits[rank] = key_value(x);
            if (sparse_row != nullptr) sparse_row[key_index(x)] = key_value(x);
        }
    }
    __syncthreads();
}

// Wide lists: cuts the cnt (> k) unique nonzero keys of buf back to a set
// that holds its best k, moved to buf[0..), and returns its size and the new
// entry bound (a later key enters only if it is above the bound).
// One warp.  The cut is found one digit at a time, two bits per step from
// three independent counts, each step reading the buffer from shared
// memory: first the top 16 bits of the high word (the ordered logit); if
// the keys at or above that coarse threshold are at most `room`, they are
// kept (at least k of them).  Otherwise the rest of the high word and then,
// when several keys share the k-th logit, the low word (the inverted row)
// give the exact k-th key, and exactly k keys are kept.
struct CutBack {
    int n;
    uint64_t bound;
};
static __device__ __noinline__ CutBack warp_cut_back(uint64_t *buf, int cnt, int k, int room, int lane) {
    __syncwarp();
    const uint32_t *w32 = reinterpret_cast<const uint32_t *>(buf);
    auto count3 = [&](uint32_t c1, uint32_t c2, uint32_t c3, int &n1, int &n2, int &n3) {
        n1 = n2 = n3 = 0;
#pragma unroll 4
        for (int e = lane; e < cnt; e += 32) {
            const uint32_t hi = w32[2 * e + 1];
            n1 += hi >= c1 ? 1 : 0;
            n2 += hi >= c2 ? 1 : 0;
            n3 += hi >= c3 ? 1 : 0;
        }
        n1 = static_cast<int>(__reduce_add_sync(0xFFFFFFFFu, n1));
        n2 = static_cast<int>(__reduce_add_sync(0xFFFFFFFFu, n2));
        n3 = static_cast<int>(__reduce_add_sync(0xFFFFFFFFu, n3));
    };
    uint32_t th = 0;
    int n1, n2, n3;
#pragma unroll 1
    for (int bit = 30; bit >= 16; bit -= 2) {
        const uint32_t c1 = th | (1u << bit), c2 = th | (2u << bit), c3 = th | (3u << bit);
        count3(c1, c2, c3, n1, n2, n3);
        th = n3 >= k ? c3 : (n2 >= k ? c2 : (n1 >= k ? c1 : th));
    }
    int n_ge = 0;
    for (int e = lane; e < cnt; e += 32) n_ge += w32[2 * e + 1] >= th ? 1 : 0;
    n_ge = static_cast<int>(__reduce_add_sync(0xFFFFFFFFu, n_ge));
    uint64_t T;
    if (th != 0 && n_ge <= room) {
        T = static_cast<uint64_t>(th) << 32;  // keys >= T: n_ge of them, at least k
    } else {
#pragma unroll 1
        for (int bit = 14; bit >= 0; bit -= 2) {
            const uint32_t c1 = th | (1u << bit), c2 = th | (2u << bit), c3 = th | (3u << bit);
            count3(c1, c2, c3, n1, n2, n3);
            th = n3 >= k ? c3 : (n2 >= k ? c2 : (n1 >= k ? c1 : th));
        }
        int n_gt = 0;
        n_ge = 0;
        for (int e = lane; e < cnt; e += 32) {
            const uint32_t hi = w32[2 * e + 1];
            n_gt += hi > th ? 1 : 0;
            n_ge += hi >= th ? 1 : 0;
        }
        n_gt = static_cast<int>(__reduce_add_sync(0xFFFFFFFFu, n_gt));
        n_ge = static_cast<int>(__reduce_add_sync(0xFFFFFFFFu, n_ge));
        uint32_t tl = 0;
        if (n_ge > k) {
            const int need = k - n_gt;  // keys still needed among those with logit th
#pragma unroll 1
            for (int bit = 30; bit >= 0; bit -= 2) {
                const uint32_t c1 = tl | (1u << bit), c2 = tl | (2u << bit), c3 = tl | (3u << bit);
                int m1 = 0, m2 = 0, m3 = 0;
                for (int e = lane; e < cnt; e += 32) {
                    if (w32[2 * e + 1] != th) continue;
                    const uint32_t lo = w32[2 * e];
                    m1 += lo >= c1 ? 1 : 0;
                    m2 += lo >= c2 ? 1 : 0;
                    m3 += lo >= c3 ? 1 : 0;
                }
                m1 = static_cast<int>(__reduce_add_sync(0xFFFFFFFFu, m1));
                m2 = static_cast<int>(__reduce_add_sync(0xFFFFFFFFu, m2));
                m3 = static_cast<int>(__reduce_add_sync(0xFFFFFFFFu, m3));
                tl = m3 >= need ? c3 : (m2 >= need ? c2 : (m1 >= need ? c1 : tl));
            }
        }
        T = (static_cast<uint64_t>(th) << 32) | tl;  // the k-th key: exactly k keys >= T
    }
    // in place: every write lands at or below the position it was read from
    // in this pass, after the whole warp has read that block of 32
    const unsigned lt_mask = (1u << lane) - 1u;
    int base = 0;
    for (int e0 = 0; e0 < cnt; e0 += 32) {
        const int e = e0 + lane;
        const uint64_t v = e < cnt ? buf[e] : 0ull;
        const bool in = v >= T && v != 0;
        const unsigned m = __ballot_sync(0xFFFFFFFFu, in);
        if (in) buf[base + __popc(m & lt_mask)] = v;
        base += __popc(m);
    }
    __syncwarp();
    // entry bound: a key enters if > bound, i.e. >= T (keys are never equal)
    return CutBack{base, T - 1};
}

// Wide lists, after the stream: the sorted list of one query's buffer (cnt
// unique nonzero keys; cnt may exceed k) written best first to dst[0..k)
// (zeros after the real keys) and its first kFastE keys to head.  Every
// thread of the CTA calls it.  win (room for the power of two >= k, at least
// kSelRun keys) and hist (256 words) are free shared memory; buf (room for
// 2k keys) is sorted in place when it holds at most k keys.
__device__ inline void write_cta_list(uint64_t *buf, int cnt, int k, uint32_t *hist, uint64_t *win,
                                      MiscSmem *ms, uint64_t *dst, uint64_t *head) {
    const int tid = threadIdx.x, nthr = static_cast<int>(blockDim.x);
    uint64_t *a = buf;
    int m = cnt;
    if (cnt > k) {
        // exactly k keys are >= T (keys are unique)
        const uint64_t T = block_radix_threshold(SmemKeys{buf}, cnt, k, 1, hist, ms);
        if (tid == 0) ms->n_win = 0;
        __syncthreads();
        for (int i = tid; i < cnt; i += nthr) {
            const uint64_t x = buf[i];
            if (x >= T) win[atomicAdd(&ms->n_win, 1)] = x;
        }
        a = win;
        m = k;
    }
    __syncthreads();
    block_sort_desc(a, m);  // room: win holds k keys; buf at least 2k when cnt <= k
    for (int i = tid; i < m; i += nthr) {
        dst[i] = a[i];
        if (i < kFastE) head[i] = a[i];
    }
    for (int i = m + tid; i < k; i += nthr) dst[i] = 0ull;
    for (int i = m + tid; i < kFastE; i += nthr) head[i] = 0ull;
}

// Shared-memory buffers of the merge.
struct MergeBufs {
    uint64_t *pref, *cands, *win;
    int *counts, *offsets;
    uint32_t *hist;
};

// Merges the G sorted lists of one query (G x k keys, `lists`) into the
// exact top-k.  Keys = SmemKeys when the lists were staged in shared memory.
template <class Keys>
__device__ void merge_lists(Keys lists, int G, int k, const MergeBufs &mb, MiscSmem *ms,
                            int32_t *oi, float *ol, float *sp) {
    const int tid = threadIdx.x;
    const int J = (k + G - 1) / G;
    const int P = G * J;

    // 1. tau*: k-th largest among the first J entries of every list
    uint64_t tau = 0;
    const bool have_pref = P <= kMergePrefixCap;
    if (have_pref) {
        for (int i = tid; i < P; i += static_cast<int>(blockDim.x)) {
            const int c = i / J, j = i - c * J;
            mb.pref[i] = lists[c * k + j];
        }
        if (tid == 0) ms->tau = 0;
        __syncthreads();
        if (P <= kRankCountMax) {
            for (int i = tid; i < P; i += static_cast<int>(blockDim.x)) {
                const uint64_t x = mb.pref[i];
                if (x != 0 && rank_among(mb.pref, P, x) == k - 1) ms->tau = x;
            }
            __syncthreads();
            tau = ms->tau;
        } else {
            int nz = 0;  // nonzero keys among the prefixes
            for (int i = 0; i < P; ++i) nz += mb.pref[i] != 0;
            tau = (nz >= k) ? block_radix_threshold(SmemKeys{mb.pref}, P, k, 1, mb.hist, ms) : 0;
        }
    }
    // 2. per-list count of keys >= tau* (lists are sorted descending); the
    //    first J entries are in the prefix buffer, deeper entries are read
    //    eight at a time with independent loads.
    const uint64_t lo = tau > 0 ? tau : 1;
    for (int c = tid; c < G; c += static_cast<int>(blockDim.x)) {
        int n = 0;
        if (have_pref)
            while (n < J && mb.pref[c * J + n] >= lo) ++n;
        if (!have_pref || n == J) {
            for (int b = n; b < k && n == b; b += 8) {
                uint64_t e[8];
#pragma unroll
                for (int q = 0; q < 8; ++q) e[q] = (b + q < k) ? lists[c * k + b + q] : 0;
#pragma unroll
                for (int q = 0; q < 8; ++q)
                    if (n == b + q && b + q < k && e[q] >= lo) ++n;
            }
        }
        mb.counts[c] = n;
    }
    __syncthreads();
    if (tid < 32) {
        // exclusive scan of counts[0..G) by one warp, a run of lists per lane
        const int per = (G + 31) / 32;
        const int b0 = tid * per;
        int local = 0;
        for (int c = b0; c < min(G, b0 + per); ++c) local += mb.counts[c];
        int incl = local;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int t2 = __shfl_up_sync(0xFFFFFFFFu, incl, o);
            if (tid >= o) incl += t2;
        }
        int run = incl - local;
        for (int c = b0; c < min(G, b0 + per); ++c) {
            mb.offsets[c] = run;
            run += mb.counts[c];
        }
        if (tid == 31) ms->n_cand = incl;
    }
    __syncthreads();
    const int M = ms->n_cand;
    if (M <= kMergeCandCap) {
        // 3a. gather the candidates, exact top-k among them
        for (int c = tid; c < G; c += static_cast<int>(blockDim.x))
            for (int j = 0; j < mb.counts[c]; ++j)
                mb.cands[mb.offsets[c] + j] =
                    (have_pref && j < J) ? mb.pref[c * J + j] : lists[c * k + j];
        __syncthreads();
        block_topk_to_output(mb.cands, M, k, mb.win, mb.hist, ms, oi, ol, sp);
    } else {
        // 3b. too many candidates: radix-select the threshold over all lists
        const uint64_t T = block_radix_threshold(lists, G * k, k, lo, mb.hist, ms);
        if (tid == 0) ms->n_win = 0;
        __syncthreads();
        for (int i = tid; i < G * k; i += static_cast<int>(blockDim.x)) {
            const uint64_t x = lists[i];
            if (x >= T && x >= lo) mb.win[atomicAdd(&ms->n_win, 1)] = x;
        }
        __syncthreads();
        block_topk_to_output(mb.win, k, k, mb.win, mb.hist, ms, oi, ol, sp);
    }
}

// The zeroed counters merge_fast_query starts from (every thread calls it;
// callers overlap it with the loads that stage the lists' heads).
__device__ __forceinline__ void merge_fast_reset(int *rank_part, MiscSmem *ms) {
    if (threadIdx.x == 0) {
        ms->tau_v = 0;
        ms->n_cand = 0;
        ms->overflow = 0;
    }
    for (int i = threadIdx.x; i < kFastE * kThreads / 2; i += static_cast<int>(blockDim.x))
        rank_part[i] = 0;  // M <= G * kFastE <= kFastE * kThreads / 2
}

// Latency-lean merge of one query for small k, spread over every warp of
// the CTA.  fe = the first kFastE keys of each of the G sorted lists, hv =
// their heads' value bits (padded with 0 to a multiple of 8).  tau = the
// k-th largest head value counted with multiplicity: at least k keys are
// >= (tau << 32), so every top-k key is too, and each list contributes its
// prefix of keys above that bound.  Returns false (writing nothing) if some
// list might hold more than kFastE such keys or fewer than k heads are
// real; the caller then merges in full.  Requires 2 * G <= kThreads, and
// the state merge_fast_reset sets, made visible by a bar.sync.
__device__ inline bool merge_fast_query(const uint64_t *fe, const uint32_t *hv, int G, int k,
                                        uint64_t *cands, int *rank_part, MiscSmem *ms, int32_t *oi,
                                        float *ol, float *sp) {
    const int tid = threadIdx.x, lane = tid & 31;
    const int G8 = (G + 7) & ~7;
    // tau: thread pair (2c, 2c+1) counts the heads >= head c, half each
    {
        const int c = tid >> 1, half = tid & 1;
        const bool real = c < G && fe[c * kFastE] != 0;
        const uint32_t v = c < G ? hv[c] : 0xFFFFFFFFu;
        const uint4 *h4 = reinterpret_cast<const uint4 *>(hv) + half * (G8 / 8);
        int ge = 0;
#pragma unroll 4
        for (int j = 0; j < G8 / 8; ++j) {
            const uint4 q = h4[j];
            ge += (q.x >= v) + (q.y >= v) + (q.z >= v) + (q.w >= v);
        }
        ge += __shfl_xor_sync(0xFFFFFFFFu, ge, 1);
        uint32_t best = (real && ge >= k) ? v : 0u;
        best = __reduce_max_sync(0xFFFFFFFFu, best);
        if (lane == 0 && best != 0) atomicMax(&ms->tau_v, best);
    }
    __syncthreads();
    const uint32_t tv = ms->tau_v;
    if (tv == 0) return false;  // uniform: fewer than k real heads
    const uint64_t lo = static_cast<uint64_t>(tv) << 32;
    const int En = k < kFastE ? k : kFastE;
    // gather: list c's keys >= lo, slots taken per warp
    {
        const int c = tid;
        int n = 0;
        if (c < G)
            while (n < En && fe[c * kFastE + n] >= lo) ++n;
        if (n == En && k > En) ms->overflow = 1;
        int incl = n;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int t = __shfl_up_sync(0xFFFFFFFFu, incl, o);
            if (lane >= o) incl += t;
        }
        int base = 0;
        if (lane == 31 && incl > 0) base = atomicAdd(&ms->n_cand, incl);
        base = __shfl_sync(0xFFFFFFFFu, base, 31);
        for (int j = 0; j < n; ++j) cands[base + incl - n + j] = fe[c * kFastE + j];
    }
    __syncthreads();
    if (ms->overflow) return false;
    const int M = ms->n_cand;
    // rank: candidate i is counted by up to kRankSplit threads, each over a
    // slice of the candidates; partial counts meet in shared memory
    constexpr int kRankSplit = 5;
    const int per = (M + kRankSplit - 1) / kRankSplit;
    for (int t = tid; t < M * kRankSplit; t += static_cast<int>(blockDim.x)) {
        const int i = t % M, part = t / M;
        const uint64_t x = cands[i];
        const int j0 = part * per, j1 = min(M, j0 + per);
        int r = 0;
#pragma unroll 4
        for (int j = j0; j < j1; ++j) r += (cands[j] > x) ? 1 : 0;
        if (r) atomicAdd(&rank_part[i], r);
    }
    __syncthreads();
    for (int i = tid; i < M; i += static_cast<int>(blockDim.x)) {
        const int rank = rank_part[i];
        if (rank < k) {
            const uint64_t x = cands[i];
            oi[rank] = key_index(x);
            ol[rank] = key_value(x);
            if (sp != nullptr) sp[key_index(x)] = key_value(x);
        }
    }
    __syncthreads();
    return true;
}

// Merges the per-CTA lists of queries 0..nq-1 (query q's G lists of k keys
// at cand + q*G*k) into each query's exact top-k, written best first to
// out_idx / out_logits + q*k and, if sparse is set, into row q of the sparse
// tensor.  `ws` is merge_bytes of shared memory for the working buffers.
// Small k: one pass of independent L2 loads fetches the first kFastE
// entries of every list of every query (thread c: list c), then each query
// is merged in shared memory; a query the fast merge cannot settle is merged
// in full.  Called by every thread of one CTA of at least kThreads threads.
__device__ inline void merge_queries(const uint64_t *cand, const uint64_t *heads, int nq, int G,
                                     int k, int64_t V,
                                     unsigned char *ws, uint32_t merge_bytes, MiscSmem *ms,
                                     int32_t *out_idx, float *out_logits, float *sparse) {
    const int tid = threadIdx.x;
    MergeBufs mb;
    mb.pref = reinterpret_cast<uint64_t *>(ws);
    mb.cands = mb.pref + kMergePrefixCap;
    mb.win = mb.cands + kMergeCandCap;
    mb.counts = reinterpret_cast<int *>(mb.win + 1024);
    mb.offsets = mb.counts + kMaxLists;
    mb.hist = reinterpret_cast<uint32_t *>(mb.offsets + kMaxLists);
    uint64_t *staged = reinterpret_cast<uint64_t *>(ws + SmemLayout::merge_fixed_bytes());
    const int stage_cap = static_cast<int>((merge_bytes - SmemLayout::merge_fixed_bytes()) / 8);

    const int G8 = (G + 7) & ~7;
    const bool fast = k <= kFastMaxK && G >= k && 2 * G <= kThreads &&
                      nq * (G * kFastE * 8 + G8 * 4) <= stage_cap * 8;
    uint32_t fast_done = 0;  // bit nb: query nb settled by the fast merge
    if (fast) {
        uint64_t *fe = staged;                                             // [nq][G][E]
        uint32_t *hv = reinterpret_cast<uint32_t *>(fe + nq * G * kFastE);  // [nq][G8]
        for (int q = 0; q < nq; ++q) {
            uint64_t key[kFastE];
            if (tid < G8) {
                // list tid's first keys from the heads area: rows of 32 bytes
                const ulonglong2 *hq = reinterpret_cast<const ulonglong2 *>(heads) +
                                       (static_cast<size_t>(q) * G + tid) * (kFastE / 2);
#pragma unroll
                for (int e = 0; e < kFastE; e += 2) {
                    const ulonglong2 x = tid < G ? __ldcg(hq + e / 2) : make_ulonglong2(0ull, 0ull);
                    key[e] = x.x;
                    key[e + 1] = x.y;
                }
            }
            if (q == 0) merge_fast_reset(mb.counts, ms);  // while the loads are in flight
            if (tid < G8) {
                if (tid < G) {
#pragma unroll
                    for (int e = 0; e < kFastE; ++e) fe[(q * G + tid) * kFastE + e] = key[e];
                }
                hv[q * G8 + tid] = tid < G ? static_cast<uint32_t>(key[0] >> 32) : 0u;
            }
        }
        __syncthreads();
        for (int nb = 0; nb < nq; ++nb) {
            int32_t *oi = out_idx + static_cast<size_t>(nb) * k;
            float *ol = out_logits + static_cast<size_t>(nb) * k;
            float *sp = sparse != nullptr ? sparse + static_cast<int64_t>(nb) * V : nullptr;
            if (nb > 0) {  // every thread is done with the previous query's counters
                __syncthreads();
                merge_fast_reset(mb.counts, ms);
                __syncthreads();
            }
            if (merge_fast_query(fe + nb * G * kFastE, hv + nb * G8, G, k, mb.cands, mb.counts, ms,
                                 oi, ol, sp))
                fast_done |= 1u << nb;
        }
    }
    for (int nb = 0; nb < nq; ++nb) {
        if (fast_done & (1u << nb)) continue;
        const uint64_t *lists = cand + static_cast<size_t>(nb) * G * k;
        int32_t *oi = out_idx + static_cast<size_t>(nb) * k;
        float *ol = out_logits + static_cast<size_t>(nb) * k;
        float *sp = sparse != nullptr ? sparse + static_cast<int64_t>(nb) * V : nullptr;
        const int n_all = G * k;
        if (n_all <= stage_cap) {
            // one pass of independent L2 loads brings every list in
            const unsigned long long *src = reinterpret_cast<const unsigned long long *>(lists);
            if ((reinterpret_cast<uintptr_t>(src) & 15u) == 0) {
                const ulonglong2 *src2 = reinterpret_cast<const ulonglong2 *>(src);
                ulonglong2 *dst2 = reinterpret_cast<ulonglong2 *>(staged);
                for (int i = tid; i < (n_all >> 1); i += static_cast<int>(blockDim.x)) dst2[i] = __ldcg(src2 + i);
                if ((n_all & 1) && tid == 0) staged[n_all - 1] = __ldcg(src + n_all - 1);
            } else {
                for (int i = tid; i < n_all; i += static_cast<int>(blockDim.x)) staged[i] = __ldcg(src + i);
            }
            __syncthreads();
            merge_lists(SmemKeys{staged}, G, k, mb, ms, oi, ol, sp);
        } else {
            merge_lists(GlobalKeys{lists}, G, k, mb, ms, oi, ol, sp);
        }
    }
}

// --------------------------------------------------------------------------
// Merge of one query from published lists (every thread of the merging CTA).
// CTA c publishes its lists with a release store of `target` (the launch's
// epoch + 1) into flags[c] once they and its sparse fill are written; words
// left by earlier launches hold older epochs.  Thread c polls flags[c] with
// acquire loads and, one iteration after it sees the value (so that load
// overlaps the next polls), copies list c's first kFastE keys (heads_q + c *
// kFastE) into fe, where the fast merge finds them.  When every list is in,
// the fast merge settles the query, or (a list that may hold more than
// kFastE of the top k, or fewer than k real heads) the lists (lists_q, G x k
// keys) are merged in full.  ws holds the merge buffers (merge_fixed_bytes);
// fe holds G * kFastE keys and then ceil(G/8)*8 head words.  Every wait is
// bounded; a list that never arrives is reported in *err and counted empty.
__device__ inline void merge_published(const uint32_t *flags, uint32_t target, const uint64_t *heads_q,
                                       const uint64_t *lists_q, int G, int k, unsigned char *ws,
                                       uint64_t *fe, MiscSmem *ms, uint32_t *err, int32_t *oi, float *ol,
                                       float *sp) {
    const int tid = threadIdx.x;
    MergeBufs mb;
    mb.pref = reinterpret_cast<uint64_t *>(ws);
    mb.cands = mb.pref + kMergePrefixCap;
    mb.win = mb.cands + kMergeCandCap;
    mb.counts = reinterpret_cast<int *>(mb.win + 1024);
    mb.offsets = mb.counts + kMaxLists;
    mb.hist = reinterpret_cast<uint32_t *>(mb.offsets + kMaxLists);
    const int G8 = (G + 7) & ~7;
    uint32_t *hv = reinterpret_cast<uint32_t *>(fe + G * kFastE);  // [G8]
    const ulonglong2 *heads2 = reinterpret_cast<const ulonglong2 *>(heads_q);

    // empty lists until they arrive; the fast merge's counters
    for (int i = tid; i < G * kFastE; i += static_cast<int>(blockDim.x)) fe[i] = 0ull;
    for (int i = tid; i < G8; i += static_cast<int>(blockDim.x)) hv[i] = 0u;
    merge_fast_reset(mb.counts, ms);
    bool pending = tid < G;  // thread c watches list c
    bool have = false;       // list c seen, its heads not copied yet
    const uint64_t t0 = global_timer_ns();
    for (;;) {
        const bool load_now = have;
        ulonglong2 e[kFastE / 2];
        if (load_now) {
#pragma unroll
            for (int j = 0; j < kFastE / 2; ++j) e[j] = __ldcg(heads2 + static_cast<size_t>(tid) * (kFastE / 2) + j);
            have = false;
        }
        if (pending) {
            if (ld_acquire_gpu(flags + tid) == target) {
                pending = false;
                have = true;
            } else if (global_timer_ns() - t0 > kWaitLimitNs) {
                pending = false;
                atomicOr(err, kErrWaitTimeout);
            }
        }
        if (load_now) {
            ulonglong2 *dst = reinterpret_cast<ulonglong2 *>(fe + tid * kFastE);
#pragma unroll
            for (int j = 0; j < kFastE / 2; ++j) dst[j] = e[j];
            hv[tid] = static_cast<uint32_t>(e[0].x >> 32);
        }
        if (__syncthreads_count((pending || have) ? 1 : 0) == 0) break;
    }
    // every list is in: the barrier above ordered each thread's acquire (and
    // the fast merge's reset) before what follows
    const bool fast_ok = k <= G && 2 * G <= static_cast<int>(blockDim.x);
    if (!(fast_ok && merge_fast_query(fe, hv, G, k, mb.cands, mb.counts, ms, oi, ol, sp)))
        merge_lists(GlobalKeys{lists_q}, G, k, mb, ms, oi, ol, sp);
}

// --------------------------------------------------------------------------
// Rows of the stage that starts at row0: whole chunks (RS rows) in the
// round-robin part, pool pieces (RSH rows) behind it, and never past the
// vocabulary.
__device__ __forceinline__ int stage_rows(int64_t row0, int64_t pool_row0, int RS, int RSH, int64_t V) {
    const int64_t len = row0 < pool_row0 ? RS : RSH;
    return static_cast<int>(min(len, V - row0));
}

// e4m3 x4 (one 32-bit word, element 0 in the low byte) times h.x..h.w into a,
// in element order; each e4m3 value is exact in fp16 and fp32.  (Decoding by
// integer shifts into fp32 bits instead took more instructions per weight
// than these conversions.)
__device__ __forceinline__ float fma_e4m3x4(uint32_t w, float4 h, float a) {
    const float2 lo = __half22float2(__half2(__nv_cvt_fp8x2_to_halfraw2(
        static_cast<__nv_fp8x2_storage_t>(w & 0xFFFFu), __NV_E4M3)));
    const float2 hi = __half22float2(__half2(__nv_cvt_fp8x2_to_halfraw2(
        static_cast<__nv_fp8x2_storage_t>(w >> 16), __NV_E4M3)));
    a = fmaf(lo.x, h.x, a);
    a = fmaf(lo.y, h.y, a);
    a = fmaf(hi.x, h.z, a);
    a = fmaf(hi.y, h.w, a);
    return a;
}

// Q8: rows of e4m3 codes (16 per 16-byte chunk) with one fp32 scale per row,
// logit = scale * sum; otherwise bf16 rows (8 per chunk).
template <int NB, int MM, int R, bool Q8>
__global__ void __launch_bounds__(threads_for<NB>(), 1) stream_topk_kernel(const StreamTopkParams p) {
    constexpr int NS = sel_warps<NB>(), T = threads_for<NB>(), QPS = NB / NS;
    extern __shared__ __align__(128) unsigned char smem[];
    const int RS = p.rows_per_stage;  // <= 8 * R
    const int S = p.stages;
    const int row_bytes = Q8 ? p.d_pad : p.d_pad * 2;
    constexpr int kEPC = Q8 ? 16 : 8;  // weights per 16-byte chunk
    const SmemLayout L(NB, p.d_pad, RS, S, row_bytes, MM == 0 ? p.sel_cap : 0);
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + L.bars);
    uint64_t *empty = full + kMaxStages;
    uint64_t *sfull = empty + kMaxStages;
    uint64_t *sempty = sfull + kScoreStages;
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
    const int RSH = p.pool_rows;  // rows of a pool piece
    const int64_t pool_row0 = static_cast<int64_t>(G) * p.static_chunks * RS;
    const int C = p.d_pad / kEPC;  // 16-byte chunks per row
    const int stage_bytes = RS * row_bytes;

    if (tid == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], kDotWarps);
        }
        for (int s = 0; s < kScoreStages; ++s) {
            mbar_init(&sfull[s], kDotWarps);
            mbar_init(&sempty[s], NS);
        }
        ms->abort = 0;
        ms->is_last = 0;
        if (p.early || p.pmerge) ms->epoch = *reinterpret_cast<volatile uint32_t *>(p.epoch);
        fence_mbar_init();
        griddep_launch_dependents();  // a kernel launched after this one may be scheduled now
    }
    // h -> shared memory as [nb][part][chunk][4] (2 parts of 4 for bf16 rows,
    // 4 for e4m3 rows) so a lane's float4 loads of one chunk fall in distinct
    // bank groups; zero pad, zero unused queries.  Asynchronous copies by warps 1.. issued before the producer
    // starts, so h is ahead of the weight stream in the memory queues; those
    // warps wait for them after the barrier (bar.sync 1 below).
    if (warp > 0) {
        for (int i = tid - 32; i < NB * p.d_pad; i += T - 32) {
            const int nb = i / p.d_pad, j = i - nb * p.d_pad;
            const bool real = nb < p.nq && j < p.d;
            const float *src = real ? p.h + static_cast<int64_t>(nb) * p.d + j : p.h;
            const int c = j / kEPC, e = j - c * kEPC;
            cp_async_4_zfill(h_s + (nb * (kEPC / 4) + (e >> 2)) * (C * 4) + c * 4 + (e & 3), src, real);
        }
        cp_async_commit();
    }
    __syncthreads();

    if (warp == 0) {
        // ---------------- producer ----------------
        if (lane == 0) {
            const uint64_t pol = l2_evict_first_policy();
            const unsigned char *W = reinterpret_cast<const unsigned char *>(p.W);
            const int Ns = p.static_chunks;
            // the early merger (CTA 0) streams its round-robin chunks only
            const bool pool = !(p.early && cta == 0);
            // first draw from the pool, issued early so its latency is hidden
            uint32_t draw = (Ns == 0 && pool) ? atomic_add_relaxed_gpu(p.next_chunk, 1u) : 0u;
            int issued = 0;
            bool ok = true;
            for (int t = 0;; ++t) {
                int64_t row0;
                if (t < Ns) {
                    row0 = static_cast<int64_t>(t * G + cta) * RS;
                } else if (pool) {
                    row0 = pool_row0 + static_cast<int64_t>(draw) * RSH;
                    if (row0 >= p.V) row0 = -1;
                } else {
                    row0 = -1;
                }
                const int s = t % S, u = t / S;
                if (t >= S && !mbar_wait(&empty[s], (u - 1) & 1, abort_flag)) {
                    ok = false;
                    break;
                }
                ms->chunk_w[s] = static_cast<int>(row0);
                if (row0 < 0) {
                    mbar_arrive(&full[s]);  // closes the stream: no bytes
                    break;
                }
                const int rows = stage_rows(row0, pool_row0, RS, RSH, p.V);
                const uint32_t bytes = static_cast<uint32_t>(rows) * row_bytes;
                mbar_arrive_expect_tx(&full[s], bytes);
                bulk_g2s(ring + s * stage_bytes, W + row0 * row_bytes, bytes, &full[s], pol);
                issued = t + 1;
                if (t + 1 >= Ns && pool) draw = atomic_add_relaxed_gpu(p.next_chunk, 1u);
            }
            if (!ok) {
                atomicOr(p.err, kErrWaitTimeout);
                ms->abort = 1;
                // drain: copies still in flight must land before the CTA exits
                const int never = 0;
                for (int t2 = max(0, issued - S); t2 < issued; ++t2)
                    mbar_wait(&full[t2 % S], (t2 / S) & 1, const_cast<volatile int *>(&never));
            }
        }
        // the other lanes wait for the producer lane here, so the whole warp
        // reaches the CTA barrier below together (bar.sync counts warps)
        __syncwarp();
    } else {
        // fused sparse output: a fixed slice of every query row = -inf
        if (p.sparse != nullptr) {
            const float ninf = __uint_as_float(0xFF800000u);
            const int64_t base = p.V / G, rem = p.V % G;
            const int64_t f0 = cta * base + (cta < rem ? cta : rem);
            const int64_t fn = base + (cta < rem ? 1 : 0);
            for (int q = 0; q < p.nq; ++q) {
                float *row = p.sparse + static_cast<int64_t>(q) * p.V + f0;
                for (int64_t i = tid - 32; i < fn; i += T - 32) row[i] = ninf;
            }
        }
        cp_async_wait_all();
        named_barrier_sync(1, T - 32);  // h in shared memory for warps 1..
        if (warp <= NS) {
            const int sw = NS == 1 ? 0 : warp - 1;  // this selector's query slots: sw, sw + NS, ...
            if constexpr (MM == 0) {
                // ---------------- selector (wide lists) ----------------
                uint64_t *sbuf = reinterpret_cast<uint64_t *>(smem + L.sel);
                const int cap = p.sel_cap;
                const unsigned lt_mask = (1u << lane) - 1u;
                int cnt[QPS];
                uint64_t tau[QPS];
#pragma unroll
                for (int j = 0; j < QPS; ++j) {
                    cnt[j] = 0;
                    tau[j] = 0;
                }
                for (int t = 0;; ++t) {
                    const int s = t % kScoreStages, u = t / kScoreStages;
                    if (!mbar_wait(&sfull[s], u & 1, abort_flag)) {
                        if (lane == 0) {
                            atomicOr(p.err, kErrWaitTimeout);
                            ms->abort = 1;
                        }
                        break;
                    }
                    const int chunk = ms->chunk_s[s];
                    if (chunk < 0) break;
                    const int64_t row0 = chunk;
                    const int rows = stage_rows(row0, pool_row0, RS, RSH, p.V);
                    const float *sc = scores + s * RS * NB;
#pragma unroll
                    for (int j = 0; j < QPS; ++j) {
                        const int nb = sw + j * NS;
                        if (nb >= p.nq) break;
                        uint64_t *buf = sbuf + nb * cap;
                        for (int rb = 0; rb < rows; rb += 32) {
                            if (cnt[j] > cap - 32) {  // no room for another 32 keys: cut back
                                const CutBack cb = warp_cut_back(buf, cnt[j], p.k, (cap + p.k) / 2, lane);
                                cnt[j] = cb.n;
                                tau[j] = cb.bound;
                            }
                            const int r = rb + lane;
                            const uint64_t key =
                                (r < rows) ? make_key(sc[r * NB + nb], static_cast<uint32_t>(row0 + r)) : 0;
                            const bool in = key > tau[j];
                            const unsigned m = __ballot_sync(0xFFFFFFFFu, in);
                            if (in) buf[cnt[j] + __popc(m & lt_mask)] = key;
                            cnt[j] += __popc(m);
                        }
                    }
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&sempty[s]);
                }
                if (lane == 0) {
#pragma unroll
                    for (int j = 0; j < QPS; ++j) ms->sel_cnt[sw + j * NS] = sw + j * NS < p.nq ? cnt[j] : 0;
                }
            } else {
                // ---------------- selector ----------------
                WarpList<MM> list[QPS];
                uint64_t tau[QPS];
#pragma unroll
                for (int j = 0; j < QPS; ++j) {
                    list[j].clear();
                    tau[j] = 0;
                }
                for (int t = 0;; ++t) {
                    const int s = t % kScoreStages, u = t / kScoreStages;
                    if (!mbar_wait(&sfull[s], u & 1, abort_flag)) {
                        if (lane == 0) {
                            atomicOr(p.err, kErrWaitTimeout);
                            ms->abort = 1;
                        }
                        break;
                    }
                    const int chunk = ms->chunk_s[s];
                    if (chunk < 0) break;
                    const int64_t row0 = chunk;
                    const int rows = stage_rows(row0, pool_row0, RS, RSH, p.V);
                    const float *sc = scores + s * RS * NB;
#pragma unroll
                    for (int j = 0; j < QPS; ++j) {
                        const int nb = sw + j * NS;
                        if (nb >= p.nq) break;
                        for (int rb = 0; rb < rows; rb += 32) {
                            const int r = rb + lane;
                            const uint64_t key =
                                (r < rows) ? make_key(sc[r * NB + nb], static_cast<uint32_t>(row0 + r)) : 0;
                            unsigned m = __ballot_sync(0xFFFFFFFFu, key > tau[j]);
                            while (m) {
                                const int srcl = __ffs(m) - 1;
                                m &= m - 1;
                                const uint64_t x = shfl_u64(key, srcl);
                                if (x > tau[j]) {
                                    list[j].insert(x, lane);
                                    tau[j] = list[j].at(p.k - 1);
                                }
                            }
                        }
                    }
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&sempty[s]);
                }
                // this CTA's sorted top-k per query -> scratch (every slot,
                // zeros for the unused ones)
#pragma unroll
                for (int j = 0; j < QPS; ++j) {
                    const int nb = sw + j * NS;
                    uint64_t *dst = p.cand + (static_cast<size_t>(nb) * G + cta) * p.k;
                    uint64_t *head = p.heads + (static_cast<size_t>(nb) * G + cta) * kFastE;
#pragma unroll
                    for (int s = 0; s < MM; ++s) {
                        const int pos = lane * MM + s;
                        if (pos < p.k) dst[pos] = list[j].v[s];
                        if (pos < kFastE) head[pos] = pos < p.k ? list[j].v[s] : 0ull;
                    }
                }
            }
        } else {
            // ---------------- projection ----------------
            const int w = warp - 1 - NS;
            int t = 0;
            for (;; ++t) {
                const int s = t % S, u = t / S;
                if (!mbar_wait(&full[s], u & 1, abort_flag)) {
                    if (lane == 0) {
                        atomicOr(p.err, kErrWaitTimeout);
                        ms->abort = 1;
                    }
                    break;
                }
                const int chunk = ms->chunk_w[s];
                if (chunk < 0) break;
                const int64_t row0 = chunk;
                const int rows = stage_rows(row0, pool_row0, RS, RSH, p.V);
                const unsigned char *stage = ring + s * stage_bytes;
                // Warp w owns rows w, w + 8, ... (at most R of them) of the
                // stage.  SPLIT = 1: the whole warp works on each row, lane
                // l on chunks l, l + 32, ...  SPLIT = 2: the half-warps take
                // the two rows of a pair (w + 8(2i), w + 8(2i+1)), half-lane l
                // on chunks l, l + 16, ..., so rows of 16 * odd chunks leave
                // no lane idle on the last pass.  Either way every row sums
                // its products in the same order wherever it sits.
                auto project = [&](auto split) -> bool {
                    constexpr int SPLIT = decltype(split)::value;
                    constexpr int RL = R / SPLIT;   // rows per lane
                    constexpr int LW = 32 / SPLIT;  // lanes per row
                    const int sub = lane / LW, sl = lane % LW;
                    int rr[RL];
#pragma unroll
                    for (int i = 0; i < RL; ++i) rr[i] = min(w + (i * SPLIT + sub) * kDotWarps, rows - 1);
                    float acc[RL][NB];
#pragma unroll
                    for (int i = 0; i < RL; ++i)
#pragma unroll
                        for (int nb = 0; nb < NB; ++nb) acc[i][nb] = 0.0f;
                    float rscale[RL];  // e4m3 rows: their scales, loaded under the FMA loop
#pragma unroll
                    for (int i = 0; i < RL; ++i) rscale[i] = Q8 ? __ldg(p.row_scale + row0 + rr[i]) : 1.0f;
                    if (w < rows) {
                        for (int c = sl; c < C; c += LW) {
                            uint4 wv[RL];
#pragma unroll
                            for (int i = 0; i < RL; ++i)
                                wv[i] = *reinterpret_cast<const uint4 *>(stage + rr[i] * row_bytes + c * 16);
#pragma unroll
                            for (int nb = 0; nb < NB; ++nb) {
                                if constexpr (Q8) {
                                    const float *hq = h_s + nb * 4 * (C * 4) + c * 4;
                                    const float4 h0 = *reinterpret_cast<const float4 *>(hq);
                                    const float4 h1 = *reinterpret_cast<const float4 *>(hq + 1 * (C * 4));
                                    const float4 h2 = *reinterpret_cast<const float4 *>(hq + 2 * (C * 4));
                                    const float4 h3 = *reinterpret_cast<const float4 *>(hq + 3 * (C * 4));
#pragma unroll
                                    for (int i = 0; i < RL; ++i) {
                                        float a = acc[i][nb];
                                        a = fma_e4m3x4(wv[i].x, h0, a);
                                        a = fma_e4m3x4(wv[i].y, h1, a);
                                        a = fma_e4m3x4(wv[i].z, h2, a);
                                        a = fma_e4m3x4(wv[i].w, h3, a);
                                        acc[i][nb] = a;
                                    }
                                } else {
                                    const float4 ha = *reinterpret_cast<const float4 *>(
                                        h_s + (nb * 2 + 0) * (C * 4) + c * 4);
                                    const float4 hb = *reinterpret_cast<const float4 *>(
                                        h_s + (nb * 2 + 1) * (C * 4) + c * 4);
#pragma unroll
                                    for (int i = 0; i < RL; ++i) {
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
                        }
                    }
                    // every read of the weight stage has retired: hand it back
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&empty[s]);
#pragma unroll
                    for (int i = 0; i < RL; ++i)
#pragma unroll
                        for (int nb = 0; nb < NB; ++nb) {
                            float a = acc[i][nb];
#pragma unroll
                            for (int o = LW / 2; o >= 1; o >>= 1) a += __shfl_xor_sync(0xFFFFFFFFu, a, o);
                            acc[i][nb] = a;
                        }
                    const int ss = t % kScoreStages, su = t / kScoreStages;
                    if (t >= kScoreStages && !mbar_wait(&sempty[ss], (su - 1) & 1, abort_flag)) {
                        if (lane == 0) {
                            atomicOr(p.err, kErrWaitTimeout);
                            ms->abort = 1;
                        }
                        return false;
                    }
                    float *sc = scores + ss * RS * NB;
                    if (sl == 0) {
                        if (w == 0 && sub == 0) ms->chunk_s[ss] = chunk;
#pragma unroll
                        for (int i = 0; i < RL; ++i) {
                            const int r = w + (i * SPLIT + sub) * kDotWarps;
                            if (r < rows) {
#pragma unroll
                                for (int nb = 0; nb < NB; ++nb)
                                    sc[r * NB + nb] = Q8 ? acc[i][nb] * rscale[i] : acc[i][nb];
                            }
                        }
                    }
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&sfull[ss]);
                    return true;
                };
                const bool ok = (R >= 2 && p.half_rows)
                                    ? project(std::integral_constant<int, (R >= 2 ? 2 : 1)>{})
                                    : project(std::integral_constant<int, 1>{});
                if (!ok) break;
            }
            // pass the end of the stream on to the selector
            if (!*abort_flag) {
                const int ss = t % kScoreStages, su = t / kScoreStages;
                if (t < kScoreStages || mbar_wait(&sempty[ss], (su - 1) & 1, abort_flag)) {
                    if (lane == 0) {
                        if (w == 0) ms->chunk_s[ss] = -1;
                        mbar_arrive(&sfull[ss]);
                    }
                } else if (lane == 0) {
                    atomicOr(p.err, kErrWaitTimeout);
                    ms->abort = 1;
                }
            }
        }
    }

    // ---------------- wide lists: buffers -> sorted lists ----------------
    // (the ring is free: every stage was consumed before its role ended)
    if constexpr (MM == 0) {
        __syncthreads();
        uint32_t *hist = reinterpret_cast<uint32_t *>(smem + L.ring);
        uint64_t *win = reinterpret_cast<uint64_t *>(smem + L.ring + 1024);
        uint64_t *sbuf = reinterpret_cast<uint64_t *>(smem + L.sel);
        for (int nb = 0; nb < p.nq; ++nb)
            write_cta_list(sbuf + nb * p.sel_cap, ms->sel_cnt[nb], p.k, hist, win, ms,
                           p.cand + (static_cast<size_t>(nb) * G + cta) * p.k,
                           p.heads + (static_cast<size_t>(nb) * G + cta) * kFastE);
    }

    // ---------------- early merge (one query, k <= 64) ----------------
    // bar.sync orders every thread's writes (list, heads, sparse fill) before
    // thread 0's release store of this launch's epoch + 1; CTA 0 acquires each
    // word before it reads that CTA's list, and a bar.sync orders all of
    // those acquires before its output writes.  Words left by earlier
    // launches hold older epochs, so nothing needs clearing.
    if (p.early) {
        __syncthreads();
        const uint32_t target = ms->epoch + 1u;
        if (tid == 0) st_release_gpu(p.flags + cta, target);
        if (cta != 0) return;
        unsigned char *ws = smem + L.merge;
        merge_published(p.flags, target, p.heads, p.cand, G, p.k, ws,
                        reinterpret_cast<uint64_t *>(ws + SmemLayout::merge_fixed_bytes()), ms, p.err,
                        p.out_idx, p.out_logits, p.sparse);
        if (tid == 0) {
            *p.next_chunk = 0;  // re-arm the pool for the next launch
            *reinterpret_cast<volatile uint32_t *>(p.epoch) = target;
        }
        return;
    }

    // ---------------- publication, then the merge (first X CTAs) ----------------
    // Several queries: the release store and the epoch as in the early merge;
    // a relaxed ticket ranks the CTAs by finishing order, the first X merge
    // (queries m, m + X, ...) while the others still stream, and the last
    // re-arms the pool and the ticket and advances the epoch (every CTA has
    // drawn its last chunk and taken its ticket by then).
    if (p.pmerge) {
        __syncthreads();
        const int X = min(p.nq, G);
        const uint32_t target = ms->epoch + 1u;
        if (tid == 0) {
            st_release_gpu(p.flags + cta, target);
            const uint32_t ticket = atomic_add_relaxed_gpu(p.ticket, 1u);
            if (ticket == static_cast<uint32_t>(G - 1)) {
                *p.next_chunk = 0;
                *p.ticket = 0;
                *reinterpret_cast<volatile uint32_t *>(p.epoch) = target;
            }
            ms->merger = ticket < static_cast<uint32_t>(X) ? static_cast<int>(ticket) : -1;
        }
        __syncthreads();
        const int mg = ms->merger;
        if (mg < 0) return;
        unsigned char *ws = smem + L.merge;
        uint64_t *fe = reinterpret_cast<uint64_t *>(ws + SmemLayout::merge_fixed_bytes());
        for (int q = mg; q < p.nq; q += X) {
            merge_published(p.flags, target, p.heads + static_cast<size_t>(q) * G * kFastE,
                            p.cand + static_cast<size_t>(q) * G * p.k, G, p.k, ws, fe, ms, p.err,
                            p.out_idx + static_cast<size_t>(q) * p.k, p.out_logits + static_cast<size_t>(q) * p.k,
                            p.sparse != nullptr ? p.sparse + static_cast<int64_t>(q) * p.V : nullptr);
            __syncthreads();
        }
        return;
    }

    // ---------------- completion ticket ----------------
    // bar.sync orders every thread's writes (lists, sparse fill) before
    // thread 0's release; its acquire, then bar.sync, orders the merging
    // CTA's reads after every other CTA's writes.
    __syncthreads();
    if (tid == 0) {
        const uint32_t ticket = atomic_add_acq_rel_gpu(p.ticket, 1u);
        ms->is_last = (ticket == static_cast<uint32_t>(G - 1)) ? 1 : 0;
    }
    __syncthreads();
    if (!ms->is_last) return;

    // ---------------- global merge (last CTA) ----------------
    // Every CTA wrote a full list (valid keys or zeros) even if it gave up on
    // a wait, so the merge stays in bounds; such a call is reported through
    // the device flag and its outputs are unspecified.
    merge_queries(p.cand, p.heads, p.nq, G, p.k, p.V, smem + L.merge, L.total - L.merge, ms, p.out_idx,
                      p.out_logits, p.sparse);
    if (tid == 0) {
        *p.ticket = 0;  // re-arm both counters for the next launch
        *p.next_chunk = 0;
    }
}

}  // namespace vie
