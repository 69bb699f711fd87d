// vie_tc_topk.cu - launchers of the tensor-core head: hi/lo query prep, and
// the tcgen05 projection with per-CTA top-k and the merge in its last CTA.
#include <cuda_bf16.h>

#include "vie_launch.h"
#include "vie_tc_launch.cuh"

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

template <int NQ, bool Q8>
void tc_sizes(int *slot_bytes, int *min_slots, int *buf_bytes, int *kb_w_bytes, int *kb_h_bytes) {
    *slot_bytes = TcShape<NQ, Q8>::kSlotBytes;
    *min_slots = TcShape<NQ, Q8>::kMinSlots;
    *buf_bytes = TcShape<NQ, Q8>::kBufBytes;
    *kb_w_bytes = TcShape<NQ, Q8>::kStageA;
    *kb_h_bytes = TcShape<NQ, Q8>::kStageB;
}

bool tc_sizes_of(int nq_tmpl, bool q8, int *slot_bytes, int *min_slots, int *buf_bytes, int *kb_w, int *kb_h) {
    switch (q8 ? -nq_tmpl : nq_tmpl) {
        case 8: tc_sizes<8, false>(slot_bytes, min_slots, buf_bytes, kb_w, kb_h); return true;
        case 16: tc_sizes<16, false>(slot_bytes, min_slots, buf_bytes, kb_w, kb_h); return true;
        case 32: tc_sizes<32, false>(slot_bytes, min_slots, buf_bytes, kb_w, kb_h); return true;
        case 64: tc_sizes<64, false>(slot_bytes, min_slots, buf_bytes, kb_w, kb_h); return true;
        case -4: tc_sizes<4, true>(slot_bytes, min_slots, buf_bytes, kb_w, kb_h); return true;
        case -8: tc_sizes<8, true>(slot_bytes, min_slots, buf_bytes, kb_w, kb_h); return true;
        case -16: tc_sizes<16, true>(slot_bytes, min_slots, buf_bytes, kb_w, kb_h); return true;
        case -32: tc_sizes<32, true>(slot_bytes, min_slots, buf_bytes, kb_w, kb_h); return true;
        default: return false;
    }
}

// The 4-query e4m3 tile builds its whole query operand in shared memory (no
// prep kernel; the ring holds weights only) when it takes at most 48 KB of
// pieces (d_pad <= 3072).
int tc_hres_bytes(int nq_tmpl, bool q8, int n_kb) {
    if (!q8 || nq_tmpl != 4) return 0;
    const int b = n_kb * TcShape<4, true>::kStageB;
    return b <= 48 * 1024 ? b : 0;
}

// The ring first (as many stages as fit beside the fewest score slots), then
// as many score slots as the shared memory left over holds.
bool tc_shape(int nq_tmpl, bool q8, int kps, int hres_bytes, int *stages, int *slots, uint32_t *smem) {
    int slot_bytes = 0, min_slots = 0, buf_bytes = 0, kb_w = 0, kb_h = 0;
    if (!tc_sizes_of(nq_tmpl, q8, &slot_bytes, &min_slots, &buf_bytes, &kb_w, &kb_h)) return false;
    const int stage_bytes = kps * (hres_bytes > 0 ? kb_w : kb_w + kb_h);
    for (int s = kTcMaxStages; s >= 2; --s) {
        const TcSmemLayout L(min_slots * slot_bytes, buf_bytes, s, stage_bytes, hres_bytes);
        if (L.total <= 232448u) {
            int sl = min_slots;
            while (sl < kTcScoreSlots &&
                   TcSmemLayout((sl + 1) * slot_bytes, buf_bytes, s, stage_bytes, hres_bytes).total <= 232448u)
                ++sl;
            *stages = s;
            *slots = sl;
            *smem = TcSmemLayout(sl * slot_bytes, buf_bytes, s, stage_bytes, hres_bytes).total;
            return true;
        }
    }
    return false;
}

int tc_tile_rows(int nq_tmpl, bool q8) {
    switch (q8 ? -nq_tmpl : nq_tmpl) {
        case 8: return TcShape<8>::kTileRows;
        case 16: return TcShape<16>::kTileRows;
        case 32: return TcShape<32>::kTileRows;
        case 64: return TcShape<64>::kTileRows;
        case -4: return TcShape<4, true>::kTileRows;
        case -8: return TcShape<8, true>::kTileRows;
        case -16: return TcShape<16, true>::kTileRows;
        case -32: return TcShape<32, true>::kTileRows;
        default: return 0;
    }
}

int tc_max_k(int nq_tmpl, bool q8) {
    switch (q8 ? -nq_tmpl : nq_tmpl) {
        case 8: return TcShape<8>::kMaxK;
        case 16: return TcShape<16>::kMaxK;
        case 32: return TcShape<32>::kMaxK;
        case 64: return TcShape<64>::kMaxK;
        case -4: return TcShape<4, true>::kMaxK;
        case -8: return TcShape<8, true>::kMaxK;
        case -16: return TcShape<16, true>::kMaxK;
        case -32: return TcShape<32, true>::kMaxK;
        default: return 0;
    }
}

cudaError_t launch_tc_topk(int nq_tmpl, bool q8, const CUtensorMap &mapW, const CUtensorMap &mapH,
                           const TcParams &p, int grid, uint32_t smem, cudaStream_t stream) {
    if (q8) return launch_tc_topk_e4m3(nq_tmpl, mapW, mapH, p, grid, smem, stream);
    switch (nq_tmpl) {
        case 8: return launch_tc_one<8, false>(mapW, mapH, p, grid, smem, stream);
        case 16: return launch_tc_one<16, false>(mapW, mapH, p, grid, smem, stream);
        case 32: return launch_tc_one<32, false>(mapW, mapH, p, grid, smem, stream);
        case 64: return launch_tc_one<64, false>(mapW, mapH, p, grid, smem, stream);
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
