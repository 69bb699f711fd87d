// vie_head.cu - the C ABI declared in include/vie_head.h: argument checks,
// handle life cycle, launch configuration, weight-layout preparation and
// the sparse-logit scatter kernel.
#include <cuda_fp8.h>
#include <cuda_runtime.h>

#include <atomic>
#include <climits>
#include <cmath>
#include <cstdarg>
#include <cstdint>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <new>

#include "vie_head.h"
#include "vie_launch.h"
#include "vie_tc_topk.cuh"

namespace {

thread_local char g_err[512] = "";

vie_status fail(vie_status st, const char *fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof g_err, fmt, ap);
    va_end(ap);
    return st;
}

vie_status fail_cuda(cudaError_t e, const char *what) {
    return fail(e == cudaErrorMemoryAllocation ? VIE_ERR_OOM : VIE_ERR_CUDA, "%s: %s (%s)", what,
                cudaGetErrorString(e), cudaGetErrorName(e));
}

// Library-wide device flag word (used by kernels that have no handle).
__device__ uint32_t g_dev_err = 0;

constexpr int kMaxSmem = 232448;  // 227 KB opt-in dynamic shared memory per CTA
constexpr int kMaxNB = 8;
// The tensor-core path keeps [NQ][G][k] lists (NQ * k <= kTcListKeys) and
// [NQ <= 64][G][4] heads in
// the same scratch as the streaming path's [kMaxNB][G][VIE_K_MAX] lists.
static_assert(vie::kTcListKeys + (vie::kTcHRows / 2) * vie::kTcMergeE <= kMaxNB * VIE_K_MAX,
              "tensor-core lists must fit the candidate scratch");
constexpr int kMaxHBytes = 64 * 1024;  // shared-memory budget for staged queries
constexpr int kMaxSelBytes = 32 * 1024;  // ... and for the wide lists' candidate buffers
// Scratch words of a handle: [0] completion ticket, [1] device flag word,
// [2] chunk / tile pool counter, [4] launch epoch, [8 ..] one publication
// word per CTA (a CTA's lists are ready once its word holds the epoch + 1).
constexpr int kEpochWord = 4;
constexpr int kFlagWords = 8;
constexpr int kNumWords = kFlagWords + vie::kMaxLists;

}  // namespace

struct vie_head {
    int device;
    int64_t V;
    int32_t d, d_pad;
    int num_sms;
    int G;
    uint16_t *W;        // [V, d_pad] bf16 bits, or e4m3 codes (bytes) when scale is set
    float *scale;       // e4m3 heads: fp32 scale per row [V]; nullptr for bf16 heads
    uint64_t *cand;     // [kMaxNB][G][VIE_K_MAX] ranking keys, then [kMaxNB][G][kFastE] heads
    uint32_t *words;    // kNumWords scratch words (see kEpochWord, kFlagWords)
    int64_t scratch_bytes;
    // tensor-core path (batches): hi/lo bf16 query matrix and TMA descriptors
    void *hB;             // [kTcHRows][d_pad] bf16, or e4m3 query pieces [4 NQ][d_pad]
    float *qscale;        // e4m3 heads: [32][kQ8Pieces] piece scales of the query group
    bool tc_ready;
    CUtensorMap mapW;     // W as [V][d_pad], box 128 rows x 128 bytes, 128-byte swizzle
    CUtensorMap mapH[4];  // hB, box 16 / 32 / 64 / 128 rows x 128 bytes
    // vie_head_topk_host: device staging of queries and top-k (grown on demand)
    float *stage_h;
    int32_t *stage_idx;
    float *stage_logits;
    size_t stage_h_elems, stage_out_elems;
};

// ---------------------------------------------------------------------------
// Row quantisation to e4m3: one warp per row of bf16 W [V, d] (any 2-byte
// alignment).  scale = max |w| / 448 in fp32 (1 for a zero row); each code is
// w / scale rounded to the nearest e4m3 value (ties to even, saturated), the
// row padded to d_pad (a multiple of 16) with zero codes.
__global__ void quantize_e4m3_kernel(const uint16_t *__restrict__ src, int64_t V, int d, int d_pad,
                                     uint8_t *__restrict__ q, float *__restrict__ scale) {
    const int lane = threadIdx.x & 31;
    const int64_t warps = static_cast<int64_t>(gridDim.x) * (blockDim.x >> 5);
    for (int64_t row = blockIdx.x * static_cast<int64_t>(blockDim.x >> 5) + (threadIdx.x >> 5);
         row < V; row += warps) {
        const uint16_t *wr = src + row * d;
        float amax = 0.0f;
        for (int j = lane; j < d; j += 32)
            amax = fmaxf(amax, fabsf(__uint_as_float(static_cast<uint32_t>(wr[j]) << 16)));
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xFFFFFFFFu, amax, o));
        const float sc = amax > 0.0f ? amax / 448.0f : 1.0f;
        uint8_t *qr = q + row * d_pad;
        for (int j = lane; j < d_pad; j += 32) {
            const float x = j < d ? __uint_as_float(static_cast<uint32_t>(wr[j]) << 16) / sc : 0.0f;
            qr[j] = static_cast<uint8_t>(__nv_cvt_float_to_fp8(x, __NV_SATFINITE, __NV_E4M3));
        }
        if (lane == 0) scale[row] = sc;
    }
}

// ---------------------------------------------------------------------------
// Weight-layout preparation: [V, d] (any 2-byte alignment) -> [V, d_pad]
// with 16-byte rows, pad columns = +0.  One thread per 16-byte output chunk.
__global__ void prep_weights_kernel(const uint16_t *__restrict__ src, int64_t V, int d, int d_pad,
                                    uint16_t *__restrict__ dst) {
    const int C = d_pad >> 3;
    const int64_t n = V * C;
    for (int64_t id = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; id < n;
         id += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t row = id / C;
        const int c = static_cast<int>(id - row * C);
        uint16_t v[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const int col = c * 8 + e;
            v[e] = col < d ? src[row * d + col] : static_cast<uint16_t>(0);
        }
        uint4 o;
        o.x = v[0] | (static_cast<uint32_t>(v[1]) << 16);
        o.y = v[2] | (static_cast<uint32_t>(v[3]) << 16);
        o.z = v[4] | (static_cast<uint32_t>(v[5]) << 16);
        o.w = v[6] | (static_cast<uint32_t>(v[7]) << 16);
        reinterpret_cast<uint4 *>(dst)[id] = o;
    }
}

// ---------------------------------------------------------------------------
// Sparse full-vocabulary logits (paper, Section 3): row b of `out` becomes
// -inf everywhere, then logits[b, j] lands at idx[b, j].  Each CTA owns a
// contiguous slice of one row: it fills the slice, synchronises, then writes
// the retrieved logits that fall inside the slice, so every fill of a slot
// happens before its value is written.
__global__ void scatter_sparse_kernel(const int32_t *__restrict__ idx,
                                      const float *__restrict__ logits, int k, int64_t V,
                                      int64_t per_cta, float *__restrict__ out, int batch_base,
                                      uint32_t *err) {
    const int b = batch_base + blockIdx.y;
    float *row = out + static_cast<int64_t>(b) * V;
    const int64_t lo = blockIdx.x * per_cta;
    const int64_t hi = min(V, lo + per_cta);
    const float ninf = __uint_as_float(0xFF800000u);
    if (lo < hi) {
        // scalar head up to 16-byte alignment, float4 body, scalar tail
        const uintptr_t a = reinterpret_cast<uintptr_t>(row + lo);
        int64_t head = static_cast<int64_t>(((16 - (a & 15)) & 15) >> 2);
        if (head > hi - lo) head = hi - lo;
        for (int64_t i = threadIdx.x; i < head; i += blockDim.x) row[lo + i] = ninf;
        const int64_t body0 = lo + head;
        const int64_t nvec = (hi - body0) >> 2;
        float4 *vp = reinterpret_cast<float4 *>(row + body0);
        const float4 f4 = make_float4(ninf, ninf, ninf, ninf);
        for (int64_t i = threadIdx.x; i < nvec; i += blockDim.x) vp[i] = f4;
        for (int64_t i = body0 + nvec * 4 + threadIdx.x; i < hi; i += blockDim.x) row[i] = ninf;
    }
    __syncthreads();
    for (int j = threadIdx.x; j < k; j += blockDim.x) {
        const int32_t t = idx[static_cast<int64_t>(b) * k + j];
        if (t < 0 || static_cast<int64_t>(t) >= V) {
            if (blockIdx.x == 0) atomicOr(err, vie::kErrScatterIndex);
            continue;
        }
        if (t >= lo && t < hi) row[t] = logits[static_cast<int64_t>(b) * k + j];
    }
}

// ---------------------------------------------------------------------------
namespace {

// Selector of the streaming kernel: register lists of 2 keys per lane for
// k <= 64, else (0) the shared-memory candidate buffers of the wide lists.
int pick_mm(int k) { return k <= vie::kFastMaxK ? 2 : 0; }

// Keys per query of a launch's candidate buffers (wide lists): a single
// query gets about 4k (its first cut-back comes early in the stream, where it
// is hidden, and usually stays the only one; the CTA's final selection then
// sorts a few k keys, not every row it streamed), groups the least size for k.
int sel_cap_launch(int nb, int k) {
    const int c = vie::sel_cap_for(k);
    if (nb != 1 || c == 0) return c;
    const int c4 = (4 * k + 63) & ~63;
    return c4 > kMaxSelBytes / 8 ? kMaxSelBytes / 8 : c4;
}

// Widest query group for a row width and k: the staged queries and the wide
// lists' candidate buffers must fit their shared-memory budgets.
int nb_cap_for(int d_pad, int k) {
    int nb = kMaxNB;
    while (nb > 1 && (nb * d_pad * 4 > kMaxHBytes || nb * vie::sel_cap_for(k) * 8 > kMaxSelBytes)) nb >>= 1;
    return nb;
}

// Launch-shape options (they change speed, never results), set through
// vie_set_launch_option.  Process-wide; each call reads them when it plans
// its launches.  The defaults are the measured best shapes.
struct OptionSpec {
    int dflt, lo, hi;
};
constexpr OptionSpec kOptionSpec[VIE_OPT_COUNT] = {
    {48, 1, 227},      // VIE_OPT_STAGE_MIN_KB
    {85, 0, 100},      // VIE_OPT_STATIC_PCT
    {1, 1, 64},        // VIE_OPT_POOL_DIV
    {2, 1, INT32_MAX}, // VIE_OPT_TC_MIN_BATCH
    {4, 1, 4},         // VIE_OPT_TC_KPS
    {1, 1, INT32_MAX}, // VIE_OPT_TC_MIN_BATCH_E4M3
    {-1, -1, 1},       // VIE_OPT_HALF_ROWS
    {1, 0, 1},         // VIE_OPT_HOST_H_DIRECT
    {1, 0, 1},         // VIE_OPT_EARLY_MERGE
};
std::atomic<int> g_options[VIE_OPT_COUNT] = {
    {kOptionSpec[0].dflt}, {kOptionSpec[1].dflt}, {kOptionSpec[2].dflt}, {kOptionSpec[3].dflt},
    {kOptionSpec[4].dflt}, {kOptionSpec[5].dflt}, {kOptionSpec[6].dflt}, {kOptionSpec[7].dflt},
    {kOptionSpec[8].dflt}};
static_assert(VIE_OPT_COUNT == 9, "one default per option");

int opt(vie_launch_option o) { return g_options[o].load(std::memory_order_relaxed); }

// Whether the streaming projection gives each half-warp its own row: with
// 16-byte chunks c per row, a full warp's last pass over a row runs c mod 32
// lanes; at most 16 of them means half-warps finish the row in one fewer
// lane slot per row pair.  Needs two rows per warp (R >= 2).
int half_rows_for(int r, int chunks) {
    if (r < 2) return 0;
    const int v = opt(VIE_OPT_HALF_ROWS);
    if (v >= 0) return v > 0 ? 1 : 0;
    const int tail = chunks % 32;
    return (tail != 0 && tail <= 16) ? 1 : 0;
}

// Rows of a pool piece for stages of rs rows.
int pool_rows_for(int rs) {
    int div = opt(VIE_OPT_POOL_DIV);
    div = div > rs ? rs : div;
    return (rs + div - 1) / div;
}

struct LaunchShape {
    int r, rs, stages;
    uint32_t smem;
};

// Rows per warp per stage (R), stage rows (8*R, fewer for very wide rows),
// and ring depth (deepest that fits) for one launch.
bool pick_shape(int nb, int d_pad, int row_bytes, int sel_cap, LaunchShape *out) {
    const int r_max = nb == 1 ? 8 : 4;  // 8 rows per warp only for single-query launches
    int r = 1;
    while (r < r_max && 8 * r * row_bytes < opt(VIE_OPT_STAGE_MIN_KB) * 1024) r <<= 1;
    for (int rs = 8 * r; rs >= 1; --rs) {
        for (int s = vie::kMaxStages; s >= 2; --s) {
            const vie::SmemLayout L(nb, d_pad, rs, s, row_bytes, sel_cap);
            if (L.total <= static_cast<uint32_t>(kMaxSmem)) {
                out->r = r;
                out->rs = rs;
                out->stages = s;
                out->smem = L.total;
                return true;
            }
        }
    }
    return false;
}

vie_status check_device(const vie_head *hd) {
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return fail_cuda(e, "cudaGetDevice");
    if (dev != hd->device)
        return fail(VIE_ERR_INVALID_ARG, "handle lives on device %d but device %d is current",
                    hd->device, dev);
    return VIE_OK;
}

// cuTensorMapEncodeTiled from the driver, looked up once.
using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                   const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                   const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn encode_tiled() {
    static EncodeTiledFn fn = []() -> EncodeTiledFn {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess)
            return nullptr;
        return reinterpret_cast<EncodeTiledFn>(p);
    }();
    return fn;
}

// 2-D uint8 tensor map [rows][cols] (cols contiguous, pitch bytes), box
// box_rows x 128 columns, 128-byte swizzle, out-of-range elements read as 0.
bool make_map_u8(CUtensorMap *m, void *base, uint64_t rows, uint64_t cols, uint64_t pitch,
                 uint32_t box_rows) {
    EncodeTiledFn fn = encode_tiled();
    if (fn == nullptr) return false;
    const cuuint64_t dims[2] = {cols, rows};
    const cuuint64_t strides[1] = {pitch};
    const cuuint32_t box[2] = {128u, box_rows};
    const cuuint32_t estr[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, base, dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 2-D bf16 tensor map [rows][cols] (cols contiguous, pitch bytes), box
// box_rows x 64 columns, 128-byte swizzle, out-of-range elements read as 0.
bool make_map_bf16(CUtensorMap *m, void *base, uint64_t rows, uint64_t cols, uint64_t pitch,
                   uint32_t box_rows) {
    EncodeTiledFn fn = encode_tiled();
    if (fn == nullptr) return false;
    const cuuint64_t dims[2] = {cols, rows};
    const cuuint64_t strides[1] = {pitch};
    const cuuint32_t box[2] = {static_cast<cuuint32_t>(vie::kTcKBlock), box_rows};
    const cuuint32_t estr[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

extern "C" {

const char *vie_last_error(void) { return g_err; }

vie_status vie_set_launch_option(vie_launch_option option, int32_t value) {
    if (static_cast<int>(option) < 0 || option >= VIE_OPT_COUNT)
        return fail(VIE_ERR_INVALID_ARG, "vie_set_launch_option: unknown option %d", static_cast<int>(option));
    const OptionSpec &sp = kOptionSpec[option];
    if (value == VIE_OPT_DEFAULT) value = sp.dflt;
    if (value < sp.lo || value > sp.hi)
        return fail(VIE_ERR_INVALID_ARG, "vie_set_launch_option: value %d of option %d outside [%d, %d]",
                    value, static_cast<int>(option), sp.lo, sp.hi);
    g_options[option].store(value, std::memory_order_relaxed);
    return VIE_OK;
}

vie_status vie_get_launch_option(vie_launch_option option, int32_t *value) {
    if (static_cast<int>(option) < 0 || option >= VIE_OPT_COUNT || value == nullptr)
        return fail(VIE_ERR_INVALID_ARG, "vie_get_launch_option: bad option %d or NULL value",
                    static_cast<int>(option));
    *value = opt(option);
    return VIE_OK;
}

static vie_status create_head(const void *W_out, int64_t V, int32_t d, vie_dtype dtype, bool e4m3,
                              vie_head **out) {
    if (out == nullptr) return fail(VIE_ERR_INVALID_ARG, "vie_head_create: out is NULL");
    *out = nullptr;
    if (W_out == nullptr) return fail(VIE_ERR_INVALID_ARG, "vie_head_create: W_out is NULL");
    if (V < 1 || V > static_cast<int64_t>(INT32_MAX) - 1)
        return fail(VIE_ERR_INVALID_ARG, "vie_head_create: V=%lld outside [1, 2^31-2]",
                    static_cast<long long>(V));
    if (d < 1 || d > VIE_D_MAX)
        return fail(VIE_ERR_INVALID_ARG, "vie_head_create: d=%d outside [1, %d]", d, VIE_D_MAX);
    if (dtype != VIE_DTYPE_BF16)
        return fail(VIE_ERR_UNSUPPORTED, "vie_head_create: dtype %d is not supported (bf16 only)",
                    static_cast<int>(dtype));
    if (reinterpret_cast<uintptr_t>(W_out) & 1u)
        return fail(VIE_ERR_INVALID_ARG, "vie_head_create: W_out is not 2-byte aligned");

    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return fail_cuda(e, "cudaGetDevice");
    cudaPointerAttributes pa;
    e = cudaPointerGetAttributes(&pa, W_out);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return fail(VIE_ERR_INVALID_ARG, "vie_head_create: W_out is not a CUDA pointer");
    }
    if ((pa.type != cudaMemoryTypeDevice && pa.type != cudaMemoryTypeManaged) || pa.device != dev)
        return fail(VIE_ERR_INVALID_ARG,
                    "vie_head_create: W_out must be device memory of the current device %d", dev);

    int sms = 0;
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return fail_cuda(e, "cudaDeviceGetAttribute");

    vie_head *hd = new (std::nothrow) vie_head();
    if (hd == nullptr) return fail(VIE_ERR_OOM, "vie_head_create: host allocation failed");
    hd->device = dev;
    hd->V = V;
    hd->d = d;
    hd->d_pad = e4m3 ? (d + 15) & ~15 : (d + 7) & ~7;  // 16-byte rows either way
    hd->num_sms = sms;
    int64_t g = (V + 63) / 64;
    if (g > sms) g = sms;
    if (g > vie::kMaxLists) g = vie::kMaxLists;
    hd->G = static_cast<int>(g < 1 ? 1 : g);

    const size_t wbytes = static_cast<size_t>(V) * hd->d_pad * (e4m3 ? 1 : 2);
    const size_t cbytes =
        static_cast<size_t>(kMaxNB) * hd->G * (VIE_K_MAX + vie::kFastE) * sizeof(uint64_t);
    hd->scratch_bytes = static_cast<int64_t>(cbytes + kNumWords * sizeof(uint32_t));
    e = cudaMalloc(&hd->W, wbytes);
    if (e == cudaSuccess && e4m3) e = cudaMalloc(&hd->scale, static_cast<size_t>(V) * sizeof(float));
    if (e == cudaSuccess) e = cudaMalloc(&hd->cand, cbytes);
    if (e == cudaSuccess) e = cudaMemset(hd->cand, 0, cbytes);  // empty lists until written
    if (e == cudaSuccess) e = cudaMalloc(&hd->words, kNumWords * sizeof(uint32_t));
    if (e == cudaSuccess)
        e = cudaMalloc(&hd->hB, static_cast<size_t>(vie::kTcHRows) * hd->d_pad * 2);
    if (e == cudaSuccess) e = cudaMemset(hd->hB, 0, static_cast<size_t>(vie::kTcHRows) * hd->d_pad * 2);
    if (e == cudaSuccess && e4m3) e = cudaMalloc(&hd->qscale, 32 * vie::kQ8Pieces * sizeof(float));
    if (e == cudaSuccess) e = cudaMemset(hd->words, 0, kNumWords * sizeof(uint32_t));
    if (e == cudaSuccess && e4m3) {
        int64_t blocks = (V + 7) / 8;  // 8 rows (warps) per block
        if (blocks > 64LL * sms) blocks = 64LL * sms;
        quantize_e4m3_kernel<<<static_cast<unsigned>(blocks), 256>>>(
            static_cast<const uint16_t *>(W_out), V, d, hd->d_pad, reinterpret_cast<uint8_t *>(hd->W),
            hd->scale);
        e = cudaGetLastError();
    } else if (e == cudaSuccess) {
        const int64_t chunks = V * (hd->d_pad >> 3);
        int64_t blocks = (chunks + 255) / 256;
        if (blocks > 32LL * sms) blocks = 32LL * sms;
        prep_weights_kernel<<<static_cast<unsigned>(blocks), 256>>>(
            static_cast<const uint16_t *>(W_out), V, d, hd->d_pad, hd->W);
        e = cudaGetLastError();
    }
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    if (e != cudaSuccess) {
        const vie_status st = fail_cuda(e, "vie_head_create");
        cudaFree(hd->W);
        cudaFree(hd->scale);
        cudaFree(hd->cand);
        cudaFree(hd->words);
        cudaFree(hd->hB);
        cudaFree(hd->qscale);
        delete hd;
        return st;
    }
    if (e4m3) {  // kind::f8f6f4 maps: codes [V][d_pad] and the query pieces, 128-byte rows
        const uint64_t pitch8 = static_cast<uint64_t>(hd->d_pad);
        hd->tc_ready = hd->d_pad >= 128 &&
                       make_map_u8(&hd->mapW, hd->W, static_cast<uint64_t>(V), hd->d_pad, pitch8, vie::kTcTile);
        for (int i = 0; i < 4 && hd->tc_ready; ++i)
            hd->tc_ready = make_map_u8(&hd->mapH[i], hd->hB, vie::kTcHRows, hd->d_pad, pitch8, 16u << i);
        *out = hd;
        return VIE_OK;
    }
    const uint64_t pitch = static_cast<uint64_t>(hd->d_pad) * 2;
    hd->tc_ready = make_map_bf16(&hd->mapW, hd->W, static_cast<uint64_t>(V), hd->d_pad, pitch,
                                 vie::kTcTile);
    for (int i = 0; i < 4 && hd->tc_ready; ++i)
        hd->tc_ready = make_map_bf16(&hd->mapH[i], hd->hB, vie::kTcHRows, hd->d_pad, pitch, 16u << i);
    *out = hd;
    return VIE_OK;
}

vie_status vie_head_create(const void *W_out, int64_t V, int32_t d, vie_dtype dtype,
                           vie_head **out) {
    return create_head(W_out, V, d, dtype, false, out);
}

vie_status vie_head_create_e4m3(const void *W_out, int64_t V, int32_t d, vie_head **out) {
    return create_head(W_out, V, d, VIE_DTYPE_BF16, true, out);
}

vie_status vie_head_export_e4m3(const vie_head *head, uint8_t *codes, float *scales,
                                vie_stream stream) {
    const char *fn = "vie_head_export_e4m3";
    if (head == nullptr || codes == nullptr || scales == nullptr)
        return fail(VIE_ERR_INVALID_ARG, "%s: NULL argument", fn);
    if (head->scale == nullptr) return fail(VIE_ERR_INVALID_ARG, "%s: not an e4m3 head", fn);
    vie_status st = check_device(head);
    if (st != VIE_OK) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = cudaMemcpy2DAsync(codes, static_cast<size_t>(head->d), head->W,
                                      static_cast<size_t>(head->d_pad), static_cast<size_t>(head->d),
                                      static_cast<size_t>(head->V), cudaMemcpyDeviceToDevice, s);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(scales, head->scale, static_cast<size_t>(head->V) * sizeof(float),
                            cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess) return fail_cuda(e, fn);
    return VIE_OK;
}

vie_status vie_head_destroy(vie_head *head) {
    if (head == nullptr) return VIE_OK;
    cudaFree(head->W);
    cudaFree(head->scale);
    cudaFree(head->cand);
    cudaFree(head->words);
    cudaFree(head->hB);
    cudaFree(head->qscale);
    cudaFree(head->stage_h);
    cudaFree(head->stage_idx);
    cudaFree(head->stage_logits);
    delete head;
    return VIE_OK;
}

vie_status vie_head_get_props(const vie_head *head, vie_head_props *props) {
    if (head == nullptr || props == nullptr)
        return fail(VIE_ERR_INVALID_ARG, "vie_head_get_props: NULL argument");
    props->V = head->V;
    props->d = head->d;
    props->d_pad = head->d_pad;
    props->ctas = head->G;
    props->device = head->device;
    props->weight_bytes = head->scale != nullptr ? head->V * head->d_pad + head->V * 4
                                                 : head->V * head->d_pad * 2;
    props->scratch_bytes = head->scratch_bytes;
    return VIE_OK;
}

// The launch plan of a top-k call (path, query groups, launches).
// Query slots per tensor-core launch: the smallest tile that holds the batch;
// 64 (one pass over W for up to 64 queries) only where k fits its lists.
// e4m3 heads: up to 32 (four accumulator columns per query).
static int tc_group(int32_t batch, int32_t k, bool q8) {
    if (q8 && batch <= 4) return 4;
    if (batch <= 8) return 8;
    if (batch <= 16) return 16;
    if (q8 || batch <= 32 || k > vie::tc_max_k(64)) return 32;
    return 64;
}

static bool use_tc(const vie_head *head, int32_t batch, int32_t k) {
    const bool q8 = head->scale != nullptr;
    return head->tc_ready && batch >= (q8 ? opt(VIE_OPT_TC_MIN_BATCH_E4M3) : opt(VIE_OPT_TC_MIN_BATCH)) &&
           k <= vie::tc_max_k(32, q8) && head->d_pad >= (q8 ? 128 : 64);
}

// Bytes of the query operand each CTA of a group of nqt slots builds itself
// (0: a prep kernel writes it).
static int tc_hres(const vie_head *head, int nqt) {
    const bool q8 = head->scale != nullptr;
    const int n_kb = (head->d_pad + (q8 ? 127 : 63)) / (q8 ? 128 : 64);
    return vie::tc_hres_bytes(nqt, q8, n_kb);
}

static vie_topk_plan make_plan(const vie_head *head, int32_t batch, int32_t k) {
    vie_topk_plan pl;
    if (use_tc(head, batch, k)) {
        const int nqt = tc_group(batch, k, head->scale != nullptr);
        pl.path = 1;
        pl.groups = (batch + nqt - 1) / nqt;
        // per group: the query prep (unless the CTAs build the operand), then
        // projection, per-CTA top-k and merge in one launch
        pl.launches = (tc_hres(head, nqt) > 0 ? 1 : 2) * pl.groups;
    } else {
        const int cap = nb_cap_for(head->d_pad, k);
        pl.path = 0;
        pl.groups = (batch + cap - 1) / cap;
        pl.launches = pl.groups;
    }
    return pl;
}

// Batches on the tensor cores: per group of up to 32 queries, the hi/lo
// query matrix, then the tcgen05 projection with per-CTA top-k and the merge.
static vie_status run_topk_tc(const char *fn, vie_head *head, const float *h, int32_t batch,
                              int32_t k, int32_t *out_idx, float *out_logits, float *sparse,
                              cudaStream_t s) {
    const bool q8 = head->scale != nullptr;
    const int nqt = tc_group(batch, k, q8);
    // K-blocks per stage: the most that still leave a ring of two stages
    // (larger stages beat deeper rings of small ones); the query boxes stay
    // resident in shared memory when they are small (e4m3 rows)
    int stages = 0, kps = 0, slots = 0;
    uint32_t smem = 0;
    int kps_max = opt(VIE_OPT_TC_KPS);
    kps_max = kps_max > vie::kTcMaxKPS ? vie::kTcMaxKPS : kps_max;
    const int hres_bytes = tc_hres(head, nqt);
    for (int c = kps_max; c >= 1 && kps == 0; --c) {
        if (vie::tc_shape(nqt, q8, c, hres_bytes, &stages, &slots, &smem)) kps = c;
    }
    if (kps == 0) return fail(VIE_ERR_UNSUPPORTED, "%s: no tensor-core layout", fn);
    const int tile_rows = vie::tc_tile_rows(nqt, q8);
    const int n_tiles = static_cast<int>((head->V + tile_rows - 1) / tile_rows);
    const int pct = opt(VIE_OPT_STATIC_PCT);
    const int n_h = (q8 ? vie::kQ8Pieces : 2) * nqt;  // query rows: boxes of 16 / 32 / 64 / 128
    const CUtensorMap &mapH = head->mapH[n_h == 16 ? 0 : (n_h == 32 ? 1 : (n_h == 64 ? 2 : 3))];
    for (int q0 = 0; q0 < batch; q0 += nqt) {
        const int nq = batch - q0 < nqt ? batch - q0 : nqt;
        const float *hq = h + static_cast<int64_t>(q0) * head->d;
        cudaError_t e = cudaSuccess;
        if (hres_bytes == 0)
            e = q8 ? vie::launch_prep_queries_e4m3(hq, nq, nqt, head->d, head->d_pad, head->hB, head->qscale, s)
                   : vie::launch_prep_queries(hq, nq, head->d, head->d_pad, 2 * nqt, head->hB, head->num_sms, s);
        if (e != cudaSuccess) return fail_cuda(e, fn);
        vie::TcParams p;
        p.V = head->V;
        p.d_pad = head->d_pad;
        p.k = k;
        p.nq = nq;
        p.stages = stages;
        p.kb_per_stage = kps;
        p.score_slots = slots;
        p.static_tiles = static_cast<int32_t>(static_cast<int64_t>(n_tiles) * pct / 100 / head->G);
        p.cand = head->cand;  // [NQ][G][k] keys (NQ * k <= kTcListKeys), then the heads
        p.heads = head->cand + static_cast<size_t>(vie::kTcListKeys) * head->G;
        p.ticket = head->words;
        p.next_tile = head->words + 2;
        p.err = head->words + 1;
        p.epoch = head->words + kEpochWord;
        p.flags = head->words + kFlagWords;
        p.out_idx = out_idx + static_cast<int64_t>(q0) * k;
        p.out_logits = out_logits + static_cast<int64_t>(q0) * k;
        p.sparse = sparse != nullptr ? sparse + static_cast<int64_t>(q0) * head->V : nullptr;
        p.row_scale = head->scale;
        p.qscale = head->qscale;
        p.h_resident = hres_bytes > 0 ? 1 : 0;
        p.h = hq;
        p.d = head->d;
        e = vie::launch_tc_topk(nqt, q8, head->mapW, mapH, p, head->G, smem, s);
        if (e != cudaSuccess) return fail_cuda(e, fn);
    }
    return VIE_OK;
}

static vie_status run_topk(const char *fn, vie_head *head, const float *h, int32_t batch,
                           int32_t k, int32_t *out_idx, float *out_logits, float *sparse,
                           vie_stream stream) {
    if (head == nullptr) return fail(VIE_ERR_INVALID_ARG, "%s: head is NULL", fn);
    if (h == nullptr || out_idx == nullptr || out_logits == nullptr)
        return fail(VIE_ERR_INVALID_ARG, "%s: NULL buffer", fn);
    if (batch < 1 || batch > VIE_BATCH_MAX)
        return fail(VIE_ERR_INVALID_ARG, "%s: batch=%d outside [1, %d]", fn, batch, VIE_BATCH_MAX);
    if (k < 1 || k > VIE_K_MAX || static_cast<int64_t>(k) > head->V)
        return fail(VIE_ERR_INVALID_ARG, "%s: k=%d outside [1, min(V=%lld, %d)]", fn, k,
                    static_cast<long long>(head->V), VIE_K_MAX);
    if ((reinterpret_cast<uintptr_t>(h) | reinterpret_cast<uintptr_t>(out_idx) |
         reinterpret_cast<uintptr_t>(out_logits) | reinterpret_cast<uintptr_t>(sparse)) & 3u)
        return fail(VIE_ERR_INVALID_ARG, "%s: buffers must be 4-byte aligned", fn);
    vie_status st = check_device(head);
    if (st != VIE_OK) return st;

    const int mm = pick_mm(k);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (use_tc(head, batch, k)) return run_topk_tc(fn, head, h, batch, k, out_idx, out_logits, sparse, s);
    const int cap = nb_cap_for(head->d_pad, k);
    for (int q0 = 0; q0 < batch; q0 += cap) {
        const int nq = batch - q0 < cap ? batch - q0 : cap;
        int nb = 1;
        while (nb < nq) nb <<= 1;
        LaunchShape shp;
        if (!pick_shape(nb, head->d_pad, head->d_pad * (head->scale != nullptr ? 1 : 2), sel_cap_launch(nb, k),
                        &shp))
            return fail(VIE_ERR_UNSUPPORTED, "%s: no shared-memory layout for d=%d", fn, head->d);
        vie::StreamTopkParams p;
        p.W = head->W;
        p.row_scale = head->scale;
        p.h = h + static_cast<int64_t>(q0) * head->d;
        p.nq = nq;
        p.V = head->V;
        p.d = head->d;
        p.d_pad = head->d_pad;
        p.k = k;
        p.rows_per_stage = shp.rs;
        p.stages = shp.stages;
        const int64_t n_chunks = (head->V + shp.rs - 1) / shp.rs;
        const int pct = opt(VIE_OPT_STATIC_PCT);
        p.static_chunks = static_cast<int32_t>(n_chunks * pct / 100 / head->G);
        p.pool_rows = pool_rows_for(shp.rs);
        p.half_rows = half_rows_for(shp.r, head->d_pad / (head->scale != nullptr ? 16 : 8));
        p.sel_cap = sel_cap_launch(nb, k);
        p.cand = head->cand;
        p.heads = head->cand + static_cast<size_t>(kMaxNB) * head->G * VIE_K_MAX;
        p.ticket = head->words;
        p.err = head->words + 1;
        p.next_chunk = head->words + 2;
        // one query, k <= 64: CTA 0 merges the lists as they arrive (its
        // merge buffers and every list's first keys in the ring's shared memory)
        const vie::SmemLayout L(nb, head->d_pad, shp.rs, shp.stages,
                                head->d_pad * (head->scale != nullptr ? 1 : 2), p.sel_cap);
        const uint32_t early_bytes = vie::SmemLayout::merge_fixed_bytes() + 8u * vie::kFastE * head->G +
                                     4u * ((head->G + 7) & ~7);
        p.early = (opt(VIE_OPT_EARLY_MERGE) != 0 && nq == 1 && k <= vie::kFastMaxK && head->G >= 2 &&
                   2 * head->G <= vie::kThreads && L.total - L.merge >= early_bytes) ? 1 : 0;
        // several queries: the first CTAs to finish merge them in parallel
        p.pmerge = (nq > 1 && head->G <= vie::kThreads && L.total - L.merge >= early_bytes) ? 1 : 0;
        p.epoch = head->words + kEpochWord;
        p.flags = head->words + kFlagWords;
        p.out_idx = out_idx + static_cast<int64_t>(q0) * k;
        p.out_logits = out_logits + static_cast<int64_t>(q0) * k;
        p.sparse = sparse != nullptr ? sparse + static_cast<int64_t>(q0) * head->V : nullptr;
        const cudaError_t e = vie::launch_stream_topk(nb, mm, shp.r, p, head->G, shp.smem, s);
        if (e != cudaSuccess) return fail_cuda(e, fn);
    }
    return VIE_OK;
}

vie_status vie_head_plan(const vie_head *head, int32_t batch, int32_t k, vie_topk_plan *plan) {
    if (head == nullptr || plan == nullptr)
        return fail(VIE_ERR_INVALID_ARG, "vie_head_plan: NULL argument");
    if (batch < 1 || batch > VIE_BATCH_MAX)
        return fail(VIE_ERR_INVALID_ARG, "vie_head_plan: batch=%d outside [1, %d]", batch,
                    VIE_BATCH_MAX);
    if (k < 1 || k > VIE_K_MAX || static_cast<int64_t>(k) > head->V)
        return fail(VIE_ERR_INVALID_ARG, "vie_head_plan: k=%d outside [1, min(V=%lld, %d)]", k,
                    static_cast<long long>(head->V), VIE_K_MAX);
    *plan = make_plan(head, batch, k);
    return VIE_OK;
}

vie_status vie_head_topk(vie_head *head, const float *h, int32_t batch, int32_t k,
                         int32_t *out_idx, float *out_logits, vie_stream stream) {
    return run_topk("vie_head_topk", head, h, batch, k, out_idx, out_logits, nullptr, stream);
}

vie_status vie_head_topk_many(vie_head *head, const float *h, int64_t n, int32_t k,
                              int32_t *out_idx, float *out_logits, vie_stream stream) {
    const char *fn = "vie_head_topk_many";
    if (n < 1 || n > VIE_MANY_MAX)
        return fail(VIE_ERR_INVALID_ARG, "%s: n=%lld outside [1, %d]", fn, static_cast<long long>(n),
                    VIE_MANY_MAX);
    if (head == nullptr) return fail(VIE_ERR_INVALID_ARG, "%s: head is NULL", fn);
    for (int64_t q0 = 0; q0 < n; q0 += VIE_BATCH_MAX) {
        const int32_t b = static_cast<int32_t>(n - q0 < VIE_BATCH_MAX ? n - q0 : VIE_BATCH_MAX);
        const vie_status st =
            run_topk(fn, head, h == nullptr ? nullptr : h + q0 * head->d, b, k,
                     out_idx == nullptr ? nullptr : out_idx + q0 * k,
                     out_logits == nullptr ? nullptr : out_logits + q0 * k, nullptr, stream);
        if (st != VIE_OK) return st;
    }
    return VIE_OK;
}

vie_status vie_head_topk_sparse(vie_head *head, const float *h, int32_t batch, int32_t k,
                                int32_t *out_idx, float *out_logits, float *out_sparse,
                                vie_stream stream) {
    if (out_sparse == nullptr)
        return fail(VIE_ERR_INVALID_ARG, "vie_head_topk_sparse: out_sparse is NULL");
    return run_topk("vie_head_topk_sparse", head, h, batch, k, out_idx, out_logits, out_sparse,
                    stream);
}

vie_status vie_sample_topk(const int32_t *idx, const float *logits, int32_t batch, int32_t k,
                           float temperature, float top_p, float min_p, uint64_t seed,
                           uint64_t step, int32_t *out_token, float *out_prob, vie_stream stream) {
    const char *fn = "vie_sample_topk";
    if (idx == nullptr || logits == nullptr || out_token == nullptr || out_prob == nullptr)
        return fail(VIE_ERR_INVALID_ARG, "%s: NULL buffer", fn);
    if (batch < 1) return fail(VIE_ERR_INVALID_ARG, "%s: batch=%d < 1", fn, batch);
    if (k < 1 || k > VIE_K_MAX)
        return fail(VIE_ERR_INVALID_ARG, "%s: k=%d outside [1, %d]", fn, k, VIE_K_MAX);
    if (!(temperature > 0.0f) || !std::isfinite(temperature))
        return fail(VIE_ERR_INVALID_ARG, "%s: temperature=%g must be positive and finite", fn,
                    static_cast<double>(temperature));
    if (!(top_p > 0.0f && top_p <= 1.0f))
        return fail(VIE_ERR_INVALID_ARG, "%s: top_p=%g outside (0, 1]", fn, static_cast<double>(top_p));
    if (!(min_p >= 0.0f && min_p <= 1.0f))
        return fail(VIE_ERR_INVALID_ARG, "%s: min_p=%g outside [0, 1]", fn, static_cast<double>(min_p));
    if ((reinterpret_cast<uintptr_t>(idx) | reinterpret_cast<uintptr_t>(logits) |
         reinterpret_cast<uintptr_t>(out_token) | reinterpret_cast<uintptr_t>(out_prob)) & 3u)
        return fail(VIE_ERR_INVALID_ARG, "%s: buffers must be 4-byte aligned", fn);
    const cudaError_t e = vie::launch_sample_topk(idx, logits, batch, k, temperature, top_p, min_p,
                                                  seed, step, out_token, out_prob,
                                                  static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return fail_cuda(e, fn);
    return VIE_OK;
}

vie_status vie_recall_hits(const int32_t *exact, int32_t k, const int32_t *approx, int32_t m,
                           int64_t n, int32_t *out_hits, vie_stream stream) {
    const char *fn = "vie_recall_hits";
    if (exact == nullptr || approx == nullptr || out_hits == nullptr)
        return fail(VIE_ERR_INVALID_ARG, "%s: NULL buffer", fn);
    if (n < 1 || n > VIE_RECALL_N_MAX)
        return fail(VIE_ERR_INVALID_ARG, "%s: n=%lld outside [1, %d]", fn, static_cast<long long>(n),
                    VIE_RECALL_N_MAX);
    if (k < 1 || k > VIE_K_MAX)
        return fail(VIE_ERR_INVALID_ARG, "%s: k=%d outside [1, %d]", fn, k, VIE_K_MAX);
    if (m < 1 || m > VIE_RECALL_M_MAX)
        return fail(VIE_ERR_INVALID_ARG, "%s: m=%d outside [1, %d]", fn, m, VIE_RECALL_M_MAX);
    if ((reinterpret_cast<uintptr_t>(exact) | reinterpret_cast<uintptr_t>(approx) |
         reinterpret_cast<uintptr_t>(out_hits)) & 3u)
        return fail(VIE_ERR_INVALID_ARG, "%s: buffers must be 4-byte aligned", fn);
    const cudaError_t e = vie::launch_recall_hits(exact, k, approx, m, n, out_hits,
                                                  static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return fail_cuda(e, fn);
    return VIE_OK;
}

vie_status vie_head_topk_sample(vie_head *head, const float *h, int32_t batch, int32_t k,
                                float temperature, float top_p, float min_p, uint64_t seed,
                                uint64_t step, int32_t *out_idx, float *out_logits,
                                float *out_sparse, int32_t *out_token, float *out_prob,
                                vie_stream stream) {
    const char *fn = "vie_head_topk_sample";
    if (out_token == nullptr || out_prob == nullptr)
        return fail(VIE_ERR_INVALID_ARG, "%s: NULL buffer", fn);
    if (!(temperature > 0.0f) || !std::isfinite(temperature) || !(top_p > 0.0f && top_p <= 1.0f) ||
        !(min_p >= 0.0f && min_p <= 1.0f))
        return fail(VIE_ERR_INVALID_ARG, "%s: temperature=%g top_p=%g min_p=%g out of range", fn,
                    static_cast<double>(temperature), static_cast<double>(top_p),
                    static_cast<double>(min_p));
    vie_status st = run_topk(fn, head, h, batch, k, out_idx, out_logits, out_sparse, stream);
    if (st != VIE_OK) return st;
    return vie_sample_topk(out_idx, out_logits, batch, k, temperature, top_p, min_p, seed, step,
                           out_token, out_prob, stream);
}

// The device address of pinned (page-locked, mapped) host memory, or nullptr
// for memory the device cannot address directly.
static void *mapped_view(const void *host_ptr) {
    cudaPointerAttributes a;
    if (cudaPointerGetAttributes(&a, host_ptr) != cudaSuccess) {
        cudaGetLastError();
        return nullptr;
    }
    return a.type == cudaMemoryTypeHost ? a.devicePointer : nullptr;
}

vie_status vie_head_topk_host(vie_head *head, const float *h_host, int32_t batch, int32_t k,
                              int32_t *idx_host, float *logits_host, float *out_sparse,
                              vie_stream stream) {
    const char *fn = "vie_head_topk_host";
    if (head == nullptr) return fail(VIE_ERR_INVALID_ARG, "%s: head is NULL", fn);
    if (h_host == nullptr || idx_host == nullptr || logits_host == nullptr)
        return fail(VIE_ERR_INVALID_ARG, "%s: NULL buffer", fn);
    if (batch < 1 || batch > VIE_BATCH_MAX)
        return fail(VIE_ERR_INVALID_ARG, "%s: batch=%d outside [1, %d]", fn, batch, VIE_BATCH_MAX);
    if (k < 1 || k > VIE_K_MAX || static_cast<int64_t>(k) > head->V)
        return fail(VIE_ERR_INVALID_ARG, "%s: k=%d outside [1, min(V=%lld, %d)]", fn, k,
                    static_cast<long long>(head->V), VIE_K_MAX);
    vie_status st = check_device(head);
    if (st != VIE_OK) return st;
    const size_t nh = static_cast<size_t>(batch) * head->d, no = static_cast<size_t>(batch) * k;
    // pinned buffers are used in place: the kernels read the queries from
    // host memory (measured faster than a copy in first) and the merging CTA
    // writes the top-k there (no copies back); VIE_OPT_HOST_H_DIRECT = 0
    // copies pinned queries in all the same
    int32_t *idx_dev = static_cast<int32_t *>(mapped_view(idx_host));
    float *logits_dev = static_cast<float *>(mapped_view(logits_host));
    const bool out_direct = idx_dev != nullptr && logits_dev != nullptr;
    const float *h_dev = opt(VIE_OPT_HOST_H_DIRECT) != 0 ? static_cast<const float *>(mapped_view(h_host)) : nullptr;
    if (h_dev == nullptr && head->stage_h_elems < nh) {
        cudaFree(head->stage_h);
        head->stage_h = nullptr;
        head->stage_h_elems = 0;
        if (cudaMalloc(&head->stage_h, nh * sizeof(float)) != cudaSuccess) {
            cudaGetLastError();
            return fail(VIE_ERR_OOM, "%s: cannot allocate %zu bytes of query staging", fn,
                        nh * sizeof(float));
        }
        head->stage_h_elems = nh;
    }
    if (!out_direct && head->stage_out_elems < no) {
        cudaFree(head->stage_idx);
        cudaFree(head->stage_logits);
        head->stage_idx = nullptr;
        head->stage_logits = nullptr;
        head->stage_out_elems = 0;
        if (cudaMalloc(&head->stage_idx, no * sizeof(int32_t)) != cudaSuccess ||
            cudaMalloc(&head->stage_logits, no * sizeof(float)) != cudaSuccess) {
            cudaGetLastError();
            return fail(VIE_ERR_OOM, "%s: cannot allocate %zu bytes of output staging", fn,
                        no * 8);
        }
        head->stage_out_elems = no;
    }
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = cudaSuccess;
    if (h_dev == nullptr) {
        e = cudaMemcpyAsync(head->stage_h, h_host, nh * sizeof(float), cudaMemcpyHostToDevice, s);
        if (e != cudaSuccess) return fail_cuda(e, "vie_head_topk_host: copy of h");
    }
    st = run_topk(fn, head, h_dev != nullptr ? h_dev : head->stage_h, batch, k,
                  out_direct ? idx_dev : head->stage_idx, out_direct ? logits_dev : head->stage_logits,
                  out_sparse, stream);
    if (st != VIE_OK) return st;
    if (!out_direct) {
        e = cudaMemcpyAsync(idx_host, head->stage_idx, no * sizeof(int32_t), cudaMemcpyDeviceToHost, s);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(logits_host, head->stage_logits, no * sizeof(float), cudaMemcpyDeviceToHost, s);
    }
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return fail_cuda(e, "vie_head_topk_host: copy of the top-k");
    return VIE_OK;
}

vie_status vie_scatter_sparse_logits(const int32_t *idx, const float *logits, int32_t batch,
                                     int32_t k, int64_t V, float *out, vie_stream stream) {
    if (idx == nullptr || logits == nullptr || out == nullptr)
        return fail(VIE_ERR_INVALID_ARG, "vie_scatter_sparse_logits: NULL buffer");
    if (batch < 1 || k < 1 || V < 1)
        return fail(VIE_ERR_INVALID_ARG, "vie_scatter_sparse_logits: batch=%d k=%d V=%lld", batch,
                    k, static_cast<long long>(V));
    if (V > INT64_MAX / batch)
        return fail(VIE_ERR_INVALID_ARG, "vie_scatter_sparse_logits: batch*V overflows");
    if ((reinterpret_cast<uintptr_t>(idx) | reinterpret_cast<uintptr_t>(logits) |
         reinterpret_cast<uintptr_t>(out)) & 3u)
        return fail(VIE_ERR_INVALID_ARG, "vie_scatter_sparse_logits: buffers must be 4-byte aligned");
    uint32_t *err = nullptr;
    cudaError_t e = cudaGetSymbolAddress(reinterpret_cast<void **>(&err), g_dev_err);
    if (e != cudaSuccess) return fail_cuda(e, "cudaGetSymbolAddress");
    // ~16 KB of output per CTA, at most 1024 CTAs per row
    int64_t per = 4096;
    int64_t bx = (V + per - 1) / per;
    if (bx > 1024) {
        bx = 1024;
        per = (V + bx - 1) / bx;
        per = (per + 3) & ~static_cast<int64_t>(3);
    }
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    for (int b0 = 0; b0 < batch; b0 += 65535) {
        const int by = batch - b0 < 65535 ? batch - b0 : 65535;
        scatter_sparse_kernel<<<dim3(static_cast<unsigned>(bx), by), 256, 0, s>>>(
            idx, logits, k, V, per, out, b0, err);
        e = cudaGetLastError();
        if (e != cudaSuccess) return fail_cuda(e, "vie_scatter_sparse_logits launch");
    }
    return VIE_OK;
}

vie_status vie_device_status(vie_stream stream) {
    cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return fail_cuda(e, "vie_device_status: stream synchronize");
    uint32_t w = 0;
    e = cudaMemcpyFromSymbol(&w, g_dev_err, sizeof w);
    if (e != cudaSuccess) return fail_cuda(e, "vie_device_status: read flag");
    if (w == 0) return VIE_OK;
    const uint32_t zero = 0;
    e = cudaMemcpyToSymbol(g_dev_err, &zero, sizeof zero);
    if (e != cudaSuccess) return fail_cuda(e, "vie_device_status: clear flag");
    return fail(VIE_ERR_DEVICE, "device flag 0x%x:%s%s", w,
                (w & vie::kErrScatterIndex) ? " scatter index outside [0, V)" : "",
                (w & vie::kErrWaitTimeout) ? " pipeline wait timed out" : "");
}

vie_status vie_head_device_status(vie_head *head, vie_stream stream) {
    if (head == nullptr) return fail(VIE_ERR_INVALID_ARG, "vie_head_device_status: head is NULL");
    vie_status st = check_device(head);
    if (st != VIE_OK) return st;
    st = vie_device_status(stream);
    uint32_t words[2] = {0, 0};
    cudaError_t e = cudaMemcpy(words, head->words, sizeof words, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return fail_cuda(e, "vie_head_device_status: read flag");
    if (words[1] != 0) {
        e = cudaMemset(head->words, 0, 4 * sizeof(uint32_t));
        if (e != cudaSuccess) return fail_cuda(e, "vie_head_device_status: clear flag");
        return fail(VIE_ERR_DEVICE, "handle device flag 0x%x:%s%s", words[1],
                    (words[1] & vie::kErrWaitTimeout) ? " pipeline wait timed out" : "",
                    (words[1] & vie::kErrScatterIndex) ? " scatter index outside [0, V)" : "");
    }
    return st;
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Top-k without any device allocation: the same kernel as vie_head_topk, with
// its scratch (ticket and pool counters, per-CTA candidate lists) placed in a
// fixed array that lives in this module instead of memory from cudaMalloc.
namespace {

constexpr size_t kNoAllocScratchBytes = size_t(1) << 20;  // 1 MiB per device
constexpr size_t kNoAllocCounterBytes = 256;              // counters, then the lists

// Host code sees only a stand-in for this array; kernels get its device
// address, looked up once per device below.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

struct NoAllocDevice {
    std::once_flag once;
    cudaError_t setup_error = cudaSuccess;
    unsigned char *scratch = nullptr;  // device address of g_noalloc_scratch
    uint32_t *flag = nullptr;          // device address of g_dev_err
    int sms = 0;
};
NoAllocDevice g_noalloc[64];

}  // namespace

extern "C" vie_status vie_head_topk_noalloc(const void *W_out, int64_t V, int32_t d, const float *h,
                                           int32_t batch, int32_t k, int32_t *out_idx,
                                           float *out_logits, vie_stream stream) {
    const char *fn = "vie_head_topk_noalloc";
    if (W_out == nullptr || h == nullptr || out_idx == nullptr || out_logits == nullptr)
        return fail(VIE_ERR_INVALID_ARG, "%s: NULL buffer", fn);
    if (V < 1 || V > static_cast<int64_t>(INT32_MAX) - 1)
        return fail(VIE_ERR_INVALID_ARG, "%s: V=%lld outside [1, 2^31-2]", fn,
                    static_cast<long long>(V));
    if (d < 8 || d > VIE_D_MAX || (d & 7) != 0)
        return fail(VIE_ERR_INVALID_ARG, "%s: d=%d must be a multiple of 8 in [8, %d]", fn, d,
                    VIE_D_MAX);
    if (reinterpret_cast<uintptr_t>(W_out) & 15u)
        return fail(VIE_ERR_INVALID_ARG, "%s: W_out must be 16-byte aligned", fn);
    if (batch < 1 || batch > VIE_BATCH_MAX)
        return fail(VIE_ERR_INVALID_ARG, "%s: batch=%d outside [1, %d]", fn, batch, VIE_BATCH_MAX);
    if (k < 1 || k > VIE_K_MAX || static_cast<int64_t>(k) > V)
        return fail(VIE_ERR_INVALID_ARG, "%s: k=%d outside [1, min(V, %d)]", fn, k, VIE_K_MAX);
    if ((reinterpret_cast<uintptr_t>(h) | reinterpret_cast<uintptr_t>(out_idx) |
         reinterpret_cast<uintptr_t>(out_logits)) & 3u)
        return fail(VIE_ERR_INVALID_ARG, "%s: buffers must be 4-byte aligned", fn);

    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return fail_cuda(e, "cudaGetDevice");
    if (dev < 0 || dev >= 64) return fail(VIE_ERR_UNSUPPORTED, "%s: device %d", fn, dev);
    // the weights are streamed by bulk copies: device (or managed) memory of
    // this device only (the query may be page-locked host memory)
    cudaPointerAttributes pa;
    e = cudaPointerGetAttributes(&pa, W_out);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return fail(VIE_ERR_INVALID_ARG, "%s: W_out is not a CUDA pointer", fn);
    }
    if ((pa.type != cudaMemoryTypeDevice && pa.type != cudaMemoryTypeManaged) || pa.device != dev)
        return fail(VIE_ERR_INVALID_ARG, "%s: W_out must be device memory of the current device %d", fn,
                    dev);
    NoAllocDevice &nd = g_noalloc[dev];
    std::call_once(nd.once, [&nd, dev]() {
        nd.setup_error = cudaGetSymbolAddress(reinterpret_cast<void **>(&nd.scratch), g_noalloc_scratch);
        if (nd.setup_error == cudaSuccess)
            nd.setup_error = cudaGetSymbolAddress(reinterpret_cast<void **>(&nd.flag), g_dev_err);
        if (nd.setup_error == cudaSuccess)
            nd.setup_error = cudaDeviceGetAttribute(&nd.sms, cudaDevAttrMultiProcessorCount, dev);
    });
    if (nd.setup_error != cudaSuccess) return fail_cuda(nd.setup_error, "vie_head_topk_noalloc set-up");

    int64_t g = (V + 63) / 64;
    if (g > nd.sms) g = nd.sms;
    if (g > vie::kMaxLists) g = vie::kMaxLists;
    const int G = static_cast<int>(g < 1 ? 1 : g);
    const int mm = pick_mm(k);
    const int cap = nb_cap_for(d, k);
    int nb_max = 1;
    while (nb_max < cap && nb_max < batch) nb_max <<= 1;
    // lists [nb_max][G][k], then the heads [nb_max][G][kFastE], which the
    // merge reads 16 bytes at a time: the list area is rounded up to an even
    // number of keys so the heads start on a 16-byte boundary
    const size_t list_keys = (static_cast<size_t>(nb_max) * G * k + 1) & ~static_cast<size_t>(1);
    const size_t lists_bytes =
        (list_keys + static_cast<size_t>(nb_max) * G * vie::kFastE) * sizeof(uint64_t);
    if (lists_bytes > kNoAllocScratchBytes - kNoAllocCounterBytes)
        return fail(VIE_ERR_UNSUPPORTED,
                    "%s: needs %zu bytes of scratch (%d query slots x %d CTAs x (k=%d + %d) x 8, "
                    "lists rounded to 16 bytes), more than the fixed %zu; use vie_head_topk or a "
                    "smaller batch or k",
                    fn, lists_bytes, nb_max, G, k, vie::kFastE,
                    kNoAllocScratchBytes - kNoAllocCounterBytes);
    uint64_t *cand = reinterpret_cast<uint64_t *>(nd.scratch + kNoAllocCounterBytes);
    uint64_t *heads = cand + list_keys;
    if ((reinterpret_cast<uintptr_t>(cand) | reinterpret_cast<uintptr_t>(heads)) & 15u)
        return fail(VIE_ERR_UNSUPPORTED, "%s: scratch lists not 16-byte aligned", fn);

    cudaStream_t s = static_cast<cudaStream_t>(stream);
    uint32_t *counters = reinterpret_cast<uint32_t *>(nd.scratch);
    e = cudaMemsetAsync(counters, 0, 4 * sizeof(uint32_t), s);  // ticket and pool start at 0
    if (e != cudaSuccess) return fail_cuda(e, "vie_head_topk_noalloc clear");
    for (int q0 = 0; q0 < batch; q0 += cap) {
        const int nq = batch - q0 < cap ? batch - q0 : cap;
        int nb = 1;
        while (nb < nq) nb <<= 1;
        LaunchShape shp;
        if (!pick_shape(nb, d, d * 2, sel_cap_launch(nb, k), &shp))
            return fail(VIE_ERR_UNSUPPORTED, "%s: no shared-memory layout for d=%d", fn, d);
        vie::StreamTopkParams p;
        p.W = static_cast<const uint16_t *>(W_out);
        p.row_scale = nullptr;
        p.h = h + static_cast<int64_t>(q0) * d;
        p.nq = nq;
        p.V = V;
        p.d = d;
        p.d_pad = d;
        p.k = k;
        p.rows_per_stage = shp.rs;
        p.stages = shp.stages;
        const int64_t n_chunks = (V + shp.rs - 1) / shp.rs;
        const int pct = opt(VIE_OPT_STATIC_PCT);
        p.static_chunks = static_cast<int32_t>(n_chunks * pct / 100 / G);
        p.pool_rows = pool_rows_for(shp.rs);
        p.half_rows = half_rows_for(shp.r, d / 8);
        p.sel_cap = sel_cap_launch(nb, k);
        p.cand = cand;
        p.heads = heads;
        p.ticket = counters;
        p.next_chunk = counters + 2;
        p.err = nd.flag;
        p.early = 0;  // the last-ticket merge: no per-CTA words in the fixed array
        p.pmerge = 0;
        p.epoch = nullptr;
        p.flags = nullptr;
        p.out_idx = out_idx + static_cast<int64_t>(q0) * k;
        p.out_logits = out_logits + static_cast<int64_t>(q0) * k;
        p.sparse = nullptr;
        e = vie::launch_stream_topk(nb, mm, shp.r, p, G, shp.smem, s);
        if (e != cudaSuccess) return fail_cuda(e, fn);
    }
    return VIE_OK;
}

namespace vie {
cudaError_t launch_stream_topk(int nb, int mm, int r, const StreamTopkParams &p, int grid,
                               uint32_t smem, cudaStream_t stream) {
    if (p.row_scale != nullptr) {
        switch (nb) {
            case 1: return launch_stream_topk_e4m3_nb1(mm, r, p, grid, smem, stream);
            case 2: return launch_stream_topk_e4m3_nb2(mm, r, p, grid, smem, stream);
            case 4: return launch_stream_topk_e4m3_nb4(mm, r, p, grid, smem, stream);
            case 8: return launch_stream_topk_e4m3_nb8(mm, r, p, grid, smem, stream);
            default: return cudaErrorInvalidValue;
        }
    }
    switch (nb) {
        case 1: return launch_stream_topk_nb1(mm, r, p, grid, smem, stream);
        case 2: return launch_stream_topk_nb2(mm, r, p, grid, smem, stream);
        case 4: return launch_stream_topk_nb4(mm, r, p, grid, smem, stream);
        case 8: return launch_stream_topk_nb8(mm, r, p, grid, smem, stream);
        default: return cudaErrorInvalidValue;
    }
}
}  // namespace vie
