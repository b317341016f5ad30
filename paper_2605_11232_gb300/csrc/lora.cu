// lora.cu -- segmented multi-adapter LoRA projection on the tensor cores.
//
// One base model serves several LoRA adapters, and a mixed request runs as
// per-adapter batches (Sec. 5.6, the adapter-first dispatch of
// pkv_lora_dispatch).  For the tokens t of a segment with adapter a:
//     y_t = W x_t + s_a B_a (A_a x_t)      (a = -1: y_t = W x_t)
// One CTA computes a 128-row x 256-column tile of y for one segment:
//   - a TMA producer thread streams 64-wide K chunks of the token rows X, of
//     W's 256 output rows and of A_a's rank rows into a 4-stage ring
//     (128-byte swizzle);
//   - one MMA thread issues Y += X.W^T (N = 256) and U += X.A_a^T (N = rank)
//     into tensor memory for each chunk;
//   - after the last chunk the 128 threads (thread = row) scale U by s_a,
//     round it to bf16 and stage it in shared memory beside B_a's 256 rows
//     (held in registers since the start; both go where the ring's first
//     stage was), and the MMA thread adds Y += U.B_a^T (K = rank, padded to
//     64 with zeros);
//   - the epilogue rounds Y to bf16 and stores the segment's rows.
// The low-rank update rides on the base GEMM's tile: x is read once for
// both products and the delta never leaves the SM.
#include "../../include/pkv.h"

#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <cstdarg>
#include <cstdio>

#include "pkv_device.cuh"
#include "pkv_internal.h"
#include "tc_ptx.cuh"

namespace pkv {
namespace {

using namespace tc;

constexpr int kThreads = 128;
constexpr int kBM = 128, kBN = 256, kBK = 64, kStages = 4;
constexpr int kMaxRank = 64;
constexpr uint64_t kWaitLimitNs = 2000000000ull;
constexpr uint64_t kDrainLimitNs = 200000000ull;
// shared memory: stages of [X 128 x 64 | W 256 x 64 | A 64 x 64], all bf16
// K-major, 128-byte swizzle.  Once every MMA of the main loop is done, U
// (128 x 64) takes stage 0's X part and B_a's tile (256 x 64) its W part.
// Four stages against three with U and B_a in their own space (the ring's
// bytes in flight then cover about 1.3 us of MMA work instead of 1 us):
// Case C1 595 -> 541 us, a 64-prompt request 2.94 -> 2.70 ms.
constexpr int kXBytes = kBM * kBK * 2, kWBytes = kBN * kBK * 2, kABytes = kMaxRank * kBK * 2;
constexpr int kStageBytes = kXBytes + kWBytes + kABytes;
constexpr int kUOff = 0;
constexpr int kBtOff = kXBytes;
static_assert(kBM * kBK * 2 <= kXBytes && kBN * kBK * 2 <= kWBytes, "U and B_a fit stage 0");
constexpr int kBarOff = kStages * kStageBytes;   // full[kStages] empty[kStages] done1 done2
constexpr int kSmemBytes = kBarOff + 8 * (2 * kStages + 2) + 16 + 1024;
static_assert(kSmemBytes <= 227 * 1024, "shared memory of the LoRA tile");

struct Tile {
    int32_t row0, rows, adapter;
    float scale;
};
struct TileList {
    int32_t n, pad[3];
    Tile t[PKV_LORA_MAX_TILES];
};

__device__ __forceinline__ uint32_t sw128(int row, int chunk) {
    return (uint32_t)(row * 128 + (((chunk & 7) ^ (row & 7)) << 4));
}

__global__ void __launch_bounds__(kThreads, 1)
    lora_tile_kernel(const __grid_constant__ CUtensorMap tmx, const __grid_constant__ CUtensorMap tmw,
                     const __grid_constant__ CUtensorMap tma, const uint16_t *__restrict__ lora_b,
                     uint16_t *__restrict__ y, int32_t d_in, int32_t d_out, int32_t rank, int *err,
                     const __grid_constant__ TileList tiles) {
    pdl_wait();
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                ~uintptr_t(1023));
    const uint32_t sb = smem_u32(smem);
    __shared__ uint32_t tmem_slot;
    __shared__ int abort_flag;
    const int warp = threadIdx.x >> 5, t = threadIdx.x;
    const Tile tile = tiles.t[blockIdx.y];
    const int n0 = blockIdx.x * kBN;
    const bool lora = tile.adapter >= 0;
    const int nk = d_in / kBK;
    const uint32_t bar_full = sb + kBarOff, bar_empty = bar_full + 8 * kStages,
                   bar_done1 = bar_full + 16 * kStages, bar_done2 = bar_done1 + 8;
    if (t == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(bar_full + 8 * s, 1);
            mbar_init(bar_empty + 8 * s, 1);
        }
        mbar_init(bar_done1, 1);
        mbar_init(bar_done2, 1);
        abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 0) {
        tmem_alloc(smem_u32(&tmem_slot), 512);   // Y in columns [0, 256), U in [256, 256 + rank)
        tmem_relinquish();
    }
    // B_a's rows n0 .. n0 + 255 (rank values each), zero past the rank:
    // thread t holds 16-byte chunk t % 8 of rows t / 8 + 16 i, in flight
    // during the main loop and staged once the ring is free
    constexpr int kBRegs = kBN * 8 / kThreads;
    uint4 breg[kBRegs];
    {
        const int c = t & 7;
#pragma unroll
        for (int i = 0; i < kBRegs; ++i) {
            const int row = (t >> 3) + i * (kThreads / 8);
            breg[i] = (lora && c < rank / 8)
                          ? ldg16(lora_b + ((int64_t)tile.adapter * d_out + n0 + row) * rank + c * 8)
                          : make_uint4(0, 0, 0, 0);
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;
    volatile int *abort = &abort_flag;

    if (t == 0) {
        // ---- TMA producer
        prefetch_tmap(&tmx);
        prefetch_tmap(&tmw);
        if (lora) prefetch_tmap(&tma);
        const uint32_t bytes = kXBytes + kWBytes + (lora ? (uint32_t)rank * kBK * 2 : 0u);
        int issued = 0;
        for (int kb = 0; kb < nk; ++kb) {
            const int s = kb % kStages;
            if (kb >= kStages && !mbar_wait(bar_empty + 8 * s, ((kb / kStages) - 1) & 1, abort, kWaitLimitNs)) break;
            const uint32_t st = sb + s * kStageBytes;
            mbar_arrive_expect_tx(bar_full + 8 * s, bytes);
            tma_load_2d(st, &tmx, kb * kBK, tile.row0, bar_full + 8 * s);
            tma_load_2d(st + kXBytes, &tmw, kb * kBK, n0, bar_full + 8 * s);
            if (lora) tma_load_2d(st + kXBytes + kWBytes, &tma, kb * kBK, tile.adapter * rank, bar_full + 8 * s);
            issued = kb + 1;
        }
        // let this CTA's own copies land before its shared memory is released
        int quiet = 0;
        for (int kb = issued > kStages ? issued - kStages : 0; kb < issued; ++kb)
            mbar_wait(bar_full + 8 * (kb % kStages), (kb / kStages) & 1, &quiet, kDrainLimitNs);
    } else if (t == 32) {
        // ---- MMA issuer
        const uint32_t id_y = idesc_bf16_f32(kBM, kBN, false);
        const uint32_t id_u = idesc_bf16_f32(kBM, rank, false);
        for (int kb = 0; kb < nk; ++kb) {
            const int s = kb % kStages;
            if (!mbar_wait(bar_full + 8 * s, (kb / kStages) & 1, abort, kWaitLimitNs)) break;
            tc_fence_after();
            const uint32_t st = sb + s * kStageBytes;
            const uint64_t xd = smem_desc_sw128(st, 16, 1024);
            const uint64_t wd = smem_desc_sw128(st + kXBytes, 16, 1024);
            const uint64_t ad = smem_desc_sw128(st + kXBytes + kWBytes, 16, 1024);
#pragma unroll
            for (int kk = 0; kk < kBK / 16; ++kk)
                mma_ss(tmem, xd + 2 * kk, wd + 2 * kk, id_y, (kb | kk) ? 1u : 0u);
            if (lora) {
#pragma unroll
                for (int kk = 0; kk < kBK / 16; ++kk)
                    mma_ss(tmem + kBN, xd + 2 * kk, ad + 2 * kk, id_u, (kb | kk) ? 1u : 0u);
            }
            mma_commit(bar_empty + 8 * s);
        }
        mma_commit(bar_done1);   // also arrives if the loop stopped early: its MMAs are done
    }
    __syncwarp();
    // ---- U = s_a * (X A_a^T) rounded to bf16, staged as the A operand of U.B_a^T
    const uint32_t lane_off = (uint32_t)(warp * 32) << 16;
    bool ok = __all_sync(0xffffffffu, mbar_wait(bar_done1, 0, abort, kWaitLimitNs));
    if (ok && lora) {
        tc_fence_after();
        uint32_t u[2][32];
        tmem_ld32(tmem + lane_off + kBN, u[0]);
        tmem_ld32(tmem + lane_off + kBN + 32, u[1]);
        tmem_wait_ld();
#pragma unroll
        for (int c = 0; c < 8; ++c) {
            uint32_t w4[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int col = c * 8 + 2 * e;
                const float lo = col < rank ? __uint_as_float(u[col >> 5][col & 31]) * tile.scale : 0.f;
                const float hi = col + 1 < rank ? __uint_as_float(u[(col + 1) >> 5][(col + 1) & 31]) * tile.scale : 0.f;
                w4[e] = pack_bf16x2(lo, hi);
            }
            *reinterpret_cast<uint4 *>(smem + kUOff + sw128(t, c)) = make_uint4(w4[0], w4[1], w4[2], w4[3]);
        }
#pragma unroll
        for (int i = 0; i < kBRegs; ++i)
            *reinterpret_cast<uint4 *>(smem + kBtOff + sw128((t >> 3) + i * (kThreads / 8), t & 7)) = breg[i];
        fence_proxy_async_smem();
    }
    tc_fence_before();
    __syncthreads();
    if (ok && lora) {
        if (t == 32) {
            tc_fence_after();
            const uint32_t id_y = idesc_bf16_f32(kBM, kBN, false);
            const uint64_t ud = smem_desc_sw128(sb + kUOff, 16, 1024);
            const uint64_t bd = smem_desc_sw128(sb + kBtOff, 16, 1024);
#pragma unroll
            for (int kk = 0; kk < kBK / 16; ++kk) mma_ss(tmem, ud + 2 * kk, bd + 2 * kk, id_y, 1u);
            mma_commit(bar_done2);
        }
        __syncwarp();
        ok = __all_sync(0xffffffffu, mbar_wait(bar_done2, 0, abort, kWaitLimitNs));
    }
    // ---- epilogue: row t of the tile, 256 columns, bf16
    if (ok) {
        tc_fence_after();
        const bool row_ok = t < tile.rows;
        uint16_t *dst = y + (int64_t)(tile.row0 + t) * d_out + n0;
#pragma unroll 1
        for (int c = 0; c < kBN / 32; ++c) {
            uint32_t v[32];
            tmem_ld32(tmem + lane_off + c * 32, v);
            tmem_wait_ld();
            if (row_ok) {
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    uint4 w;
                    w.x = pack_bf16x2(__uint_as_float(v[8 * q + 0]), __uint_as_float(v[8 * q + 1]));
                    w.y = pack_bf16x2(__uint_as_float(v[8 * q + 2]), __uint_as_float(v[8 * q + 3]));
                    w.z = pack_bf16x2(__uint_as_float(v[8 * q + 4]), __uint_as_float(v[8 * q + 5]));
                    w.w = pack_bf16x2(__uint_as_float(v[8 * q + 6]), __uint_as_float(v[8 * q + 7]));
                    *reinterpret_cast<uint4 *>(dst + c * 32 + q * 8) = w;
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
    if (t == 0 && abort_flag) latch_error(err, kDevTimeout);
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    // looked up once (thread-safe static initialisation); null if absent
    static const PFN_cuTensorMapEncodeTiled_v12000 fn = []() -> PFN_cuTensorMapEncodeTiled_v12000 {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
        return nullptr;
    }();
    return fn;
}

// 2-D row-major bf16 matrix [rows][cols], box {64 columns, box_rows rows}, 128-byte swizzle
bool map_2d(CUtensorMap *m, const void *base, int64_t rows, int64_t cols, uint32_t box_rows) {
    auto enc = encode_fn();
    if (!enc) return false;
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
    cuuint32_t box[2] = {64, box_rows};
    cuuint32_t es[2] = {1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int fail(int code, const char *fmt, ...) {
    char buf[256];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    return set_last_error(code, buf);
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace
}  // namespace pkv

extern "C" int pkv_lora_sgmv(const void *x, const void *w, const void *lora_a, const void *lora_b,
                             const float *scale, const int32_t *seg_start, const int32_t *seg_adapter,
                             int32_t num_segments, int32_t num_tokens, int32_t d_in, int32_t d_out,
                             int32_t rank, int32_t num_adapters, void *y, int32_t *error_word,
                             pkv_stream_t stream) {
    using namespace pkv;
    if (num_segments < 0 || num_tokens < 0 || d_in <= 0 || d_out <= 0 || num_adapters < 0)
        return fail(PKV_ERR_INVALID_ARG, "pkv_lora_sgmv: bad sizes");
    if (d_in % kBK != 0 || d_out % kBN != 0)
        return fail(PKV_ERR_UNSUPPORTED, "pkv_lora_sgmv: d_in must be a multiple of 64 and d_out of 256");
    if (rank != 16 && rank != 32 && rank != 48 && rank != 64)
        return fail(PKV_ERR_UNSUPPORTED, "pkv_lora_sgmv: rank must be 16, 32, 48 or 64");
    if (!seg_start || (num_segments > 0 && !seg_adapter))
        return fail(PKV_ERR_INVALID_ARG, "pkv_lora_sgmv: NULL segment arrays");
    if (seg_start[0] != 0 || seg_start[num_segments] != num_tokens)
        return fail(PKV_ERR_INVALID_ARG, "pkv_lora_sgmv: segments must cover rows 0 .. num_tokens");
    TileList tl{};
    for (int32_t s = 0; s < num_segments; ++s) {
        const int32_t a = seg_start[s], e = seg_start[s + 1], ad = seg_adapter[s];
        if (e < a) return fail(PKV_ERR_INVALID_ARG, "pkv_lora_sgmv: segment %d ends before it starts", s);
        if (ad < -1 || ad >= num_adapters)
            return fail(PKV_ERR_INVALID_ARG, "pkv_lora_sgmv: segment %d names adapter %d of %d", s, ad, num_adapters);
        if (ad >= 0 && !scale) return fail(PKV_ERR_INVALID_ARG, "pkv_lora_sgmv: NULL scale");
        for (int32_t r = a; r < e; r += kBM) {
            if (tl.n == PKV_LORA_MAX_TILES)
                return fail(PKV_ERR_UNSUPPORTED, "pkv_lora_sgmv: more than %d row tiles; split the call",
                            PKV_LORA_MAX_TILES);
            tl.t[tl.n++] = Tile{r, e - r < kBM ? e - r : kBM, ad, ad >= 0 ? scale[ad] : 0.f};
        }
    }
    if (tl.n == 0) return set_last_error(PKV_OK, "");
    if (!x || !w || !y || (num_adapters > 0 && (!lora_a || !lora_b)))
        return fail(PKV_ERR_INVALID_ARG, "pkv_lora_sgmv: NULL buffer");
    if (!aligned16(x) || !aligned16(w) || !aligned16(y) || (lora_a && !aligned16(lora_a)) ||
        (lora_b && !aligned16(lora_b)))
        return fail(PKV_ERR_INVALID_ARG, "pkv_lora_sgmv: buffers must be 16-byte aligned");
    CUtensorMap mx, mw, ma;
    bool okm = map_2d(&mx, x, num_tokens, d_in, kBM) && map_2d(&mw, w, d_out, d_in, kBN);
    if (okm && num_adapters > 0) okm = map_2d(&ma, lora_a, (int64_t)num_adapters * rank, d_in, (uint32_t)rank);
    else ma = mx;   // never read: no tile has an adapter
    if (!okm) return fail(PKV_ERR_CUDA, "pkv_lora_sgmv: cuTensorMapEncodeTiled failed");
    static SmemLimit limit;
    cudaError_t e = limit.ensure(reinterpret_cast<const void *>(lora_tile_kernel), kSmemBytes);
    if (e == cudaSuccess)
        e = launch_pdl(lora_tile_kernel, dim3((unsigned)(d_out / kBN), (unsigned)tl.n), dim3(kThreads), kSmemBytes,
                       static_cast<cudaStream_t>(stream), mx, mw, ma, static_cast<const uint16_t *>(lora_b),
                       static_cast<uint16_t *>(y), d_in, d_out, rank, reinterpret_cast<int *>(error_word), tl);
    if (e != cudaSuccess) return fail(PKV_ERR_CUDA, "pkv_lora_sgmv launch: %s", cudaGetErrorString(e));
    return set_last_error(PKV_OK, "");
}
