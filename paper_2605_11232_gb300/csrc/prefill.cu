// prefill.cu -- suffix/chunk prefill over a paged, prefix-cached KV cache on
// the 5th-generation tensor cores (tcgen05, TMEM, TMA).
//
// The paper's serving stack reuses the KV blocks of a shared policy prefix and
// computes only the case-specific suffix (Sec. 5.4; the "enable APC" row of
// the bottleneck table): every new token attends to the whole cached context
// plus, causally, to the new tokens before it.  One CTA computes one 128-row
// tile of (new token, q head) pairs for one kv head: the g q heads of a kv
// head are packed next to each other (row = token * g + head), so one K/V tile
// serves all of them (GQA packing).
//
// Pipeline (one CTA, 6 warps):
//   warp 0   TMA producer: for each 128-key tile, 8 paged blocks x (head-dim
//            halves) of K and of V, each a 16-row x 128-byte box read through
//            the block table, into a 2-stage ring (128-byte swizzle).
//   warp 1   MMA issuer (one thread): S = Q K^T into TMEM (double-buffered),
//            then O += P V with P read from TMEM and V from shared memory.
//   warps 2-5  softmax: thread = row; S row from TMEM, scale, causal mask,
//            online max/sum in base 2, P (bf16) written back over S in TMEM;
//            O is rescaled in TMEM only when the running max grows by more
//            than 2^8 (otherwise the stale max is kept -- exact, since the same
//            max normalises O and l).  Epilogue: O / l -> bf16, LSE.
// Every mbarrier wait is bounded; on a timeout the CTA stops, drains its own
// TMA copies and MMAs, frees TMEM and latches PKV_ERR_DEVICE_TIMEOUT.
#include <math.h>

#include "pkv_device.cuh"
#include "pkv_internal.h"
#include "tc_ptx.cuh"

namespace pkv {

namespace {

using namespace tc;

constexpr int kThreads = 192;
constexpr int kRows = 128;            // M of the tile
constexpr int kKeys = 128;            // keys per tile (N of Q.K^T)
constexpr uint32_t kTmemCols = 512;   // S0 [0,128) S1 [128,256) O [256, 256+D)
constexpr uint64_t kWaitLimitNs = 2000000000ull;
constexpr uint64_t kDrainLimitNs = 200000000ull;
constexpr int kMaxItemBlocks = 2048;  // keys of one work item <= 32768

template <int D>
struct Layout {
    static constexpr int kHalves = D / 64;            // 64-element (128-byte) column halves
    static constexpr int kHalfBytes = 128 * 128;      // 128 rows x 128 bytes
    static constexpr int kQ = 0;
    static constexpr int kTile = kHalves * kHalfBytes;  // one Q, K or V tile
    static constexpr int kK0 = kQ + kTile;
    static constexpr int kV0 = kK0 + 2 * kTile;
    static constexpr int kBar = kV0 + 2 * kTile;
    // barrier block: k_full[2] v_full[2] kv_empty[2] s_full[2] p_full[2] o_ready[2] done
    static constexpr int kKFull = kBar + 0, kVFull = kBar + 16, kKvEmpty = kBar + 32;
    static constexpr int kSFull = kBar + 48, kPFull = kBar + 64, kOReady = kBar + 80;
    static constexpr int kDone = kBar + 96, kTmemSlot = kBar + 104, kAbort = kBar + 108;
    static constexpr int kBlkIds = kBar + 128;        // int32 [kMaxItemBlocks]
    static constexpr int kBytes = kBlkIds + 4 * kMaxItemBlocks;
    static constexpr int kDynSmem = kBytes + 1024;    // room to align the base to 1 KiB
};

struct KernelParams {
    const uint16_t *q;
    uint16_t *out;
    float *lse;
    const int32_t *cu_seqlens_q;
    const int32_t *context_lens;
    const int32_t *block_table;
    int32_t max_blocks;
    int32_t Hq, Hkv, g, tpt;   // tpt: tokens per 128-row tile
    int32_t num_blocks_pool;
    float scale_log2;
    int *err;
    // shared-prefix decode pass only
    const int32_t *group_start;
    const int32_t *member_req;
    const int32_t *group_blocks;
    int32_t num_requests;       // decode batch size (member ids must be below it)
    int32_t blocks_per_part;    // prefix blocks per key split
    int32_t parts_per_head;     // partial slots per (request, q head)
    float *o_part;              // [R*Hq*parts][D] unnormalised O
    float2 *ml_part;            // [R*Hq*parts] (running max (base 2), sum)
};

// 2^x on the FMA pipe, to offload part of the exponentials from the
// special-function unit (which alone would need as many cycles per score as
// the two MMAs take).  x = n + f with n = round(x) found by adding
// 1.5 * 2^23 (the sum's low mantissa bits are n), 2^f by a cubic fitted on
// [-0.5, 0.5] (max relative error 7.5e-5; Lawson-weighted least squares on
// Chebyshev nodes, see fit_exp2_poly.py), and n added into the exponent field.
// x is clamped to -125 so the result stays a normal number; masked scores
// (-inf) give exactly 0.
__device__ __forceinline__ float poly_exp2(float x) {
    const float xc = fmaxf(x, -125.0f);
    const float t = xc + 12582912.0f;
    const float n = t - 12582912.0f;
    const float f = xc - n;
    float p = fmaf(0.0551716648f, f, 0.2426111251f);
    p = fmaf(p, f, 0.6932609677f);
    p = fmaf(p, f, 0.9999280572f);
    const uint32_t e = (uint32_t)(__float_as_int(t) - 0x4B400000) << 23;
    const float r = __uint_as_float(__float_as_uint(p) + e);
    return x < -125.0f ? 0.0f : r;
}

// TMEM address of the c-th 32-column chunk of the O accumulator in this
// warp's lane quarter.
__device__ __forceinline__ uint32_t o_addr(uint32_t tmem, uint32_t lane_off, int c) {
    return tmem + lane_off + 256 + c * 32;
}

__device__ __forceinline__ bool wait_bar(uint32_t bar, uint32_t parity, volatile int *abort) {
    return mbar_wait(bar, parity, abort, kWaitLimitNs);
}

// Whole-warp wait with a warp-uniform outcome, so that the .sync.aligned
// tcgen05 instructions after it are reached by all lanes or by none.
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int *abort) {
    return __all_sync(0xffffffffu, wait_bar(bar, parity, abort));
}

// PREFIX = false: suffix prefill.  CTA (request r, kv head h, token tile);
//   row i = token (i / g) of the tile, q head h*g + i % g; keys 0 .. pos(i).
// PREFIX = true: shared-prefix pass of decode.  CTA (group, kv head, member
//   tile, key split); row i = member request (i / g) of the tile; keys = the
//   split's range of the group's prefix blocks (read through the first
//   member's table row), all visible; writes unnormalised partials.
template <int D, bool PREFIX>
__global__ void __launch_bounds__(kThreads, 1)
    attn_tile_kernel(const __grid_constant__ CUtensorMap tmk, const __grid_constant__ CUtensorMap tmv,
                     const KernelParams p) {
    using Ly = Layout<D>;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int h = blockIdx.x % p.Hkv;
    int rows_valid, nblk, kv_end, q_pos0 = 0, blk_off = 0, cu0 = 0, tok0 = 0, m0 = 0;
    const int32_t *trow;
    if constexpr (!PREFIX) {
        const int r = blockIdx.x / p.Hkv;
        const int tile = gridDim.y - 1 - blockIdx.y;      // heaviest tiles first
        cu0 = __ldg(p.cu_seqlens_q + r);
        const int n_r = __ldg(p.cu_seqlens_q + r + 1) - cu0;
        tok0 = tile * p.tpt;
        if (tok0 >= n_r) return;
        const int ntok = min(p.tpt, n_r - tok0);
        const int L = __ldg(p.context_lens + r);
        if (L < n_r || L > 16 * p.max_blocks) {
            if (threadIdx.x == 0) latch_error(p.err, kDevBounds);
            return;
        }
        q_pos0 = L - n_r + tok0;          // absolute position of the tile's first token
        kv_end = q_pos0 + ntok;           // keys [0, kv_end) are visible to some row
        nblk = (kv_end + 15) >> 4;
        rows_valid = ntok * p.g;
        trow = p.block_table + (int64_t)r * p.max_blocks;
    } else {
        const int grp = blockIdx.x / p.Hkv;
        const int gs = __ldg(p.group_start + grp);
        const int nm = __ldg(p.group_start + grp + 1) - gs;
        const int mt0 = blockIdx.y * p.tpt;
        if (mt0 >= nm) return;
        const int gb = __ldg(p.group_blocks + grp);
        blk_off = blockIdx.z * p.blocks_per_part;
        if (blk_off >= gb) return;
        if (gb > p.max_blocks) {
            if (threadIdx.x == 0) latch_error(p.err, kDevBounds);
            return;
        }
        nblk = min(p.blocks_per_part, gb - blk_off);
        kv_end = nblk * 16;
        rows_valid = min(p.tpt, nm - mt0) * p.g;
        m0 = gs + mt0;
        // every member id of this tile (and the first member, whose table row
        // names the prefix blocks) must be a request of the batch
        bool ids_ok = true;
        const int r_first = __ldg(p.member_req + gs);
        if (r_first < 0 || r_first >= p.num_requests) ids_ok = false;
        for (int i = 0; i < rows_valid; i += p.g) {
            const int rm = __ldg(p.member_req + m0 + i / p.g);
            if (rm < 0 || rm >= p.num_requests) ids_ok = false;
        }
        if (!ids_ok) {
            if (threadIdx.x == 0) latch_error(p.err, kDevBounds);
            return;
        }
        trow = p.block_table + (int64_t)r_first * p.max_blocks;
    }
    if (nblk > kMaxItemBlocks) {
        if (threadIdx.x == 0) latch_error(p.err, kDevBounds);
        return;
    }
    const int nkt = (kv_end + kKeys - 1) / kKeys;
    // global q row of tile row i (decode q is [R][Hq][D], prefill q is [T][Hq][D])
    auto q_row = [&](int i) -> int64_t {
        if constexpr (PREFIX)
            return (int64_t)__ldg(p.member_req + m0 + i / p.g) * p.Hq + h * p.g + i % p.g;
        else
            return (int64_t)(cu0 + tok0 + i / p.g) * p.Hq + h * p.g + i % p.g;
    };

    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                ~uintptr_t(1023));
    const uint32_t sb = smem_u32(smem);
    volatile int *abort = reinterpret_cast<volatile int *>(smem + Ly::kAbort);
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + Ly::kTmemSlot);

    if (threadIdx.x == 0) {
        for (int i = 0; i < 2; ++i) {
            mbar_init(sb + Ly::kKFull + 8 * i, 1);
            mbar_init(sb + Ly::kVFull + 8 * i, 1);
            mbar_init(sb + Ly::kKvEmpty + 8 * i, 1);
            mbar_init(sb + Ly::kSFull + 8 * i, 1);
            mbar_init(sb + Ly::kPFull + 8 * i, 128);
            mbar_init(sb + Ly::kOReady + 8 * i, 1);
        }
        mbar_init(sb + Ly::kDone, 1);
        *abort = 0;
        fence_barrier_init();
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(tmem_slot), kTmemCols);
        tmem_relinquish();
    }
    // Q tile -> shared memory, K-major with the 128-byte swizzle (16-byte
    // chunk c of row i goes to chunk c ^ (i % 8) of its 128-byte row).  All
    // loads are issued before the first store so their latencies overlap.
    {
        constexpr int kChunks = D / 8;
        constexpr int kIters = (kRows * kChunks + kThreads - 1) / kThreads;
        uint4 v[kIters];
#pragma unroll
        for (int k = 0; k < kIters; ++k) {
            const int idx = threadIdx.x + k * kThreads;
            const int i = idx / kChunks, c = idx % kChunks;
            v[k] = make_uint4(0, 0, 0, 0);
            if (idx < kRows * kChunks && i < rows_valid) v[k] = ldg16(p.q + q_row(i) * D + c * 8);
        }
#pragma unroll
        for (int k = 0; k < kIters; ++k) {
            const int idx = threadIdx.x + k * kThreads;
            if (idx < kRows * kChunks) {
                const int i = idx / kChunks, c = idx % kChunks;
                const int half = c >> 3, cc = c & 7;
                *reinterpret_cast<uint4 *>(smem + Ly::kQ + half * Ly::kHalfBytes + i * 128 +
                                           ((cc ^ (i & 7)) << 4)) = v[k];
            }
        }
        fence_proxy_async_smem();
    }
    // the item's physical block ids, checked once, for the producer
    int32_t *blk_ids = reinterpret_cast<int32_t *>(smem + Ly::kBlkIds);
    if (warp == 0) {
        for (int b = lane; b < nblk; b += 32) {
            int32_t id = __ldg(trow + blk_off + b);
            if (id < 0 || id >= p.num_blocks_pool) {
                latch_error(p.err, kDevBounds);
                id = 0;
            }
            blk_ids[b] = id;
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            prefetch_tmap(&tmk);
            prefetch_tmap(&tmv);
            int issued = 0;
            for (int j = 0; j < nkt; ++j) {
                const int s = j & 1;
                if (j >= 2 && !wait_bar(sb + Ly::kKvEmpty + 8 * s, ((j >> 1) - 1) & 1, abort)) break;
                const int b0 = j * 8, nb = min(8, nblk - b0);
                const uint32_t bytes = (uint32_t)nb * Ly::kHalves * 2048u;
                const uint32_t kdst = sb + Ly::kK0 + s * Ly::kTile;
                const uint32_t vdst = sb + Ly::kV0 + s * Ly::kTile;
                int32_t phys[8];
                for (int b = 0; b < nb; ++b) phys[b] = blk_ids[b0 + b];
                mbar_arrive_expect_tx(sb + Ly::kKFull + 8 * s, bytes);
                for (int b = 0; b < nb; ++b)
                    for (int hf = 0; hf < Ly::kHalves; ++hf)
                        tma_load_4d(kdst + hf * Ly::kHalfBytes + b * 2048, &tmk, hf * 64, 0, h,
                                    phys[b], sb + Ly::kKFull + 8 * s);
                mbar_arrive_expect_tx(sb + Ly::kVFull + 8 * s, bytes);
                for (int b = 0; b < nb; ++b)
                    for (int hf = 0; hf < Ly::kHalves; ++hf)
                        tma_load_4d(vdst + hf * Ly::kHalfBytes + b * 2048, &tmv, hf * 64, 0, h,
                                    phys[b], sb + Ly::kVFull + 8 * s);
                issued = j + 1;
            }
            // let this CTA's own copies land before its shared memory is released
            int quiet = 0;
            for (int j = max(0, issued - 2); j < issued; ++j) {
                mbar_wait(sb + Ly::kKFull + 8 * (j & 1), (j >> 1) & 1, &quiet, kDrainLimitNs);
                mbar_wait(sb + Ly::kVFull + 8 * (j & 1), (j >> 1) & 1, &quiet, kDrainLimitNs);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        const uint32_t id_qk = idesc_bf16_f32(kRows, kKeys, false);
        const uint32_t id_pv = idesc_bf16_f32(kRows, D, true);
        const uint32_t o_col = tmem + 256;
        bool ok = true;
        auto issue_pv = [&](int jj) -> bool {
            const int s = jj & 1;
            if (!warp_wait(sb + Ly::kVFull + 8 * s, (jj >> 1) & 1, abort)) return false;
            if (!warp_wait(sb + Ly::kPFull + 8 * s, (jj >> 1) & 1, abort)) return false;
            const uint32_t vbase = sb + Ly::kV0 + s * Ly::kTile;
            if (jj == nkt - 1) {
                // keys past the context: p = 0 there, but their V rows may hold
                // anything (0 * NaN = NaN in the MMA), so clear them
                const int first = kv_end - jj * kKeys;
                uint8_t *vs = smem + Ly::kV0 + s * Ly::kTile;
                for (int row = first + lane; row < kKeys; row += 32)
                    for (int hf = 0; hf < Ly::kHalves; ++hf) {
                        uint4 *d4 = reinterpret_cast<uint4 *>(vs + hf * Ly::kHalfBytes + row * 128);
#pragma unroll
                        for (int c = 0; c < 8; ++c) d4[c] = make_uint4(0, 0, 0, 0);
                    }
                fence_proxy_async_smem();
                __syncwarp();
            }
            tc_fence_after();
            if (lane == 0) {
#pragma unroll
                for (int kk = 0; kk < kKeys / 16; ++kk) {
                    // V is N-major (head dim contiguous): LBO = stride between the
                    // 64-wide head-dim halves, SBO = stride between 8-key groups
                    const uint64_t bdesc = smem_desc_sw128(vbase + kk * 2048, Ly::kHalfBytes, 1024);
                    mma_ts(o_col, tmem + s * 128 + kk * 8, bdesc, id_pv, (jj > 0 || kk > 0) ? 1u : 0u);
                }
                mma_commit(sb + Ly::kKvEmpty + 8 * s);
                mma_commit(sb + Ly::kOReady + 8 * (jj & 1));
            }
            __syncwarp();
            return true;
        };
        for (int j = 0; j < nkt && ok; ++j) {
            const int s = j & 1;
            if (!warp_wait(sb + Ly::kKFull + 8 * s, (j >> 1) & 1, abort)) { ok = false; break; }
            tc_fence_after();
            if (lane == 0) {
                const uint32_t qbase = sb + Ly::kQ, kbase = sb + Ly::kK0 + s * Ly::kTile;
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk) {
                    const uint32_t off = (kk >> 2) * Ly::kHalfBytes + (kk & 3) * 32;
                    mma_ss(tmem + s * 128, smem_desc_sw128(qbase + off, 16, 1024),
                           smem_desc_sw128(kbase + off, 16, 1024), id_qk, kk > 0 ? 1u : 0u);
                }
                mma_commit(sb + Ly::kSFull + 8 * s);
            }
            __syncwarp();
            if (j >= 1) ok = issue_pv(j - 1);
        }
        if (ok) ok = issue_pv(nkt - 1);
        // all MMAs issued by this thread must finish before TMEM is freed
        if (lane == 0) mma_commit(sb + Ly::kDone);
        __syncwarp();
        int quiet = 0;
        mbar_wait(sb + Ly::kDone, 0, &quiet, kDrainLimitNs);
    } else {
        // ------------------------------------------------------------ softmax
        const int quarter = warp & 3;                 // TMEM lanes this warp may touch
        const int row = quarter * 32 + lane;
        const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;
        const bool valid = row < rows_valid;
        // last visible key (tile-local numbering of the item's key range)
        const int pos = (!PREFIX && valid) ? q_pos0 + row / p.g : kv_end - 1;
        float m = -INFINITY, l = 0.f;
        bool ok = true;
        // P.V(k) completes o_ready[k & 1].  Waiting for P.V(k) is unambiguous
        // when P.V(k - 2) is known complete, which holds wherever it is used
        // below: Q.K(j) is issued after P.V(j - 2), and S(j) is in hand.
        auto wait_pv = [&](int k) -> bool {
            return warp_wait(sb + Ly::kOReady + 8 * (k & 1), (k >> 1) & 1, abort);
        };
        for (int j = 0; j < nkt; ++j) {
            const int b = j & 1;
            if (!warp_wait(sb + Ly::kSFull + 8 * b, (j >> 1) & 1, abort)) { ok = false; break; }
            tc_fence_after();
            uint32_t sr[4][32];
#pragma unroll
            for (int c = 0; c < 4; ++c) tmem_ld32(tmem + lane_off + b * 128 + c * 32, sr[c]);
            tmem_wait_ld();
            const int kb = j * kKeys;
            const int lim = pos - kb;                 // keys with column index <= lim are visible
            float mx = -INFINITY;
            if (__all_sync(0xffffffffu, lim >= kKeys - 1)) {
                // every key of the tile is visible to every row of this warp
#pragma unroll
                for (int c = 0; c < 4; ++c)
#pragma unroll
                    for (int e = 0; e < 32; ++e) mx = fmaxf(mx, __uint_as_float(sr[c][e]));
            } else {
#pragma unroll
                for (int c = 0; c < 4; ++c)
#pragma unroll
                    for (int e = 0; e < 32; ++e) {
                        const float v = (c * 32 + e <= lim) ? __uint_as_float(sr[c][e]) : -INFINITY;
                        sr[c][e] = __float_as_uint(v);
                        mx = fmaxf(mx, v);
                    }
            }
            mx *= p.scale_log2;                       // scale > 0 commutes with max
            // conditional rescale: keep a stale max unless it grows by > 8 (x256)
            const float m_new = (mx > m + 8.0f) ? mx : m;
            const bool grow = (m_new != m) && (j > 0);
            float alpha = grow ? fast_exp2(m - m_new) : 1.0f;
            if (__any_sync(0xffffffffu, grow)) {
                // O must hold P.V(j-1) before it is rescaled
                if (!wait_pv(j - 1)) { ok = false; break; }
                tc_fence_after();
#pragma unroll
                for (int c = 0; c < D / 32; ++c) {
                    uint32_t o[32];
                    tmem_ld32(o_addr(tmem, lane_off, c), o);
                    tmem_wait_ld();
#pragma unroll
                    for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
                    tmem_st32(o_addr(tmem, lane_off, c), o);
                }
            }
            m = m_new;
            float sum = 0.f;
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                uint32_t pk[16];
#pragma unroll
                for (int e = 0; e < 16; ++e) {
                    const float x0 = fmaf(__uint_as_float(sr[c][2 * e]), p.scale_log2, -m);
                    const float x1 = fmaf(__uint_as_float(sr[c][2 * e + 1]), p.scale_log2, -m);
                    // one in four exponentials on the FMA pipe
                    const float p0 = fast_exp2(x0);
                    const float p1 = (e & 1) ? poly_exp2(x1) : fast_exp2(x1);
                    sum += p0 + p1;
                    pk[e] = pack_bf16x2(p0, p1);
                }
                tmem_st16(tmem + lane_off + b * 128 + c * 16, pk);
            }
            l = l * alpha + sum;
            tmem_wait_st();
            tc_fence_before();
            mbar_arrive(sb + Ly::kPFull + 8 * b);
        }
        if (ok && wait_pv(nkt - 1)) {
            tc_fence_after();
            const int64_t orow = valid ? q_row(row) : 0;
            if constexpr (!PREFIX) {
                const float inv = 1.0f / l;
#pragma unroll
                for (int c = 0; c < D / 32; ++c) {
                    uint32_t o[32];
                    tmem_ld32(o_addr(tmem, lane_off, c), o);
                    tmem_wait_ld();
                    if (valid) {
                        uint4 *dst = reinterpret_cast<uint4 *>(p.out + orow * D + c * 32);
#pragma unroll
                        for (int v = 0; v < 4; ++v) {
                            uint4 w;
                            w.x = pack_bf16x2(__uint_as_float(o[8 * v + 0]) * inv, __uint_as_float(o[8 * v + 1]) * inv);
                            w.y = pack_bf16x2(__uint_as_float(o[8 * v + 2]) * inv, __uint_as_float(o[8 * v + 3]) * inv);
                            w.z = pack_bf16x2(__uint_as_float(o[8 * v + 4]) * inv, __uint_as_float(o[8 * v + 5]) * inv);
                            w.w = pack_bf16x2(__uint_as_float(o[8 * v + 6]) * inv, __uint_as_float(o[8 * v + 7]) * inv);
                            dst[v] = w;
                        }
                    }
                }
                if (valid && p.lse) p.lse[orow] = (m + __log2f(l)) * 0.69314718055994530942f;
            } else {
                // unnormalised partial of key split blockIdx.z, merged by the combine
                const int64_t slot = orow * p.parts_per_head + blockIdx.z;
#pragma unroll
                for (int c = 0; c < D / 32; ++c) {
                    uint32_t o[32];
                    tmem_ld32(o_addr(tmem, lane_off, c), o);
                    tmem_wait_ld();
                    if (valid) {
                        uint4 *dst = reinterpret_cast<uint4 *>(p.o_part + slot * D + c * 32);
#pragma unroll
                        for (int v = 0; v < 8; ++v)
                            dst[v] = make_uint4(o[4 * v], o[4 * v + 1], o[4 * v + 2], o[4 * v + 3]);
                    }
                }
                if (valid) p.ml_part[slot] = make_float2(m, l);
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
    if (threadIdx.x == 0 && *abort) latch_error(p.err, kDevTimeout);
}

}  // namespace

template <int D, bool PREFIX>
static cudaError_t launch_tile_kernel(dim3 grid, const CUtensorMap &tk, const CUtensorMap &tv,
                                      const KernelParams &p, cudaStream_t stream) {
    static bool attr = false;
    // the d = 64 tile is smaller; ask for the d = 128 footprint anyway so one
    // CTA owns an SM (its 512 TMEM columns never wait on a neighbour)
    if (!attr) {
        cudaError_t e = cudaFuncSetAttribute(attn_tile_kernel<D, PREFIX>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             Layout<128>::kDynSmem);
        if (e != cudaSuccess) return e;
        attr = true;
    }
    attn_tile_kernel<D, PREFIX><<<grid, kThreads, Layout<128>::kDynSmem, stream>>>(tk, tv, p);
    return cudaGetLastError();
}

cudaError_t launch_prefill(const PrefillArgs &a, cudaStream_t stream, Tracer *tr) {
    const int g = a.Hq / a.Hkv;
    KernelParams p{};
    p.q = static_cast<const uint16_t *>(a.q);
    p.out = static_cast<uint16_t *>(a.out);
    p.lse = a.lse;
    p.cu_seqlens_q = a.cu_seqlens_q;
    p.context_lens = a.context_lens;
    p.block_table = a.block_table;
    p.max_blocks = a.max_blocks;
    p.Hq = a.Hq; p.Hkv = a.Hkv; p.g = g; p.tpt = kRows / g;
    p.num_blocks_pool = a.num_blocks_pool;
    p.scale_log2 = a.scale_log2;
    p.err = a.err;
    const int tiles = (a.max_seqlen_q + p.tpt - 1) / p.tpt;
    if (tiles <= 0 || a.R <= 0) return cudaSuccess;
    if (tiles > 65535) return cudaErrorInvalidConfiguration;
    dim3 grid((unsigned)(a.R * a.Hkv), (unsigned)tiles);
    if (tr) tr->begin(kKernelPrefill, stream);
    cudaError_t e = a.d == 128 ? launch_tile_kernel<128, false>(grid, *a.tmap_k, *a.tmap_v, p, stream)
                               : launch_tile_kernel<64, false>(grid, *a.tmap_k, *a.tmap_v, p, stream);
    if (tr) tr->end(kKernelPrefill, stream);
    return e;
}

cudaError_t launch_decode_prefix(const DecodeLayout &L, const DecodeArgs &a,
                                 int32_t num_blocks_pool, cudaStream_t stream, Tracer *tr) {
    KernelParams p{};
    p.q = static_cast<const uint16_t *>(a.q);
    p.block_table = a.block_table;
    p.max_blocks = a.max_blocks;
    p.Hq = L.Hq; p.Hkv = L.Hkv; p.g = L.g; p.tpt = kRows / L.g;
    p.num_blocks_pool = num_blocks_pool;
    p.scale_log2 = a.scale_log2;
    p.err = a.err;
    p.group_start = a.group_start;
    p.member_req = a.member_req;
    p.group_blocks = a.group_blocks;
    p.num_requests = L.R;
    p.blocks_per_part = L.prefix_blocks_per_part;
    p.parts_per_head = L.parts_per_head;
    p.o_part = reinterpret_cast<float *>(static_cast<char *>(a.ws) + L.off_o);
    p.ml_part = reinterpret_cast<float2 *>(static_cast<char *>(a.ws) + L.off_ml);
    const int mtiles = (a.max_group_members + p.tpt - 1) / p.tpt;
    if (mtiles <= 0 || L.prefix_parts <= 0) return cudaSuccess;
    if (mtiles > 65535) return cudaErrorInvalidConfiguration;
    dim3 grid((unsigned)(a.num_groups * L.Hkv), (unsigned)mtiles, (unsigned)L.prefix_parts);
    if (tr) tr->begin(kKernelDecodePrefix, stream);
    cudaError_t e = L.d == 128 ? launch_tile_kernel<128, true>(grid, *a.tmap_k, *a.tmap_v, p, stream)
                               : launch_tile_kernel<64, true>(grid, *a.tmap_k, *a.tmap_v, p, stream);
    if (tr) tr->end(kKernelDecodePrefix, stream);
    return e;
}

}  // namespace pkv
