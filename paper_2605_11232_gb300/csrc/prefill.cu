// prefill.cu -- attention tiles over a paged, prefix-cached KV cache on the
// 5th-generation tensor cores (tcgen05, TMEM, TMA): the suffix/chunk prefill
// and the shared-prefix pass of decode.
//
// The paper's serving stack reuses the KV blocks of a shared policy prefix and
// computes only the case-specific suffix (Sec. 5.4; the "enable APC" row of
// the bottleneck table): every new token attends to the whole cached context
// plus, causally, to the new tokens before it.  One CTA computes a work item
// of two 128-row tiles (A and B) of (query, q head) pairs for one kv head:
// the g q heads of a kv head sit next to each other (row = query * g + head),
// so every K/V tile read serves all of them (GQA packing) and both tiles.
//
// Pipeline (one CTA per SM, 12 warps = 3 warpgroups):
//   warp 0     TMA producer: per 128-key tile, 8 paged blocks x head-dim
//              halves of K and of V, each a 16-row x 128-byte box read
//              through the block table, into a 2-stage ring (128-byte
//              swizzle); the lanes issue a tile's boxes together.
//   warp 1     MMA issuer (one thread), ping-pong between the tiles:
//                P.V_A(j), Q.K_A(j+1), P.V_B(j), Q.K_B(j+1), ...
//              so the tensor core runs one tile's MMAs while the other tile's
//              softmax runs.  S = Q.K^T lands in TMEM; P.V reads P from TMEM
//              and V from shared memory.
//   warps 2-3  idle
//   warps 4-7  softmax of tile A, warps 8-11 of tile B: thread = row.  S row
//              from TMEM, causal mask, online softmax in base 2, P (bf16)
//              written back over S in TMEM.  After the first key tile one
//              pass computes P against the running max, however stale (exact:
//              the same max normalises O and the row sum); only when the
//              tile's row sum shows a P above 2^15 is the row max found, O
//              rescaled in TMEM and the pass redone.
//              The exponentials run on the SFU.  The two softmax warpgroups
//              run concurrently (their work is staggered by the MMA order).
// All warps keep the launch allocation of 168 registers: moving registers
// from the control warps to the softmax warps (setmaxnreg) measured slower,
// since the MMA issuer then spills in its issue loop.
// Every mbarrier wait is bounded; on a timeout the CTA stops, drains its own
// TMA copies and MMAs, frees TMEM and latches PKV_ERR_DEVICE_TIMEOUT.
#include <math.h>

#include "pkv_device.cuh"
#include "pkv_internal.h"
#include "tc_ptx.cuh"

namespace pkv {

namespace {

using namespace tc;

constexpr int kThreads = 384;
constexpr int kRows = 128;            // M of one tile
constexpr int kKeys = 128;            // keys per K/V tile (N of Q.K^T)
constexpr uint32_t kTmemCols = 512;   // S_A [0,128) S_B [128,256) O_A [256,384) O_B [384,512)
constexpr uint64_t kWaitLimitNs = 2000000000ull;
constexpr uint64_t kDrainLimitNs = 200000000ull;
constexpr int kMaxItemBlocks = kPrefillMaxBlocks;  // keys of one work item <= 32768
template <int D>
struct Layout {
    static constexpr int kHalves = D / 64;            // 64-element (128-byte) column halves
    static constexpr int kHalfBytes = 128 * 128;      // 128 rows x 128 bytes
    static constexpr int kTile = kHalves * kHalfBytes;  // one Q, K or V tile
    static constexpr int kQ = 0;                      // Q_A, then Q_B
    static constexpr int kK0 = kQ + 2 * kTile;
    static constexpr int kV0 = kK0 + 2 * kTile;
    static constexpr int kBar = kV0 + 2 * kTile;
    // barriers: k_full[2] v_full[2] k_empty[2] v_empty[2] s_full[A,B] p_full[A,B]
    // o_done[A,B] done
    static constexpr int kKFull = kBar + 0, kVFull = kBar + 16, kKEmpty = kBar + 32;
    static constexpr int kVEmpty = kBar + 48, kSFull = kBar + 64, kPFull = kBar + 80;
    static constexpr int kODone = kBar + 96, kDone = kBar + 112;
    static constexpr int kTmemSlot = kBar + 120, kAbort = kBar + 124;
    static constexpr int kBlkIds = kBar + 128;        // int32 [kMaxItemBlocks]
    static constexpr int kRowIdx = kBlkIds + 4 * kMaxItemBlocks;   // int64 [2 * kRows]
    static constexpr int kBytes = kRowIdx + 8 * 2 * kRows;
    static constexpr int kDynSmem = kBytes + 1024;    // room to align the base to 1 KiB
    // UMMA descriptors hold address / 16 in 14 bits; k-steps add to that field
    static_assert(kDynSmem < 256 * 1024, "shared addresses must stay below 256 KiB");
};

struct KernelParams {
    const uint16_t *q;
    uint16_t *out;
    float *lse;
    const int32_t *cu_seqlens_q;
    const int32_t *context_lens;
    const int32_t *block_table;
    int32_t max_blocks;
    int32_t Hq, Hkv, g, tpt;   // tpt: queries per 128-row tile
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
    // suffix prefill only: null, or [T] draft masks (bit j of new token t's
    // mask: t sees new token j of its request; at most 64 new tokens each)
    const unsigned long long *tree_mask;
    // suffix prefill with the new tokens' K/V fused in: keys at positions
    // >= L - n_r come from k_new / v_new (tensor maps tmkn / tmvn), and each
    // CTA stores its own queries' K/V rows into the pool
    int32_t fused;
    const uint16_t *k_new, *v_new;   // [T][Hkv][D]
    uint16_t *k_cache, *v_cache;     // the pool
    // shared-prefix pass over draft tokens (grouped verification): the table
    // row naming each group's prefix blocks (null: the first member's row,
    // the member ids being requests) and the number of table rows
    const int32_t *group_row;
    int32_t num_table_rows;
    // private pass of grouped verification (PART): each request's keys after
    // its group's shared blocks, written as part slot private_part
    const int32_t *request_group;    // [R] group of each request, -1: none
    int32_t private_part;
    int32_t prefix_parts;            // prefix part slots (their count per request goes to nparts)
    int32_t *nparts;                 // [T * Hkv] part counts (private | prefix << 16)
    int32_t num_rows;                // T: tokens the workspace holds partials for
    int32_t after_prefix;            // a shared-prefix pass precedes (and started) this pass
    int32_t lpt;                     // suffix prefill: CTAs take items longest first (prefill_lpt_select)
};

// Row maximum of the 128 raw scores a thread holds (8 independent chains).
__device__ __forceinline__ float row_max(const uint32_t (&sr)[4][32]) {
    float mx8[8];
#pragma unroll
    for (int t = 0; t < 8; ++t) mx8[t] = -INFINITY;
#pragma unroll
    for (int c = 0; c < 4; ++c)
#pragma unroll
        for (int e = 0; e < 32; e += 2)
            mx8[(e >> 1) & 7] = fmax3(mx8[(e >> 1) & 7], __uint_as_float(sr[c][e]), __uint_as_float(sr[c][e + 1]));
    return fmaxf(fmax3(mx8[0], mx8[1], mx8[2]), fmax3(fmax3(mx8[3], mx8[4], mx8[5]), mx8[6], mx8[7]));
}

// One softmax pass over a thread's row of 128 scores: P = 2^(s * scale_log2 -
// mref) written as bf16 over the row's S columns in TMEM, and the row sum of
// P returned.  Exponentials on the SFU, so masked scores (-inf) give exactly 0.
__device__ __forceinline__ float softmax_pass(const uint32_t (&sr)[4][32], float scale_log2, float mref,
                                              uint32_t s_addr) {
    const float2 sc2 = make_float2(scale_log2, scale_log2);
    const float2 nm2 = make_float2(-mref, -mref);
    float2 sum2[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
    for (int c = 0; c < 4; ++c) {
        uint32_t pk[16];
#pragma unroll
        for (int e = 0; e < 16; ++e) {
            const float2 sv = make_float2(__uint_as_float(sr[c][2 * e]), __uint_as_float(sr[c][2 * e + 1]));
            const float2 xv = ffma2(sv, sc2, nm2);
            const float2 pp = make_float2(fast_exp2(xv.x), fast_exp2(xv.y));
            sum2[e & 1] = fadd2(sum2[e & 1], pp);
            pk[e] = pack_bf16x2(pp.x, pp.y);
        }
        tmem_st16(s_addr + c * 16, pk);
    }
    const float2 s2 = fadd2(sum2[0], sum2[1]);
    return s2.x + s2.y;
}

__device__ __forceinline__ bool wait_bar(uint32_t bar, uint32_t parity, volatile int *abort) {
    return mbar_wait(bar, parity, abort, kWaitLimitNs);
}

// Whole-warp wait with a warp-uniform outcome, so that the .sync.aligned
// tcgen05 instructions after it are reached by all lanes or by none.
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int *abort) {
    return __all_sync(0xffffffffu, wait_bar(bar, parity, abort));
}

// Longest-first order of a suffix prefill's CTAs.  Item i of request r (n
// new tokens, context L, P = 2 * tpt queries per item, m = ceil(n / P)
// items) ends at key e(i) = min(L, L - n + (i + 1) P) and costs t(i) =
// ceil(e(i) / 128) key tiles, increasing in i.  CTA u of the grid takes the
// item of rank u / Hkv in the order (t descending, r, i) and kv head
// u % Hkv, so the heaviest CTAs start first whatever the requests' lengths
// (a short grid's last wave then holds its lightest CTAs).  Warp-wide (all 32
// lanes): returns false for a spare CTA.
__device__ __forceinline__ int prefill_items_from(int c, int n, int L, int P) {
    // items of a request with t(i) >= c
    if (n <= 0 || L <= 128 * (c - 1)) return 0;
    const int m = (n + P - 1) / P;
    const int A = 128 * (c - 1) - (L - n);
    return A < 0 ? m : max(0, m - A / P);
}

__device__ __forceinline__ bool prefill_lpt_select(const int32_t *__restrict__ cu_seqlens,
                                                   const int32_t *__restrict__ context_lens, int R, int Hkv,
                                                   int P, int64_t u, int *r_out, int *item_out, int *h_out) {
    const int lane = threadIdx.x & 31;
    // a request's keys are taken as at least its new tokens, so that every
    // item of a request with new tokens is scheduled even where the lengths
    // are inconsistent (the kernel then latches DEVICE_BOUNDS for it)
    auto keys_of = [&](int r, int n) -> int { return max(__ldg(context_lens + r), n); };
    // up to 32 requests: one per lane, held in registers
    const bool one = R <= 32;
    const int n1 = one && lane < R ? __ldg(cu_seqlens + lane + 1) - __ldg(cu_seqlens + lane) : 0;
    const int L1 = one && lane < R ? keys_of(lane, n1) : 0;
    auto count_ge = [&](int c) -> int64_t {   // items with t >= c, over all requests
        int64_t s = 0;
        if (one) {
            s = prefill_items_from(c, n1, L1, P);
        } else {
            for (int r = lane; r < R; r += 32) {
                const int n = __ldg(cu_seqlens + r + 1) - __ldg(cu_seqlens + r);
                s += prefill_items_from(c, n, keys_of(r, n), P);
            }
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
        return s;
    };
    int cmax = one ? max(1, (L1 + 127) / 128) : 1;
    if (!one)
        for (int r = lane; r < R; r += 32)
            cmax = max(cmax, (keys_of(r, __ldg(cu_seqlens + r + 1) - __ldg(cu_seqlens + r)) + 127) / 128);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) cmax = max(cmax, __shfl_xor_sync(0xffffffffu, cmax, off));
    const int64_t k = u / Hkv;
    if (k >= count_ge(1)) return false;
    // the item's cost: the largest c with more than k items of cost >= c
    int lo = 1, hi = cmax;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (count_ge(mid) > k) lo = mid; else hi = mid - 1;
    }
    const int c = lo;
    int64_t skip = k - count_ge(c + 1);   // among the items of cost exactly c, in (r, i) order
    int64_t base = 0;
    bool found = false;
    for (int r0 = 0; r0 < R && !found; r0 += 32) {
        const int r = r0 + lane;
        int e = 0, first = 0;
        if (r < R) {
            const int n = one ? n1 : __ldg(cu_seqlens + r + 1) - __ldg(cu_seqlens + r);
            const int L = one ? L1 : keys_of(r, n);
            const int m = n > 0 ? (n + P - 1) / P : 0;
            const int ge = prefill_items_from(c, n, L, P);
            e = ge - prefill_items_from(c + 1, n, L, P);
            first = m - ge;
        }
        int64_t incl = e;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const int64_t v = __shfl_up_sync(0xffffffffu, incl, off);
            if (lane >= off) incl += v;
        }
        const bool mine = e > 0 && skip >= base + incl - e && skip < base + incl;
        const unsigned who = __ballot_sync(0xffffffffu, mine);
        if (who) {
            const int src = __ffs(who) - 1;
            const int it = first + (int)(skip - (base + incl - e));
            *r_out = __shfl_sync(0xffffffffu, r, src);
            *item_out = __shfl_sync(0xffffffffu, it, src);
            found = true;
        }
        base += __shfl_sync(0xffffffffu, incl, 31);
    }
    *h_out = (int)(u % Hkv);
    return found;
}

// PREFIX = false: suffix prefill.  CTA (request r, kv head h, query item);
//   tile X row i = query X*tpt + i / g of the item, q head h*g + i % g;
//   keys 0 .. pos(query).
// PREFIX = true: shared-prefix pass of decode.  CTA (group, kv head, member
//   item, key split); tile X row i = member X*tpt + i / g of the item; keys =
//   the split's range of the group's prefix blocks (read through the first
//   member's table row), all visible; writes unnormalised partials.
template <int D, bool PREFIX, bool TREE = false, bool FUSED = false, bool PART = false>
__global__ void __launch_bounds__(kThreads, 1)
    attn_tile_kernel(const __grid_constant__ CUtensorMap tmk, const __grid_constant__ CUtensorMap tmv,
                     const __grid_constant__ CUtensorMap tmkn, const __grid_constant__ CUtensorMap tmvn,
                     const KernelParams p) {
    using Ly = Layout<D>;
    // The private pass of grouped verification runs beside the shared-prefix
    // pass, which started it after its own wait: nothing read here is written
    // by that pass, so it waits for it only before leaving (the combine needs
    // both).  Every other mode, and a private pass with no prefix pass before
    // it, waits for the preceding kernel first.
    if (!PART || !p.after_prefix) pdl_wait();
    // The shared-prefix pass lets the split pass launch at once: it reads
    // nothing this pass writes and waits for it only before exiting.  Its
    // CTAs are launched once every CTA of this pass has started, so they take
    // the SMs this pass leaves idle at once and the others as its CTAs exit.
    if constexpr (PREFIX) pdl_trigger();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    int h = blockIdx.x % p.Hkv;
    int nq, nblk, kv_end, q_pos0 = 0, blk_off = 0, cu0 = 0, q0 = 0, m0 = 0, new_blk0 = 1 << 30, cached = 0;
    const int32_t *trow;
    if constexpr (!PREFIX) {
        int r = blockIdx.x / p.Hkv;
        int item = gridDim.y - 1 - blockIdx.y;            // heaviest items of each request first
        if (!PART && p.lpt) {
            // longest first over all requests (prefill_lpt_select)
            __shared__ int s_sel[3];
            if (warp == 0) {
                int sr = -1, si = 0, sh = 0;
                const bool ok = prefill_lpt_select(p.cu_seqlens_q, p.context_lens, (int)gridDim.x / p.Hkv, p.Hkv,
                                                   2 * p.tpt, (int64_t)blockIdx.y * gridDim.x + blockIdx.x, &sr,
                                                   &si, &sh);
                if (lane == 0) { s_sel[0] = ok ? sr : -1; s_sel[1] = si; s_sel[2] = sh; }
            }
            __syncthreads();
            if (s_sel[0] < 0) return;     // spare CTA
            r = s_sel[0]; item = s_sel[1]; h = s_sel[2];
        }
        cu0 = __ldg(p.cu_seqlens_q + r);
        const int n_r = __ldg(p.cu_seqlens_q + r + 1) - cu0;
        q0 = item * 2 * p.tpt;
        if (q0 >= n_r) {
            if constexpr (PART) pdl_wait();
            return;
        }
        nq = min(2 * p.tpt, n_r - q0);
        const int L = __ldg(p.context_lens + r);
        if (L < n_r || L > 16 * p.max_blocks) {
            if (threadIdx.x == 0) latch_error(p.err, kDevBounds);
            if constexpr (PART) pdl_wait();
            return;
        }
        cached = L - n_r;                 // keys before the request's new tokens
        if constexpr (FUSED) {
            // new keys come from k_new in whole 16-token blocks
            if (cached & 15) {
                if (threadIdx.x == 0) latch_error(p.err, kDevBounds);
                return;
            }
            new_blk0 = cached >> 4;
        }
        q_pos0 = L - n_r + q0;            // absolute position of the item's first query
        kv_end = q_pos0 + nq;             // keys [0, kv_end) are visible to some row
        if constexpr (PART) {
            // keys from the end of the group's shared blocks; positions from
            // here on count from there
            const int grp = p.request_group ? __ldg(p.request_group + r) : -1;
            blk_off = grp >= 0 ? __ldg(p.group_blocks + grp) : 0;
            // the partials of rows cu0 .. cu0 + n_r - 1 must lie in the
            // workspace, sized for num_rows tokens
            if (blk_off < 0 || blk_off * 16 > q_pos0 || cu0 < 0 || cu0 + n_r > p.num_rows) {
                if (threadIdx.x == 0) latch_error(p.err, kDevBounds);
                pdl_wait();
                return;
            }
            q_pos0 -= blk_off * 16;
            kv_end -= blk_off * 16;
        }
        nblk = (kv_end + 15) >> 4;
        trow = p.block_table + (int64_t)r * p.max_blocks;
    } else {
        const int grp = blockIdx.x / p.Hkv;
        const int gs = __ldg(p.group_start + grp);
        const int nm = __ldg(p.group_start + grp + 1) - gs;
        const int mt0 = blockIdx.y * 2 * p.tpt;
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
        nq = min(2 * p.tpt, nm - mt0);
        m0 = gs + mt0;
        // every member id of this item must be below num_requests, and the
        // table row naming the prefix blocks (the first member's, or the
        // group's own) a row of the table: thread i checks member i
        // (nq <= 256 < kThreads)
        const int r_first = p.group_row ? __ldg(p.group_row + grp) : __ldg(p.member_req + gs);
        bool bad = r_first < 0 || r_first >= (p.group_row ? p.num_table_rows : p.num_requests);
        if (threadIdx.x < nq) {
            const int rm = __ldg(p.member_req + m0 + threadIdx.x);
            bad = bad || rm < 0 || rm >= p.num_requests;
        }
        if (__syncthreads_or(bad)) {
            if (threadIdx.x == 0) latch_error(p.err, kDevBounds);
            return;
        }
        trow = p.block_table + (int64_t)r_first * p.max_blocks;
    }
    if (nblk > kMaxItemBlocks) {
        if (threadIdx.x == 0) latch_error(p.err, kDevBounds);
        if constexpr (PART) pdl_wait();
        return;
    }
    const int nkt = (kv_end + kKeys - 1) / kKeys;
    const bool has_b = nq > p.tpt;        // tile B holds at least one query
    const int rows_a = min(nq, p.tpt) * p.g;
    const int rows_b = max(0, nq - p.tpt) * p.g;
    // global q row of the item's query qi (0 <= qi < nq), q head h*g + hd
    auto q_row = [&](int qi, int hd) -> int64_t {
        if constexpr (PREFIX)
            return (int64_t)__ldg(p.member_req + m0 + qi) * p.Hq + h * p.g + hd;
        else
            return (int64_t)(cu0 + q0 + qi) * p.Hq + h * p.g + hd;
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
            mbar_init(sb + Ly::kKEmpty + 8 * i, 1);
            mbar_init(sb + Ly::kVEmpty + 8 * i, 1);
            mbar_init(sb + Ly::kSFull + 8 * i, 1);
            mbar_init(sb + Ly::kPFull + 8 * i, 128);
            mbar_init(sb + Ly::kODone + 8 * i, 1);
        }
        mbar_init(sb + Ly::kDone, 1);
        *abort = 0;
        fence_barrier_init();
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(tmem_slot), kTmemCols);
        tmem_relinquish();
    }
    // global q row of every tile row (-1: no query), looked up once; the Q
    // loads and the epilogue stores use this table.  Thread t < 256 also
    // copies tile row t of Q into shared memory (asynchronously, while the
    // block ids below are read): K-major with the 128-byte swizzle, 16-byte
    // chunk c of row i at chunk c ^ (i % 8) of its 128-byte row; rows
    // without a query are zero-filled.
    int64_t *row_idx = reinterpret_cast<int64_t *>(smem + Ly::kRowIdx);
    if (threadIdx.x < 2 * kRows) {
        const int x = threadIdx.x >> 7, i = threadIdx.x & 127;
        const int64_t qr = i < (x ? rows_b : rows_a) ? q_row(x * p.tpt + i / p.g, i % p.g) : -1;
        row_idx[threadIdx.x] = qr;
        const uint16_t *src = p.q + (qr >= 0 ? qr : 0) * D;
        const uint32_t dst_row = sb + Ly::kQ + x * Ly::kTile + i * 128;
#pragma unroll
        for (int c = 0; c < D / 8; ++c)
            cp_async16(dst_row + (c >> 3) * Ly::kHalfBytes + (((c & 7) ^ (i & 7)) << 4), src + c * 8, qr >= 0);
    }
    // the item's physical block ids, checked once, for the producer
    int32_t *blk_ids = reinterpret_cast<int32_t *>(smem + Ly::kBlkIds);
    for (int b = threadIdx.x - 2 * kRows; b >= 0 && b < nblk; b += kThreads - 2 * kRows) {
        int32_t id = __ldg(trow + blk_off + b);
        if (id < 0 || id >= p.num_blocks_pool) {
            latch_error(p.err, kDevBounds);
            id = 0;
        }
        blk_ids[b] = id;
    }
    __syncthreads();
    // The producer issues the K/V loads of the first two key tiles now, so
    // that their latency overlaps the Q copies still in flight.
    auto issue_kv = [&](int j, bool k_side) {
        const int s = j & 1;
        const int b0 = j * 8, nb = min(8, nblk - b0);
        const uint32_t bytes = (uint32_t)nb * Ly::kHalves * 2048u;
        const uint32_t bar = sb + (k_side ? Ly::kKFull : Ly::kVFull) + 8 * s;
        const uint32_t dst = sb + (k_side ? Ly::kK0 : Ly::kV0) + s * Ly::kTile;
        // Warp 0, all lanes: lane 0 posts the byte count, then lane l issues
        // box l (block l / kHalves, half l % kHalves).  One thread issuing
        // a tile's 16-32 boxes in turn measured 7 % slower on prefill (the
        // next tiles' copies started later) and 6 us slower on the decode
        // step's shared-prefix pass.
        if (lane == 0) mbar_arrive_expect_tx(bar, bytes);
        __syncwarp();
        // cached blocks from the pool; with the fused write, the request's
        // new blocks (from new_blk0 on) from k_new / v_new, 16 tokens each
        const int nb_pool = FUSED ? min(nb, max(0, new_blk0 - b0)) : nb;
        if (lane < nb * Ly::kHalves) {
            const int b = lane / Ly::kHalves, hf = lane % Ly::kHalves;
            if (b < nb_pool)
                tma_load_4d(dst + hf * Ly::kHalfBytes + b * 2048, k_side ? &tmk : &tmv, hf * 64, 0, h,
                            blk_ids[b0 + b], bar);
            else if constexpr (FUSED)
                tma_load_3d(dst + hf * Ly::kHalfBytes + b * 2048, k_side ? &tmkn : &tmvn, hf * 64, h,
                            cu0 + (b0 + b) * 16 - cached, bar);
        }
    };
    const int early = min(2, nkt);
    if (warp == 0) {
        if (lane == 0) {
            prefetch_tmap(&tmk);
            prefetch_tmap(&tmv);
            if constexpr (FUSED) {
                prefetch_tmap(&tmkn);
                prefetch_tmap(&tmvn);
            }
        }
        for (int j = 0; j < early; ++j) {
            issue_kv(j, true);
            issue_kv(j, false);
        }
    }
    // the Q rows are in shared memory once every thread's copies have landed
    cp_async_wait_all();
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp < 4) {
      if (warp == 0) {
        // ------------------------------------------------------------ producer
        // the whole warp: key tiles 0 and 1 were issued before the Q load
        int issued = early, issued_k_only = 0;
        for (int j = early; j < nkt; ++j) {
            const int s = j & 1;
            // K(j) may replace K(j-2) once both Q.K MMAs of tile j-2 are
            // done; V(j) replaces V(j-2) after both P.V MMAs of tile j-2
            if (!warp_wait(sb + Ly::kKEmpty + 8 * s, ((j >> 1) - 1) & 1, abort)) break;
            issue_kv(j, true);
            if (!warp_wait(sb + Ly::kVEmpty + 8 * s, ((j >> 1) - 1) & 1, abort)) {
                issued_k_only = j + 1;
                break;
            }
            issue_kv(j, false);
            issued = j + 1;
        }
        if (lane == 0) {
            // let this CTA's own copies land before its shared memory is released
            int quiet = 0;
            for (int j = max(0, issued - 2); j < issued; ++j) {
                mbar_wait(sb + Ly::kKFull + 8 * (j & 1), (j >> 1) & 1, &quiet, kDrainLimitNs);
                mbar_wait(sb + Ly::kVFull + 8 * (j & 1), (j >> 1) & 1, &quiet, kDrainLimitNs);
            }
            if (issued_k_only) {
                const int j = issued_k_only - 1;
                mbar_wait(sb + Ly::kKFull + 8 * (j & 1), (j >> 1) & 1, &quiet, kDrainLimitNs);
            }
            if constexpr (FUSED) {
                // Whole blocks of the item's own new tokens are in the last
                // two stages (an item has at most 64 tokens, so its blocks lie
                // in the last two key tiles, whose stages are never reloaded):
                // store them into the pool from there.  Blocks only partly
                // the item's go by plain stores (warps 2-3).
                if (!*abort && issued == nkt) {
                    const int bfirst = (q_pos0 + 15) >> 4, blast = kv_end >> 4;   // [bfirst, blast)
                    for (int bi = bfirst; bi < blast; ++bi) {
                        const int j = bi >> 3, bb = bi & 7, st = j & 1;
                        for (int hf = 0; hf < Ly::kHalves; ++hf) {
                            const uint32_t off = st * Ly::kTile + hf * Ly::kHalfBytes + bb * 2048;
                            tma_store_4d(&tmk, sb + Ly::kK0 + off, hf * 64, 0, h, blk_ids[bi]);
                            tma_store_4d(&tmv, sb + Ly::kV0 + off, hf * 64, 0, h, blk_ids[bi]);
                        }
                    }
                    bulk_commit();
                    bulk_wait();
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        // Lane 0 alone runs the issue loop: tcgen05.mma and commit are
        // per-thread, and warp-wide waits and syncs around every group of
        // MMAs measured 6 % slower on prefill.
        if (lane == 0) {
        const uint32_t id_qk = idesc_bf16_f32(kRows, kKeys, false);
        const uint32_t id_pv = idesc_bf16_f32(kRows, D, true);
        bool ok = true;
        // S_X = Q_X . K(j)^T; the last tile to read K(j) releases its stage
        auto issue_qk = [&](int x, int j) {
            tc_fence_after();
            // one descriptor per operand tile; a k-step adds its byte offset / 16
            // to the start-address field (shared addresses < 256 KiB: no carry)
            const uint64_t qd = smem_desc_sw128(sb + Ly::kQ + x * Ly::kTile, 16, 1024);
            const uint64_t kd = smem_desc_sw128(sb + Ly::kK0 + (j & 1) * Ly::kTile, 16, 1024);
            const uint32_t dt = tmem + x * 128;
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk) {
                const uint32_t off = ((kk >> 2) * Ly::kHalfBytes + (kk & 3) * 32) >> 4;
                mma_ss(dt, qd + off, kd + off, id_qk, kk > 0 ? 1u : 0u);
            }
            mma_commit(sb + Ly::kSFull + 8 * x);
            if (x == 1 || !has_b) mma_commit(sb + Ly::kKEmpty + 8 * (j & 1));
        };
        // O_X += P_X . V(j)
        auto issue_pv = [&](int x, int j) {
            tc_fence_after();
            // V is N-major (head dim contiguous): LBO = stride between the
            // 64-wide head-dim halves, SBO = stride between 8-key groups; a
            // 16-key step advances the start address by 2 KiB
            const uint64_t vd = smem_desc_sw128(sb + Ly::kV0 + (j & 1) * Ly::kTile, Ly::kHalfBytes, 1024);
            const uint32_t dt = tmem + 256 + x * 128, at = tmem + x * 128;
#pragma unroll
            for (int kk = 0; kk < kKeys / 16; ++kk)
                mma_ts(dt, at + kk * 8, vd + (uint64_t)((kk * 2048) >> 4), id_pv, (j > 0 || kk > 0) ? 1u : 0u);
            if (j == nkt - 1) mma_commit(sb + Ly::kODone + 8 * x);
        };
        if (wait_bar(sb + Ly::kKFull, 0, abort)) {
            issue_qk(0, 0);
            if (has_b) issue_qk(1, 0);
        } else {
            ok = false;
        }
        for (int j = 0; j < nkt && ok; ++j) {
            const int s = j & 1;
            if (!wait_bar(sb + Ly::kVFull + 8 * s, (j >> 1) & 1, abort)) { ok = false; break; }
            if (j == nkt - 1) {
                // keys past the item's range: p = 0 there, but their V rows may
                // hold anything (0 * NaN = NaN in the MMA), so clear them
                const int first = kv_end - j * kKeys;
                uint8_t *vs = smem + Ly::kV0 + s * Ly::kTile;
                for (int row = first; row < kKeys; ++row)
                    for (int hf = 0; hf < Ly::kHalves; ++hf) {
                        uint4 *d4 = reinterpret_cast<uint4 *>(vs + hf * Ly::kHalfBytes + row * 128);
#pragma unroll
                        for (int c = 0; c < 8; ++c) d4[c] = make_uint4(0, 0, 0, 0);
                    }
                fence_proxy_async_smem();
            }
            const bool more = j + 1 < nkt;
            // tile A: P.V(j) as soon as P is ready, then Q.K(j+1) into the S
            // it just consumed once K(j+1) has landed (measured: K(j+1)
            // arrives up to ~0.5 us after P(j); waiting for it before P.V(j)
            // kept the tensor core idle for that long every key tile)
            if (!wait_bar(sb + Ly::kPFull, j & 1, abort)) { ok = false; break; }
            issue_pv(0, j);
            if (more && !wait_bar(sb + Ly::kKFull + 8 * (s ^ 1), ((j + 1) >> 1) & 1, abort)) {
                ok = false;
                break;
            }
            if (more) issue_qk(0, j + 1);
            if (has_b) {
                if (!wait_bar(sb + Ly::kPFull + 8, j & 1, abort)) { ok = false; break; }
                issue_pv(1, j);
                if (more) issue_qk(1, j + 1);
            }
            mma_commit(sb + Ly::kVEmpty + 8 * s);    // V(j) consumed
        }
        // all MMAs issued by this thread must finish before TMEM is freed
        mma_commit(sb + Ly::kDone);
        int quiet = 0;
        mbar_wait(sb + Ly::kDone, 0, &quiet, kDrainLimitNs);
        }
        __syncwarp();
      } else if constexpr (FUSED) {
        {
            // ------------------------------------------------ store (warps 2-3)
            // the K/V rows of this item's own queries (kv head h) that lie in
            // blocks only partly the item's (the producer stores the whole
            // ones by TMA); every new token belongs to exactly one item per head
            constexpr int CPR = D / 8;
            const int t0 = threadIdx.x - 64;
            const int head_rows = min(nq, ((q_pos0 + 15) & ~15) - q_pos0);   // before the first whole block
            const int tail0 = max(head_rows, (kv_end & ~15) - q_pos0);       // from the last partial block
            const int n_plain = head_rows + (nq - tail0);
            for (int i = t0; i < n_plain * 2 * CPR; i += 64) {
                const int k = i / (2 * CPR), rem = i - k * 2 * CPR;
                const int qi = k < head_rows ? k : tail0 + (k - head_rows);
                const int isv = rem >= CPR, c = rem - isv * CPR;
                const int pos = q_pos0 + qi;
                const int64_t src = ((int64_t)(cu0 + q0 + qi) * p.Hkv + h) * D + c * 8;
                const int64_t dst = (((int64_t)blk_ids[pos >> 4] * p.Hkv + h) * 16 + (pos & 15)) * D + c * 8;
                const uint4 v = ldg_stream((isv ? p.v_new : p.k_new) + src);
                *reinterpret_cast<uint4 *>((isv ? p.v_cache : p.k_cache) + dst) = v;
            }
        }
      }
    } else {
        // ------------------------------------------------------------ softmax
        const int x = (warp - 4) >> 2;                // tile A (warps 4-7) or B (8-11)
        const int quarter = warp & 3;                 // TMEM lanes this warp may touch
        const int row = quarter * 32 + lane;
        const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;
        const uint32_t s_addr = tmem + lane_off + x * 128;
        const uint32_t o_addr = tmem + lane_off + 256 + x * 128;
        const int rows_x = x ? rows_b : rows_a;
        const bool valid = row < rows_x;
        const int qi = x * p.tpt + row / p.g;         // query of the item behind this row
        // last visible key (item-local numbering of the key range)
        const int pos = (!PREFIX && valid) ? q_pos0 + qi : kv_end - 1;
        // tree-shaped drafts: new token qi sees the request's new tokens whose
        // bits are set in its mask (its ancestors and itself), all context keys
        constexpr bool tree = !PREFIX && TREE;
        const int new0 = q_pos0 - q0;                 // position of the request's first new token
        const unsigned long long tmask = (tree && valid) ? __ldg(p.tree_mask + cu0 + q0 + qi) : ~0ull;
        const bool active = (x == 0) || has_b;
        float m = -INFINITY, l = 0.f;
        bool ok = active;
        for (int j = 0; j < nkt && ok; ++j) {
            if (!warp_wait(sb + Ly::kSFull + 8 * x, j & 1, abort)) { ok = false; break; }
            tc_fence_after();
            uint32_t sr[4][32];
#pragma unroll
            for (int c = 0; c < 4; ++c) tmem_ld32(s_addr + c * 32, sr[c]);
            tmem_wait_ld();
            const int lim = pos - j * kKeys;          // keys with column index <= lim are visible
            const int d0 = new0 - j * kKeys;          // column of the first new token (may be < 0)
            const bool tree_tile = tree && d0 < kKeys;
            const bool all_visible = __all_sync(0xffffffffu, lim >= kKeys - 1 && !tree_tile);
            if (!all_visible) {
#pragma unroll
                for (int c = 0; c < 4; ++c)
#pragma unroll
                    for (int e = 0; e < 32; ++e) {
                        const int col = c * 32 + e;
                        bool vis = col <= lim;
                        // col - d0 <= pos - new0 < 64 whenever col <= lim
                        if (vis && tree_tile && col >= d0) vis = (tmask >> (col - d0)) & 1ull;
                        if (!vis) sr[c][e] = __float_as_uint(-INFINITY);
                    }
            }
            // The first tile finds its row max before the pass.  Later tiles
            // compute P against the running max m, however stale: the same m
            // normalises O and the row sum, so the result is exact as long as
            // no P overflows.  The row sum bounds every P of the tile: a sum
            // of at most 2^15 means every P <= 2^15 (harmless in bf16 and in
            // the fp32 accumulators); above it, the row's max is found, O is
            // rescaled in TMEM and the pass redone with the new max (after
            // which the sum is at most 128).
            if (j == 0) m = row_max(sr) * p.scale_log2;   // scale > 0 commutes with max
            float tile_sum = softmax_pass(sr, p.scale_log2, m, s_addr);
            const bool grow = tile_sum > 32768.0f;
            if (__any_sync(0xffffffffu, grow)) {
                // P.V(j-1) has completed: Q.K(j), which produced S(j), was issued after it
                const float m_new = grow ? fmaxf(m, row_max(sr) * p.scale_log2) : m;
                const float alpha = fast_exp2(m - m_new);
                tmem_wait_st();
#pragma unroll 1
                for (int c = 0; c < D / 32; ++c) {
                    uint32_t o[32];
                    tmem_ld32(o_addr + c * 32, o);
                    tmem_wait_ld();
#pragma unroll
                    for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
                    tmem_st32(o_addr + c * 32, o);
                }
                l *= alpha;
                m = m_new;
                tile_sum = softmax_pass(sr, p.scale_log2, m, s_addr);
            }
            l += tile_sum;
            tmem_wait_st();
            tc_fence_before();
            mbar_arrive(sb + Ly::kPFull + 8 * x);
        }
        if (ok && warp_wait(sb + Ly::kODone + 8 * x, 0, abort)) {
            tc_fence_after();
            // Epilogue through shared memory: every MMA reading Q_X has
            // finished, so this tile's Q buffer holds the rows while they are
            // turned from one-row-per-thread into whole-row 16-byte stores.
            // Staged rows are RB = 2*D bytes (128 rows fill the Q tile); 16-byte
            // chunk c of row i sits at chunk c ^ (i % CPR), so both the
            // per-row writes and the per-chunk reads avoid bank conflicts.
            uint8_t *stage = smem + Ly::kQ + x * Ly::kTile;
            constexpr int RB = 2 * D, CPR = RB / 16, RPI = 32 / CPR;
            static_assert(kRows * RB == Ly::kTile, "staging rows must fill the Q tile");
            auto row_chunk = [&](int i, int c) -> uint4 * {
                return reinterpret_cast<uint4 *>(stage + i * RB + ((c ^ (i & (CPR - 1))) << 4));
            };
            // drain the staged rows of this warp: lane -> (row, chunk)
            auto drain = [&](auto &&dst_of) {
                __syncwarp();
#pragma unroll
                for (int it = 0; it < 32 / RPI; ++it) {
                    const int i = quarter * 32 + it * RPI + lane / CPR, c = lane % CPR;
                    const uint4 v = *row_chunk(i, c);
                    if (i < rows_x) *dst_of(i, c) = v;
                }
                __syncwarp();
            };
            if constexpr (!PREFIX && !PART) {
                const float inv = 1.0f / l;
                // bf16 rows of D values: D * 2 bytes <= RB
#pragma unroll
                for (int c = 0; c < D / 32; ++c) {
                    uint32_t o[32];
                    tmem_ld32(o_addr + c * 32, o);
                    tmem_wait_ld();
#pragma unroll
                    for (int v = 0; v < 4; ++v) {
                        uint4 w;
                        w.x = pack_bf16x2(__uint_as_float(o[8 * v + 0]) * inv, __uint_as_float(o[8 * v + 1]) * inv);
                        w.y = pack_bf16x2(__uint_as_float(o[8 * v + 2]) * inv, __uint_as_float(o[8 * v + 3]) * inv);
                        w.z = pack_bf16x2(__uint_as_float(o[8 * v + 4]) * inv, __uint_as_float(o[8 * v + 5]) * inv);
                        w.w = pack_bf16x2(__uint_as_float(o[8 * v + 6]) * inv, __uint_as_float(o[8 * v + 7]) * inv);
                        *row_chunk(row, 4 * c + v) = w;
                    }
                }
                drain([&](int i, int c) {
                    return reinterpret_cast<uint4 *>(p.out + row_idx[x * kRows + i] * D) + c;
                });
                if (valid && p.lse) p.lse[row_idx[x * kRows + row]] = (m + __log2f(l)) * 0.69314718055994530942f;
            } else {
                // unnormalised fp32 partial (of key split blockIdx.z, or the
                // private part), merged by the combine; staged D/2 columns
                // (RB bytes) at a time
                const int part = PREFIX ? (int)blockIdx.z : p.private_part;
#pragma unroll
                for (int hc = 0; hc < 2; ++hc) {
#pragma unroll
                    for (int cc = 0; cc < D / 64; ++cc) {
                        uint32_t o[32];
                        tmem_ld32(o_addr + hc * (D / 2) + cc * 32, o);
                        tmem_wait_ld();
#pragma unroll
                        for (int v = 0; v < 8; ++v)
                            *row_chunk(row, 8 * cc + v) = make_uint4(o[4 * v], o[4 * v + 1], o[4 * v + 2], o[4 * v + 3]);
                    }
                    drain([&](int i, int c) {
                        const int64_t slot = row_idx[x * kRows + i] * p.parts_per_head + part;
                        return reinterpret_cast<uint4 *>(p.o_part + slot * D + hc * (D / 2)) + c;
                    });
                }
                if (valid) p.ml_part[row_idx[x * kRows + row] * p.parts_per_head + part] = make_float2(m, l);
                if constexpr (PART) {
                    // the token's part counts for the combine: one private
                    // part, and the prefix partials of its group
                    if (valid && row % p.g == 0) {
                        const int n_pre = blk_off > 0 ? min((blk_off + p.blocks_per_part - 1) / p.blocks_per_part,
                                                            p.prefix_parts)
                                                      : 0;
                        p.nparts[(int64_t)(cu0 + q0 + qi) * p.Hkv + h] = 1 | (n_pre << 16);
                    }
                }
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
    if constexpr (PART) pdl_wait();
}

}  // namespace

template <int D, bool PREFIX, bool TREE = false, bool FUSED = false, bool PART = false>
static cudaError_t launch_tile_kernel(dim3 grid, const CUtensorMap &tk, const CUtensorMap &tv,
                                      const CUtensorMap &tkn, const CUtensorMap &tvn,
                                      const KernelParams &p, cudaStream_t stream) {
    // the d = 64 tiles are smaller; ask for the d = 128 footprint anyway so
    // one CTA owns an SM (its 512 TMEM columns never wait on a neighbour)
    static SmemLimit limit;
    cudaError_t e = limit.ensure(reinterpret_cast<const void *>(attn_tile_kernel<D, PREFIX, TREE, FUSED, PART>),
                                 Layout<128>::kDynSmem);
    if (e != cudaSuccess) return e;
    return launch_pdl(attn_tile_kernel<D, PREFIX, TREE, FUSED, PART>, grid, dim3(kThreads), Layout<128>::kDynSmem, stream,
                      tk, tv, tkn, tvn, p);
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
    p.tree_mask = a.tree_mask;
    p.fused = a.k_new != nullptr;
    p.k_new = static_cast<const uint16_t *>(a.k_new);
    p.v_new = static_cast<const uint16_t *>(a.v_new);
    p.k_cache = static_cast<uint16_t *>(a.k_cache);
    p.v_cache = static_cast<uint16_t *>(a.v_cache);
    // without the fused write the new-token maps are never read
    const CUtensorMap &tkn = p.fused ? *a.tmap_kn : *a.tmap_k, &tvn = p.fused ? *a.tmap_vn : *a.tmap_v;
    const int items = (a.max_seqlen_q + 2 * p.tpt - 1) / (2 * p.tpt);
    if (items <= 0 || a.R <= 0) return cudaSuccess;
    if (items > 65535) return cudaErrorInvalidConfiguration;
    dim3 grid((unsigned)(a.R * a.Hkv), (unsigned)items);
    // Few waves: a wave's worth of light CTAs at the end costs a whole CTA's
    // time; taking the items longest first packs the last wave (measured on
    // the Qwen chunks: 3.2 waves, 315 -> 255 us predicted from the CTAs' own
    // durations).  Many waves, or many requests (the selection's cost grows
    // with them): launch order.
    p.lpt = (int64_t)grid.x * grid.y <= 8LL * a.num_sms && a.R <= 256;
    if (tr) tr->begin(kKernelPrefill, stream);
    cudaError_t e;
    if (p.fused)
        e = a.d == 128 ? launch_tile_kernel<128, false, false, true>(grid, *a.tmap_k, *a.tmap_v, tkn, tvn, p, stream)
                       : launch_tile_kernel<64, false, false, true>(grid, *a.tmap_k, *a.tmap_v, tkn, tvn, p, stream);
    else if (p.tree_mask)
        e = a.d == 128 ? launch_tile_kernel<128, false, true>(grid, *a.tmap_k, *a.tmap_v, tkn, tvn, p, stream)
                       : launch_tile_kernel<64, false, true>(grid, *a.tmap_k, *a.tmap_v, tkn, tvn, p, stream);
    else
        e = a.d == 128 ? launch_tile_kernel<128, false>(grid, *a.tmap_k, *a.tmap_v, tkn, tvn, p, stream)
                       : launch_tile_kernel<64, false>(grid, *a.tmap_k, *a.tmap_v, tkn, tvn, p, stream);
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
    const int mitems = (a.max_group_members + 2 * p.tpt - 1) / (2 * p.tpt);
    if (mitems <= 0 || L.prefix_parts <= 0) return cudaSuccess;
    if (mitems > 65535) return cudaErrorInvalidConfiguration;
    dim3 grid((unsigned)(a.num_groups * L.Hkv), (unsigned)mitems, (unsigned)L.prefix_parts);
    // The split pass starts beside this pass (see the trigger in the kernel).
    // With a grid that leaves at least a quarter of the SMs free, the split
    // pass's grid covers just those; with one that fills the device, its grid
    // covers every SM and its CTAs take the SMs as this pass's CTAs exit
    // (measured on clock-stamped steps against starting it after this pass:
    // Llama-3-70B decode 314 -> 285 us, Qwen2.5-7B mixed decode 99.5 -> 85 us).
    p.group_row = a.group_row;
    p.num_table_rows = a.num_table_rows;
    if (tr) tr->begin(kKernelDecodePrefix, stream);
    cudaError_t e = L.d == 128
                        ? launch_tile_kernel<128, true>(grid, *a.tmap_k, *a.tmap_v, *a.tmap_k, *a.tmap_v, p, stream)
                        : launch_tile_kernel<64, true>(grid, *a.tmap_k, *a.tmap_v, *a.tmap_k, *a.tmap_v, p, stream);
    if (tr) tr->end(kKernelDecodePrefix, stream);
    return e;
}

cudaError_t launch_verify_grouped(const DecodeLayout &L, const DecodeArgs &a, const PrefillArgs &pa,
                                  const int32_t *request_group, cudaStream_t stream, Tracer *tr) {
    // the shared prefixes, once per group: rows = draft tokens x heads
    const bool prefix = L.prefix_parts > 0 && a.num_groups > 0 && request_group;
    cudaError_t e = prefix ? launch_decode_prefix(L, a, pa.num_blocks_pool, stream, tr) : cudaSuccess;
    if (e != cudaSuccess) return e;
    // each request's private keys and drafts, under the draft masks, into
    // the private part slot (beside the prefix pass when it leaves SMs free)
    KernelParams p{};
    p.q = static_cast<const uint16_t *>(pa.q);
    p.cu_seqlens_q = pa.cu_seqlens_q;
    p.context_lens = pa.context_lens;
    p.block_table = pa.block_table;
    p.max_blocks = pa.max_blocks;
    p.Hq = pa.Hq; p.Hkv = pa.Hkv; p.g = pa.Hq / pa.Hkv; p.tpt = kRows / p.g;
    p.num_blocks_pool = pa.num_blocks_pool;
    p.scale_log2 = pa.scale_log2;
    p.err = pa.err;
    p.tree_mask = pa.tree_mask;
    p.group_blocks = a.group_blocks;
    p.request_group = prefix ? request_group : nullptr;   // no prefix pass: every key here
    p.after_prefix = prefix ? 1 : 0;
    p.blocks_per_part = L.prefix_blocks_per_part;
    p.prefix_parts = L.prefix_parts;
    p.parts_per_head = L.parts_per_head;
    p.private_part = L.prefix_parts;
    p.o_part = reinterpret_cast<float *>(static_cast<char *>(a.ws) + L.off_o);
    p.ml_part = reinterpret_cast<float2 *>(static_cast<char *>(a.ws) + L.off_ml);
    p.nparts = reinterpret_cast<int32_t *>(static_cast<char *>(a.ws) + L.off_nparts);
    p.num_rows = L.R;
    const int items = (pa.max_seqlen_q + 2 * p.tpt - 1) / (2 * p.tpt);
    if (items <= 0 || pa.R <= 0) return cudaSuccess;
    if (items > 65535) return cudaErrorInvalidConfiguration;
    dim3 grid((unsigned)(pa.R * pa.Hkv), (unsigned)items);
    if (tr) tr->begin(kKernelPrefill, stream);
    e = pa.d == 128 ? launch_tile_kernel<128, false, true, false, true>(grid, *pa.tmap_k, *pa.tmap_v, *pa.tmap_k,
                                                                         *pa.tmap_v, p, stream)
                    : launch_tile_kernel<64, false, true, false, true>(grid, *pa.tmap_k, *pa.tmap_v, *pa.tmap_k,
                                                                        *pa.tmap_v, p, stream);
    if (tr) tr->end(kKernelPrefill, stream);
    if (e != cudaSuccess) return e;
    return launch_decode_combine(L, a, stream, tr);
}

}  // namespace pkv
