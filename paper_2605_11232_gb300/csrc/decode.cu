// decode.cu -- split-KV paged decode attention (one query token per request).
//
// The decode step of the paper's short structured outputs (Sec. 5.3) reads
// each request's whole block list (PagedAttention, Sec. 2 / Sec. 5.4) for one
// query token.  With GQA the g q-heads of a kv head share every K/V row, so
// the arithmetic intensity is ~g FLOP per byte: HBM-bound once the dot
// products run on tensor cores.
//
// Work split ("pieces").  The private blocks of all (request, kv head) pairs
// form one stream of W blocks, segment (r, h) after segment.  Warp w of the
// grid takes the contiguous range [w*per, (w+1)*per) of that stream, so every
// warp moves the same number of bytes whatever the length mix; a warp whose
// range crosses segment boundaries emits one unnormalised partial (O, m, l)
// per segment it touches.  The combine kernel merges a head's partials with
// log-sum-exp weights.  The grid covers the SMs the shared-prefix pass leaves
// free (all of them without one), so all warps start together and end
// together; beside a prefix pass that fills the device it covers every SM,
// its CTAs starting as the prefix pass's CTAs exit.
//
// Data path (per warp).  The (block, kv head) K and V tiles of the warp's
// range are copied by TMA, with the 128-byte swizzle, into a ring of stages
// in shared memory, issued by the warp itself a few blocks ahead of the one
// it computes on; the ring runs on across piece boundaries, and the piece
// metadata (request, head, shared-block offset, block ids) is looked up ahead
// of the copies, so a new segment costs no pipeline restart.
//
// Inner loop (one 16-token block per step):
//   S^T[16 keys x 8 heads] = K_blk[16 x d] . Q^T[d x 8]   (mma m16n8k16, A = K)
//   online softmax per head column (shuffles across the 8 row groups)
//   O^T[d x 8] += V_blk^T[d x 16] . P^T[16 x 8]           (A = V^T, B = P^T)
// A fragments come from the swizzled stages by ldmatrix (V through its
// transposing form); the S^T accumulator becomes the P^T operand through one
// movmatrix transpose per 8x8 quadrant.
//
// Fused write.  With the query tokens' own K/V given (paged_attn_decode_append),
// the warp that reaches a request's last block stores the new row (position
// L - 1) into the pool and over the stale row of its shared-memory stage
// before computing on it, so no separate cache-write kernel precedes the pass.
#include <math.h>

#include <algorithm>

#include "pkv_device.cuh"
#include "pkv_internal.h"
#include "tc_ptx.cuh"

namespace pkv {

namespace {

using namespace tc;

constexpr int kWarps = 8;
constexpr int kThreads = kWarps * 32;
constexpr uint64_t kWaitLimitNs = 2000000000ull;
constexpr uint64_t kDrainLimitNs = 200000000ull;

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2,
                                        uint32_t &r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2,
                                          uint32_t &r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

// Byte offset of 16-byte chunk c (head-dim elements 8c..8c+7) of key row
// `row` inside a (block, head) tile as TMA lays it out: 64-column boxes of
// 16 rows x 128 bytes, chunk position XORed with row % 8 (128-byte swizzle).
__device__ __forceinline__ uint32_t tile_off(int row, int c) {
    return (uint32_t)((c >> 3) * 2048 + row * 128 + (((c & 7) ^ (row & 7)) << 4));
}

// What the producer records for each stage when it issues the copies.
struct SlotDesc {
    int32_t r, h;
    int32_t phys;      // physical block id
    int32_t info;      // valid keys | kFirst | kLast | kWrite | kSegFirst
    int32_t part;      // part slot of the piece's partial
    int32_t nparts;    // part-count word of the segment (private | prefix << 16)
    int32_t pad0, pad1;
};
constexpr int32_t kValidMask = 31;
constexpr int32_t kFirst = 1 << 8;      // first block of a piece: reset the state, new Q
constexpr int32_t kLast = 1 << 9;       // last block of a piece: emit the partial
constexpr int32_t kWrite = 1 << 10;     // holds the request's query token: store k_new / v_new
constexpr int32_t kSegFirst = 1 << 11;  // the piece starts the segment: write its part counts
constexpr int32_t kWriteSoon = 1 << 12; // first block of a piece that ends with kWrite

template <int D>
struct SoftmaxState {
    float m[2];   // running max (base 2, scaled) of heads 2*(lane%4) + {0, 1}
    float l[2];   // thread-partial sums
    float o[D / 16][4];
};

// One 16-key block from a stage: K tile at kb, V tile at vb (shared addresses).
template <int D>
__device__ __forceinline__ void attend_block(SoftmaxState<D> &st, uint32_t kb, uint32_t vb,
                                             const uint32_t (&qf)[D / 16][2], int lane, int valid,
                                             float scale_log2) {
    float sacc[4] = {0.f, 0.f, 0.f, 0.f};
    {
        // matrices (keys 0-7 | 8-15) x (head-dim chunk 2kk | 2kk+1): A fragment of K
        const int row = (lane & 7) + ((lane >> 3) & 1) * 8;
        const int hi = lane >> 4;
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
            uint32_t a0, a1, a2, a3;
            ldsm_x4(kb + tile_off(row, 2 * kk + hi), a0, a1, a2, a3);
            mma_bf16_16816(sacc, a0, a1, a2, a3, qf[kk][0], qf[kk][1]);
        }
    }
    // thread (lane): keys lane/4 and lane/4 + 8, heads 2*(lane%4) + {0, 1}
    const int key0 = lane >> 2, key1 = key0 + 8;
    const bool ok0 = key0 < valid, ok1 = key1 < valid;
    const float s00 = ok0 ? sacc[0] * scale_log2 : -INFINITY;
    const float s01 = ok0 ? sacc[1] * scale_log2 : -INFINITY;
    const float s10 = ok1 ? sacc[2] * scale_log2 : -INFINITY;
    const float s11 = ok1 ? sacc[3] * scale_log2 : -INFINITY;
    float mx0 = fmaxf(s00, s10), mx1 = fmaxf(s01, s11);
#pragma unroll
    for (int off = 4; off < 32; off <<= 1) {
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, off));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, off));
    }
    // mn is finite: every processed block has at least one valid key
    const float mn0 = fmaxf(st.m[0], mx0), mn1 = fmaxf(st.m[1], mx1);
    const float a0 = fast_exp2(st.m[0] - mn0), a1 = fast_exp2(st.m[1] - mn1);
    st.m[0] = mn0;
    st.m[1] = mn1;
    const float p00 = fast_exp2(s00 - mn0), p10 = fast_exp2(s10 - mn0);
    const float p01 = fast_exp2(s01 - mn1), p11 = fast_exp2(s11 - mn1);
    st.l[0] = st.l[0] * a0 + (p00 + p10);
    st.l[1] = st.l[1] * a1 + (p01 + p11);
#pragma unroll
    for (int i = 0; i < D / 16; ++i) {
        st.o[i][0] *= a0;
        st.o[i][2] *= a0;
        st.o[i][1] *= a1;
        st.o[i][3] *= a1;
    }
    // P^T fragments: transpose the two 8x8 quadrants (keys 0-7, 8-15) of P
    const uint32_t t0 = movmatrix_trans(pack_bf16x2(p00, p01));
    const uint32_t t1 = movmatrix_trans(pack_bf16x2(p10, p11));
    {
        // matrices (head-dim chunk 2mt | 2mt+1) x (keys 0-7 | 8-15) of V^T,
        // read from V's key rows by the transposing ldmatrix
        const int j = lane >> 3, r = lane & 7;
        const int key = 8 * (j >> 1) + r;
#pragma unroll
        for (int mt = 0; mt < D / 16; ++mt) {
            uint32_t v0, v1, v2, v3;
            ldsm_x4_t(vb + tile_off(key, 2 * mt + (j & 1)), v0, v1, v2, v3);
            mma_bf16_16816(st.o[mt], v0, v1, v2, v3, t0, t1);
        }
    }
}

// Q fragments (B operand of S^T = K.Q^T) from a stage's copy of the g q-head
// rows of (request, kv head): thread (lane) gets head lane/4, head-dim
// elements 16kk + 2(lane%4) + {0, 1} and + 8.  Rows g..7 of the area hold
// stale data: those heads' columns of S^T, P^T and O^T are never written out
// (an MMA column depends on its own B column only).
template <int D>
__device__ __forceinline__ void load_q_smem(uint32_t (&qf)[D / 16][2], uint32_t qa, int lane) {
    // matrices: head rows 0-7 x head-dim chunks c0 .. c0+3 (two k-steps)
    const uint32_t row = qa + (uint32_t)(lane & 7) * (D * 2);
#pragma unroll
    for (int kk = 0; kk < D / 16; kk += 2)
        ldsm_x4(row + (uint32_t)(2 * kk + (lane >> 3)) * 16, qf[kk][0], qf[kk][1], qf[kk + 1][0], qf[kk + 1][1]);
}

// Block-wide plan: P[r] = sum of the private block counts of requests < r,
// P[R] = their total; Ls[r] = context_lens[r] when Ls is not null;
// *max_n_out = the largest count.
__device__ void build_plan(int32_t *P, int32_t *Ls, int32_t R, const int32_t *__restrict__ context_lens,
                           const int32_t *__restrict__ group_of_req,
                           const int32_t *__restrict__ group_blocks, int32_t num_groups,
                           int32_t max_blocks, int32_t *max_n_out, int *err) {
    __shared__ int32_t warp_tot[kWarps];
    __shared__ int32_t warp_max[kWarps];
    __shared__ int32_t s_gb[kThreads];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    // Up to kThreads groups: their shared block counts go to shared memory,
    // loaded beside each thread's first request, so that no load waits on
    // another.  More groups: a dependent load per request.
    const bool gb_smem = num_groups <= kThreads;
    if (num_groups > 0 && gb_smem && tid < num_groups) s_gb[tid] = __ldg(group_blocks + tid);
    int32_t L0 = 0, gi0 = -1;
    if (tid < R) {
        L0 = __ldg(context_lens + tid);
        if (num_groups > 0) gi0 = __ldg(group_of_req + tid);
    }
    __syncthreads();
    // private block counts, request r on thread r % kThreads (independent
    // loads, in flight together), kept in P for now
    for (int r = tid; r < R; r += kThreads) {
        const int32_t L = r == tid ? L0 : __ldg(context_lens + r);
        int32_t nblk = (L + 15) >> 4;
        if (nblk > max_blocks) {   // context longer than the table row
            latch_error(err, kDevBounds);
            nblk = max_blocks;
        }
        int32_t sh = 0;
        if (num_groups > 0) {
            const int32_t gi = r == tid ? gi0 : __ldg(group_of_req + r);
            if (gi >= 0 && gi < num_groups) sh = gb_smem ? s_gb[gi] : __ldg(group_blocks + gi);
        }
        int32_t n = nblk - sh;
        if (L < 1 || n < 1 || sh < 0) {   // decode needs a private tail block holding the query
            latch_error(err, kDevBounds);
            n = 1;
        }
        P[r] = n;
        if (Ls) Ls[r] = L;
    }
    __syncthreads();
    // exclusive prefix sum over contiguous ranges of requests per thread
    const int per_thread = (R + kThreads - 1) / kThreads;
    const int r0 = min(R, tid * per_thread), r1 = min(R, r0 + per_thread);
    int32_t run = 0, mx = 0;
    for (int r = r0; r < r1; ++r) {
        run += P[r];
        mx = max(mx, P[r]);
    }
    int32_t incl = run;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const int32_t v = __shfl_up_sync(0xffffffffu, incl, off);
        if (lane >= off) incl += v;
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) mx = max(mx, __shfl_xor_sync(0xffffffffu, mx, off));
    if (lane == 31) warp_tot[warp] = incl;
    if (lane == 0) warp_max[warp] = mx;
    __syncthreads();
    int32_t base = 0, total = 0, gmax = 0;
    for (int w = 0; w < kWarps; ++w) {
        if (w < warp) base += warp_tot[w];
        total += warp_tot[w];
        gmax = max(gmax, warp_max[w]);
    }
    int32_t acc = base + incl - run;   // exclusive prefix at r0
    for (int r = r0; r < r1; ++r) {
        const int32_t n = P[r];
        P[r] = acc;
        acc += n;
    }
    if (tid == 0) {
        P[R] = total;
        *max_n_out = gmax;
    }
    __syncthreads();
}

// The split pass: per warp, a contiguous range of the block stream through a
// TMA ring (see the file comment).  Ranges are equal in cost: a block costs
// one unit and each segment kPieceCost more (its Q rows, its partial and the
// ramp of a new piece), so warps whose range crosses many short segments
// take fewer blocks.
constexpr int32_t kPieceCost = 1;

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    decode_split_kernel(const __grid_constant__ CUtensorMap tmk, const __grid_constant__ CUtensorMap tmv,
                        const DecodeArgs a, const DecodeLayout lay, int32_t num_blocks_pool,
                        int32_t after_prefix) {
    constexpr int kHalves = D / 64;
    constexpr uint32_t kTileBytes = kHalves * 2048;   // one K or V tile of a (block, kv head)
    constexpr uint32_t kSlotBytes = 2 * kTileBytes;
    constexpr int CPR = D / 8;                        // 16-byte chunks per key row
    const uint32_t kQBytes = (uint32_t)lay.qbytes;    // Q area of a stage: 4 or 8 head rows
    const int S = lay.stages;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                ~uintptr_t(1023));
    // K/V stages [kWarps][S] | Q areas [kWarps][S] | slack | descriptors
    // [kWarps][S] | full barriers [kWarps][S] | plan [R + 1] | context lengths
    // [R] (if they fit).  The Q fragments are read as 8 head rows; with 4-row
    // areas (g <= 4) rows 4-7 come from the next area, or from the slack after
    // the last one, and feed only head columns that are never written out.
    const uint32_t qbase = smem_u32(smem) + (uint32_t)(kWarps * S) * kSlotBytes;
    SlotDesc *descs = reinterpret_cast<SlotDesc *>(smem + (size_t)kWarps * S * (kSlotBytes + kQBytes) +
                                                   (8 * D * 2 - kQBytes));
    uint64_t *bars = reinterpret_cast<uint64_t *>(descs + kWarps * S);
    int32_t *P = reinterpret_cast<int32_t *>(bars + kWarps * S);
    int32_t *Ls = lay.lens_in_smem ? P + lay.R + 1 : nullptr;
    __shared__ int32_t s_max_n;
    __shared__ int abort_flag;

    // After a shared-prefix pass, which starts this kernel once it has seen
    // everything before it complete, nothing read here is written by that
    // pass: wait for it only before exiting (the combine needs both).
    // Without one, wait for the preceding kernel first.
    if (!after_prefix) pdl_wait();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    {
        // Warm L2 with the block table while the plan is built: its lines are
        // split over the CTAs, one 128-byte line per thread and pass (tables
        // up to 16 MiB).
        const int64_t lines = min(((int64_t)lay.R * a.max_blocks * 4 + 127) >> 7, (int64_t)1 << 17);
        const char *base = reinterpret_cast<const char *>(a.block_table);
        for (int64_t i = (int64_t)blockIdx.x * kThreads + threadIdx.x; i < lines; i += (int64_t)gridDim.x * kThreads)
            prefetch_l2(base + (i << 7));
    }
    if (threadIdx.x == 0) {
        abort_flag = 0;
        prefetch_tmap(&tmk);   // the descriptors are fetched while the plan is built
        prefetch_tmap(&tmv);
    }
    const uint32_t mybar = smem_u32(bars + warp * S);
    if (lane == 0) {
        for (int s = 0; s < S; ++s) mbar_init(mybar + 8 * s, 1);
        fence_barrier_init();
    }
    const int32_t R = lay.R, Hkv = lay.Hkv, Hq = lay.Hq, g = lay.g;
    build_plan(P, Ls, R, a.context_lens, a.group_of_req, a.group_blocks, a.num_groups, a.max_blocks,
               &s_max_n, a.err);   // ends with __syncthreads: the barriers are initialised
    // cost stream: segment (r, h) spans [Hkv (P[r] + c r) + h (n_r + c), + n_r + c),
    // its blocks the last n_r positions
    constexpr int32_t c = kPieceCost;
    const int64_t W = (int64_t)Hkv * ((int64_t)P[R] + (int64_t)c * R);
    const int64_t nwarps = (int64_t)gridDim.x * kWarps;
    int64_t per = (W + nwarps - 1) / nwarps;
    const int64_t need = (s_max_n - 1 + kMaxPrivateParts - 3) / (kMaxPrivateParts - 2);
    if (per < need) per = need;
    if (per < kMinBlocksPerPiece) per = kMinBlocksPerPiece;
    const int64_t gw = (int64_t)blockIdx.x * kWarps + warp;
    const int64_t x0 = gw * per, x1 = min(x0 + per, W);
    // cost positions below 2^31 (every realistic batch) divide in 32 bits
    const bool narrow = W < ((int64_t)1 << 31);
    auto div_per = [&](int64_t v) -> int64_t {   // v >= 0
        return narrow ? (int64_t)((uint32_t)v / (uint32_t)per) : v / per;
    };

    if (x0 < x1) {
        float *o_part = reinterpret_cast<float *>(static_cast<char *>(a.ws) + lay.off_o);
        float2 *ml_part = reinterpret_cast<float2 *>(static_cast<char *>(a.ws) + lay.off_ml);
        int32_t *nparts = reinterpret_cast<int32_t *>(static_cast<char *>(a.ws) + lay.off_nparts);
        const uint32_t ring = smem_u32(smem) + (uint32_t)(warp * S) * kSlotBytes;
        const uint32_t qarea = qbase + (uint32_t)(warp * S) * kQBytes;
        const uint32_t qbytes = (uint32_t)g * D * 2;
        SlotDesc *mydesc = descs + warp * S;
        const bool fused = a.k_new != nullptr;

        // ---- the warp's pieces, 32 at a time: lane k describes the piece of
        // segment seg_base + k (segment (r, h) = r * Hkv + h)
        int64_t seg_base;
        {
            const int64_t xr = x0 / Hkv;
            int lo = 0, hi = R - 1;
            while (lo < hi) {
                const int mid = (lo + hi + 1) >> 1;
                if ((int64_t)P[mid] + (int64_t)c * mid <= xr) lo = mid; else hi = mid - 1;
            }
            const int32_t n0 = P[lo + 1] - P[lo];
            const int64_t off = x0 - (int64_t)Hkv * ((int64_t)P[lo] + (int64_t)c * lo);
            seg_base = (int64_t)lo * Hkv + (narrow ? (int64_t)((uint32_t)off / (uint32_t)(n0 + c)) : off / (n0 + c));
        }
        int32_t pr = 0, ph = 0, plo = 0, phi = 0, psh = 0, pL = 0, pn = 0, ppart = 0, pnw = 0;
        auto fill_list = [&]() {
            // segment ids stay below R * Hkv + 32 < 2^31
            const int32_t sg = (int32_t)(seg_base + lane);
            pr = (int32_t)((uint32_t)sg / (uint32_t)Hkv);
            ph = sg - pr * Hkv;
            plo = phi = 0;
            if (pr < R) {
                pn = P[pr + 1] - P[pr];
                // cost position of the segment's block 0
                const int64_t b0 = (int64_t)Hkv * ((int64_t)P[pr] + (int64_t)c * pr) + (int64_t)ph * (pn + c) + c;
                const int64_t lo = max(x0, b0), hi = min(x1, b0 + pn);
                if (lo < hi) {
                    plo = (int32_t)(lo - b0);
                    phi = (int32_t)(hi - b0);
                    pL = Ls ? Ls[pr] : __ldg(a.context_lens + pr);
                    const int32_t nblk = min((pL + 15) >> 4, a.max_blocks);
                    psh = max(nblk - pn, 0);
                    const int64_t w0 = div_per(b0);   // the warp whose range holds block 0
                    ppart = lay.prefix_parts + (int32_t)(gw - w0);
                    const int32_t n_priv = (int32_t)(div_per(b0 + pn - 1) - w0 + 1);
                    const int32_t n_pre = lay.prefix_parts > 0 && a.num_groups > 0
                                              ? min((psh + lay.prefix_blocks_per_part - 1) / lay.prefix_blocks_per_part,
                                                    lay.prefix_parts)
                                              : 0;
                    pnw = n_priv | (n_pre << 16);
                }
            }
        };
        fill_list();

        // block ids of a piece, 32 at a time: lane j holds block base + j
        auto load_ids = [&](int r_, int sh_, int base, int hi) -> int32_t {
            int32_t id = 0;
            if (base + lane < hi) {
                id = __ldg(a.block_table + (int64_t)r_ * a.max_blocks + sh_ + base + lane);
                if (id < 0 || id >= num_blocks_pool) {
                    latch_error(a.err, kDevBounds);
                    id = 0;
                }
            }
            return id;
        };

        // ---- producer cursor (warp-uniform): piece k of the list, next block b
        int k = -1, b = 0, b_lo = 0, b_hi = 0, cr = 0, ch = 0, csh = 0, cL = 0, cn = 0, cpart = 0, cnw = 0;
        int win_base = 0, nwin_for = -1;
        int32_t win = 0, nwin = 0;
        // the next piece of the range; false when the range is done
        auto enter_next = [&]() -> bool {
            ++k;
            if (k == 32) {
                seg_base += 32;
                fill_list();
                k = 0;
                nwin_for = -1;
            }
            b_lo = __shfl_sync(0xffffffffu, plo, k);
            b_hi = __shfl_sync(0xffffffffu, phi, k);
            if (b_lo >= b_hi) return false;   // pieces are consecutive: none follows an empty one
            cr = __shfl_sync(0xffffffffu, pr, k);
            ch = __shfl_sync(0xffffffffu, ph, k);
            csh = __shfl_sync(0xffffffffu, psh, k);
            cL = __shfl_sync(0xffffffffu, pL, k);
            cn = __shfl_sync(0xffffffffu, pn, k);
            cpart = __shfl_sync(0xffffffffu, ppart, k);
            cnw = __shfl_sync(0xffffffffu, pnw, k);
            b = b_lo;
            win_base = b_lo;
            win = nwin_for == k ? nwin : load_ids(cr, csh, b_lo, b_hi);
            // the next piece's first ids, in flight while this piece issues
            nwin_for = -1;
            if (k + 1 < 32) {
                const int r1 = __shfl_sync(0xffffffffu, pr, k + 1), sh1 = __shfl_sync(0xffffffffu, psh, k + 1);
                const int lo1 = __shfl_sync(0xffffffffu, plo, k + 1), hi1 = __shfl_sync(0xffffffffu, phi, k + 1);
                if (lo1 < hi1) {
                    nwin = load_ids(r1, sh1, lo1, hi1);
                    nwin_for = k + 1;
                }
            }
            return true;
        };
        // issue the copies of the next block into stage s; false when the
        // range is done (nothing issued)
        bool more = true;
        auto produce = [&](int s) -> bool {
            if (b == b_hi && !enter_next()) return false;
            if (b - win_base >= 32) {
                win_base = b;
                win = load_ids(cr, csh, b, b_hi);
            }
            const int32_t phys = __shfl_sync(0xffffffffu, win, b - win_base);
            const int valid = min(16, cL - (csh + b) * 16);
            int32_t info = valid;
            const bool first = b == b_lo;
            const bool write_at_end = fused && b_hi == cn && cL - (csh + cn - 1) * 16 >= 1;
            if (first) info |= kFirst | (b_lo == 0 ? kSegFirst : 0) | (write_at_end ? kWriteSoon : 0);
            if (b == b_hi - 1) info |= kLast;
            if (write_at_end && b == cn - 1) info |= kWrite;
            if (lane == 0) {
                SlotDesc dsc;
                dsc.r = cr; dsc.h = ch; dsc.phys = phys; dsc.info = info;
                dsc.part = cpart; dsc.nparts = cnw; dsc.pad0 = dsc.pad1 = 0;
                mydesc[s] = dsc;
                const uint32_t dst = ring + (uint32_t)s * kSlotBytes, bar = mybar + 8 * s;
                fence_proxy_async_smem();   // this stage's earlier generic reads / writes
                mbar_arrive_expect_tx(bar, kSlotBytes + (first ? qbytes : 0u));
                if (first)   // the piece's g q-head rows, contiguous in q
                    bulk_load(qarea + (uint32_t)s * kQBytes,
                              static_cast<const uint16_t *>(a.q) + ((int64_t)cr * Hq + (int64_t)ch * g) * D, qbytes, bar);
                // read once: marked first out of L2 (measured: the pass
                // streams faster, and the shared-prefix pass beside it too)
                const uint64_t pol = l2_evict_first_policy();
#pragma unroll
                for (int hf = 0; hf < kHalves; ++hf) {
                    tma_load_4d_hint(dst + hf * 2048, &tmk, hf * 64, 0, ch, phys, bar, pol);
                    tma_load_4d_hint(dst + kTileBytes + hf * 2048, &tmv, hf * 64, 0, ch, phys, bar, pol);
                }
            }
            __syncwarp();
            ++b;
            return true;
        };

        int64_t issued = 0;
        for (int s0 = 0; s0 < S && more; ++s0) {
            more = produce(s0);
            if (more) ++issued;
        }

        uint32_t qf[D / 16][2];
        uint4 kvn = make_uint4(0, 0, 0, 0);   // lane < CPR: k_new chunk; < 2 CPR: v_new chunk
        auto load_new = [&](const SlotDesc &d) {
            if (lane < 2 * CPR) {
                const uint16_t *src = static_cast<const uint16_t *>(lane < CPR ? a.k_new : a.v_new);
                const int cc = lane < CPR ? lane : lane - CPR;
                kvn = ldg16(src + ((int64_t)d.r * Hkv + d.h) * D + cc * 8);
            }
        };
        if (issued > 0) {
            const SlotDesc d0 = mydesc[0];
            if (d0.info & kWriteSoon) load_new(d0);
        }
        SoftmaxState<D> st;
        int s = 0;
        uint32_t phase = 0;
        int64_t u = 0;
        for (; u < issued; ++u) {
            if (!__all_sync(0xffffffffu, mbar_wait(mybar + 8 * s, phase, &abort_flag, kWaitLimitNs))) break;
            const SlotDesc d = mydesc[s];
            const int valid = d.info & kValidMask;
            const uint32_t kb = ring + (uint32_t)s * kSlotBytes, vb = kb + kTileBytes;
            if (d.info & kFirst) {
                load_q_smem<D>(qf, qarea + (uint32_t)s * kQBytes, lane);
                st.m[0] = st.m[1] = -INFINITY;
                st.l[0] = st.l[1] = 0.f;
#pragma unroll
                for (int i = 0; i < D / 16; ++i) st.o[i][0] = st.o[i][1] = st.o[i][2] = st.o[i][3] = 0.f;
                if ((d.info & kSegFirst) && lane == 0) nparts[(int64_t)d.r * Hkv + d.h] = d.nparts;
            }
            if (d.info & kWrite) {
                // the query token's K/V: into the pool at position L - 1 and
                // over the stale row of this stage
                const int off = valid - 1;
                if (lane < 2 * CPR) {
                    const bool isv = lane >= CPR;
                    const int cc = isv ? lane - CPR : lane;
                    uint16_t *cache = static_cast<uint16_t *>(const_cast<void *>(isv ? a.v_cache : a.k_cache));
                    *reinterpret_cast<uint4 *>(cache + (((int64_t)d.phys * Hkv + d.h) * 16 + off) * D + cc * 8) = kvn;
                    const uint32_t dst = (isv ? vb : kb) + tile_off(off, cc);
                    asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};" ::"r"(dst), "r"(kvn.x), "r"(kvn.y),
                                 "r"(kvn.z), "r"(kvn.w)
                                 : "memory");
                }
            }
            if (valid < 16) {
                // keys past the context: p = 0, but their V rows may hold
                // anything (0 * NaN = NaN in the MMA), so clear them
                for (int i = lane; i < (16 - max(valid, 0)) * CPR; i += 32) {
                    const int row = max(valid, 0) + i / CPR, cc = i % CPR;
                    asm volatile("st.shared.v4.u32 [%0], {%1,%1,%1,%1};" ::"r"(vb + tile_off(row, cc)), "r"(0)
                                 : "memory");
                }
            }
            if (u + 1 < issued) {
                // a piece that starts next and ends with the query token's
                // row: its new K/V in flight from now on
                const SlotDesc d1 = mydesc[s + 1 == S ? 0 : s + 1];
                if (d1.info & kWriteSoon) load_new(d1);
            }
            __syncwarp();
            attend_block<D>(st, kb, vb, qf, lane, valid, a.scale_log2);
            if (d.info & kLast) {
                // row-group reduction of the thread-partial sums, then the
                // unnormalised partial of this piece
                float l0 = st.l[0], l1 = st.l[1];
#pragma unroll
                for (int off = 4; off < 32; off <<= 1) {
                    l0 += __shfl_xor_sync(0xffffffffu, l0, off);
                    l1 += __shfl_xor_sync(0xffffffffu, l1, off);
                }
#pragma unroll
                for (int cc = 0; cc < 2; ++cc) {
                    const int hd = 2 * (lane & 3) + cc;
                    if (hd < g) {
                        const int64_t slot = ((int64_t)d.r * Hq + d.h * g + hd) * lay.parts_per_head + d.part;
                        float *dst = o_part + slot * D + (lane >> 2);
#pragma unroll
                        for (int mt = 0; mt < D / 16; ++mt) {
                            dst[16 * mt] = st.o[mt][cc];
                            dst[16 * mt + 8] = st.o[mt][2 + cc];
                        }
                        if ((lane >> 2) == 0) ml_part[slot] = make_float2(st.m[cc], cc ? l1 : l0);
                    }
                }
            }
            __syncwarp();
            if (more) {
                more = produce(s);
                if (more) ++issued;
            }
            if (++s == S) {
                s = 0;
                phase ^= 1u;
            }
        }
        if (u < issued) {
            // a wait ran out: latch it, then let this warp's copies still in
            // flight (units u .. issued - 1) land before the CTA exits
            if (lane == 0) {
                latch_error(a.err, kDevTimeout);
                int quiet = 0;
                for (int64_t v = u; v < issued; ++v) {
                    const int sv = (int)(v % S);
                    mbar_wait(mybar + 8 * sv, (uint32_t)((v / S) & 1), &quiet, kDrainLimitNs);
                }
            }
            __syncwarp();
        }
    }
    if (after_prefix) pdl_wait();
}

// Merge the partials of each (request, kv head) with log-sum-exp weights.
// The g q heads of a kv head share one list of parts (the group's prefix
// splits, then the private pieces); `wpi` warps split them, GW heads each.
// Lane k holds part slot k's (m, l) for the warp's heads; lane c holds
// elements [c*E, c*E + E) of every head's output.  With SPEC the partials of
// slots 0 .. KR-1 are loaded in the same round as the part counts and the
// (m, l): they are parts 0 .. KR-1 whenever the request's prefix partials
// fill the prefix slots or number at least KR (every request of a one-group
// batch), and are reloaded from their real slots otherwise; without it the
// first round of partials waits for the counts like the others.
template <int D, int GW, bool SPEC>
__global__ void __launch_bounds__(128) decode_combine_kernel(DecodeArgs a, DecodeLayout lay, int32_t wpi) {
    constexpr int E = D / 32;    // output elements per lane and head
    constexpr int KR = 16 / GW;  // parts per round: KR x GW element vectors in flight per lane
    pdl_wait();
    const int lane = threadIdx.x & 31;
    const int64_t wid = (int64_t)blockIdx.x * (blockDim.x / 32) + (threadIdx.x >> 5);
    const int64_t item = wpi == 2 ? wid >> 1 : wid;   // wpi is 1 or 2
    if (item >= (int64_t)lay.R * lay.Hkv) return;
    const int r = (int)(item / lay.Hkv), h = (int)(item % lay.Hkv);
    const int g = lay.g;
    const int hs = wpi == 2 ? (int)(wid & 1) * GW : 0;   // the warp's first head within the kv head
    const int ng = min(GW, g - hs);                // its heads (at least 1)
    if (ng <= 0) return;
    const int pph = lay.parts_per_head;
    const float *o_part = reinterpret_cast<const float *>(static_cast<const char *>(a.ws) + lay.off_o);
    const float2 *ml_part =
        reinterpret_cast<const float2 *>(static_cast<const char *>(a.ws) + lay.off_ml);
    const int32_t *nparts =
        reinterpret_cast<const int32_t *>(static_cast<const char *>(a.ws) + lay.off_nparts);
    const int64_t head0 = (int64_t)r * lay.Hq + (int64_t)h * g + hs;   // (request, q head) index of head 0
    auto load_part = [&](float (&dst)[E], int hd, int slot) {
        const float *src = o_part + ((head0 + hd) * pph + slot) * D + lane * E;
        if constexpr (E == 4) {
            const float4 t = *reinterpret_cast<const float4 *>(src);
            dst[0] = t.x; dst[1] = t.y; dst[2] = t.z; dst[3] = t.w;
        } else {
            const float2 t = *reinterpret_cast<const float2 *>(src);
            dst[0] = t.x; dst[1] = t.y;
        }
    };
    // one round: the part counts written by the split pass (private pieces
    // | prefix partials << 16), the (m, l) of every part slot (lane k: slot
    // k), and the partials of slots 0 .. KR-1; what lies beyond the counts
    // may hold anything and is masked or replaced below
    const int32_t counts = nparts[item];
    float2 mlv[GW];
#pragma unroll
    for (int hd = 0; hd < GW; ++hd) {
        mlv[hd] = make_float2(-INFINITY, 0.f);
        if (hd < ng && lane < pph) mlv[hd] = ml_part[(head0 + hd) * pph + lane];
    }
    float v[KR][GW][E];
#pragma unroll
    for (int u = 0; u < KR; ++u)
#pragma unroll
        for (int hd = 0; hd < GW; ++hd) {
#pragma unroll
            for (int e = 0; e < E; ++e) v[u][hd][e] = 0.f;
            if (SPEC && hd < ng && u < pph) load_part(v[u][hd], hd, u);
        }
    const int n_priv = min(max(counts & 0xFFFF, 0), pph - lay.prefix_parts);
    const int n_pre = min((counts >> 16) & 0xFFFF, lay.prefix_parts);
    const int total = min(n_pre + n_priv, 32);
    const bool live = lane < n_pre || (lane >= lay.prefix_parts && lane < lay.prefix_parts + n_priv);
    // parts in merge order: the prefix partials, then the private pieces
    auto part_lane = [&](int k) { return k < n_pre ? k : lay.prefix_parts + (k - n_pre); };
    // weights: the lane of a slot owns that slot's weight for every head
    float wk[GW], mx[GW], den[GW];
#pragma unroll
    for (int hd = 0; hd < GW; ++hd) {
        mx[hd] = (hd < ng && live) ? mlv[hd].x : -INFINITY;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) mx[hd] = fmaxf(mx[hd], __shfl_xor_sync(0xffffffffu, mx[hd], off));
    }
#pragma unroll
    for (int hd = 0; hd < GW; ++hd) {
        const float w = (hd < ng && live) ? fast_exp2(mlv[hd].x - mx[hd]) : 0.f;
        den[hd] = (hd < ng && live) ? w * mlv[hd].y : 0.f;
        wk[hd] = w;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) den[hd] += __shfl_xor_sync(0xffffffffu, den[hd], off);
    }
    float acc[GW][E];
#pragma unroll
    for (int hd = 0; hd < GW; ++hd)
#pragma unroll
        for (int e = 0; e < E; ++e) acc[hd][e] = 0.f;
    // the first round: keep what was loaded where part u sits in slot u,
    // reload it where it does not, and drop slots past the parts
#pragma unroll
    for (int u = 0; u < KR; ++u)
#pragma unroll
        for (int hd = 0; hd < GW; ++hd) {
            if (u >= total) {
#pragma unroll
                for (int e = 0; e < E; ++e) v[u][hd][e] = 0.f;
            } else if ((!SPEC || part_lane(u) != u) && hd < ng) {
                load_part(v[u][hd], hd, part_lane(u));
            }
        }
#pragma unroll
    for (int u = 0; u < KR; ++u)
#pragma unroll
        for (int hd = 0; hd < GW; ++hd) {
            const float w = __shfl_sync(0xffffffffu, wk[hd], u < total ? part_lane(u) : 0);
#pragma unroll
            for (int e = 0; e < E; ++e) acc[hd][e] += w * v[u][hd][e];
        }
    // the other parts in rounds of KR
    for (int k0 = KR; k0 < total; k0 += KR) {
#pragma unroll
        for (int u = 0; u < KR; ++u)
#pragma unroll
            for (int hd = 0; hd < GW; ++hd) {
#pragma unroll
                for (int e = 0; e < E; ++e) v[u][hd][e] = 0.f;
                if (k0 + u < total && hd < ng) load_part(v[u][hd], hd, part_lane(k0 + u));
            }
#pragma unroll
        for (int u = 0; u < KR; ++u)
#pragma unroll
            for (int hd = 0; hd < GW; ++hd) {
                const float w = __shfl_sync(0xffffffffu, wk[hd], k0 + u < total ? part_lane(k0 + u) : 0);
#pragma unroll
                for (int e = 0; e < E; ++e) acc[hd][e] += w * v[u][hd][e];
            }
    }
#pragma unroll
    for (int hd = 0; hd < GW; ++hd) {
        if (hd >= ng) break;
        const float inv = 1.f / den[hd];
        uint16_t *out = static_cast<uint16_t *>(a.out) + (head0 + hd) * D + lane * E;
        if constexpr (E == 4) {
            *reinterpret_cast<uint2 *>(out) = make_uint2(pack_bf16x2(acc[hd][0] * inv, acc[hd][1] * inv),
                                                         pack_bf16x2(acc[hd][2] * inv, acc[hd][3] * inv));
        } else {
            *reinterpret_cast<uint32_t *>(out) = pack_bf16x2(acc[hd][0] * inv, acc[hd][1] * inv);
        }
        if (a.lse && lane == 0) a.lse[head0 + hd] = (mx[hd] + __log2f(den[hd])) * 0.69314718055994530942f;
    }
}

}  // namespace

namespace {

// Shared memory of the split pass for `stages` ring stages.
// qbytes: the Q area of a stage (4 or 8 head rows of d bf16)
size_t split_smem_bytes(int32_t R, int32_t d, int stages, bool lens, size_t qbytes) {
    const size_t slot = 2 * (size_t)(d / 64) * 2048 + qbytes;   // K/V tiles + Q area
    return 1024 + (size_t)kWarps * stages * (slot + sizeof(SlotDesc) + 8) + (8 * (size_t)d * 2 - qbytes) +
           4 * ((size_t)R + 1) + (lens ? 4 * (size_t)R : 0);
}

}  // namespace

namespace {

// Workspace offsets for prefix_parts + private_parts part slots per (row, q head).
void set_part_slots(DecodeLayout &L, int private_parts) {
    L.parts_per_head = L.prefix_parts + private_parts;
    const size_t slots = (size_t)L.R * L.Hq * L.parts_per_head;
    auto up = [](size_t x) { return (x + 255) & ~(size_t)255; };
    L.off_o = 0;
    L.off_ml = up(slots * L.d * sizeof(float));
    L.off_nparts = L.off_ml + up(slots * sizeof(float2));
    L.total = L.off_nparts + up((size_t)L.R * L.Hkv * sizeof(int32_t));
}

}  // namespace

DecodeLayout decode_layout(int32_t R, int32_t Hq, int32_t Hkv, int32_t d, int32_t max_blocks,
                           int32_t num_groups, int32_t max_group_blocks, int32_t max_group_members,
                           int32_t num_sms) {
    DecodeLayout L{};
    L.R = R; L.Hq = Hq; L.Hkv = Hkv; L.d = d; L.g = Hq / Hkv;
    L.sms = num_sms > 0 ? num_sms : 148;
    const int sms = L.sms;
    L.prefix_blocks_per_part = 8;
    L.prefix_parts = 0;
    L.prefix_ctas = 0;
    L.prefix_early = 0;
    // the private split pass streams about kSplitGBsPerSM per SM, together
    // at most kSplitGBsTotal, after about kSplitStartUs of start-up; its bytes
    // are estimated from the table width (60 % of the blocks past the longest
    // prefix), which only steers choices
    constexpr double kSplitGBsPerSM = 47.0, kSplitGBsTotal = 6300.0, kSplitStartUs = 7.0;
    const double unit_bytes = 16.0 * d * 2 * 2;   // K + V of one (block, kv head)
    const double priv_blocks = 0.6 * std::max(1, max_blocks - std::max(0, max_group_blocks));
    const double split_bytes = (double)R * Hkv * priv_blocks * unit_bytes;
    auto split_us = [&](int nsm) {
        return kSplitStartUs + split_bytes / std::min(kSplitGBsTotal, kSplitGBsPerSM * nsm) * 1e-3;
    };
    if (num_groups > 0 && max_group_blocks > 0 && max_group_members > 0) {
        // Key splits of the prefix pass: one CTA per (group, kv head, member
        // tile, split), one CTA per SM.  When its grid leaves at least a
        // quarter of the SMs free, the split pass runs beside it on those
        // SMs and a step costs about max(prefix critical path, split time on
        // the free SMs); otherwise the two run one after the other.
        // Measured on GB300 with per-CTA clock stamps: a prefix CTA alone
        // costs about 11.5 us of fixed work (set-up, Q tile, pipeline fill,
        // partial writes) plus 1.7 us per key tile; beside the split pass
        // (2-stage ring) 13 us plus 2.2 us per key tile, its 2-stage K/V ring
        // then waiting on memory.
        const int per_item = 2 * (128 / L.g);   // members per work item (two 128-row tiles)
        const int64_t tiles = (int64_t)num_groups * Hkv * ((max_group_members + per_item - 1) / per_item);
        const int key_tiles = (max_group_blocks + 7) / 8;
        int best = 1;
        double best_t = 1e300;
        for (int sp = 1; sp <= kMaxPrefixParts && sp <= key_tiles; ++sp) {
            const int per = (key_tiles + sp - 1) / sp;
            const int64_t ctas = tiles * sp;
            const bool beside = 4 * ctas <= 3 * (int64_t)sms;
            const double cta_us = beside ? 13.0 + 2.2 * per : 11.5 + 1.7 * per;
            const double crit = (double)((ctas + sms - 1) / sms) * cta_us;
            const double t = beside ? std::max(crit, split_us(sms - (int)ctas)) : crit + split_us(sms);
            if (t < best_t - 1e-9) { best_t = t; best = sp; }
        }
        const int per_tiles = (key_tiles + best - 1) / best;
        L.prefix_blocks_per_part = per_tiles * 8;
        L.prefix_parts = (max_group_blocks + L.prefix_blocks_per_part - 1) / L.prefix_blocks_per_part;
        L.prefix_ctas = tiles * L.prefix_parts;
        L.prefix_early = (4 * L.prefix_ctas <= 3 * (int64_t)sms) ? 1 : 0;
    }
    L.split_grid = L.prefix_early ? sms - (int32_t)L.prefix_ctas : sms;
    // as many ring stages as fit (the plan takes 4 bytes per request)
    // Ring stages: each warp keeps S - 1 blocks in flight while it computes
    // on one.  Alone on the device the pass takes as many as fit (up to 3 of
    // 8 KB at d = 128).  Beside the shared-prefix pass it keeps to 16 KB per
    // warp: with fewer copies queued at HBM that pass's own loads wait less
    // (measured on the 64-request Llama-3-8B step: prefix pass 43 -> 38 us,
    // the split pass's end unchanged, step -3 us).
    L.qbytes = (L.g <= 4 ? 4 : 8) * d * 2;
    L.stages = 2;
    const int max_stages = d == 64 ? 4 : (L.prefix_early ? 2 : 3);
    for (int st = max_stages; st > 2; --st)
        if (split_smem_bytes(R, d, st, false, L.qbytes) <= kMaxSmemPerBlock) { L.stages = st; break; }
    // the context lengths beside the plan when they fit (saves a global read per piece list)
    L.lens_in_smem = split_smem_bytes(R, d, L.stages, true, L.qbytes) <= kMaxSmemPerBlock ? 1 : 0;
    L.split_smem = split_smem_bytes(R, d, L.stages, L.lens_in_smem != 0, L.qbytes);
    set_part_slots(L, kMaxPrivateParts);
    return L;
}

DecodeLayout verify_layout(int32_t T, int32_t Hq, int32_t Hkv, int32_t d, int32_t max_blocks,
                           int32_t num_groups, int32_t max_group_blocks, int32_t max_group_tokens,
                           int32_t num_sms) {
    // the prefix pass of decode over draft tokens, and one private part per
    // token (the tile pass over the request's keys after the shared blocks)
    DecodeLayout L = decode_layout(T, Hq, Hkv, d, max_blocks, num_groups, max_group_blocks, max_group_tokens,
                                   num_sms);
    set_part_slots(L, 1);
    return L;
}

template <int D>
static cudaError_t launch_decode_t(const DecodeLayout &L, const DecodeArgs &a, int32_t num_blocks_pool,
                                   cudaStream_t stream, Tracer *tr) {
    const bool prefix = L.prefix_parts > 0 && a.num_groups > 0;
    if (prefix) {
        cudaError_t e = launch_decode_prefix(L, a, num_blocks_pool, stream, tr);
        if (e != cudaSuccess) return e;
    }
    static SmemLimit limit;
    {
        cudaError_t e = limit.ensure(reinterpret_cast<const void *>(decode_split_kernel<D>), (int)L.split_smem);
        if (e != cudaSuccess) return e;
    }
    if (tr) tr->begin(kKernelDecodeSplit, stream);
    // the split pass runs beside the prefix pass: on the SMs that pass leaves
    // free when they are a quarter of the device, otherwise on every SM (its
    // CTAs take the SMs the prefix pass leaves idle, then those its CTAs free)
    const int grid = prefix ? L.split_grid : L.sms;
    cudaError_t e = launch_pdl(decode_split_kernel<D>, dim3(grid), dim3(kThreads), L.split_smem, stream,
                               *a.tmap_k, *a.tmap_v, a, L, num_blocks_pool, prefix ? 1 : 0);
    if (tr) tr->end(kKernelDecodeSplit, stream);
    if (e != cudaSuccess) return e;
    return launch_decode_combine(L, a, stream, tr);
}

template <int D>
static cudaError_t launch_combine_t(const DecodeLayout &L, const DecodeArgs &a, cudaStream_t stream, Tracer *tr) {
    // Four warps per CTA.  While the (request, kv head) items alone would
    // leave the device's warps idle (at most 8 items per SM), each item's
    // heads are split over two warps of 2 (g <= 4) or 4 heads, which keep 8
    // or 4 parts in flight per round, the first round loaded with the part
    // counts (measured on the Qwen2.5-7B mixed batch, 1024 items: decode
    // 89.3 -> 88.2 us); with more items one warp takes every head (the
    // split and the early round measured slower on 4096-item batches).
    const bool split = (int64_t)L.R * L.Hkv <= 8LL * L.sms;
    const int gw = split ? (L.g <= 4 ? 2 : 4) : (L.g <= 4 ? 4 : 8);
    const int32_t wpi = (L.g + gw - 1) / gw;   // 1 or 2 (g <= 8)
    const int64_t warps = (int64_t)L.R * L.Hkv * wpi;
    const int64_t cgrid = (warps + 3) / 4;
    if (cgrid > 0x7fffffff) return cudaErrorInvalidConfiguration;
    if (tr) tr->begin(kKernelDecodeCombine, stream);
    const dim3 cg((unsigned)cgrid), cb(128);
    cudaError_t e = gw == 2   ? launch_pdl(decode_combine_kernel<D, 2, true>, cg, cb, 0, stream, a, L, wpi)
                    : split   ? launch_pdl(decode_combine_kernel<D, 4, true>, cg, cb, 0, stream, a, L, wpi)
                    : gw == 4 ? launch_pdl(decode_combine_kernel<D, 4, false>, cg, cb, 0, stream, a, L, wpi)
                              : launch_pdl(decode_combine_kernel<D, 8, false>, cg, cb, 0, stream, a, L, wpi);
    if (tr) tr->end(kKernelDecodeCombine, stream);
    return e;
}

cudaError_t launch_decode_combine(const DecodeLayout &L, const DecodeArgs &a, cudaStream_t stream, Tracer *tr) {
    return L.d == 128 ? launch_combine_t<128>(L, a, stream, tr) : launch_combine_t<64>(L, a, stream, tr);
}

cudaError_t launch_decode(const DecodeLayout &L, const DecodeArgs &a, int32_t num_blocks_pool,
                          cudaStream_t stream, Tracer *tr) {
    if (L.d == 128) return launch_decode_t<128>(L, a, num_blocks_pool, stream, tr);
    return launch_decode_t<64>(L, a, num_blocks_pool, stream, tr);
}

}  // namespace pkv
