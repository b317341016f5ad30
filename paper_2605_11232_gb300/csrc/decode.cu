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
// persistent grid takes blocks [w*per, (w+1)*per) of that stream, so every
// warp moves the same number of bytes whatever the length mix; a warp that
// crosses a segment boundary emits one unnormalised partial (O, m, l) per
// segment it touches.  The combine kernel merges a head's partials with
// log-sum-exp weights.
//
// Inner loop (one 16-token block per step, per warp):
//   S^T[16 keys x 8 heads] = K_blk[16 x d] . Q^T[d x 8]   (mma m16n8k16, A = K)
//   online softmax per head column (shuffles across the 8 row groups)
//   O^T[d x 8] += V_blk^T[d x 16] . P^T[16 x 8]           (A = V^T, B = P^T)
// K and V are read with 16-byte loads straight into registers in the order
// the mma fragments need: the head dimension is a contraction index for
// Q.K and the key index one for P.V, so both may be permuted freely as long
// as both operands use the same permutation.  The S^T accumulator becomes the
// P^T operand through one movmatrix transpose per 8x8 quadrant; the key order
// sigma() of the QK^T rows is chosen so that the transposed fragments land on
// exactly the keys each thread loaded for P.V.
#include <math.h>

#include <algorithm>

#include "pkv_device.cuh"
#include "pkv_internal.h"

namespace pkv {

namespace {

constexpr int kWarps = 8;
constexpr int kThreads = kWarps * 32;
constexpr int kChunksPerWarp = 2;   // work chunks per warp of the grid (balance vs. pipeline restarts)

__device__ __forceinline__ uint32_t reg_of(const uint4 &v, int i) {
    return i == 0 ? v.x : (i == 1 ? v.y : (i == 2 ? v.z : v.w));
}

// Physical key (row of the 16-token block) behind logical QK^T row r (0..7);
// row r + 8 is sigma(r) + 2.
__device__ __forceinline__ int sigma(int r) { return 2 * r - (r & 1); }

template <int D>
struct BlockRegs {
    uint4 ka[D / 32];   // K[sigma(r)    ][chunk 4j+q]
    uint4 kb[D / 32];   // K[sigma(r) + 2][chunk 4j+q]
    uint4 va[4];        // V[4q+s][chunk r]       (d 8r..8r+7)
    uint4 vb[D == 128 ? 4 : 1];   // V[4q+s][chunk 8+r] (d 64+8r..), d = 128 only
};

template <int D>
__device__ __forceinline__ void load_block(BlockRegs<D> &b, const uint16_t *kt,
                                           const uint16_t *vt, int lr, int lq) {
    const int s0 = sigma(lr);
#pragma unroll
    for (int j = 0; j < D / 32; ++j) {
        b.ka[j] = ldg_stream(kt + s0 * D + (4 * j + lq) * 8);
        b.kb[j] = ldg_stream(kt + (s0 + 2) * D + (4 * j + lq) * 8);
    }
#pragma unroll
    for (int s = 0; s < 4; ++s) {
        b.va[s] = ldg_stream(vt + (4 * lq + s) * D + lr * 8);
        if constexpr (D == 128) b.vb[s] = ldg_stream(vt + (4 * lq + s) * D + (8 + lr) * 8);
    }
}

// Running state of one warp over one piece.  Thread (lr = lane/4, lq = lane%4)
// holds heads 2lq, 2lq+1: m, l (thread-partial sum) and O^T fragments.
template <int D>
struct SoftmaxState {
    float m[2];
    float l[2];
    float o[D / 16][4];
};

template <int D>
__device__ __forceinline__ void attend_block(SoftmaxState<D> &st, BlockRegs<D> &b,
                                             const uint32_t (&qf)[D / 32][4], int lr, int lq,
                                             int valid_keys, float scale_log2) {
    // S^T = K . Q^T
    float sacc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int s = 0; s < D / 16; ++s) {
        const int j = s >> 1, e = s & 1;
        mma_bf16_16816(sacc, reg_of(b.ka[j], 2 * e), reg_of(b.kb[j], 2 * e),
                       reg_of(b.ka[j], 2 * e + 1), reg_of(b.kb[j], 2 * e + 1), qf[j][2 * e],
                       qf[j][2 * e + 1]);
    }
    const int key0 = sigma(lr), key1 = key0 + 2;
    const bool ok0 = key0 < valid_keys, ok1 = key1 < valid_keys;
    float s00 = ok0 ? sacc[0] * scale_log2 : -INFINITY;   // key0, head 2lq
    float s01 = ok0 ? sacc[1] * scale_log2 : -INFINITY;   // key0, head 2lq+1
    float s10 = ok1 ? sacc[2] * scale_log2 : -INFINITY;   // key1, head 2lq
    float s11 = ok1 ? sacc[3] * scale_log2 : -INFINITY;   // key1, head 2lq+1
    float mx0 = fmaxf(s00, s10), mx1 = fmaxf(s01, s11);
#pragma unroll
    for (int off = 4; off < 32; off <<= 1) {
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, off));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, off));
    }
    const float mn0 = fmaxf(st.m[0], mx0), mn1 = fmaxf(st.m[1], mx1);
    // mn is finite: every processed block has at least one valid key.
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
    // P^T fragments: transpose the two 8x8 quadrants of P^T(key, head).
    const uint32_t t0 = movmatrix_trans(pack_bf16x2(p00, p01));
    const uint32_t t1 = movmatrix_trans(pack_bf16x2(p10, p11));
    // Masked keys carry p = 0, but 0 * NaN would poison O: zero their V rows.
#pragma unroll
    for (int s = 0; s < 4; ++s) {
        if (4 * lq + s >= valid_keys) {
            b.va[s] = make_uint4(0, 0, 0, 0);
            if constexpr (D == 128) b.vb[s] = make_uint4(0, 0, 0, 0);
        }
    }
    // O^T += V^T . P^T, one 16-row tile of the head dim per mma.
#pragma unroll
    for (int i = 0; i < D / 16; ++i) {
        const uint4 *src = (i < 4) ? b.va : b.vb;
        const int w = i & 3;
        const uint32_t x0 = reg_of(src[0], w), x1 = reg_of(src[1], w);
        const uint32_t x2 = reg_of(src[2], w), x3 = reg_of(src[3], w);
        mma_bf16_16816(st.o[i], __byte_perm(x0, x1, 0x5410), __byte_perm(x0, x1, 0x7632),
                       __byte_perm(x2, x3, 0x5410), __byte_perm(x2, x3, 0x7632), t0, t1);
    }
}

// Block-wide plan: P[r] = sum of the private block counts of requests < r,
// P[R] = their total; *max_n_out = the largest count.
__device__ void build_plan(int32_t *P, int32_t R, const int32_t *__restrict__ context_lens,
                           const int32_t *__restrict__ group_of_req,
                           const int32_t *__restrict__ group_blocks, int32_t num_groups,
                           int32_t max_blocks, int32_t *max_n_out, int *err) {
    __shared__ int32_t warp_tot[kWarps];
    __shared__ int32_t warp_max[kWarps];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int per_thread = (R + kThreads - 1) / kThreads;
    const int r0 = min(R, tid * per_thread), r1 = min(R, r0 + per_thread);
    int32_t run = 0, mx = 0;
    for (int r = r0; r < r1; ++r) {
        const int32_t L = __ldg(context_lens + r);
        int32_t nblk = (L + 15) >> 4;
        if (nblk > max_blocks) {   // context longer than the table row
            latch_error(err, kDevBounds);
            nblk = max_blocks;
        }
        int32_t sh = 0;
        if (num_groups > 0) {
            const int32_t gi = __ldg(group_of_req + r);
            if (gi >= 0 && gi < num_groups) sh = __ldg(group_blocks + gi);
        }
        int32_t n = nblk - sh;
        if (L < 1 || n < 1 || sh < 0) {   // decode needs a private tail block holding the query
            latch_error(err, kDevBounds);
            n = 1;
            sh = 0;
        }
        P[r] = n;   // the count for now; this thread alone touches P[r0..r1)
        run += n;
        mx = max(mx, n);
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

template <int D>
__global__ void __launch_bounds__(kThreads, 1) decode_split_kernel(DecodeArgs a, DecodeLayout lay,
                                                                  int32_t num_blocks_pool,
                                                                  int32_t after_prefix) {
    extern __shared__ int32_t P[];   // [R + 1]
    __shared__ int32_t s_max_n;
    // After a shared-prefix pass, which starts this kernel once it has seen
    // the cache write complete, nothing read here is written by that pass:
    // wait for it only before exiting (the combine needs both).  Without one,
    // wait for the cache write first.
    if (!after_prefix) pdl_wait();
    const int32_t R = lay.R, Hkv = lay.Hkv, Hq = lay.Hq, g = lay.g;
    build_plan(P, R, a.context_lens, a.group_of_req, a.group_blocks, a.num_groups, a.max_blocks,
               &s_max_n, a.err);
    const int64_t W = (int64_t)Hkv * P[R];
    const int64_t nwarps = (int64_t)gridDim.x * kWarps;
    int64_t per = (W + nwarps * kChunksPerWarp - 1) / (nwarps * kChunksPerWarp);
    const int64_t need = (s_max_n - 1 + kMaxPrivateParts - 3) / (kMaxPrivateParts - 2);
    if (per < need) per = need;
    if (per < kMinBlocksPerPiece) per = kMinBlocksPerPiece;

    const int lane = threadIdx.x & 31;
    const int lr = lane >> 2, lq = lane & 3;
    const int64_t nchunks = (W + per - 1) / per;

    const uint16_t *q = static_cast<const uint16_t *>(a.q);
    const uint16_t *kc = static_cast<const uint16_t *>(a.k_cache);
    const uint16_t *vc = static_cast<const uint16_t *>(a.v_cache);
    float *o_part = reinterpret_cast<float *>(static_cast<char *>(a.ws) + lay.off_o);
    float2 *ml_part = reinterpret_cast<float2 *>(static_cast<char *>(a.ws) + lay.off_ml);
    int32_t *nparts = reinterpret_cast<int32_t *>(static_cast<char *>(a.ws) + lay.off_nparts);

    // Chunks of `per` stream blocks are handed out by a counter, so that CTAs
    // which start late (on SMs the prefix pass still holds) take less work.
    for (;;) {
      int chunk = 0;
      if (lane == 0) chunk = atomicAdd(a.sched, 1);
      chunk = __shfl_sync(0xffffffffu, chunk, 0);
      if (chunk >= nchunks) break;
      int64_t x = (int64_t)chunk * per;
      const int64_t x_end = min(x + per, W);
      while (x < x_end) {
        // segment containing x: request r (largest r with P[r] <= x / Hkv), head h
        const int64_t xr = x / Hkv;
        int lo = 0, hi = R - 1;
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (P[mid] <= xr) lo = mid; else hi = mid - 1;
        }
        const int r = lo;
        const int32_t n = P[r + 1] - P[r];
        const int64_t seg_base = (int64_t)Hkv * P[r];
        const int h = (int)((x - seg_base) / n);
        const int64_t seg_off = seg_base + (int64_t)h * n;
        const int64_t piece_end = min(x_end, seg_off + n);
        const int b_lo = (int)(x - seg_off), b_hi = (int)(piece_end - seg_off);
        const int part = (int)(x / per - seg_off / per);

        const int32_t L = __ldg(a.context_lens + r);
        // shared leading blocks: the plan's private count n ends at the last block
        const int32_t nblk = min((L + 15) >> 4, a.max_blocks);
        const int32_t sh = max(nblk - n, 0);
        const int32_t *trow = a.block_table + (int64_t)r * a.max_blocks;

        // Q fragments of the g heads of kv head h (head lr of the group)
        uint32_t qf[D / 32][4];
        {
            const bool hv = lr < g;
            const uint16_t *qrow = q + ((int64_t)r * Hq + h * g + (hv ? lr : 0)) * D;
#pragma unroll
            for (int j = 0; j < D / 32; ++j) {
                uint4 v = hv ? ldg16(qrow + (4 * j + lq) * 8) : make_uint4(0, 0, 0, 0);
                qf[j][0] = v.x; qf[j][1] = v.y; qf[j][2] = v.z; qf[j][3] = v.w;
            }
        }
        SoftmaxState<D> st;
        st.m[0] = st.m[1] = -INFINITY;
        st.l[0] = st.l[1] = 0.f;
#pragma unroll
        for (int i = 0; i < D / 16; ++i) st.o[i][0] = st.o[i][1] = st.o[i][2] = st.o[i][3] = 0.f;

        // block ids of this piece, 32 at a time, one per lane
        int win_base = b_lo;
        int32_t my_phys = 0;
        auto refresh = [&](int base) {
            win_base = base;
            const int bi = sh + base + lane;
            int32_t p = (base + lane < b_hi) ? __ldg(trow + bi) : 0;
            if (p < 0 || p >= num_blocks_pool) {
                if (base + lane < b_hi) latch_error(a.err, kDevBounds);
                p = 0;
            }
            my_phys = p;
        };
        refresh(b_lo);
        auto tile_of = [&](int b, const uint16_t *base) {
            if (b - win_base >= 32) refresh(b);
            const int32_t phys = __shfl_sync(0xffffffffu, my_phys, b - win_base);
            return base + ((int64_t)phys * Hkv + h) * 16 * D;
        };
        auto valid_of = [&](int b) {
            const int pos0 = (sh + b) * 16;
            return min(16, L - pos0);
        };

        BlockRegs<D> b0, b1;
        load_block<D>(b0, tile_of(b_lo, kc), tile_of(b_lo, vc), lr, lq);
        for (int b = b_lo; b < b_hi; b += 2) {
            if (b + 1 < b_hi) load_block<D>(b1, tile_of(b + 1, kc), tile_of(b + 1, vc), lr, lq);
            attend_block<D>(st, b0, qf, lr, lq, valid_of(b), a.scale_log2);
            if (b + 1 >= b_hi) break;
            if (b + 2 < b_hi) load_block<D>(b0, tile_of(b + 2, kc), tile_of(b + 2, vc), lr, lq);
            attend_block<D>(st, b1, qf, lr, lq, valid_of(b + 1), a.scale_log2);
        }

        // row-group reduction of the thread-partial sums
#pragma unroll
        for (int off = 4; off < 32; off <<= 1) {
            st.l[0] += __shfl_xor_sync(0xffffffffu, st.l[0], off);
            st.l[1] += __shfl_xor_sync(0xffffffffu, st.l[1], off);
        }
        const int slot_part = lay.prefix_parts + part;
#pragma unroll
        for (int c = 0; c < 2; ++c) {
            const int hd = 2 * lq + c;
            if (hd < g) {
                const int64_t slot = ((int64_t)r * Hq + h * g + hd) * lay.parts_per_head + slot_part;
                float *dst = o_part + slot * D;
#pragma unroll
                for (int half = 0; half < D / 64; ++half) {
                    const int i0 = half * 4;
                    float4 v0 = make_float4(st.o[i0][c], st.o[i0][2 + c], st.o[i0 + 1][c],
                                            st.o[i0 + 1][2 + c]);
                    float4 v1 = make_float4(st.o[i0 + 2][c], st.o[i0 + 2][2 + c],
                                            st.o[i0 + 3][c], st.o[i0 + 3][2 + c]);
                    float4 *p4 = reinterpret_cast<float4 *>(dst + half * 64 + lr * 8);
                    p4[0] = v0;
                    p4[1] = v1;
                }
                if (lr == 0) ml_part[slot] = make_float2(st.m[c], st.l[c]);
            }
        }
        if (x == seg_off && lane == 0) {
            // the segment's part counts for the combine: private pieces in the
            // low half, the prefix pass's partials of its group in the high one
            const int32_t n_priv = (int32_t)((seg_off + n - 1) / per - seg_off / per + 1);
            const int32_t n_pre = lay.prefix_parts > 0 && a.num_groups > 0
                                      ? min((sh + lay.prefix_blocks_per_part - 1) / lay.prefix_blocks_per_part,
                                            lay.prefix_parts)
                                      : 0;
            nparts[(int64_t)r * Hkv + h] = n_priv | (n_pre << 16);
        }
        x = piece_end;
      }
    }
    // the last warp out leaves both counters at zero for the next call
    if (lane == 0 && atomicAdd(a.sched + 1, 1) == (int)(gridDim.x * kWarps) - 1) {
        atomicExch(a.sched, 0);
        atomicExch(a.sched + 1, 0);
    }
    if (after_prefix) pdl_wait();
}

// Merge the partials of each (request, kv head) with log-sum-exp weights:
// one warp per (request, kv head) merges the g q heads of that kv head, which
// share one list of parts (the group's prefix splits, then the private
// pieces).  Lane k holds part k's (m, l) for every head; lane c holds
// elements [c*E, c*E + E) of every head's output.  All loads of a round are
// in flight together.
template <int D, int G>
__global__ void __launch_bounds__(128) decode_combine_kernel(DecodeArgs a, DecodeLayout lay) {
    constexpr int E = D / 32;   // output elements per lane and head
    // G: q heads per kv head rounded up to 4 or 8 (g <= G)
    pdl_wait();
    const int lane = threadIdx.x & 31;
    const int64_t item = (int64_t)blockIdx.x * (blockDim.x / 32) + (threadIdx.x >> 5);
    if (item >= (int64_t)lay.R * lay.Hkv) return;
    const int r = (int)(item / lay.Hkv), h = (int)(item % lay.Hkv);
    const int g = lay.g;
    const float *o_part = reinterpret_cast<const float *>(static_cast<const char *>(a.ws) + lay.off_o);
    const float2 *ml_part =
        reinterpret_cast<const float2 *>(static_cast<const char *>(a.ws) + lay.off_ml);
    const int32_t *nparts =
        reinterpret_cast<const int32_t *>(static_cast<const char *>(a.ws) + lay.off_nparts);
    // The part counts written by the split pass (private pieces | prefix
    // partials << 16) and, in the same round of loads, the (m, l) of every
    // part slot: lane k holds slot k (prefix partials from 0, private pieces
    // from prefix_parts); slots beyond the counts are masked once they are
    // known (they may hold anything).
    const int32_t counts = nparts[item];
    const int64_t head0 = (int64_t)r * lay.Hq + (int64_t)h * g;   // (request, q head) index of head 0
    float2 mlv[G];
#pragma unroll
    for (int hd = 0; hd < G; ++hd) {
        mlv[hd] = make_float2(-INFINITY, 0.f);
        if (hd < g && lane < lay.parts_per_head) mlv[hd] = ml_part[(head0 + hd) * lay.parts_per_head + lane];
    }
    const int n_priv = min(max(counts & 0xFFFF, 0), kMaxPrivateParts);
    const int n_pre = min((counts >> 16) & 0xFFFF, lay.prefix_parts);
    const int total = min(n_pre + n_priv, 32);
    const bool live = lane < n_pre || (lane >= lay.prefix_parts && lane < lay.prefix_parts + n_priv);
    // parts in merge order: the prefix partials, then the private pieces
    auto part_lane = [&](int k) { return k < n_pre ? k : lay.prefix_parts + (k - n_pre); };
    auto part_slot = [&](int hd, int k) { return (head0 + hd) * lay.parts_per_head + part_lane(k); };
    // weights: the lane of a slot owns that slot's weight for every head
    float wk[G], mx[G], den[G];
#pragma unroll
    for (int hd = 0; hd < G; ++hd) {
        mx[hd] = (hd < g && live) ? mlv[hd].x : -INFINITY;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) mx[hd] = fmaxf(mx[hd], __shfl_xor_sync(0xffffffffu, mx[hd], off));
    }
#pragma unroll
    for (int hd = 0; hd < G; ++hd) {
        const float w = (hd < g && live) ? fast_exp2(mlv[hd].x - mx[hd]) : 0.f;
        den[hd] = (hd < g && live) ? w * mlv[hd].y : 0.f;
        wk[hd] = w;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) den[hd] += __shfl_xor_sync(0xffffffffu, den[hd], off);
    }
    float acc[G][E];
#pragma unroll
    for (int hd = 0; hd < G; ++hd)
#pragma unroll
        for (int e = 0; e < E; ++e) acc[hd][e] = 0.f;
    // parts in rounds of KR (KR x G element vectors in flight per lane)
    constexpr int KR = 16 / G;
    for (int k0 = 0; k0 < total; k0 += KR) {
        float v[KR][G][E];
#pragma unroll
        for (int u = 0; u < KR; ++u)
#pragma unroll
            for (int hd = 0; hd < G; ++hd) {
#pragma unroll
                for (int e = 0; e < E; ++e) v[u][hd][e] = 0.f;
                if (k0 + u < total && hd < g) {
                    const float *src = o_part + part_slot(hd, k0 + u) * D + lane * E;
                    if constexpr (E == 4) {
                        const float4 t = *reinterpret_cast<const float4 *>(src);
                        v[u][hd][0] = t.x; v[u][hd][1] = t.y; v[u][hd][2] = t.z; v[u][hd][3] = t.w;
                    } else {
                        const float2 t = *reinterpret_cast<const float2 *>(src);
                        v[u][hd][0] = t.x; v[u][hd][1] = t.y;
                    }
                }
            }
#pragma unroll
        for (int u = 0; u < KR; ++u)
#pragma unroll
            for (int hd = 0; hd < G; ++hd) {
                const float w = __shfl_sync(0xffffffffu, wk[hd], k0 + u < total ? part_lane(k0 + u) : 0);
#pragma unroll
                for (int e = 0; e < E; ++e) acc[hd][e] += w * v[u][hd][e];
            }
    }
#pragma unroll
    for (int hd = 0; hd < G; ++hd) {
        if (hd >= g) break;
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

DecodeLayout decode_layout(int32_t R, int32_t Hq, int32_t Hkv, int32_t d, int32_t max_blocks,
                           int32_t num_groups, int32_t max_group_blocks, int32_t max_group_members,
                           int32_t num_sms) {
    DecodeLayout L{};
    L.R = R; L.Hq = Hq; L.Hkv = Hkv; L.d = d; L.g = Hq / Hkv;
    L.sms = num_sms > 0 ? num_sms : 148;
    L.prefix_blocks_per_part = 8;
    L.prefix_parts = 0;
    if (num_groups > 0 && max_group_blocks > 0 && max_group_members > 0) {
        // Key splits of the prefix pass: one CTA per (group, kv head, member
        // tile, split), one CTA per SM.  The private split pass runs on the
        // SMs the prefix pass leaves free (it starts as soon as the prefix
        // pass has), so a step costs about
        //   max(prefix critical path, (prefix SM-time + split SM-time) / SMs).
        // Measured on GB300: a prefix CTA costs about 13 us of fixed work
        // (set-up, Q tile, pipeline fill, partial writes) plus 2.1 us per key
        // tile; the split pass streams about 41 GB/s per SM.  The private
        // work is estimated from the table width (60 % of the blocks past the
        // longest prefix), which only steers the split count.
        const int per_item = 2 * (128 / L.g);   // members per work item (two 128-row tiles)
        const int64_t tiles = (int64_t)num_groups * Hkv * ((max_group_members + per_item - 1) / per_item);
        const int sms = num_sms > 0 ? num_sms : 148;
        const int key_tiles = (max_group_blocks + 7) / 8;
        const double unit_bytes = 16.0 * d * 2 * 2;   // K + V of one (block, kv head)
        const double priv_blocks = 0.6 * std::max(1, max_blocks - max_group_blocks);
        const double split_sm_us = (double)R * Hkv * priv_blocks * unit_bytes / 41e3;
        int best = 1;
        double best_t = 1e300;
        for (int sp = 1; sp <= kMaxPrefixParts && sp <= key_tiles; ++sp) {
            const int per = (key_tiles + sp - 1) / sp;
            const int64_t ctas = tiles * sp;
            const double cta_us = 13.0 + 2.1 * per;
            const double crit = (double)((ctas + sms - 1) / sms) * cta_us;
            const double t = std::max(crit, (ctas * cta_us + split_sm_us) / sms);
            if (t < best_t - 1e-9) { best_t = t; best = sp; }
        }
        const int per_tiles = (key_tiles + best - 1) / best;
        L.prefix_blocks_per_part = per_tiles * 8;
        L.prefix_parts = (max_group_blocks + L.prefix_blocks_per_part - 1) / L.prefix_blocks_per_part;
    }
    L.parts_per_head = L.prefix_parts + kMaxPrivateParts;
    const size_t slots = (size_t)R * Hq * L.parts_per_head;
    auto up = [](size_t x) { return (x + 255) & ~(size_t)255; };
    L.off_o = 0;
    L.off_ml = up(slots * d * sizeof(float));
    L.off_nparts = L.off_ml + up(slots * sizeof(float2));
    L.total = L.off_nparts + up((size_t)R * Hkv * sizeof(int32_t));
    return L;
}

template <int D>
static cudaError_t launch_decode_t(const DecodeLayout &L, const DecodeArgs &a, int num_sms,
                                   int32_t num_blocks_pool, cudaStream_t stream, Tracer *tr) {
    if (L.prefix_parts > 0 && a.num_groups > 0) {
        cudaError_t e = launch_decode_prefix(L, a, num_blocks_pool, stream, tr);
        if (e != cudaSuccess) return e;
    }
    const size_t smem = (size_t)(L.R + 1) * sizeof(int32_t);
    static size_t attr_bytes = 0;
    if (smem > 48 * 1024 && smem > attr_bytes) {
        cudaError_t e = cudaFuncSetAttribute(decode_split_kernel<D>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        attr_bytes = smem;
    }
    if (tr) tr->begin(kKernelDecodeSplit, stream);
    const int32_t after_prefix = (L.prefix_parts > 0 && a.num_groups > 0) ? 1 : 0;
    cudaError_t e = launch_pdl(decode_split_kernel<D>, dim3(num_sms), dim3(kThreads), smem, stream,
                               a, L, num_blocks_pool, after_prefix);
    if (tr) tr->end(kKernelDecodeSplit, stream);
    if (e != cudaSuccess) return e;
    // four warps per CTA: small batches spread over more SMs
    const int64_t items = (int64_t)L.R * L.Hkv;
    const int64_t grid = (items + 3) / 4;
    if (grid > 0x7fffffff) return cudaErrorInvalidConfiguration;
    if (tr) tr->begin(kKernelDecodeCombine, stream);
    e = L.g <= 4 ? launch_pdl(decode_combine_kernel<D, 4>, dim3((unsigned)grid), dim3(128), 0, stream, a, L)
                 : launch_pdl(decode_combine_kernel<D, 8>, dim3((unsigned)grid), dim3(128), 0, stream, a, L);
    if (tr) tr->end(kKernelDecodeCombine, stream);
    return e;
}

cudaError_t launch_decode(const DecodeLayout &L, const DecodeArgs &a, int num_sms,
                          int32_t num_blocks_pool, cudaStream_t stream, Tracer *tr) {
    if (L.d == 128) return launch_decode_t<128>(L, a, num_sms, num_blocks_pool, stream, tr);
    return launch_decode_t<64>(L, a, num_sms, num_blocks_pool, stream, tr);
}

}  // namespace pkv
