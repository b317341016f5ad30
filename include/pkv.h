/*
 * pkv.h -- C ABI of the prefix-cached paged-attention library (libpkv.so).
 *
 * The library implements the data-parallel hot path of the "Reuse plane" of
 * the compliance serving stack of arXiv 2605.11232 (Fig. 1): attention over a
 * KV cache kept in fixed-size physical blocks addressed through per-request
 * block tables (PagedAttention, Sec. 2 and Sec. 5.4), whose leading blocks can
 * be a policy/schema prefix shared by many requests and stored once
 * (Automatic Prefix Caching, Sec. 2 and Sec. 5.4; the design rule at the end
 * of Sec. 3 that shared prefixes are not recomputed).
 *
 * Contents: the block pool and its reference counts (kv_pool_*), slot
 * mapping (kv_slot_mapping), the prefix-caching index (pkv_prefix_cache_*)
 * and the prefix groups of a decode batch (pkv_prefix_groups_build),
 * the adapter-first, length-bucketed dispatch of a multi-adapter request
 * (pkv_lora_dispatch) and the segmented multi-adapter LoRA projection
 * (pkv_lora_sgmv), the cache write (kv_cache_write), suffix prefill
 * (paged_attn_prefill; with the write fused in: paged_attn_prefill_append;
 * tree-shaped draft verification: paged_attn_verify_tree, pkv_tree_masks;
 * with each group's shared prefix read once: paged_attn_verify_tree_grouped,
 * pkv_verify_groups_build),
 * decode (paged_attn_decode; with the write fused in:
 * paged_attn_decode_append; without a caller workspace:
 * paged_attn_decode_noalloc; one host-driven step with its copies:
 * paged_attn_decode_step), KV-block transfer between pools
 * (pkv_blocks_gather / pkv_blocks_scatter), per-kernel tracing
 * (pkv_trace_*), device error reporting (pkv_check_device_errors), the host
 * check of block tables (pkv_check_block_table) and a test aid for the
 * bounded waits (pkv_selftest_wait_timeout).
 *
 * Conventions for every call
 *  - All device buffers are owned by the caller.  The library keeps host
 *    metadata (free list, reference counts, TMA descriptors) and one 4-byte
 *    device word per pool (its error word), allocated by kv_pool_create.
 *  - "device" pointers are CUDA global-memory addresses on the pool's device;
 *    "host" pointers are ordinary CPU memory.  Device buffers must be 16-byte
 *    aligned and contiguous in the stated layout.
 *  - Kernels are enqueued on `stream` (a cudaStream_t; NULL is the legacy
 *    default stream) and return before they run.  Argument errors are found
 *    on the host and returned before anything is enqueued; errors seen by a
 *    kernel (an out-of-range slot or block id, a bounded wait that ran out)
 *    are latched in the pool's device error word and reported by
 *    pkv_check_device_errors.
 *  - Every call returns PKV_OK (0) or a negative pkv_status; pkv_last_error()
 *    then gives a message (per thread).  No C++ exception crosses the ABI.
 *  - Element type: bf16 only.  Block size: 16 tokens.  Head dim: 64 or 128.
 *    num_q_heads must be a multiple of num_kv_heads; q heads h belong to kv
 *    head h / (num_q_heads / num_kv_heads) (contiguous GQA grouping).
 *  - A pool handle is not thread-safe; calls on one handle must not overlap
 *    in time on the host.  On the GPU the kernels of one pool share only its
 *    error word, so launches on several streams may be in flight together as
 *    long as each has its own workspace and outputs and they write no common
 *    slots.  Different pools may be used from different host threads.
 */
#ifndef PKV_H
#define PKV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct pkv_pool *pkv_pool_t;
typedef void *pkv_stream_t; /* a cudaStream_t */
typedef void *pkv_event_t;  /* a cudaEvent_t */

typedef enum {
    PKV_OK = 0,
    PKV_ERR_INVALID_ARG = -1,        /* null pointer, bad size or layout        */
    PKV_ERR_OUT_OF_BLOCKS = -2,      /* free list cannot satisfy an allocation   */
    PKV_ERR_REFCOUNT = -3,           /* release of a free block, bad id          */
    PKV_ERR_SHARED_BLOCK_WRITE = -4, /* a slot lies in a block with refcount > 1 */
    PKV_ERR_CUDA = -5,               /* a CUDA runtime/driver call failed        */
    PKV_ERR_UNSUPPORTED = -6,        /* shape outside what the kernels handle    */
    PKV_ERR_WORKSPACE = -7,          /* workspace missing or too small           */
    PKV_ERR_DEVICE_TIMEOUT = -8,     /* a bounded device wait ran out            */
    PKV_ERR_DEVICE_BOUNDS = -9       /* a kernel met an out-of-range slot/block  */
} pkv_status;

enum { PKV_DTYPE_BF16 = 1 };

/* Physical block pool.  K and V caches are separate device arrays of
 * num_blocks * num_kv_heads * block_size * head_dim bf16 values laid out as
 * [num_blocks][num_kv_heads][block_size][head_dim]: the 16 tokens of one
 * (block, kv head) pair are one contiguous tile (4 KiB at head_dim 128). */
typedef struct {
    int32_t num_blocks;      /* > 0                                              */
    int32_t block_size;      /* must be 16                                       */
    int32_t num_kv_heads;    /* > 0                                              */
    int32_t head_dim;        /* 64 or 128                                        */
    int32_t dtype;           /* PKV_DTYPE_BF16                                   */
    int32_t reserved;        /* 0                                                */
    uint64_t placement_seed; /* 0: blocks are handed out as 0,1,2,...; otherwise
                                the initial free list is a permutation drawn
                                from this seed (splitmix64 + Fisher-Yates)      */
} pkv_pool_desc;

/* Shared-prefix groups of a decode batch (APC, Sec. 5.4).  Group g owns the
 * first group_blocks[g] table entries of each of its member requests: those
 * entries are the same physical blocks for every member, hold full 16-token
 * blocks of the shared prefix, and are never written.  With groups, decode
 * reads each shared block once per group and kv head instead of once per
 * request.  All arrays are device arrays.  The two host bounds size the
 * workspace and the prefix pass's grid; the device arrays are not read on the
 * host, so a group with more blocks or members than the bounds is not
 * detected: the kernels stay inside the workspace and the tables, but the
 * blocks or members past a bound are left out of that request's attention.
 * pkv_prefix_groups_build returns exact bounds. */
typedef struct {
    int32_t num_groups;        /* G >= 0; 0 means no sharing information         */
    int32_t max_group_blocks;  /* host upper bound on group_blocks[g]            */
    int32_t max_group_members; /* host upper bound on members of one group       */
    int32_t reserved;          /* 0                                              */
    const int32_t *group_start;  /* [G+1] CSR offsets into member_req            */
    const int32_t *member_req;   /* [group_start[G]] request indices, by group   */
    const int32_t *group_blocks; /* [G] shared leading blocks of group g (>= 0)  */
    const int32_t *group_of_req; /* [num_requests] group of request r, -1: none  */
} pkv_prefix_groups;

/* ---- a1: pool and reference counts (host) ------------------------------- */

/* Create a pool over caller-owned device caches (Sec. 2, Sec. 5.4: paged KV
 * memory).  k_cache/v_cache: device, layout above; both NULL gives a
 * metadata-only pool (allocation calls work, kernel calls fail with
 * PKV_ERR_INVALID_ARG).  On success *out owns host metadata and 16 bytes of
 * device words (error word, split-pass counters); free it with
 * kv_pool_destroy.  Errors: INVALID_ARG, UNSUPPORTED
 * (block_size != 16, head_dim not 64/128, dtype not bf16), CUDA. */
int kv_pool_create(const pkv_pool_desc *desc, void *k_cache, void *v_cache, pkv_pool_t *out);

/* Free the host metadata and the device words (not the caches).  NULL is a no-op. */
int kv_pool_destroy(pkv_pool_t pool);

/* Take n free blocks; their ids go to ids_out (host, n entries), each with
 * reference count 1.  All or nothing: OUT_OF_BLOCKS leaves the pool as it was. */
int kv_pool_alloc(pkv_pool_t pool, int32_t n, int32_t *ids_out);

/* Add one reference to each listed block (host ids): a request that reuses a
 * cached prefix holds its blocks this way (APC, Sec. 5.4).  REFCOUNT if an id
 * is out of range or free; nothing changes on error. */
int kv_pool_retain(pkv_pool_t pool, const int32_t *ids, int32_t n);

/* Drop one reference from each listed block (host ids); a block whose count
 * reaches 0 returns to the free list.  REFCOUNT on a free or out-of-range id,
 * or on an id listed more times than it has references; nothing changes on
 * error. */
int kv_pool_release(pkv_pool_t pool, const int32_t *ids, int32_t n);

/* Reference count of one block (0 = free).  INVALID_ARG on a bad id. */
int kv_pool_refcount(pkv_pool_t pool, int32_t id, int32_t *out);

/* Number of free blocks. */
int kv_pool_num_free(pkv_pool_t pool, int32_t *out);

/* One request's block-table row (a1 + a2): retain the n_prefix shared prefix
 * blocks `prefix_ids` (host; may be NULL when n_prefix is 0), allocate
 * n_blocks - n_prefix private blocks, and write the row to row_out (host,
 * n_blocks entries): prefix ids first, then the new private ids in order.
 * All or nothing. */
int kv_pool_alloc_sequence(pkv_pool_t pool, const int32_t *prefix_ids, int32_t n_prefix,
                           int32_t n_blocks, int32_t *row_out);

/* ---- a2: slot mapping (host) -------------------------------------------- */

/* Slot of every new token (PagedAttention addressing, Sec. 2): new token i of
 * request r is at position p = context_lens[r] - new_lens[r] + i and goes to
 * slot block_table[r][p / 16] * 16 + p % 16.  Tokens are numbered request
 * after request.  All arrays are host arrays; block_table is [R][max_blocks]
 * row-major; slots_out has sum(new_lens) entries.  With a pool (non-NULL),
 * every target block must be allocated and unshared: a slot in a block with
 * reference count > 1 returns SHARED_BLOCK_WRITE (shared prefix blocks are
 * immutable), a free block REFCOUNT, a block id outside the pool INVALID_ARG.
 * pool may be NULL (no ownership checks). */
int kv_slot_mapping(pkv_pool_t pool, const int32_t *block_table, int32_t max_blocks,
                    const int32_t *context_lens, const int32_t *new_lens, int32_t num_requests,
                    int64_t *slots_out);

/* Host check of a batch's block tables before a launch (the kernels check
 * every block id they read as well, latching DEVICE_BOUNDS): for each request
 * r, the entries a kernel reads, block_table[r][0 .. ceil(context_lens[r] /
 * 16)), must name allocated blocks of the pool; later entries are never read
 * and are not checked.  block_table: host int32 [num_requests][max_blocks];
 * context_lens: host int32 [num_requests].  Returns PKV_OK, INVALID_ARG (a
 * negative context, one longer than 16 * max_blocks, or a block id outside
 * the pool: the condition the kernels latch as DEVICE_BOUNDS) or REFCOUNT (a
 * free block); *bad_request_out (may be NULL) gets the first offending
 * request, -1 when none. */
int pkv_check_block_table(pkv_pool_t pool, const int32_t *block_table, int32_t max_blocks,
                          int32_t num_requests, const int32_t *context_lens, int32_t *bad_request_out);

/* ---- automatic prefix caching (host) -------------------------------------- */

/* An index of cached full blocks of a pool, keyed by token prefix: the prefix
 * reuse of Automatic Prefix Caching (Sec. 5.4).  A request's tokens are cut
 * into blocks of 16; a full block is keyed by its whole token prefix (its own
 * 16 tokens and all before them).  The index holds one reference on every
 * block it caches, so a cached block outlives the request that wrote it;
 * blocks that only the index holds are evicted least recently used first.
 * Keys are chained 64-bit hashes checked token by token, so a collision never
 * shares a block.  Host only; a handle is not thread-safe, and the pool must
 * outlive it. */
typedef struct pkv_prefix_cache *pkv_prefix_cache_t;

/* flags for pkv_prefix_cache_create: test aid that keeps 4 bits of every key,
 * so that most lookups meet colliding keys. */
#define PKV_PREFIX_CACHE_WEAK_HASH 1

int pkv_prefix_cache_create(pkv_pool_t pool, int32_t flags, pkv_prefix_cache_t *out);
/* Drops the index's reference on every cached block. NULL is a no-op. */
int pkv_prefix_cache_destroy(pkv_prefix_cache_t cache);
/* The longest run of cached full blocks that begins tokens[0 .. n_tokens):
 * their ids (at most max_ids) go to ids_out[0 .. *n_ids_out), each retained
 * once more for the caller's request (refcount + 1), so they can head its
 * block-table row; the rest of the row comes from kv_pool_alloc, and the
 * request releases the whole row when it ends.  Marks them used. */
int pkv_prefix_cache_match(pkv_prefix_cache_t cache, const int32_t *tokens, int32_t n_tokens,
                           int32_t *ids_out, int32_t max_ids, int32_t *n_ids_out);
/* Register the full blocks of tokens[0 .. n_tokens) held in ids[0 .. n_ids)
 * (block j holds tokens [16j, 16j + 16); the caller holds every id and has
 * written its K/V).  A block whose prefix is not cached yet is added and
 * retained by the index; a prefix already cached keeps its block.  Every
 * block of the path is marked used.  *n_added_out (may be NULL) counts the
 * new entries.  Errors: REFCOUNT for a free id, INVALID_ARG. */
int pkv_prefix_cache_insert(pkv_prefix_cache_t cache, const int32_t *tokens, int32_t n_tokens,
                            const int32_t *ids, int32_t n_ids, int32_t *n_added_out);
/* Evict up to n_wanted cached blocks that no request holds (the index's
 * reference is the only one) and whose cached successors are gone: least
 * recently used first, then the deeper block, then the older entry.  Each is
 * released to the pool's free list; their ids go to ids_out[0 ..
 * *n_evicted_out). */
int pkv_prefix_cache_evict(pkv_prefix_cache_t cache, int32_t n_wanted, int32_t *ids_out,
                           int32_t *n_evicted_out);
/* Number of cached blocks. */
int pkv_prefix_cache_size(pkv_prefix_cache_t cache, int32_t *n_cached_out);

/* Prefix groups of a decode batch from its block tables (host; the
 * descriptor that paged_attn_decode's shared-prefix pass takes): requests
 * whose rows begin with the same physical blocks, e.g. blocks handed out by
 * pkv_prefix_cache_match, share those blocks.  Rule: candidates are grouped
 * by their first block id (in request order).  A member's shareable run is
 * the run of equal leading ids it has with the group's first candidate,
 * capped at (context_lens[r] - 1) / 16 blocks so that the block holding its
 * query token stays private; candidates whose run is shorter than
 * min_shared_blocks (>= 1) stay out; the group shares the shortest run of
 * its members; groups of one member are dropped (their request gets -1).
 *  block_table: host int32 [R][max_blocks]; context_lens: host int32 [R].
 *  Outputs (host): group_of_req_out [R] (-1: no group), group_start_out
 *  [R + 1] (CSR offsets into member_req_out; G + 1 used), member_req_out [R],
 *  group_blocks_out [R] (G used), *num_groups_out = G, and the largest group
 *  blocks and member counts. */
int pkv_prefix_groups_build(const int32_t *block_table, int32_t max_blocks, int32_t num_requests,
                            const int32_t *context_lens, int32_t min_shared_blocks,
                            int32_t *group_of_req_out, int32_t *group_start_out,
                            int32_t *member_req_out, int32_t *group_blocks_out,
                            int32_t *num_groups_out, int32_t *max_group_blocks_out,
                            int32_t *max_group_members_out);

/* ---- multi-adapter dispatch (host) ---------------------------------------- */

/* Batches of a request whose items go to different LoRA adapters (Sec. 5.6:
 * group the items by adapter, bucket each group by prompt length, run each
 * bucket as one batch call, return the results in request order).
 *  adapter_id, prompt_len: host int32 [n], both >= 0.
 *  bucket_edges: host int32 [n_edges], strictly ascending (may be NULL when
 *    n_edges is 0); an item of length L goes to bucket
 *    #{j : L >= bucket_edges[j]} (edges {512, 2048}: short, medium, long).
 *  max_batch: > 0 caps a batch at that many items (a larger bucket runs as
 *    consecutive batches, the last one shorter); 0 leaves buckets whole.
 * Order: adapters by their first item in the request, buckets of an adapter
 * from the shortest range up, items of a bucket in request order.
 * Outputs (host, caller-sized): order_out [n] (the request index of the k-th
 * item executed: result k belongs to item order_out[k]), batch_start_out
 * [n + 1] (batch b is order_out[batch_start_out[b] .. batch_start_out[b+1])),
 * batch_adapter_out [n], batch_bucket_out [n], *n_batches_out.
 * Errors: INVALID_ARG (negative sizes, ids or lengths; edges not ascending);
 * nothing is written then except the message. */
int pkv_lora_dispatch(const int32_t *adapter_id, const int32_t *prompt_len, int32_t n,
                      const int32_t *bucket_edges, int32_t n_edges, int32_t max_batch,
                      int32_t *order_out, int32_t *batch_start_out, int32_t *batch_adapter_out,
                      int32_t *batch_bucket_out, int32_t *n_batches_out);

/* ---- multi-adapter LoRA projection (device) ---------------------------------- */

/* The segmented multi-adapter LoRA projection of Sec. 5.6 (one base model,
 * several adapters, a mixed request run as the per-adapter batches of
 * pkv_lora_dispatch): for the tokens t of segment s with adapter
 * a = seg_adapter[s],
 *     y_t = W x_t + scale[a] * B_a (A_a x_t)     (a = -1: y_t = W x_t).
 * The paper names LoRA adapters but prints no formula; this is the standard
 * low-rank update.  Both products run on the tensor cores in one kernel (bf16
 * operands, fp32 accumulation); A_a x_t is scaled and rounded to bf16 before
 * its product with B_a; y is rounded to bf16.
 *  x: device bf16 [num_tokens][d_in]; w: device bf16 [d_out][d_in];
 *  lora_a: device bf16 [num_adapters][rank][d_in];
 *  lora_b: device bf16 [num_adapters][d_out][rank];
 *  y: device bf16 [num_tokens][d_out]; all 16-byte aligned.
 *  scale: host float [num_adapters]; seg_start: host int32 [num_segments + 1]
 *  from 0 to num_tokens, non-decreasing; seg_adapter: host int32
 *  [num_segments], each in [-1, num_adapters).
 *  error_word: device int32 the kernel latches DEVICE_TIMEOUT into if a
 *  bounded wait runs out (may be NULL).
 * Limits: d_in a multiple of 64, d_out of 256, rank 16, 32, 48 or 64
 * (UNSUPPORTED otherwise); each segment is cut into 128-row tiles, at most
 * PKV_LORA_MAX_TILES per call (UNSUPPORTED beyond: split the call).
 * Errors: INVALID_ARG, UNSUPPORTED, CUDA. */
#define PKV_LORA_MAX_TILES 1024
int pkv_lora_sgmv(const void *x, const void *w, const void *lora_a, const void *lora_b,
                  const float *scale, const int32_t *seg_start, const int32_t *seg_adapter,
                  int32_t num_segments, int32_t num_tokens, int32_t d_in, int32_t d_out,
                  int32_t rank, int32_t num_adapters, void *y, int32_t *error_word,
                  pkv_stream_t stream);

/* ---- a3: cache write (device) ------------------------------------------- */

/* Scatter new-token keys and values into their slots (bit-exact copy).
 * k_new, v_new: device bf16 [num_tokens][num_kv_heads][head_dim].
 * slot_mapping: device int64 [num_tokens]; slot s goes to block s / 16, offset
 * s % 16; s < 0 skips the token; s >= num_blocks * 16 is skipped and latches
 * DEVICE_BOUNDS.  Two tokens with the same slot: undefined which one lands.
 * num_tokens == 0 is a no-op. */
int kv_cache_write(pkv_pool_t pool, const void *k_new, const void *v_new,
                   const int64_t *slot_mapping, int32_t num_tokens, pkv_stream_t stream);

/* ---- a4: suffix prefill over cached context (device) -------------------- */

/* Attention of the new (suffix or chunk) tokens of each request: new token i
 * of request r, at position p = context_lens[r] - n_r + i with
 * n_r = cu_seqlens_q[r+1] - cu_seqlens_q[r], attends to every cached key of
 * the request (shared prefix included) and causally to the new keys, i.e. to
 * positions 0..p, read through the block table (Sec. 5.4: the cached prefix
 * is reused, only the suffix is computed).  The new tokens' K/V must already
 * be in the cache (kv_cache_write).
 *  q, out: device bf16 [T][num_q_heads][head_dim], T = cu_seqlens_q[R].
 *  lse: device fp32 [T][num_q_heads] natural-log log-sum-exp, or NULL.
 *  cu_seqlens_q: device int32 [R+1], non-decreasing from 0.
 *  context_lens: device int32 [R], context_lens[r] >= n_r (includes them).
 *  block_table: device int32 [R][max_blocks]; entries past ceil(L/16) unread.
 *  max_seqlen_q: host upper bound on n_r (sizes the grid); requests with
 *  n_r = 0 are skipped.
 *  scale: softmax scale (normally 1/sqrt(head_dim)).
 * Errors: INVALID_ARG, UNSUPPORTED (num_q_heads / num_kv_heads > 128), CUDA. */
int paged_attn_prefill(pkv_pool_t pool, const void *q, void *out, float *lse,
                       const int32_t *cu_seqlens_q, const int32_t *context_lens,
                       const int32_t *block_table, int32_t max_blocks, int32_t num_requests,
                       int32_t max_seqlen_q, int32_t num_q_heads, float scale,
                       pkv_stream_t stream);

/* paged_attn_prefill with the cache write of the new tokens fused in (Sec.
 * 5.4: only the new tokens cost anything once the prefix is cached): new
 * token i of request r is stored into its slot (position
 * context_lens[r] - n_r + i, through block_table) by the prefill kernel, and
 * the new keys and values are read from k_new / v_new while attending.  The
 * outputs, and the pool afterwards, equal kv_cache_write of those tokens
 * followed by paged_attn_prefill.
 *  k_new, v_new: device bf16 [num_new_tokens][num_kv_heads][head_dim],
 *  16-byte aligned, rows in q's order (num_new_tokens = cu_seqlens_q[R]).
 *  Each request's cached part, context_lens[r] - n_r, must be whole blocks (a
 *  multiple of 16, as prefix caching leaves it): a request that is not is
 *  skipped and latches DEVICE_BOUNDS.  The blocks of the new tokens must be
 *  the request's own (reference count 1).
 * Every other argument and the errors are those of paged_attn_prefill. */
int paged_attn_prefill_append(pkv_pool_t pool, const void *q, const void *k_new, const void *v_new,
                              int32_t num_new_tokens, void *out, float *lse, const int32_t *cu_seqlens_q,
                              const int32_t *context_lens, const int32_t *block_table, int32_t max_blocks,
                              int32_t num_requests, int32_t max_seqlen_q, int32_t num_q_heads, float scale,
                              pkv_stream_t stream);

/* ---- speculative-decode verification with tree-shaped drafts (device) ---- */

/* paged_attn_prefill where each request's new tokens are draft tokens of a
 * tree (Sec. 5.3: speculative decoding verifies several drafts in one pass):
 * new token i of a request sees every context token and exactly the new
 * tokens j whose bit j is set in tree_mask[cu_seqlens_q[r] + i] (its
 * ancestors and itself; pkv_tree_masks builds them from parent indices).
 * tree_mask: device uint64 [T], 8-byte aligned.  At most 64 new tokens per
 * request (max_seqlen_q <= 64, else UNSUPPORTED).  Every other argument,
 * layout and error as paged_attn_prefill.  A chain mask (bits 0..i for token
 * i) gives paged_attn_prefill's causal result. */
int paged_attn_verify_tree(pkv_pool_t pool, const void *q, void *out, float *lse,
                           const int32_t *cu_seqlens_q, const int32_t *context_lens,
                           const int32_t *block_table, int32_t max_blocks, int32_t num_requests,
                           int32_t max_seqlen_q, int32_t num_q_heads, float scale,
                           const uint64_t *tree_mask, pkv_stream_t stream);

/* Shared-prefix groups of a verification batch (Sec. 5.3 with Sec. 5.4):
 * the draft tokens of the requests that share a cached prefix, grouped so
 * that the prefix is read once per group and kv head rather than once per
 * request.  Group g's requests all name the same group_blocks[g] physical
 * blocks first in their table rows (full blocks of the shared prefix, before
 * every draft); member_token lists the draft tokens (rows of q) of those
 * requests.  All arrays are device arrays; pkv_verify_groups_build makes them
 * (on the host) from each request's group.  As with pkv_prefix_groups, the
 * host bounds size the workspace and the grid and are not checked against
 * the device arrays: members or blocks past a bound are left out. */
typedef struct {
    int32_t num_groups;        /* G >= 0; 0: no sharing, every key in the private pass */
    int32_t max_group_blocks;  /* host upper bound on group_blocks[g]             */
    int32_t max_group_tokens;  /* host upper bound on the draft tokens of a group */
    int32_t reserved;          /* 0                                               */
    const int32_t *group_start;   /* [G+1] CSR offsets into member_token          */
    const int32_t *member_token;  /* [group_start[G]] draft-token rows, by group  */
    const int32_t *group_blocks;  /* [G] shared leading blocks of group g         */
    const int32_t *group_row;     /* [G] a block-table row (request) of group g   */
    const int32_t *request_group; /* [num_requests] group of request r, -1: none  */
} pkv_verify_groups;

/* Bytes of workspace paged_attn_verify_tree_grouped needs (host call).
 * num_tokens: draft tokens of the batch (cu_seqlens_q[num_requests]); groups
 * may be NULL.  Errors: INVALID_ARG. */
int paged_attn_verify_tree_workspace_size(pkv_pool_t pool, int32_t num_tokens, int32_t num_q_heads,
                                          int32_t max_blocks, const pkv_verify_groups *groups,
                                          size_t *bytes_out);

/* paged_attn_verify_tree with the shared prefix of each group read once per
 * group and kv head: a tensor-core pass over each group's draft tokens and
 * its shared blocks (all visible to every draft), a pass over each request's
 * keys after them (its private context and its drafts, under the draft
 * masks), and the log-sum-exp merge of the two.  Same result as
 * paged_attn_verify_tree up to rounding (the merge of two partial softmaxes).
 *  num_tokens: cu_seqlens_q[num_requests] (host); the workspace holds
 *  partials for that many rows, and a request whose rows reach past it is
 *  skipped and latches DEVICE_BOUNDS.  groups: as above, or NULL.
 *  A grouped request's cached part, context_lens[r] - n_r, must cover its
 *  group's blocks (else it latches DEVICE_BOUNDS and its outputs are
 *  undefined).
 *  workspace: device, 256-byte aligned, at least
 *  paged_attn_verify_tree_workspace_size() bytes; holds partials between the
 *  passes.
 * Errors: those of paged_attn_verify_tree; UNSUPPORTED beyond 8 q heads per kv
 * head; WORKSPACE. */
int paged_attn_verify_tree_grouped(pkv_pool_t pool, const void *q, void *out, float *lse,
                                   const int32_t *cu_seqlens_q, const int32_t *context_lens,
                                   const int32_t *block_table, int32_t max_blocks, int32_t num_requests,
                                   int32_t num_tokens, int32_t max_seqlen_q, int32_t num_q_heads, float scale,
                                   const uint64_t *tree_mask, const pkv_verify_groups *groups,
                                   void *workspace, size_t workspace_bytes, pkv_stream_t stream);

/* Token groups of a verification batch (host): from cu_seqlens ([R+1],
 * cu_seqlens[0] = 0) and request_group ([R], values in [-1, num_groups)),
 * writes group_start_out [num_groups + 1], member_token_out
 * [cu_seqlens[R]] (the draft tokens of group 0's requests in request order,
 * then group 1's, ...; tokens of ungrouped requests are not listed),
 * group_row_out [num_groups] (the group's first request, -1 if it has none)
 * and *max_group_tokens_out.  All host arrays.  Errors: INVALID_ARG. */
int pkv_verify_groups_build(const int32_t *cu_seqlens, const int32_t *request_group, int32_t num_requests,
                            int32_t num_groups, int32_t *group_start_out, int32_t *member_token_out,
                            int32_t *group_row_out, int32_t *max_group_tokens_out);

/* Draft masks of tree-shaped drafts (host): parent[cu_seqlens[r] + i] is the
 * draft that draft i of request r continues (-1: the context), an earlier
 * draft of the same request; masks_out[cu_seqlens[r] + i] gets bit j set for
 * each draft j on i's path, itself included.  parent, cu_seqlens
 * ([num_requests + 1], cu_seqlens[0] = 0), masks_out: host arrays.  At most
 * 64 drafts per request.  Errors: INVALID_ARG. */
int pkv_tree_masks(const int32_t *parent, const int32_t *cu_seqlens, int32_t num_requests,
                   uint64_t *masks_out);

/* ---- a5-a7: decode (device) ---------------------------------------------- */

/* Bytes of workspace paged_attn_decode needs for these shapes (host call).
 * groups may be NULL. */
int paged_attn_decode_workspace_size(pkv_pool_t pool, int32_t num_requests,
                                     int32_t num_q_heads, int32_t max_blocks,
                                     const pkv_prefix_groups *groups, size_t *bytes_out);

/* One query token per request attends to all context_lens[r] keys of its
 * block list (the decode step of Sec. 5.3's short structured outputs).  The
 * query token's own K/V must already be in the cache.  Keys are split into
 * ranges processed in parallel, each producing an unnormalised partial output
 * with its running max and sum; a combine pass merges them by log-sum-exp
 * weights.  With groups, the shared prefix blocks of each group are processed
 * once per group for all member requests.
 *  q, out: device bf16 [R][num_q_heads][head_dim].
 *  lse: device fp32 [R][num_q_heads] (natural log) or NULL.
 *  context_lens: device int32 [R], each >= 1 (and > 16 * shared blocks).
 *  block_table: device int32 [R][max_blocks].
 *  groups: NULL, or a descriptor as above.
 *  workspace: device scratch of at least paged_attn_decode_workspace_size()
 *  bytes, 256-byte aligned; its contents need no initialisation and are
 *  clobbered.
 * Errors: INVALID_ARG, UNSUPPORTED (group size g > 8), WORKSPACE, CUDA. */
int paged_attn_decode(pkv_pool_t pool, const void *q, void *out, float *lse,
                      const int32_t *context_lens, const int32_t *block_table,
                      int32_t max_blocks, int32_t num_requests, int32_t num_q_heads,
                      float scale, const pkv_prefix_groups *groups, void *workspace,
                      size_t workspace_bytes, pkv_stream_t stream);

/* paged_attn_decode with the cache write of the query tokens fused in: each
 * request's own key and value (the token it decodes, at position
 * context_lens[r] - 1) are stored into the pool by the decode kernels instead
 * of a kv_cache_write launch beforehand, then all context_lens[r] keys are
 * attended to as by paged_attn_decode (Sec. 5.3's decode step; Sec. 5.4's
 * paged cache).  The result, and the pool afterwards, equal kv_cache_write of
 * those tokens to slots block_table[r][(L - 1) / 16] * 16 + (L - 1) % 16
 * followed by paged_attn_decode.
 *  k_new, v_new: device bf16 [R][num_kv_heads][head_dim], 16-byte aligned.
 *  The block holding position L - 1 must be the request's own (reference
 *  count 1; the decode requires its last block private in any case).
 * Every other argument, the workspace and the errors are those of
 * paged_attn_decode. */
int paged_attn_decode_append(pkv_pool_t pool, const void *q, const void *k_new, const void *v_new,
                             void *out, float *lse, const int32_t *context_lens,
                             const int32_t *block_table, int32_t max_blocks, int32_t num_requests,
                             int32_t num_q_heads, float scale, const pkv_prefix_groups *groups,
                             void *workspace, size_t workspace_bytes, pkv_stream_t stream);

/* ---- a decode step from host memory --------------------------------------- */

/* Byte offsets of one step's inputs inside a packed buffer, each a multiple
 * of 16: q bf16 [R][num_q_heads][head_dim], k_new and v_new bf16
 * [T][num_kv_heads][head_dim], slot_mapping int64 [T], context_lens int32
 * [R]; bytes = the size of the whole buffer. */
typedef struct pkv_step_layout {
    size_t q, k_new, v_new, slot_mapping, context_lens;
    size_t bytes;
    uint64_t flags;   /* PKV_STEP_* */
} pkv_step_layout;

/* The step's new tokens are the requests' query tokens (num_new_tokens ==
 * num_requests, token r at position context_lens[r] - 1): the decode kernels
 * store them (paged_attn_decode_append) instead of kv_cache_write; the
 * slot_mapping region is not read. */
#define PKV_STEP_FUSED_WRITE 1u

/* One decode step of a serving loop from host memory (Sec. 5.3's decode with
 * the paged cache of Sec. 5.4), all enqueued on `stream`; the call does not
 * wait for the GPU:
 *   1. one copy of layout->bytes bytes from host_in to dev_in (host_in should
 *      be pinned for the copy to be asynchronous; dev_in is device memory,
 *      16-byte aligned, with the same layout),
 *   2. kv_cache_write of the T = num_new_tokens new tokens in dev_in (with
 *      PKV_STEP_FUSED_WRITE in layout->flags: stored by step 3 instead),
 *   3. paged_attn_decode of the R = num_requests queries in dev_in over
 *      block_table (device int32 [R][max_blocks]) into out (device bf16) and
 *      lse (device fp32, or NULL),
 *   4. a copy of out to host_out, and of lse to host_lse when both are
 *      non-NULL (host_out may be NULL: no copy).
 * wait_event (a cudaEvent_t, or NULL): the kernels wait for it after the
 * input copy.  done_event (or NULL): recorded once the kernels are done,
 * before the output copy.  With two streams taking alternate steps, each
 * with its own dev_in, out and lse, and each step waiting for the previous
 * step's done_event, a step's copies overlap the other stream's kernels
 * while the kernels themselves stay in order (so the steps may share one
 * workspace).
 * The caller keeps host_in, host_out and host_lse untouched until the stream
 * has passed the step (an event recorded after the call).  Other arguments
 * and the errors are those of kv_cache_write and paged_attn_decode;
 * INVALID_ARG also for a layout whose regions are misaligned or outside
 * layout->bytes, CUDA for a failed copy.  The paper has no counterpart: this
 * composes the entry points above for callers that drive the step from the
 * host. */
int paged_attn_decode_step(pkv_pool_t pool, const void *host_in, void *dev_in,
                           const pkv_step_layout *layout, int32_t num_new_tokens,
                           const int32_t *block_table, int32_t max_blocks, int32_t num_requests,
                           int32_t num_q_heads, float scale, const pkv_prefix_groups *groups,
                           void *workspace, size_t workspace_bytes, void *out, float *lse,
                           void *host_out, float *host_lse, pkv_event_t wait_event,
                           pkv_event_t done_event, pkv_stream_t stream);

/* ---- decode without a caller workspace ------------------------------------ */

/* paged_attn_decode for callers that cannot allocate device memory when they
 * decode (work recorded into a CUDA graph, inference plugins whose framework
 * owns all device buffers, processes with a fixed up-front memory budget).
 * The paper has no counterpart: this is a deployment convenience of the
 * library.  Arguments and results are those of paged_attn_decode; the
 * split-KV scratch comes from a 64 MiB static device array instead of a
 * caller workspace, and the call allocates no device memory.
 *  - Shapes whose workspace (paged_attn_decode_workspace_size) exceeds
 *    64 MiB are refused with PKV_ERR_WORKSPACE.
 *  - The first call on a device looks up the array's device address
 *    (cudaGetSymbolAddress, with that device made current for the lookup);
 *    make that first call before any stream capture.
 *  - All calls share the one array: calls that may overlap on the GPU (other
 *    streams, other threads, other pools on the same device) race on it and
 *    must be serialised by the caller.
 *  - Every GPU that loads the library holds the 64 MiB until process exit. */
int paged_attn_decode_noalloc(pkv_pool_t pool, const void *q, void *out, float *lse,
                              const int32_t *context_lens, const int32_t *block_table,
                              int32_t max_blocks, int32_t num_requests, int32_t num_q_heads,
                              float scale, const pkv_prefix_groups *groups, pkv_stream_t stream);

/* ---- test aid ------------------------------------------------------------ */

/* Make one bounded device wait run out: a single thread waits, with the same
 * bounded mbarrier wait as the kernels, on a phase that nothing completes,
 * for limit_us microseconds (0 .. 1e6), then latches DEVICE_TIMEOUT into the
 * pool's error word and returns (no copy, MMA or tensor memory involved).
 * pkv_check_device_errors then reports PKV_ERR_DEVICE_TIMEOUT, and the
 * context stays usable.  Errors: INVALID_ARG, CUDA. */
int pkv_selftest_wait_timeout(pkv_pool_t pool, int32_t limit_us, pkv_stream_t stream);

/* ---- tracing -------------------------------------------------------------- */

/* Per-kernel device time of the launches made while tracing was on. */
typedef struct {
    char name[32];       /* "kv_cache_write", "decode_split", "decode_combine",
                            "decode_prefix", "prefill" */
    int32_t launches;    /* launches recorded since the last read            */
    int32_t reserved;
    double total_ms;     /* sum of CUDA-event durations of those launches    */
} pkv_kernel_time;

/* Turn per-launch timing on or off for kernels launched through this pool.
 * While on, every kernel launch is bracketed by a CUDA event pair recorded on
 * its stream (the observability of Fig. 1: per-stage latency).  Turning it
 * off synchronises the device and drops unread records. */
int pkv_trace_enable(pkv_pool_t pool, int32_t enable);

/* Synchronise on the recorded events and report, per kernel, the launches
 * and their summed duration since the previous read; then clear the records.
 * out: host array of max_entries; *n_out gets the number filled.
 * INVALID_ARG if tracing is off. */
int pkv_trace_read(pkv_pool_t pool, pkv_kernel_time *out, int32_t max_entries, int32_t *n_out);

/* ---- errors --------------------------------------------------------------- */

/* ---- KV-block transfer between pools (device) -------------------------------- */

/* Prefill/decode disaggregation (Sec. 2; Sec. 7) moves a request's KV blocks
 * from the pool of the instance that prefilled it to the pool of the one that
 * decodes it.  The blocks are gathered into one contiguous staging buffer
 * (the unit a peer or network copy moves) and scattered from it into blocks
 * allocated in the destination pool (kv_pool_alloc); the caller then
 * releases the source blocks (kv_pool_release), which moves the references.
 * Staging layout: [n][2][num_kv_heads][16][head_dim] bf16, block i's K tile
 * (all kv heads) then its V tile: the blocks' bytes as they are in the
 * pools, so both copies are bit-exact.  The two pools need the same
 * num_kv_heads and head_dim.  The paper gives the mechanism, not a layout or
 * an interface; these calls are this library's.
 *
 * Bytes of staging for n blocks of this pool's geometry (host call). */
int pkv_blocks_staging_size(pkv_pool_t pool, int32_t n, size_t *bytes_out);

/* Copy the n blocks block_ids[0..n) of the pool into staging.
 *  block_ids: device int32 [n]; an id outside [0, num_blocks) is skipped and
 *  latches DEVICE_BOUNDS.
 *  staging: device, 16-byte aligned, pkv_blocks_staging_size(n) bytes.
 * Asynchronous on `stream`.  Errors: INVALID_ARG, CUDA. */
int pkv_blocks_gather(pkv_pool_t pool, const int32_t *block_ids, int32_t n, void *staging,
                      pkv_stream_t stream);

/* Copy staging (as written by pkv_blocks_gather) into the n blocks
 * block_ids[0..n) of the pool: every K and V row of each block.  The target
 * blocks should be allocated and private (reference count 1): shared blocks
 * are immutable.  Arguments, bounds and errors as pkv_blocks_gather. */
int pkv_blocks_scatter(pkv_pool_t pool, const int32_t *block_ids, int32_t n, const void *staging,
                       pkv_stream_t stream);

/* Synchronise `stream`, then read and clear the pool's device error word.
 * *code_out gets PKV_OK or the first latched device status (DEVICE_BOUNDS,
 * DEVICE_TIMEOUT).  The return value reports failures of the call itself. */
int pkv_check_device_errors(pkv_pool_t pool, pkv_stream_t stream, int32_t *code_out);

/* Message of the last failing call on this thread ("" if none). */
const char *pkv_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* PKV_H */
