// pkv_api.cpp -- the C ABI of include/pkv.h: host-side pool, argument checks
// and kernel dispatch.  Host metadata only; device buffers belong to the caller.
#include "../../include/pkv.h"

#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <climits>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include "pkv_internal.h"

namespace pkv {
const char *const kKernelNames[kNumKernelIds] = {"kv_cache_write", "decode_split", "decode_combine",
                                                 "decode_prefix", "prefill", "block_copy"};
}

namespace {

// Records a CUDA event pair around each launch while enabled; times are
// read (after a synchronize) by pkv_trace_read.
struct EventTracer final : pkv::Tracer {
    struct Rec {
        int kid;
        cudaEvent_t a, b;
    };
    std::vector<Rec> recs;
    std::vector<cudaEvent_t> spare;
    cudaEvent_t pending = nullptr;
    cudaError_t err = cudaSuccess;

    cudaEvent_t get() {
        if (!spare.empty()) {
            cudaEvent_t e = spare.back();
            spare.pop_back();
            return e;
        }
        cudaEvent_t e = nullptr;
        cudaError_t r = cudaEventCreate(&e);
        if (r != cudaSuccess && err == cudaSuccess) err = r;
        return e;
    }
    void begin(int, cudaStream_t s) override {
        pending = get();
        if (pending) cudaEventRecord(pending, s);
    }
    void end(int kid, cudaStream_t s) override {
        cudaEvent_t b = get();
        if (!pending || !b) return;
        cudaEventRecord(b, s);
        recs.push_back({kid, pending, b});
        pending = nullptr;
    }
    void recycle() {
        for (auto &r : recs) {
            spare.push_back(r.a);
            spare.push_back(r.b);
        }
        recs.clear();
    }
    ~EventTracer() override {
        recycle();
        for (cudaEvent_t e : spare) cudaEventDestroy(e);
    }
};

}  // namespace

struct pkv_pool {
    pkv_pool_desc desc;
    void *k_cache = nullptr;
    void *v_cache = nullptr;
    std::vector<int32_t> refcnt;     // 0 = free
    std::vector<int32_t> free_list;  // back() is handed out next
    int *d_err = nullptr;            // device error word (latched by the kernels)
    int device = -1;
    int num_sms = 0;
    bool tmaps_ready = false;
    CUtensorMap tmap_k;
    CUtensorMap tmap_v;
    EventTracer *tracer = nullptr;   // non-null while tracing is enabled
};

namespace {

thread_local std::string g_last_error;

int fail(int code, const char *fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    g_last_error = buf;
    return code;
}

int ok() {
    g_last_error.clear();
    return PKV_OK;
}

int cuda_fail(cudaError_t e, const char *what) {
    return fail(PKV_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// splitmix64 (Steele, Lea, Flood 2014): the seeded stream of the placement.
uint64_t splitmix64(uint64_t &s) {
    uint64_t z = (s += 0x9E3779B97F4A7C15ull);
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

int check_kernel_pool(pkv_pool_t pool) {
    if (!pool) return fail(PKV_ERR_INVALID_ARG, "pool is NULL");
    if (!pool->k_cache || !pool->v_cache)
        return fail(PKV_ERR_INVALID_ARG, "pool has no device caches (metadata-only pool)");
    return PKV_OK;
}

int set_device(pkv_pool_t pool) {
    int cur = -1;
    cudaError_t e = cudaGetDevice(&cur);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if (cur != pool->device) {
        e = cudaSetDevice(pool->device);
        if (e != cudaSuccess) return cuda_fail(e, "cudaSetDevice");
    }
    return PKV_OK;
}

// TMA descriptors over the pool: a 4-D view {d, 16 slots, Hkv, num_blocks} of
// each cache, box {64 elements, 16 slots, 1, 1} = one (block, head) half-row
// tile of 2 KiB with the 128-byte swizzle the tensor-core operands use.
int build_tmaps(pkv_pool_t pool) {
    if (pool->tmaps_ready) return PKV_OK;
    void *fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000,
                                                     cudaEnableDefault, &q);
    if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !fn)
        return fail(PKV_ERR_CUDA, "cuTensorMapEncodeTiled entry point not found");
    auto encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    const pkv_pool_desc &d = pool->desc;
    cuuint64_t dims[4] = {(cuuint64_t)d.head_dim, 16, (cuuint64_t)d.num_kv_heads,
                          (cuuint64_t)d.num_blocks};
    cuuint64_t strides[3] = {(cuuint64_t)d.head_dim * 2, (cuuint64_t)d.head_dim * 2 * 16,
                             (cuuint64_t)d.head_dim * 2 * 16 * d.num_kv_heads};
    cuuint32_t box[4] = {64, 16, 1, 1};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    for (int which = 0; which < 2; ++which) {
        CUresult r = encode(which ? &pool->tmap_v : &pool->tmap_k,
                            CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4,
                            which ? pool->v_cache : pool->k_cache, dims, strides, box, estr,
                            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                            CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        if (r != CUDA_SUCCESS) return fail(PKV_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", (int)r);
    }
    pool->tmaps_ready = true;
    return PKV_OK;
}

}  // namespace

namespace pkv {
cudaError_t SmemLimit::ensure(const void *func, int need) {
    if (need <= 48 * 1024) return cudaSuccess;   // no opt-in below the default limit
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    if (bytes[dev].load(std::memory_order_acquire) >= need) return cudaSuccess;
    std::lock_guard<std::mutex> lock(mu);
    const int have = bytes[dev].load(std::memory_order_relaxed);
    if (have >= need) return cudaSuccess;
    e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, need);
    if (e == cudaSuccess) bytes[dev].store(need, std::memory_order_release);
    return e;
}

// Record a failure message for pkv_last_error() from another translation unit.
int set_last_error(int code, const char *msg) {
    g_last_error = msg ? msg : "";
    return code;
}

int pool_device(pkv_pool_t pool, int *dev) {
    int rc = check_kernel_pool(pool);
    if (rc != PKV_OK) return rc;
    *dev = pool->device;
    return PKV_OK;
}

int pool_device_error_word(pkv_pool_t pool, int **err) {
    int rc = check_kernel_pool(pool);
    if (rc != PKV_OK) return rc;
    if ((rc = set_device(pool)) != PKV_OK) return rc;
    *err = pool->d_err;
    return PKV_OK;
}
}  // namespace pkv

extern "C" {

const char *pkv_last_error(void) { return g_last_error.c_str(); }

int kv_pool_create(const pkv_pool_desc *desc, void *k_cache, void *v_cache, pkv_pool_t *out) {
    if (!desc || !out) return fail(PKV_ERR_INVALID_ARG, "desc and out must be non-NULL");
    *out = nullptr;
    if (desc->num_blocks <= 0 || desc->num_kv_heads <= 0)
        return fail(PKV_ERR_INVALID_ARG, "num_blocks and num_kv_heads must be positive");
    if (desc->block_size != 16) return fail(PKV_ERR_UNSUPPORTED, "block_size must be 16");
    if (desc->head_dim != 64 && desc->head_dim != 128)
        return fail(PKV_ERR_UNSUPPORTED, "head_dim must be 64 or 128");
    if (desc->dtype != PKV_DTYPE_BF16) return fail(PKV_ERR_UNSUPPORTED, "dtype must be bf16");
    if ((k_cache == nullptr) != (v_cache == nullptr))
        return fail(PKV_ERR_INVALID_ARG, "give both caches or neither");
    if (k_cache && (!aligned16(k_cache) || !aligned16(v_cache)))
        return fail(PKV_ERR_INVALID_ARG, "caches must be 16-byte aligned");
    pkv_pool *p = new pkv_pool();
    p->desc = *desc;
    p->k_cache = k_cache;
    p->v_cache = v_cache;
    const int32_t n = desc->num_blocks;
    p->refcnt.assign(n, 0);
    std::vector<int32_t> order(n);
    for (int32_t i = 0; i < n; ++i) order[i] = i;
    if (desc->placement_seed != 0) {
        uint64_t s = desc->placement_seed;
        for (int32_t i = n - 1; i > 0; --i) {   // Fisher-Yates
            const int32_t j = (int32_t)(splitmix64(s) % (uint64_t)(i + 1));
            std::swap(order[i], order[j]);
        }
    }
    p->free_list.assign(order.rbegin(), order.rend());   // back() = order[0]
    if (k_cache) {
        cudaError_t e = cudaGetDevice(&p->device);
        if (e == cudaSuccess) e = cudaDeviceGetAttribute(&p->num_sms, cudaDevAttrMultiProcessorCount, p->device);
        // the device error word
        if (e == cudaSuccess) e = cudaMalloc(&p->d_err, sizeof(int));
        if (e == cudaSuccess) e = cudaMemset(p->d_err, 0, sizeof(int));
        if (e != cudaSuccess) {
            if (p->d_err) cudaFree(p->d_err);
            delete p;
            return cuda_fail(e, "kv_pool_create");
        }
    }
    *out = p;
    return ok();
}

int kv_pool_destroy(pkv_pool_t pool) {
    if (!pool) return ok();
    if (pool->d_err) cudaFree(pool->d_err);
    delete pool->tracer;
    delete pool;
    return ok();
}

int kv_pool_alloc(pkv_pool_t pool, int32_t n, int32_t *ids_out) {
    if (!pool || n < 0 || (n > 0 && !ids_out)) return fail(PKV_ERR_INVALID_ARG, "bad arguments");
    if ((size_t)n > pool->free_list.size())
        return fail(PKV_ERR_OUT_OF_BLOCKS, "need %d blocks, %zu free", n, pool->free_list.size());
    for (int32_t i = 0; i < n; ++i) {
        const int32_t id = pool->free_list.back();
        pool->free_list.pop_back();
        pool->refcnt[id] = 1;
        ids_out[i] = id;
    }
    return ok();
}

int kv_pool_retain(pkv_pool_t pool, const int32_t *ids, int32_t n) {
    if (!pool || n < 0 || (n > 0 && !ids)) return fail(PKV_ERR_INVALID_ARG, "bad arguments");
    for (int32_t i = 0; i < n; ++i) {
        const int32_t id = ids[i];
        if (id < 0 || id >= pool->desc.num_blocks)
            return fail(PKV_ERR_REFCOUNT, "block id %d out of range", id);
        if (pool->refcnt[id] <= 0) return fail(PKV_ERR_REFCOUNT, "block %d is free", id);
    }
    for (int32_t i = 0; i < n; ++i) ++pool->refcnt[ids[i]];
    return ok();
}

int kv_pool_release(pkv_pool_t pool, const int32_t *ids, int32_t n) {
    if (!pool || n < 0 || (n > 0 && !ids)) return fail(PKV_ERR_INVALID_ARG, "bad arguments");
    std::vector<int32_t> drop;   // validate first: all or nothing
    drop.reserve(n);
    for (int32_t i = 0; i < n; ++i) {
        const int32_t id = ids[i];
        if (id < 0 || id >= pool->desc.num_blocks)
            return fail(PKV_ERR_REFCOUNT, "block id %d out of range", id);
        drop.push_back(id);
    }
    std::sort(drop.begin(), drop.end());
    for (size_t i = 0; i < drop.size();) {
        size_t j = i;
        while (j < drop.size() && drop[j] == drop[i]) ++j;
        if ((int32_t)(j - i) > pool->refcnt[drop[i]])
            return fail(PKV_ERR_REFCOUNT, "block %d released %zu times with refcount %d",
                        drop[i], j - i, pool->refcnt[drop[i]]);
        i = j;
    }
    for (int32_t i = 0; i < n; ++i) {
        if (--pool->refcnt[ids[i]] == 0) pool->free_list.push_back(ids[i]);
    }
    return ok();
}

int kv_pool_refcount(pkv_pool_t pool, int32_t id, int32_t *out) {
    if (!pool || !out || id < 0 || id >= pool->desc.num_blocks)
        return fail(PKV_ERR_INVALID_ARG, "bad arguments");
    *out = pool->refcnt[id];
    return ok();
}

int kv_pool_num_free(pkv_pool_t pool, int32_t *out) {
    if (!pool || !out) return fail(PKV_ERR_INVALID_ARG, "bad arguments");
    *out = (int32_t)pool->free_list.size();
    return ok();
}

int kv_pool_alloc_sequence(pkv_pool_t pool, const int32_t *prefix_ids, int32_t n_prefix,
                           int32_t n_blocks, int32_t *row_out) {
    if (!pool || n_prefix < 0 || n_blocks < n_prefix || !row_out || (n_prefix > 0 && !prefix_ids))
        return fail(PKV_ERR_INVALID_ARG, "bad arguments");
    const int32_t n_new = n_blocks - n_prefix;
    if ((size_t)n_new > pool->free_list.size())
        return fail(PKV_ERR_OUT_OF_BLOCKS, "need %d blocks, %zu free", n_new, pool->free_list.size());
    int rc = kv_pool_retain(pool, prefix_ids, n_prefix);
    if (rc != PKV_OK) return rc;
    for (int32_t i = 0; i < n_prefix; ++i) row_out[i] = prefix_ids[i];
    return kv_pool_alloc(pool, n_new, row_out + n_prefix);
}

int kv_slot_mapping(pkv_pool_t pool, const int32_t *block_table, int32_t max_blocks,
                    const int32_t *context_lens, const int32_t *new_lens, int32_t num_requests,
                    int64_t *slots_out) {
    if (!block_table || !context_lens || !new_lens || num_requests < 0 || max_blocks <= 0)
        return fail(PKV_ERR_INVALID_ARG, "bad arguments");
    int64_t t = 0;
    for (int32_t r = 0; r < num_requests; ++r) {
        const int32_t L = context_lens[r], n = new_lens[r];
        if (n < 0 || L < n || ((int64_t)L + 15) / 16 > max_blocks)
            return fail(PKV_ERR_INVALID_ARG, "request %d: context %d, new %d, table width %d", r, L,
                        n, max_blocks);
        for (int32_t i = 0; i < n; ++i) {
            const int64_t p = (int64_t)L - n + i;
            const int32_t blk = block_table[(int64_t)r * max_blocks + p / 16];
            if (blk < 0) return fail(PKV_ERR_INVALID_ARG, "request %d: no block for position %lld", r, (long long)p);
            if (pool) {
                if (blk >= pool->desc.num_blocks)
                    return fail(PKV_ERR_INVALID_ARG, "request %d: block id %d is outside the pool", r, blk);
                if (pool->refcnt[blk] == 0)
                    return fail(PKV_ERR_REFCOUNT, "request %d: block %d is not allocated", r, blk);
                if (pool->refcnt[blk] > 1)
                    return fail(PKV_ERR_SHARED_BLOCK_WRITE,
                                "request %d: position %lld maps into shared block %d", r,
                                (long long)p, blk);
            }
            if (slots_out) slots_out[t] = (int64_t)blk * 16 + p % 16;
            ++t;
        }
    }
    return ok();
}

int pkv_check_block_table(pkv_pool_t pool, const int32_t *block_table, int32_t max_blocks,
                          int32_t num_requests, const int32_t *context_lens, int32_t *bad_request_out) {
    if (bad_request_out) *bad_request_out = -1;
    if (!pool || num_requests < 0 || max_blocks <= 0 ||
        (num_requests > 0 && (!block_table || !context_lens)))
        return fail(PKV_ERR_INVALID_ARG, "bad arguments");
    for (int32_t r = 0; r < num_requests; ++r) {
        const int32_t L = context_lens[r];
        const int64_t nblk = ((int64_t)L + 15) / 16;
        int rc = PKV_OK;
        if (L < 0 || nblk > max_blocks) {
            rc = fail(PKV_ERR_INVALID_ARG, "request %d: context %d does not fit %d table entries", r, L,
                      max_blocks);
        } else {
            const int32_t *row = block_table + (int64_t)r * max_blocks;
            for (int64_t j = 0; j < nblk && rc == PKV_OK; ++j) {
                const int32_t id = row[j];
                if (id < 0 || id >= pool->desc.num_blocks)
                    rc = fail(PKV_ERR_INVALID_ARG, "request %d: entry %lld holds block id %d, outside the pool",
                              r, (long long)j, id);
                else if (pool->refcnt[id] == 0)
                    rc = fail(PKV_ERR_REFCOUNT, "request %d: entry %lld holds free block %d", r,
                              (long long)j, id);
            }
        }
        if (rc != PKV_OK) {
            if (bad_request_out) *bad_request_out = r;
            return rc;
        }
    }
    return ok();
}

int kv_cache_write(pkv_pool_t pool, const void *k_new, const void *v_new,
                   const int64_t *slot_mapping, int32_t num_tokens, pkv_stream_t stream) {
    int rc = check_kernel_pool(pool);
    if (rc != PKV_OK) return rc;
    if (num_tokens < 0) return fail(PKV_ERR_INVALID_ARG, "num_tokens < 0");
    if (num_tokens == 0) return ok();
    if (!k_new || !v_new || !slot_mapping) return fail(PKV_ERR_INVALID_ARG, "NULL buffer");
    if (!aligned16(k_new) || !aligned16(v_new) || (reinterpret_cast<uintptr_t>(slot_mapping) & 7))
        return fail(PKV_ERR_INVALID_ARG, "misaligned buffer");
    if ((rc = set_device(pool)) != PKV_OK) return rc;
    const pkv_pool_desc &d = pool->desc;
    cudaError_t e = pkv::launch_cache_write(k_new, v_new, slot_mapping, num_tokens, pool->k_cache,
                                            pool->v_cache, d.num_kv_heads, d.head_dim,
                                            (int64_t)d.num_blocks * 16, pool->d_err,
                                            static_cast<cudaStream_t>(stream), pool->tracer);
    if (e != cudaSuccess) return cuda_fail(e, "kv_cache_write launch");
    return ok();
}

}  // extern "C"

namespace {

// paged_attn_prefill, with tree-shaped draft masks when tree_mask is set
// TMA descriptor of new-token rows [T][Hkv][d] (k_new or v_new): a 3-D view
// {d, Hkv, T}, box {64, 1, 16} = 16 tokens of one kv head, laid out in shared
// memory exactly like a pool box of 16 slots (128-byte swizzle).
int new_rows_tmap(CUtensorMap *m, const void *base, int32_t T, int32_t Hkv, int32_t d) {
    void *fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
    if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !fn)
        return fail(PKV_ERR_CUDA, "cuTensorMapEncodeTiled entry point not found");
    auto encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    cuuint64_t dims[3] = {(cuuint64_t)d, (cuuint64_t)Hkv, (cuuint64_t)T};
    cuuint64_t strides[2] = {(cuuint64_t)d * 2, (cuuint64_t)d * 2 * Hkv};
    cuuint32_t box[3] = {64, 1, 16};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base), dims, strides, box,
                        estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(PKV_ERR_CUDA, "cuTensorMapEncodeTiled (new rows) failed (%d)", (int)r);
    return PKV_OK;
}

int prefill_impl(pkv_pool_t pool, const void *q, void *out, float *lse, const int32_t *cu_seqlens_q,
                 const int32_t *context_lens, const int32_t *block_table, int32_t max_blocks,
                 int32_t num_requests, int32_t max_seqlen_q, int32_t num_q_heads, float scale,
                 const uint64_t *tree_mask, const void *k_new, const void *v_new, int32_t num_new_tokens,
                 pkv_stream_t stream) {
    int rc = check_kernel_pool(pool);
    if (rc != PKV_OK) return rc;
    const pkv_pool_desc &d = pool->desc;
    if (num_requests < 0 || max_seqlen_q < 0 || max_blocks <= 0)
        return fail(PKV_ERR_INVALID_ARG, "bad sizes");
    if (num_q_heads <= 0 || num_q_heads % d.num_kv_heads != 0)
        return fail(PKV_ERR_INVALID_ARG, "num_q_heads must be a positive multiple of num_kv_heads");
    if (num_q_heads / d.num_kv_heads > 128)
        return fail(PKV_ERR_UNSUPPORTED, "more than 128 q heads per kv head");
    if (max_blocks > pkv::kPrefillMaxBlocks)
        return fail(PKV_ERR_UNSUPPORTED, "table width %d: prefill supports contexts up to %d blocks (%d tokens)",
                    max_blocks, pkv::kPrefillMaxBlocks, 16 * pkv::kPrefillMaxBlocks);
    if (!(scale > 0.f) || !std::isfinite(scale)) return fail(PKV_ERR_INVALID_ARG, "bad scale");
    if (num_requests == 0 || max_seqlen_q == 0) return ok();
    if (!q || !out || !cu_seqlens_q || !context_lens || !block_table)
        return fail(PKV_ERR_INVALID_ARG, "NULL buffer");
    if (!aligned16(q) || !aligned16(out)) return fail(PKV_ERR_INVALID_ARG, "misaligned q/out");
    if ((k_new == nullptr) != (v_new == nullptr)) return fail(PKV_ERR_INVALID_ARG, "give both k_new and v_new");
    if (k_new && (!aligned16(k_new) || !aligned16(v_new)))
        return fail(PKV_ERR_INVALID_ARG, "misaligned k_new/v_new");
    if (k_new && num_new_tokens <= 0) return fail(PKV_ERR_INVALID_ARG, "num_new_tokens must be positive");
    if ((rc = set_device(pool)) != PKV_OK) return rc;
    if ((rc = build_tmaps(pool)) != PKV_OK) return rc;
    CUtensorMap tkn, tvn;
    if (k_new) {
        if ((rc = new_rows_tmap(&tkn, k_new, num_new_tokens, d.num_kv_heads, d.head_dim)) != PKV_OK) return rc;
        if ((rc = new_rows_tmap(&tvn, v_new, num_new_tokens, d.num_kv_heads, d.head_dim)) != PKV_OK) return rc;
    }
    pkv::PrefillArgs a{};
    a.q = q; a.out = out; a.lse = lse;
    a.cu_seqlens_q = cu_seqlens_q; a.context_lens = context_lens;
    a.block_table = block_table; a.max_blocks = max_blocks;
    a.R = num_requests; a.Hq = num_q_heads; a.Hkv = d.num_kv_heads; a.d = d.head_dim;
    a.max_seqlen_q = max_seqlen_q;
    a.num_blocks_pool = d.num_blocks;
    a.scale_log2 = scale * 1.4426950408889634f;
    a.tmap_k = &pool->tmap_k; a.tmap_v = &pool->tmap_v;
    a.err = pool->d_err;
    a.tree_mask = reinterpret_cast<const unsigned long long *>(tree_mask);
    a.num_sms = pool->num_sms;
    if (k_new) {
        a.k_new = k_new; a.v_new = v_new;
        a.k_cache = pool->k_cache; a.v_cache = pool->v_cache;
        a.tmap_kn = &tkn; a.tmap_vn = &tvn;
    }
    cudaError_t e = pkv::launch_prefill(a, static_cast<cudaStream_t>(stream), pool->tracer);
    if (e != cudaSuccess) return cuda_fail(e, "paged_attn_prefill launch");
    return ok();
}

}  // namespace

extern "C" {

int paged_attn_prefill(pkv_pool_t pool, const void *q, void *out, float *lse,
                       const int32_t *cu_seqlens_q, const int32_t *context_lens,
                       const int32_t *block_table, int32_t max_blocks, int32_t num_requests,
                       int32_t max_seqlen_q, int32_t num_q_heads, float scale,
                       pkv_stream_t stream) {
    return prefill_impl(pool, q, out, lse, cu_seqlens_q, context_lens, block_table, max_blocks,
                        num_requests, max_seqlen_q, num_q_heads, scale, nullptr, nullptr, nullptr, 0, stream);
}

int paged_attn_prefill_append(pkv_pool_t pool, const void *q, const void *k_new, const void *v_new,
                              int32_t num_new_tokens, void *out, float *lse, const int32_t *cu_seqlens_q,
                              const int32_t *context_lens, const int32_t *block_table, int32_t max_blocks,
                              int32_t num_requests, int32_t max_seqlen_q, int32_t num_q_heads, float scale,
                              pkv_stream_t stream) {
    if (num_requests > 0 && max_seqlen_q > 0 && (!k_new || !v_new))
        return fail(PKV_ERR_INVALID_ARG, "NULL k_new/v_new");
    return prefill_impl(pool, q, out, lse, cu_seqlens_q, context_lens, block_table, max_blocks,
                        num_requests, max_seqlen_q, num_q_heads, scale, nullptr, k_new, v_new, num_new_tokens,
                        stream);
}

int paged_attn_verify_tree(pkv_pool_t pool, const void *q, void *out, float *lse,
                           const int32_t *cu_seqlens_q, const int32_t *context_lens,
                           const int32_t *block_table, int32_t max_blocks, int32_t num_requests,
                           int32_t max_seqlen_q, int32_t num_q_heads, float scale,
                           const uint64_t *tree_mask, pkv_stream_t stream) {
    if (max_seqlen_q > 64) return fail(PKV_ERR_UNSUPPORTED, "at most 64 draft tokens per request");
    if (num_requests > 0 && max_seqlen_q > 0 &&
        (!tree_mask || (reinterpret_cast<uintptr_t>(tree_mask) & 7)))
        return fail(PKV_ERR_INVALID_ARG, "tree_mask must be a non-NULL, 8-byte aligned device array");
    return prefill_impl(pool, q, out, lse, cu_seqlens_q, context_lens, block_table, max_blocks,
                        num_requests, max_seqlen_q, num_q_heads, scale, tree_mask, nullptr, nullptr, 0, stream);
}

int paged_attn_verify_tree_workspace_size(pkv_pool_t pool, int32_t num_tokens, int32_t num_q_heads,
                                          int32_t max_blocks, const pkv_verify_groups *groups,
                                          size_t *bytes_out) {
    if (!pool || !bytes_out || num_tokens < 0 || num_q_heads <= 0 || max_blocks <= 0)
        return fail(PKV_ERR_INVALID_ARG, "bad arguments");
    const bool grouped = groups && groups->num_groups > 0;
    pkv::DecodeLayout L = pkv::verify_layout(num_tokens, num_q_heads, pool->desc.num_kv_heads,
                                             pool->desc.head_dim, max_blocks, grouped ? groups->num_groups : 0,
                                             grouped ? groups->max_group_blocks : 0,
                                             grouped ? groups->max_group_tokens : 0, pool->num_sms);
    *bytes_out = L.total;
    return ok();
}

int paged_attn_verify_tree_grouped(pkv_pool_t pool, const void *q, void *out, float *lse,
                                   const int32_t *cu_seqlens_q, const int32_t *context_lens,
                                   const int32_t *block_table, int32_t max_blocks, int32_t num_requests,
                                   int32_t num_tokens, int32_t max_seqlen_q, int32_t num_q_heads, float scale,
                                   const uint64_t *tree_mask, const pkv_verify_groups *groups,
                                   void *workspace, size_t workspace_bytes, pkv_stream_t stream) {
    int rc = check_kernel_pool(pool);
    if (rc != PKV_OK) return rc;
    const pkv_pool_desc &d = pool->desc;
    if (num_requests < 0 || num_tokens < 0 || max_seqlen_q < 0 || max_blocks <= 0)
        return fail(PKV_ERR_INVALID_ARG, "bad sizes");
    if (num_q_heads <= 0 || num_q_heads % d.num_kv_heads != 0)
        return fail(PKV_ERR_INVALID_ARG, "num_q_heads must be a positive multiple of num_kv_heads");
    if (num_q_heads / d.num_kv_heads > 8)
        return fail(PKV_ERR_UNSUPPORTED, "grouped verification supports up to 8 q heads per kv head");
    if (max_seqlen_q > 64) return fail(PKV_ERR_UNSUPPORTED, "at most 64 draft tokens per request");
    if (max_blocks > pkv::kPrefillMaxBlocks)
        return fail(PKV_ERR_UNSUPPORTED, "table width %d: verification supports up to %d blocks", max_blocks,
                    pkv::kPrefillMaxBlocks);
    if (num_tokens > (1 << 20)) return fail(PKV_ERR_UNSUPPORTED, "more than 2^20 draft tokens");
    if (!(scale > 0.f) || !std::isfinite(scale)) return fail(PKV_ERR_INVALID_ARG, "bad scale");
    if (num_requests == 0 || max_seqlen_q == 0 || num_tokens == 0) return ok();
    if (!q || !out || !cu_seqlens_q || !context_lens || !block_table)
        return fail(PKV_ERR_INVALID_ARG, "NULL buffer");
    if (!aligned16(q) || !aligned16(out)) return fail(PKV_ERR_INVALID_ARG, "misaligned q/out");
    if (!tree_mask || (reinterpret_cast<uintptr_t>(tree_mask) & 7))
        return fail(PKV_ERR_INVALID_ARG, "tree_mask must be a non-NULL, 8-byte aligned device array");
    int32_t G = 0, mgb = 0, mgt = 0;
    if (groups && groups->num_groups > 0) {
        G = groups->num_groups;
        mgb = groups->max_group_blocks;
        mgt = groups->max_group_tokens;
        if (!groups->group_start || !groups->member_token || !groups->group_blocks || !groups->group_row ||
            !groups->request_group || mgb < 0 || mgt < 0)
            return fail(PKV_ERR_INVALID_ARG, "incomplete verification-group descriptor");
        if (mgb > max_blocks) return fail(PKV_ERR_INVALID_ARG, "max_group_blocks exceeds the table width");
        if ((int64_t)G * d.num_kv_heads > INT32_MAX) return fail(PKV_ERR_UNSUPPORTED, "too many groups");
    }
    const pkv::DecodeLayout L = pkv::verify_layout(num_tokens, num_q_heads, d.num_kv_heads, d.head_dim,
                                                   max_blocks, G, mgb, mgt, pool->num_sms);
    if (!workspace || workspace_bytes < L.total)
        return fail(PKV_ERR_WORKSPACE, "workspace of %zu bytes needed", L.total);
    if (reinterpret_cast<uintptr_t>(workspace) & 255)
        return fail(PKV_ERR_WORKSPACE, "workspace must be 256-byte aligned");
    if ((rc = set_device(pool)) != PKV_OK) return rc;
    if ((rc = build_tmaps(pool)) != PKV_OK) return rc;
    const float scale_log2 = scale * 1.4426950408889634f;
    pkv::DecodeArgs a{};
    a.q = q; a.out = out; a.lse = lse;
    a.block_table = block_table; a.max_blocks = max_blocks;
    a.scale_log2 = scale_log2;
    a.num_groups = G;
    if (G > 0) {
        a.max_group_members = mgt;
        a.group_start = groups->group_start; a.member_req = groups->member_token;
        a.group_blocks = groups->group_blocks;
        a.group_row = groups->group_row;
        a.num_table_rows = num_requests;
    }
    a.ws = workspace;
    a.err = pool->d_err;
    a.tmap_k = &pool->tmap_k; a.tmap_v = &pool->tmap_v;
    pkv::PrefillArgs pa{};
    pa.q = q;
    pa.cu_seqlens_q = cu_seqlens_q; pa.context_lens = context_lens;
    pa.block_table = block_table; pa.max_blocks = max_blocks;
    pa.R = num_requests; pa.Hq = num_q_heads; pa.Hkv = d.num_kv_heads; pa.d = d.head_dim;
    pa.max_seqlen_q = max_seqlen_q;
    pa.num_blocks_pool = d.num_blocks;
    pa.scale_log2 = scale_log2;
    pa.tmap_k = &pool->tmap_k; pa.tmap_v = &pool->tmap_v;
    pa.err = pool->d_err;
    pa.tree_mask = reinterpret_cast<const unsigned long long *>(tree_mask);
    cudaError_t e = pkv::launch_verify_grouped(L, a, pa, G > 0 ? groups->request_group : nullptr,
                                               static_cast<cudaStream_t>(stream), pool->tracer);
    if (e != cudaSuccess) return cuda_fail(e, "paged_attn_verify_tree_grouped launch");
    return ok();
}

int pkv_verify_groups_build(const int32_t *cu_seqlens, const int32_t *request_group, int32_t num_requests,
                            int32_t num_groups, int32_t *group_start_out, int32_t *member_token_out,
                            int32_t *group_row_out, int32_t *max_group_tokens_out) {
    if (num_requests < 0 || num_groups < 0 || !cu_seqlens || !group_start_out || !max_group_tokens_out ||
        (num_requests > 0 && !request_group) || (num_groups > 0 && !group_row_out))
        return fail(PKV_ERR_INVALID_ARG, "bad arguments");
    if (cu_seqlens[0] != 0) return fail(PKV_ERR_INVALID_ARG, "cu_seqlens[0] must be 0");
    std::vector<int64_t> count(num_groups, 0);
    for (int32_t r = 0; r < num_requests; ++r) {
        const int32_t n = cu_seqlens[r + 1] - cu_seqlens[r];
        if (n < 0) return fail(PKV_ERR_INVALID_ARG, "cu_seqlens decreases at request %d", r);
        const int32_t gr = request_group[r];
        if (gr < -1 || gr >= num_groups)
            return fail(PKV_ERR_INVALID_ARG, "request %d: group %d out of range", r, gr);
        if (gr >= 0) count[gr] += n;
    }
    if (num_requests > 0 && cu_seqlens[num_requests] > 0 && !member_token_out)
        return fail(PKV_ERR_INVALID_ARG, "NULL member_token_out");
    int64_t total = 0, mx = 0;
    for (int32_t g = 0; g < num_groups; ++g) {
        group_start_out[g] = (int32_t)total;
        group_row_out[g] = -1;
        total += count[g];
        mx = std::max(mx, count[g]);
    }
    group_start_out[num_groups] = (int32_t)total;
    std::vector<int64_t> fill(group_start_out, group_start_out + num_groups);
    for (int32_t r = 0; r < num_requests; ++r) {
        const int32_t gr = request_group[r];
        if (gr < 0) continue;
        if (group_row_out[gr] < 0) group_row_out[gr] = r;
        for (int32_t t = cu_seqlens[r]; t < cu_seqlens[r + 1]; ++t) member_token_out[fill[gr]++] = t;
    }
    *max_group_tokens_out = (int32_t)mx;
    return ok();
}

int pkv_tree_masks(const int32_t *parent, const int32_t *cu_seqlens, int32_t num_requests,
                   uint64_t *masks_out) {
    if (num_requests < 0 || !cu_seqlens || (num_requests > 0 && cu_seqlens[num_requests] > 0 &&
                                             (!parent || !masks_out)))
        return fail(PKV_ERR_INVALID_ARG, "bad arguments");
    if (cu_seqlens[0] != 0) return fail(PKV_ERR_INVALID_ARG, "cu_seqlens[0] must be 0");
    for (int32_t r = 0; r < num_requests; ++r) {
        const int32_t a = cu_seqlens[r], n = cu_seqlens[r + 1] - a;
        if (n < 0 || n > 64)
            return fail(PKV_ERR_INVALID_ARG, "request %d: %d drafts (0 to 64 allowed)", r, n);
        for (int32_t i = 0; i < n; ++i) {
            const int32_t pa = parent[a + i];
            if (pa < -1 || pa >= i)
                return fail(PKV_ERR_INVALID_ARG, "request %d draft %d: parent %d is not -1 or an earlier draft",
                            r, i, pa);
            masks_out[a + i] = (pa < 0 ? 0ull : masks_out[a + pa]) | (1ull << i);
        }
    }
    return ok();
}

int paged_attn_decode_workspace_size(pkv_pool_t pool, int32_t num_requests, int32_t num_q_heads,
                                     int32_t max_blocks, const pkv_prefix_groups *groups,
                                     size_t *bytes_out) {
    if (!pool || !bytes_out || num_requests < 0 || num_q_heads <= 0 || max_blocks <= 0)
        return fail(PKV_ERR_INVALID_ARG, "bad arguments");
    const int32_t G = groups ? groups->num_groups : 0;
    const int32_t mgb = groups ? groups->max_group_blocks : 0;
    const int32_t mgm = groups ? groups->max_group_members : 0;
    pkv::DecodeLayout L = pkv::decode_layout(num_requests, num_q_heads, pool->desc.num_kv_heads,
                                             pool->desc.head_dim, max_blocks, G, mgb, mgm,
                                             pool->num_sms);
    *bytes_out = L.total;
    return ok();
}

}  // extern "C"

namespace {

// Every host-side check of paged_attn_decode, then its layout and kernel
// arguments (and the pool's TMA descriptors when the prefix pass runs);
// nothing is enqueued.  *empty: no request, nothing to launch.
int prepare_decode(pkv_pool_t pool, const void *q, const void *k_new, const void *v_new, void *out,
                   float *lse, const int32_t *context_lens, const int32_t *block_table, int32_t max_blocks,
                   int32_t num_requests, int32_t num_q_heads, float scale,
                   const pkv_prefix_groups *groups, void *workspace, size_t workspace_bytes,
                   pkv::DecodeLayout *L_out, pkv::DecodeArgs *a_out, bool *empty) {
    *empty = true;
    int rc = check_kernel_pool(pool);
    if (rc != PKV_OK) return rc;
    const pkv_pool_desc &d = pool->desc;
    if (num_requests < 0 || max_blocks <= 0) return fail(PKV_ERR_INVALID_ARG, "bad sizes");
    if (num_q_heads <= 0 || num_q_heads % d.num_kv_heads != 0)
        return fail(PKV_ERR_INVALID_ARG, "num_q_heads must be a positive multiple of num_kv_heads");
    const int32_t g = num_q_heads / d.num_kv_heads;
    if (g > 8) return fail(PKV_ERR_UNSUPPORTED, "decode supports up to 8 q heads per kv head");
    if (num_requests > 16384) return fail(PKV_ERR_UNSUPPORTED, "decode supports up to 16384 requests");
    if (!(scale > 0.f) || !std::isfinite(scale)) return fail(PKV_ERR_INVALID_ARG, "bad scale");
    *empty = num_requests == 0;
    if (*empty) return ok();
    if (!q || !out || !context_lens || !block_table) return fail(PKV_ERR_INVALID_ARG, "NULL buffer");
    if (!aligned16(q) || !aligned16(out)) return fail(PKV_ERR_INVALID_ARG, "misaligned q/out");
    if ((k_new == nullptr) != (v_new == nullptr)) return fail(PKV_ERR_INVALID_ARG, "give both k_new and v_new");
    if (k_new && (!aligned16(k_new) || !aligned16(v_new)))
        return fail(PKV_ERR_INVALID_ARG, "misaligned k_new/v_new");
    int32_t G = 0, mgb = 0, mgm = 0;
    if (groups && groups->num_groups > 0) {
        G = groups->num_groups;
        mgb = groups->max_group_blocks;
        mgm = groups->max_group_members;
        if (!groups->group_start || !groups->member_req || !groups->group_blocks ||
            !groups->group_of_req || mgb < 0 || mgm < 0)
            return fail(PKV_ERR_INVALID_ARG, "incomplete prefix-group descriptor");
        if (mgb > max_blocks) return fail(PKV_ERR_INVALID_ARG, "max_group_blocks exceeds the table width");
        if ((int64_t)G * d.num_kv_heads > INT32_MAX) return fail(PKV_ERR_UNSUPPORTED, "too many groups");
    }
    pkv::DecodeLayout &L = *L_out;
    L = pkv::decode_layout(num_requests, num_q_heads, d.num_kv_heads, d.head_dim,
                                             max_blocks, G, mgb, mgm, pool->num_sms);
    if (!workspace || workspace_bytes < L.total)
        return fail(PKV_ERR_WORKSPACE, "workspace of %zu bytes needed", L.total);
    if (reinterpret_cast<uintptr_t>(workspace) & 255)
        return fail(PKV_ERR_WORKSPACE, "workspace must be 256-byte aligned");
    if ((rc = set_device(pool)) != PKV_OK) return rc;
    if ((rc = build_tmaps(pool)) != PKV_OK) return rc;
    pkv::DecodeArgs &a = *a_out;
    a = pkv::DecodeArgs{};
    a.q = q; a.out = out; a.lse = lse;
    a.context_lens = context_lens; a.block_table = block_table; a.max_blocks = max_blocks;
    a.k_cache = pool->k_cache; a.v_cache = pool->v_cache;
    a.scale_log2 = scale * 1.4426950408889634f;
    a.num_groups = G;
    if (G > 0) {
        a.max_group_members = groups->max_group_members;
        a.group_start = groups->group_start; a.member_req = groups->member_req;
        a.group_blocks = groups->group_blocks; a.group_of_req = groups->group_of_req;
    }
    a.ws = workspace;
    a.err = pool->d_err;
    a.tmap_k = &pool->tmap_k;
    a.tmap_v = &pool->tmap_v;
    a.k_new = k_new;
    a.v_new = v_new;
    return ok();
}

}  // namespace

extern "C" {

int paged_attn_decode(pkv_pool_t pool, const void *q, void *out, float *lse,
                      const int32_t *context_lens, const int32_t *block_table, int32_t max_blocks,
                      int32_t num_requests, int32_t num_q_heads, float scale,
                      const pkv_prefix_groups *groups, void *workspace, size_t workspace_bytes,
                      pkv_stream_t stream) {
    pkv::DecodeLayout L{};
    pkv::DecodeArgs a{};
    bool empty = true;
    const int rc = prepare_decode(pool, q, nullptr, nullptr, out, lse, context_lens, block_table, max_blocks,
                                  num_requests, num_q_heads, scale, groups, workspace, workspace_bytes, &L, &a,
                                  &empty);
    if (rc != PKV_OK || empty) return rc;
    cudaError_t e = pkv::launch_decode(L, a, pool->desc.num_blocks, static_cast<cudaStream_t>(stream),
                                       pool->tracer);
    if (e != cudaSuccess) return cuda_fail(e, "paged_attn_decode launch");
    return ok();
}

int paged_attn_decode_append(pkv_pool_t pool, const void *q, const void *k_new, const void *v_new,
                             void *out, float *lse, const int32_t *context_lens,
                             const int32_t *block_table, int32_t max_blocks, int32_t num_requests,
                             int32_t num_q_heads, float scale, const pkv_prefix_groups *groups,
                             void *workspace, size_t workspace_bytes, pkv_stream_t stream) {
    if (num_requests > 0 && (!k_new || !v_new)) return fail(PKV_ERR_INVALID_ARG, "NULL k_new/v_new");
    pkv::DecodeLayout L{};
    pkv::DecodeArgs a{};
    bool empty = true;
    const int rc = prepare_decode(pool, q, k_new, v_new, out, lse, context_lens, block_table, max_blocks,
                                  num_requests, num_q_heads, scale, groups, workspace, workspace_bytes, &L, &a,
                                  &empty);
    if (rc != PKV_OK || empty) return rc;
    cudaError_t e = pkv::launch_decode(L, a, pool->desc.num_blocks, static_cast<cudaStream_t>(stream),
                                       pool->tracer);
    if (e != cudaSuccess) return cuda_fail(e, "paged_attn_decode_append launch");
    return ok();
}

int paged_attn_decode_step(pkv_pool_t pool, const void *host_in, void *dev_in,
                           const pkv_step_layout *layout, int32_t num_new_tokens,
                           const int32_t *block_table, int32_t max_blocks, int32_t num_requests,
                           int32_t num_q_heads, float scale, const pkv_prefix_groups *groups,
                           void *workspace, size_t workspace_bytes, void *out, float *lse,
                           void *host_out, float *host_lse, pkv_event_t wait_event,
                           pkv_event_t done_event, pkv_stream_t stream) {
    int rc = check_kernel_pool(pool);
    if (rc != PKV_OK) return rc;
    if (!host_in || !dev_in || !layout) return fail(PKV_ERR_INVALID_ARG, "NULL step buffer or layout");
    if (num_new_tokens < 0 || num_requests < 0 || num_q_heads <= 0)
        return fail(PKV_ERR_INVALID_ARG, "bad sizes");
    if (!aligned16(dev_in)) return fail(PKV_ERR_INVALID_ARG, "dev_in must be 16-byte aligned");
    const pkv_pool_desc &d = pool->desc;
    const size_t row = (size_t)d.head_dim * 2;
    const bool fused = (layout->flags & PKV_STEP_FUSED_WRITE) != 0;
    if (layout->flags & ~(uint64_t)PKV_STEP_FUSED_WRITE) return fail(PKV_ERR_INVALID_ARG, "unknown step flags");
    if (fused && num_new_tokens != num_requests)
        return fail(PKV_ERR_INVALID_ARG, "a fused-write step has one new token per request");
    // every region 16-byte aligned and inside the buffer
    const struct { size_t off, len; } regions[] = {
        {layout->q, (size_t)num_requests * num_q_heads * row},
        {layout->k_new, (size_t)num_new_tokens * d.num_kv_heads * row},
        {layout->v_new, (size_t)num_new_tokens * d.num_kv_heads * row},
        {fused ? 0 : layout->slot_mapping, fused ? 0 : (size_t)num_new_tokens * sizeof(int64_t)},
        {layout->context_lens, (size_t)num_requests * sizeof(int32_t)},
    };
    for (const auto &g : regions)
        if (g.off % 16 != 0 || g.off > layout->bytes || g.len > layout->bytes - g.off)
            return fail(PKV_ERR_INVALID_ARG, "step layout: region at %zu (%zu bytes) misaligned or "
                        "outside the %zu-byte buffer", g.off, g.len, layout->bytes);
    // every argument check before anything is enqueued
    const char *din = static_cast<const char *>(dev_in);
    pkv::DecodeLayout L{};
    pkv::DecodeArgs a{};
    bool empty = true;
    rc = prepare_decode(pool, din + layout->q, fused ? din + layout->k_new : nullptr,
                        fused ? din + layout->v_new : nullptr, out, lse,
                        reinterpret_cast<const int32_t *>(din + layout->context_lens), block_table,
                        max_blocks, num_requests, num_q_heads, scale, groups, workspace, workspace_bytes,
                        &L, &a, &empty);
    if (rc != PKV_OK) return rc;
    if ((rc = set_device(pool)) != PKV_OK) return rc;
    const cudaStream_t st = static_cast<cudaStream_t>(stream);
    cudaError_t e = cudaMemcpyAsync(dev_in, host_in, layout->bytes, cudaMemcpyHostToDevice, st);
    if (e != cudaSuccess) return cuda_fail(e, "paged_attn_decode_step input copy");
    if (wait_event) {
        e = cudaStreamWaitEvent(st, static_cast<cudaEvent_t>(wait_event), 0);
        if (e != cudaSuccess) return cuda_fail(e, "paged_attn_decode_step wait_event");
    }
    if (!fused) {
        rc = kv_cache_write(pool, din + layout->k_new, din + layout->v_new,
                            reinterpret_cast<const int64_t *>(din + layout->slot_mapping), num_new_tokens,
                            stream);
        if (rc != PKV_OK) return rc;
    }
    if (!empty) {
        e = pkv::launch_decode(L, a, d.num_blocks, st, pool->tracer);
        if (e != cudaSuccess) return cuda_fail(e, "paged_attn_decode_step launch");
    }
    if (done_event) {
        e = cudaEventRecord(static_cast<cudaEvent_t>(done_event), st);
        if (e != cudaSuccess) return cuda_fail(e, "paged_attn_decode_step done_event");
    }
    if (host_out && num_requests > 0) {
        e = cudaMemcpyAsync(host_out, out, (size_t)num_requests * num_q_heads * row,
                            cudaMemcpyDeviceToHost, st);
        if (e == cudaSuccess && host_lse && lse)
            e = cudaMemcpyAsync(host_lse, lse, (size_t)num_requests * num_q_heads * sizeof(float),
                                cudaMemcpyDeviceToHost, st);
        if (e != cudaSuccess) return cuda_fail(e, "paged_attn_decode_step output copy");
    }
    return ok();
}

int pkv_blocks_staging_size(pkv_pool_t pool, int32_t n, size_t *bytes_out) {
    if (!pool || n < 0 || !bytes_out) return fail(PKV_ERR_INVALID_ARG, "bad arguments");
    *bytes_out = (size_t)n * 2 * pool->desc.num_kv_heads * 16 * pool->desc.head_dim * 2;
    return ok();
}

}  // extern "C"

namespace {

int block_copy(pkv_pool_t pool, const int32_t *block_ids, int32_t n, void *staging, bool to_staging,
               pkv_stream_t stream, const char *what) {
    int rc = check_kernel_pool(pool);
    if (rc != PKV_OK) return rc;
    if (n < 0) return fail(PKV_ERR_INVALID_ARG, "%s: n < 0", what);
    if (n == 0) return ok();
    if (!block_ids || !staging) return fail(PKV_ERR_INVALID_ARG, "%s: NULL buffer", what);
    if ((reinterpret_cast<uintptr_t>(block_ids) & 3) || !aligned16(staging))
        return fail(PKV_ERR_INVALID_ARG, "%s: misaligned block ids or staging", what);
    if ((rc = set_device(pool)) != PKV_OK) return rc;
    const pkv_pool_desc &d = pool->desc;
    const cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (pool->tracer) pool->tracer->begin(pkv::kKernelBlockCopy, st);
    cudaError_t e = pkv::launch_block_copy(block_ids, n, d.num_kv_heads, d.head_dim, pool->k_cache,
                                           pool->v_cache, staging, d.num_blocks, to_staging, pool->d_err,
                                           pool->num_sms, st);
    if (pool->tracer) pool->tracer->end(pkv::kKernelBlockCopy, st);
    if (e != cudaSuccess) return cuda_fail(e, what);
    return ok();
}

}  // namespace

extern "C" {

int pkv_blocks_gather(pkv_pool_t pool, const int32_t *block_ids, int32_t n, void *staging,
                      pkv_stream_t stream) {
    return block_copy(pool, block_ids, n, staging, true, stream, "pkv_blocks_gather");
}

int pkv_blocks_scatter(pkv_pool_t pool, const int32_t *block_ids, int32_t n, const void *staging,
                       pkv_stream_t stream) {
    return block_copy(pool, block_ids, n, const_cast<void *>(staging), false, stream, "pkv_blocks_scatter");
}

int pkv_check_device_errors(pkv_pool_t pool, pkv_stream_t stream, int32_t *code_out) {
    int rc = check_kernel_pool(pool);
    if (rc != PKV_OK) return rc;
    if (!code_out) return fail(PKV_ERR_INVALID_ARG, "code_out is NULL");
    if ((rc = set_device(pool)) != PKV_OK) return rc;
    cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
    int v = 0;
    e = cudaMemcpy(&v, pool->d_err, sizeof(int), cudaMemcpyDeviceToHost);
    if (e == cudaSuccess) e = cudaMemset(pool->d_err, 0, sizeof(int));
    if (e != cudaSuccess) return cuda_fail(e, "reading the device error word");
    *code_out = v;
    return ok();
}

int pkv_trace_enable(pkv_pool_t pool, int32_t enable) {
    int rc = check_kernel_pool(pool);
    if (rc != PKV_OK) return rc;
    if (enable && !pool->tracer) pool->tracer = new EventTracer();
    if (!enable && pool->tracer) {
        if ((rc = set_device(pool)) != PKV_OK) return rc;
        cudaDeviceSynchronize();
        delete pool->tracer;
        pool->tracer = nullptr;
    }
    return ok();
}

int pkv_trace_read(pkv_pool_t pool, pkv_kernel_time *out, int32_t max_entries, int32_t *n_out) {
    int rc = check_kernel_pool(pool);
    if (rc != PKV_OK) return rc;
    if (!n_out || max_entries < 0 || (max_entries > 0 && !out))
        return fail(PKV_ERR_INVALID_ARG, "bad arguments");
    *n_out = 0;
    EventTracer *t = pool->tracer;
    if (!t) return fail(PKV_ERR_INVALID_ARG, "tracing is not enabled");
    if ((rc = set_device(pool)) != PKV_OK) return rc;
    if (t->err != cudaSuccess) return cuda_fail(t->err, "trace event");
    double tot[pkv::kNumKernelIds] = {0};
    int32_t cnt[pkv::kNumKernelIds] = {0};
    for (auto &r : t->recs) {
        cudaError_t e = cudaEventSynchronize(r.b);
        float ms = 0.f;
        if (e == cudaSuccess) e = cudaEventElapsedTime(&ms, r.a, r.b);
        if (e != cudaSuccess) return cuda_fail(e, "reading trace events");
        tot[r.kid] += ms;
        cnt[r.kid] += 1;
    }
    t->recycle();
    int32_t n = 0;
    for (int k = 0; k < pkv::kNumKernelIds; ++k) {
        if (!cnt[k]) continue;
        if (n < max_entries) {
            memset(&out[n], 0, sizeof(out[n]));
            snprintf(out[n].name, sizeof(out[n].name), "%s", pkv::kKernelNames[k]);
            out[n].launches = cnt[k];
            out[n].total_ms = tot[k];
        }
        ++n;
    }
    *n_out = n < max_entries ? n : max_entries;
    return ok();
}

}  // extern "C"
