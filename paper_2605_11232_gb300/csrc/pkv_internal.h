// pkv_internal.h -- declarations shared by the host API and the kernel files.
// Not part of the public ABI (that is include/pkv.h).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>
#include <mutex>

struct pkv_pool;   // the pool handle's struct (include/pkv.h: pkv_pool_t)

namespace pkv {

// Kernels the library launches (names reported by pkv_trace_read).
enum KernelId : int {
    kKernelCacheWrite = 0,
    kKernelDecodeSplit = 1,
    kKernelDecodeCombine = 2,
    kKernelDecodePrefix = 3,
    kKernelPrefill = 4,
    kKernelBlockCopy = 5,
    kNumKernelIds = 6,
};
extern const char *const kKernelNames[kNumKernelIds];

// Optional per-launch timing: a CUDA event pair recorded on the launch stream
// around each kernel (null = tracing off).
struct Tracer {
    virtual void begin(int kernel_id, cudaStream_t s) = 0;
    virtual void end(int kernel_id, cudaStream_t s) = 0;
    virtual ~Tracer() {}
};

// Launch with programmatic dependent launch allowed: the kernel's launch is
// processed while its predecessor in the stream is still running, and its
// CTAs start as the predecessor's CTAs exit; it calls griddepcontrol.wait
// (pdl_wait) before touching any memory, so it observes everything the
// predecessor wrote.  This hides the launch gaps between the kernels of a step.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t stream, Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// A kernel's dynamic shared-memory limit (cudaFuncAttributeMaxDynamicSharedMemorySize)
// is a per-device setting.  One SmemLimit per kernel instantiation records,
// per device, the largest limit set so far; ensure() raises it on the current
// device when a launch needs more.  Thread-safe: the limit only grows, under
// the lock, so two threads launching on one device never lower each other's.
constexpr int kMaxDevices = 64;
struct SmemLimit {
    std::atomic<int> bytes[kMaxDevices] = {};
    std::mutex mu;
    cudaError_t ensure(const void *func, int need);
};

// Largest table width paged_attn_prefill accepts: a work item's block ids are
// staged in shared memory, at most kPrefillMaxBlocks of them (32768 keys).
constexpr int kPrefillMaxBlocks = 2048;

// Set the thread's pkv_last_error() message; returns code.
int set_last_error(int code, const char *msg);

// The device a pool's caches live on (the one its kernels launch on), after
// checking that the pool has device caches; PKV_OK or an error code.
int pool_device(::pkv_pool *pool, int *dev);

// The pool's device error word, after checking that the pool has device
// caches and making its device current; PKV_OK or an error code.
int pool_device_error_word(::pkv_pool *pool, int **err);

// Device error word values (a kernel latches the first one with atomicCAS).
enum : int {
    kDevOk = 0,
    kDevBounds = -9,   // PKV_ERR_DEVICE_BOUNDS
    kDevTimeout = -8,  // PKV_ERR_DEVICE_TIMEOUT
};

// Decode split-KV layout, shared by the split, prefix and combine kernels.
// Partials of request r, q-head hq live at part slots
//   [(r * Hq + hq) * parts_per_head + p]
// with p in [0, prefix_parts) for the shared-prefix pass and
// p in [prefix_parts, prefix_parts + kMaxPrivateParts) for private pieces.
constexpr int kMaxPrivateParts = 16;
constexpr int kMaxPrefixParts = 16;   // parts_per_head <= 32: one part per combine lane
constexpr int kMinBlocksPerPiece = 4;

constexpr size_t kMaxSmemPerBlock = 227 * 1024;   // opt-in dynamic shared memory per CTA

struct DecodeLayout {
    int32_t R, Hq, Hkv, d, g;
    int32_t sms;                 // SMs of the device the layout was made for
    int32_t prefix_parts;        // prefix-pass part slots per head (0 without groups)
    int32_t prefix_blocks_per_part;
    int64_t prefix_ctas;         // CTAs of the prefix pass (0 without groups)
    int32_t prefix_early;        // the prefix pass leaves a quarter of the SMs to the split pass
    int32_t split_grid;          // split-pass CTAs beside such a prefix pass (sms - prefix_ctas)
    int32_t stages;              // ring stages per warp of the split pass
    int32_t qbytes;              // bytes of a stage's Q area (4 or 8 head rows)
    int32_t lens_in_smem;        // the split pass keeps the context lengths in shared memory
    size_t split_smem;           // dynamic shared memory of the split pass
    int32_t parts_per_head;      // prefix_parts + kMaxPrivateParts
    // byte offsets inside the workspace
    size_t off_o;                // float [R*Hq*parts][d]
    size_t off_ml;               // float2 [R*Hq*parts]
    size_t off_nparts;           // int32 [R*Hkv] part counts per (r, kv head): private | prefix << 16
    size_t total;
};

DecodeLayout decode_layout(int32_t R, int32_t Hq, int32_t Hkv, int32_t d, int32_t max_blocks,
                           int32_t num_groups, int32_t max_group_blocks, int32_t max_group_members,
                           int32_t num_sms);

// Grouped verification: decode's layout with rows = draft tokens (T) and one
// private part slot per (token, q head).
DecodeLayout verify_layout(int32_t T, int32_t Hq, int32_t Hkv, int32_t d, int32_t max_blocks,
                           int32_t num_groups, int32_t max_group_blocks, int32_t max_group_tokens,
                           int32_t num_sms);

cudaError_t launch_cache_write(const void *k_new, const void *v_new, const int64_t *slots,
                               int32_t T, void *k_cache, void *v_cache, int32_t Hkv, int32_t d,
                               int64_t num_slots, int *err, cudaStream_t stream, Tracer *tr);

struct DecodeArgs {
    const void *q;
    void *out;
    float *lse;
    const int32_t *context_lens;
    const int32_t *block_table;
    int32_t max_blocks;
    const void *k_cache;
    const void *v_cache;
    float scale_log2;   // softmax scale * log2(e)
    // prefix groups (all null / 0 without groups)
    int32_t num_groups;
    int32_t max_group_members;
    const int32_t *group_start;
    const int32_t *member_req;
    const int32_t *group_blocks;
    const int32_t *group_of_req;
    void *ws;
    int *err;
    const CUtensorMap *tmap_k;   // TMA descriptors of the pool's caches
    const CUtensorMap *tmap_v;
    // the query tokens' own K/V, bf16 [R][Hkv][d], stored at position L - 1
    // by the split pass (paged_attn_decode_append); null: already in the cache
    const void *k_new;
    const void *v_new;
    // grouped verification: the table row naming each group's prefix blocks
    // (null: the first member's) and the number of table rows
    const int32_t *group_row;
    int32_t num_table_rows;
};

cudaError_t launch_decode(const DecodeLayout &L, const DecodeArgs &a, int32_t num_blocks_pool,
                          cudaStream_t stream, Tracer *tr);

// The combine alone: merge every (row, kv head)'s partials of the workspace
// into out / lse (rows = L.R; decode requests, or draft tokens).
cudaError_t launch_decode_combine(const DecodeLayout &L, const DecodeArgs &a, cudaStream_t stream, Tracer *tr);



// Bit copy of n blocks (device ids) between a pool's caches and a staging
// buffer [n][K, V][Hkv][16][d] (transfer.cu).
cudaError_t launch_block_copy(const int32_t *ids, int32_t n, int32_t Hkv, int32_t d, void *k_cache,
                              void *v_cache, void *staging, int32_t num_blocks, bool to_staging, int *err,
                              int num_sms, cudaStream_t stream);

struct PrefillArgs {
    const void *q;
    void *out;
    float *lse;
    const int32_t *cu_seqlens_q;
    const int32_t *context_lens;
    const int32_t *block_table;
    int32_t max_blocks;
    int32_t R, Hq, Hkv, d;
    int32_t max_seqlen_q;
    int32_t num_blocks_pool;
    float scale_log2;
    const CUtensorMap *tmap_k;  // host copies, passed by value to the kernel
    const CUtensorMap *tmap_v;
    int *err;
    const unsigned long long *tree_mask;   // null, or [T] draft masks (tree verification)
    // the new tokens' K/V stored by the kernel (null: already in the cache)
    const void *k_new, *v_new;             // [T][Hkv][d]
    void *k_cache, *v_cache;
    const CUtensorMap *tmap_kn;            // 3-D maps over k_new / v_new
    const CUtensorMap *tmap_vn;
    int32_t num_sms;                       // the device's SM count (0: unknown)
};

cudaError_t launch_prefill(const PrefillArgs &a, cudaStream_t stream, Tracer *tr);

// Grouped verification of tree-shaped drafts: the shared-prefix pass over each
// group's draft tokens, the private pass (keys after the shared blocks, draft
// masks) writing partial slot L.prefix_parts, then the combine over the
// tokens.  a: the decode arguments with rows = draft tokens (a.q, a.out,
// a.lse over [T]; groups over tokens, a.group_row / a.num_table_rows set);
// pa: the prefill arguments of the private pass (tree_mask set).
cudaError_t launch_verify_grouped(const DecodeLayout &L, const DecodeArgs &a, const PrefillArgs &pa,
                                  const int32_t *request_group, cudaStream_t stream, Tracer *tr);

// Shared-prefix pass of decode (tcgen05 tile kernel in prefix mode): partials
// of every group member over its group's prefix blocks, split in key ranges of
// L.prefix_blocks_per_part blocks, into part slots [0, L.prefix_parts).
cudaError_t launch_decode_prefix(const DecodeLayout &L, const DecodeArgs &a,
                                 int32_t num_blocks_pool, cudaStream_t stream, Tracer *tr);

}  // namespace pkv
