// decode_noalloc.cu -- paged_attn_decode for callers that cannot allocate
// device memory.
//
// Some callers of this library cannot call cudaMalloc at the point where
// they run decode: code recorded into a CUDA graph (an allocation would break
// or escape the capture), inference plugins whose host framework owns every
// device buffer and forbids allocations in its enqueue path, and serving
// processes that reserve a fixed memory budget up front.  For them this file
// keeps the decode split-KV scratch in one statically sized device array that
// the CUDA runtime creates when the library's module is loaded on a GPU, so
// the call itself allocates nothing.
#include "../../include/pkv.h"

#include <cuda_runtime.h>

#include <cstdio>
#include <mutex>

#include "pkv_internal.h"

namespace {

// Largest workspace this entry point can serve.  Every GPU that loads the
// library holds this array until the process exits.
constexpr size_t kScratchBytes = size_t(64) << 20;
using pkv::kMaxDevices;

__device__ __align__(256) unsigned char g_decode_scratch[kScratchBytes];

// Device address of g_decode_scratch per device, found once per device.
void *g_scratch_addr[kMaxDevices] = {};
std::mutex g_scratch_mu;

}  // namespace

extern "C" int paged_attn_decode_noalloc(pkv_pool_t pool, const void *q, void *out, float *lse,
                                         const int32_t *context_lens, const int32_t *block_table,
                                         int32_t max_blocks, int32_t num_requests,
                                         int32_t num_q_heads, float scale,
                                         const pkv_prefix_groups *groups, pkv_stream_t stream) {
    if (!pool || !q) return pkv::set_last_error(PKV_ERR_INVALID_ARG, "pool and q must be non-NULL");
    size_t need = 0;
    int rc = paged_attn_decode_workspace_size(pool, num_requests, num_q_heads, max_blocks, groups,
                                              &need);
    if (rc != PKV_OK) return rc;
    if (need > kScratchBytes) {
        char msg[200];
        snprintf(msg, sizeof msg,
                 "paged_attn_decode_noalloc: these shapes need %zu bytes of scratch, the static "
                 "scratch holds %zu; use paged_attn_decode with a caller workspace",
                 need, kScratchBytes);
        return pkv::set_last_error(PKV_ERR_WORKSPACE, msg);
    }
    // the kernels run on the pool's device: the scratch address must be that
    // device's, and q must live there too
    int dev = -1;
    rc = pkv::pool_device(pool, &dev);
    if (rc != PKV_OK) return rc;
    if (dev < 0 || dev >= kMaxDevices)
        return pkv::set_last_error(PKV_ERR_INVALID_ARG, "paged_attn_decode_noalloc: pool device out of range");
    cudaPointerAttributes attr;
    cudaError_t e = cudaPointerGetAttributes(&attr, q);
    if (e != cudaSuccess || attr.type != cudaMemoryTypeDevice || attr.device != dev) {
        cudaGetLastError();
        return pkv::set_last_error(PKV_ERR_INVALID_ARG,
                                   "paged_attn_decode_noalloc: q is not device memory of the pool's device");
    }
    void *scratch = nullptr;
    {
        // one-time set-up on this device, with the device current: the host
        // name g_decode_scratch is only a stand-in, the kernels need the
        // device address
        std::lock_guard<std::mutex> lock(g_scratch_mu);
        if (!g_scratch_addr[dev]) {
            int prev = -1;
            e = cudaGetDevice(&prev);
            if (e == cudaSuccess && prev != dev) e = cudaSetDevice(dev);
            void *p = nullptr;
            if (e == cudaSuccess) e = cudaGetSymbolAddress(&p, g_decode_scratch);
            if (prev >= 0 && prev != dev) cudaSetDevice(prev);
            if (e != cudaSuccess || !p) {
                char msg[200];
                snprintf(msg, sizeof msg,
                         "paged_attn_decode_noalloc: cudaGetSymbolAddress failed: %s",
                         cudaGetErrorString(e));
                return pkv::set_last_error(PKV_ERR_CUDA, msg);
            }
            g_scratch_addr[dev] = p;
        }
        scratch = g_scratch_addr[dev];
    }
    return paged_attn_decode(pool, q, out, lse, context_lens, block_table, max_blocks, num_requests,
                             num_q_heads, scale, groups, scratch, kScratchBytes, stream);
}
