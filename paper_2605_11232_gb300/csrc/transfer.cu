// transfer.cu -- KV-block transfer between pools through a staging buffer.
//
// Prefill/decode disaggregation (Sec. 2; Sec. 7 names it as early
// exploration) moves a request's KV cache from the pool of the instance that
// prefilled it to the pool of the instance that decodes it.  The blocks of a
// request are scattered over the source pool; a transfer gathers them into
// one contiguous staging buffer (the unit a peer or network copy moves), and
// scatters that buffer into blocks allocated in the destination pool.  Both
// are plain bit copies, one 16-byte vector per thread: HBM-bound, 2 x (read +
// write) bytes per block.
//
// Staging layout: [n][2][Hkv][16][d] bf16 -- block i's K tile (all kv heads),
// then its V tile, exactly the bytes of that block in the pool's K and V
// caches.
#include "../../include/pkv.h"

#include <cuda_runtime.h>

#include "pkv_device.cuh"
#include "pkv_internal.h"

namespace pkv {
namespace {

// to_staging: pool -> staging; otherwise staging -> pool.  chunks_per_tile:
// 16-byte chunks of one block's K (or V) tile.
__global__ void __launch_bounds__(256) block_copy_kernel(const int32_t *__restrict__ ids, int32_t n,
                                                         int64_t chunks_per_tile, uint4 *k_cache,
                                                         uint4 *v_cache, uint4 *staging,
                                                         int32_t num_blocks, int to_staging, int *err) {
    pdl_wait();
    const int64_t total = (int64_t)n * 2 * chunks_per_tile;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; c < total; c += stride) {
        const int64_t tile = c / chunks_per_tile;     // 2 i + (0: K, 1: V)
        const int64_t off = c - tile * chunks_per_tile;
        const int32_t i = (int32_t)(tile >> 1);
        const int32_t id = __ldg(ids + i);
        if (id < 0 || id >= num_blocks) {
            latch_error(err, kDevBounds);
            continue;
        }
        uint4 *cache = (tile & 1) ? v_cache : k_cache;
        uint4 *pool_chunk = cache + (int64_t)id * chunks_per_tile + off;
        if (to_staging)
            staging[c] = ldg_stream(pool_chunk);
        else
            *pool_chunk = ldg_stream(staging + c);
    }
}

}  // namespace

cudaError_t launch_block_copy(const int32_t *ids, int32_t n, int32_t Hkv, int32_t d, void *k_cache,
                              void *v_cache, void *staging, int32_t num_blocks, bool to_staging, int *err,
                              int num_sms, cudaStream_t stream) {
    if (n <= 0) return cudaSuccess;
    const int64_t chunks_per_tile = (int64_t)Hkv * 16 * d / 8;
    const int64_t total = (int64_t)n * 2 * chunks_per_tile;
    int64_t blocks = (total + 255) / 256;
    const int64_t cap = (int64_t)(num_sms > 0 ? num_sms : 148) * 8;   // grid-stride beyond 8 CTAs per SM
    if (blocks > cap) blocks = cap;
    return launch_pdl(block_copy_kernel, dim3((unsigned)blocks), dim3(256), 0, stream, ids, n, chunks_per_tile,
                      static_cast<uint4 *>(k_cache), static_cast<uint4 *>(v_cache),
                      static_cast<uint4 *>(staging), num_blocks, to_staging ? 1 : 0, err);
}

}  // namespace pkv
