// cache_write.cu -- scatter of new-token K/V rows into the paged pool.
//
// The paged KV cache of Sec. 2 / Sec. 5.4 stores each token in a slot of a
// physical block; the slot mapping names that slot.  This kernel is a plain
// bit copy, one 16-byte vector per thread: source rows [T][Hkv][d] are read
// contiguously and each (token, head) row of d bf16 lands contiguously at
// pool[slot / 16][head][slot % 16][:].  HBM-bound: 2 * (read + write) bytes.
#include "pkv_device.cuh"
#include "pkv_internal.h"

namespace pkv {

__global__ void __launch_bounds__(256) cache_write_kernel(
    const uint4 *__restrict__ k_new, const uint4 *__restrict__ v_new,
    const int64_t *__restrict__ slots, int64_t total_chunks, int32_t chunks_per_token,
    int32_t chunks_per_row, int32_t Hkv, uint4 *__restrict__ k_cache,
    uint4 *__restrict__ v_cache, int64_t num_slots, int *err) {
    pdl_wait();
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; c < total_chunks; c += stride) {
        const int64_t t = c / chunks_per_token;
        const int32_t rem = (int32_t)(c - t * chunks_per_token);
        const int32_t h = rem / chunks_per_row;
        const int32_t ch = rem - h * chunks_per_row;
        const int64_t s = __ldg(slots + t);
        if (s < 0) continue;
        if (s >= num_slots) {
            latch_error(err, kDevBounds);
            continue;
        }
        const int64_t blk = s >> 4, off = s & 15;
        const int64_t dst = ((blk * Hkv + h) * 16 + off) * chunks_per_row + ch;
        const uint4 kv = ldg_stream(k_new + c);
        const uint4 vv = ldg_stream(v_new + c);
        k_cache[dst] = kv;
        v_cache[dst] = vv;
    }
}

cudaError_t launch_cache_write(const void *k_new, const void *v_new, const int64_t *slots,
                               int32_t T, void *k_cache, void *v_cache, int32_t Hkv, int32_t d,
                               int64_t num_slots, int *err, cudaStream_t stream, Tracer *tr) {
    if (T <= 0) return cudaSuccess;
    const int32_t chunks_per_row = d / 8;
    const int32_t chunks_per_token = Hkv * chunks_per_row;
    const int64_t total = (int64_t)T * chunks_per_token;
    int64_t blocks = (total + 255) / 256;
    if (blocks > 152 * 16) blocks = 152 * 16;
    if (tr) tr->begin(kKernelCacheWrite, stream);
    cudaError_t e = launch_pdl(cache_write_kernel, dim3((unsigned)blocks), dim3(256), 0, stream,
                               reinterpret_cast<const uint4 *>(k_new),
                               reinterpret_cast<const uint4 *>(v_new), slots, total, chunks_per_token,
                               chunks_per_row, Hkv, reinterpret_cast<uint4 *>(k_cache),
                               reinterpret_cast<uint4 *>(v_cache), num_slots, err);
    if (tr) tr->end(kKernelCacheWrite, stream);
    return e;
}

}  // namespace pkv
