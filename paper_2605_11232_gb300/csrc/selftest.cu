// selftest.cu -- a test aid for the failure path of the bounded waits.
//
// Every wait of the library's kernels on an mbarrier or a counter has a time
// limit; when it runs out the kernel latches DEVICE_TIMEOUT into the pool's
// error word and returns, so that the GPU and the context stay usable.  This
// kernel makes such a wait run out on purpose, with nothing else in flight:
// one thread waits, with the library's bounded wait, on an mbarrier phase that
// nothing completes (no TMA copy, no MMA, no tensor memory).
#include "../../include/pkv.h"

#include <cuda_runtime.h>

#include "pkv_device.cuh"
#include "pkv_internal.h"
#include "tc_ptx.cuh"

namespace pkv {
namespace {

__global__ void wait_timeout_kernel(int *err, uint64_t limit_ns) {
    __shared__ __align__(8) uint64_t bar;
    __shared__ int abort_flag;
    if (threadIdx.x != 0) return;
    abort_flag = 0;
    tc::mbar_init(tc::smem_u32(&bar), 1);   // one arrival expected; none comes
    tc::fence_barrier_init();
    if (!tc::mbar_wait(tc::smem_u32(&bar), 0, &abort_flag, limit_ns)) latch_error(err, kDevTimeout);
}

}  // namespace
}  // namespace pkv

extern "C" int pkv_selftest_wait_timeout(pkv_pool_t pool, int32_t limit_us, pkv_stream_t stream) {
    if (limit_us < 0 || limit_us > 1000000)
        return pkv::set_last_error(PKV_ERR_INVALID_ARG, "limit_us must be in [0, 1e6]");
    int *err = nullptr;
    const int rc = pkv::pool_device_error_word(pool, &err);
    if (rc != PKV_OK) return rc;
    pkv::wait_timeout_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(err, (uint64_t)limit_us * 1000);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return pkv::set_last_error(PKV_ERR_CUDA, cudaGetErrorString(e));
    return PKV_OK;
}
