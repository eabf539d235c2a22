// dar_selftest.cu -- dar_check_bounded_wait: exercises the give-up path that
// every kernel of the library shares when a bounded wait runs out (report
// DAR_ERR_DEVICE, let the block's own copies land, release tensor memory,
// exit), on a barrier that nothing ever completes.
#include "dar_common.cuh"
#include "dar_launch.h"
#include "dar_sm100.cuh"

namespace dar {
namespace {

constexpr unsigned kCopyBytes = 256;
constexpr uint32_t kTmemCols = 32;  // the smallest allocation

static __device__ __align__(128) unsigned char g_copy_src[kCopyBytes];

__global__ void __launch_bounds__(64, 1) bounded_wait_check_kernel(int32_t *status, unsigned long long limit_ns)
{
    using namespace sm100;
    __shared__ __align__(128) unsigned char buf[kCopyBytes];
    __shared__ __align__(8) uint64_t bars[2];  // [0]: the copy landed; [1]: never completed
    __shared__ uint32_t tmem_slot;
    const int warp = threadIdx.x >> 5;
    if (threadIdx.x == 0) {
        mbar_init(&bars[0], 1);
        mbar_init(&bars[1], 1);
        mbar_init_fence();
    }
    if (warp == 1) {
        tmem_alloc(&tmem_slot, kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;
    if (threadIdx.x == 0) {
        // a copy of this block in flight when the wait gives up
        mbar_expect_tx(&bars[0], kCopyBytes);
        bulk_g2s(buf, g_copy_src, kCopyBytes, &bars[0]);
        // nothing arrives on bars[1]: this wait runs out after limit_ns
        if (!mbar_wait(&bars[1], 0, nullptr, limit_ns)) {
            report(status, DAR_ERR_DEVICE);
            // the give-up path: own copies land (bounded) before the block leaves
            mbar_wait(&bars[0], 0, nullptr);
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1)
        tmem_dealloc(tmem, kTmemCols);
}

}  // namespace
}  // namespace dar

extern "C" dar_status dar_check_bounded_wait(int32_t *status, uint32_t limit_us, void *stream)
{
    if (!status || limit_us < 1 || limit_us > 2000000u) {
        dar::set_last_error("dar_check_bounded_wait: status must be non-NULL and limit_us in [1, 2000000]");
        return DAR_ERR_INVALID_ARG;
    }
    dar::bounded_wait_check_kernel<<<1, 64, 0, static_cast<cudaStream_t>(stream)>>>(
        status, (unsigned long long)limit_us * 1000ull);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) {
        dar::set_last_error(cudaGetErrorString(e));
        return DAR_ERR_CUDA;
    }
    dar::set_last_error("");
    return DAR_OK;
}
