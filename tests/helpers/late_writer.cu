// Test helper: a kernel that allows the next kernel on its stream to start at
// once (griddepcontrol.launch_dependents, programmatic dependent launch), and
// only after a delay copies src to dst.  A consumer launched after it that
// reads dst before the copy would see stale data.  The delay loop is bounded.
#include <cuda_runtime.h>
#include <stdint.h>

__global__ void late_copy_kernel(const uint4 *src, uint4 *dst, int n16, unsigned long long delay_ns)
{
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    unsigned long long t0, t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t0));
    for (int k = 0; k < 50000000; ++k) {
        asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
        if (t - t0 >= delay_ns)
            break;
    }
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n16; i += gridDim.x * blockDim.x)
        dst[i] = src[i];
}

extern "C" int late_copy(const void *src, void *dst, int n16, unsigned long long delay_ns, void *stream)
{
    late_copy_kernel<<<4, 256, 0, static_cast<cudaStream_t>(stream)>>>(static_cast<const uint4 *>(src),
                                                                       static_cast<uint4 *>(dst), n16, delay_ns);
    return (int)cudaGetLastError();
}
