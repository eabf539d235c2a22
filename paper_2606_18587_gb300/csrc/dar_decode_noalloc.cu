// dar_decode_noalloc.cu -- dar_attn_decode for callers that cannot allocate
// device memory.
//
// Some callers have no way to obtain a device buffer for the decode
// workspace: code embedded in a host framework that exposes no device
// allocator, or serving loops whose policy forbids any allocation after
// start-up.  For them this entry point takes its scratch from one
// file-scope __device__ array of DAR_DECODE_NOALLOC_MAX_BYTES that every GPU
// loading the library holds until the process exits.
#include <stdio.h>

#include "dar_common.cuh"
#include "dar_launch.h"

namespace {

static __device__ __align__(256) unsigned char g_decode_scratch[DAR_DECODE_NOALLOC_MAX_BYTES];

// device address of g_decode_scratch, looked up once per device (thread-safe)
dar::PerDeviceOnce g_scratch_once;
void *g_scratch_ptr[dar::kMaxDevices] = {};

}  // namespace

extern "C" dar_status dar_attn_decode_noalloc(const dar_cache *cache, int32_t Hq, const void *q,
                                              const float *Uk, const float *Uv, float scale, void *out,
                                              void *stream)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= dar::kMaxDevices) {
        dar::set_last_error("dar_attn_decode_noalloc: no usable current device");
        return DAR_ERR_CUDA;
    }
    // One-time set-up on this device (with it current): the host-side name of
    // the array is not a device address, so ask the runtime for the address.
    const cudaError_t e = dar::per_device_once(g_scratch_once, [](int d) {
        void *p = nullptr;
        cudaError_t e2 = cudaGetSymbolAddress(&p, g_decode_scratch);
        if (e2 == cudaSuccess && !p)
            e2 = cudaErrorInvalidSymbol;
        g_scratch_ptr[d] = p;
        return e2;
    });
    if (e != cudaSuccess) {
        dar::set_last_error(cudaGetErrorString(e));
        return DAR_ERR_CUDA;
    }
    const size_t need = dar_decode_workspace_bytes(cache, Hq);
    if (need == 0)  // invalid cache or Hq: the regular entry point reports which, launching nothing
        return dar_attn_decode(cache, Hq, q, Uk, Uv, scale, out, g_scratch_ptr[dev], 0, stream);
    if (need > DAR_DECODE_NOALLOC_MAX_BYTES) {
        char msg[160];
        snprintf(msg, sizeof msg,
                 "dar_attn_decode_noalloc: this cache shape needs %zu bytes of scratch, more than the "
                 "built-in %u (use dar_attn_decode with a workspace)",
                 need, (unsigned)DAR_DECODE_NOALLOC_MAX_BYTES);
        dar::set_last_error(msg);
        return DAR_ERR_CAPACITY;
    }
    // The array keeps whatever the previous call left; the decode kernels
    // rewrite every byte of it they read, so it needs no clearing.
    return dar_attn_decode(cache, Hq, q, Uk, Uv, scale, out, g_scratch_ptr[dev], need, stream);
}
