// dar_common.cuh -- storage-type helpers shared by the DAR kernels.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "dar.h"

namespace dar {

constexpr int kHeadDim = 64;  // d, the head dimension the kernels are built for
constexpr int kPage = DAR_PAGE_SIZE;

using bf16 = __nv_bfloat16;

// Elements of T in one 16-byte granule.
template <typename T>
struct Granule;
template <>
struct Granule<float> {
    static constexpr int kElems = 4;
};
template <>
struct Granule<bf16> {
    static constexpr int kElems = 8;
};

__device__ __forceinline__ uint4 ld_stream_v4(const void *p)
{
    uint4 r;
    asm volatile("ld.global.nc.L1::no_allocate.L2::256B.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
                 : "l"(p));
    return r;
}

__device__ __forceinline__ float bf16lo(uint32_t u) { return __uint_as_float(u << 16); }
__device__ __forceinline__ float bf16hi(uint32_t u) { return __uint_as_float(u & 0xffff0000u); }

// Unpack one raw 16-byte granule into floats.
__device__ __forceinline__ void unpack(const uint4 &r, float (&x)[4], float)
{
    x[0] = __uint_as_float(r.x);
    x[1] = __uint_as_float(r.y);
    x[2] = __uint_as_float(r.z);
    x[3] = __uint_as_float(r.w);
}
__device__ __forceinline__ void unpack(const uint4 &r, float (&x)[8], bf16)
{
    x[0] = bf16lo(r.x);
    x[1] = bf16hi(r.x);
    x[2] = bf16lo(r.y);
    x[3] = bf16hi(r.y);
    x[4] = bf16lo(r.z);
    x[5] = bf16hi(r.z);
    x[6] = bf16lo(r.w);
    x[7] = bf16hi(r.w);
}

__device__ __forceinline__ float to_f32(float x) { return x; }
__device__ __forceinline__ float to_f32(bf16 x) { return __bfloat162float(x); }

template <typename T>
__device__ __forceinline__ T from_f32(float x);
template <>
__device__ __forceinline__ float from_f32<float>(float x)
{
    return x;
}
template <>
__device__ __forceinline__ bf16 from_f32<bf16>(float x)
{
    return __float2bfloat16_rn(x);
}

// First device-side error wins.
__device__ __forceinline__ void report(int32_t *status, int code)
{
    if (status)
        atomicCAS(status, 0, code);
}

}  // namespace dar
