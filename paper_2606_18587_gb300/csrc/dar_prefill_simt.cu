// dar_prefill_simt.cu -- causal DAR attention forward on the CUDA cores (fp32
// FFMA).  Used for fp32 storage, where the 1e-5 accuracy target rules out
// TF32 tensor cores.
//
// One CTA = 64 query rows of one head; key tiles of 64.  A key tile is
// all-global (every pair has i - j >= w), all-local (every pair i - j < w) or a
// band tile that holds both kinds; the element rule is Eq. 3 (local iff
// i - j < w).  Local pairs score q . k (d = 64); global pairs score
// q~ . k^D with q~ = q Uk^T (d_down; in the direct variant of Sec. 5, q~ is
// the row's own d_down query times scale_down / scale).  One online softmax covers both kinds,
// values accumulate in d (local) and d_down (global) and the global part is
// lifted once with Uv in the epilogue:  o = (o_loc + o_glob Uv) / l.
#include "dar_common.cuh"
#include "dar_launch.h"

namespace dar {

constexpr int kSimtRows = 64, kSimtKeys = 64, kSimtLd = 65;

template <int DD>
constexpr size_t simt_smem_floats()
{
    return 5 * 64 * kSimtLd + 3 * 64 * (DD + 1);
}

template <typename T, int DD>
__global__ void __launch_bounds__(256) prefill_simt_kernel(PrefillArgs a)
{
    constexpr int LDD = DD + 1;
    constexpr int OG = DD / 4;  // global accumulators per thread
    extern __shared__ float sm[];
    float *Qs = sm;                        // [64][65] scaled q
    float *Ks = Qs + kSimtRows * kSimtLd;  // [64][65]
    float *Vs = Ks + kSimtKeys * kSimtLd;  // [64][65]
    float *Ps = Vs + kSimtKeys * kSimtLd;  // [64][65] weights of local pairs
    float *Pg = Ps + kSimtRows * kSimtLd;  // [64][65] weights of global pairs
    float *Qt = Pg + kSimtRows * kSimtLd;  // [64][DD+1] scaled q~
    float *KDs = Qt + kSimtRows * LDD;     // [64][DD+1]
    float *VDs = KDs + kSimtKeys * LDD;    // [64][DD+1]

    const int N = a.N, w = a.w;
    const int bh = blockIdx.y, b = bh / a.Hq, h = bh % a.Hq, g = h / (a.Hq / a.Hkv);
    const int i0 = blockIdx.x * kSimtRows;
    const int tid = threadIdx.x, r = tid >> 2, qd = tid & 3;
    const int i = i0 + r;
    const T *q = static_cast<const T *>(a.q) + ((size_t)b * a.Hq + h) * N * kHeadDim;
    const T *k = static_cast<const T *>(a.k) + ((size_t)b * a.Hkv + g) * N * kHeadDim;
    const T *v = static_cast<const T *>(a.v) + ((size_t)b * a.Hkv + g) * N * kHeadDim;
    const T *kd = static_cast<const T *>(a.kd) + ((size_t)b * a.Hkv + g) * N * DD;
    const T *vd = static_cast<const T *>(a.vd) + ((size_t)b * a.Hkv + g) * N * DD;
    const float *Uk = a.Uk + (size_t)g * DD * kHeadDim;
    const float *Uv = a.Uv + (size_t)g * DD * kHeadDim;

    for (int idx = tid; idx < kSimtRows * kHeadDim; idx += 256) {
        const int rr = idx / kHeadDim, t = idx % kHeadDim;
        Qs[rr * kSimtLd + t] = (i0 + rr < N) ? to_f32(q[(size_t)(i0 + rr) * kHeadDim + t]) * a.qscale : 0.f;
    }
    __syncthreads();
    for (int idx = tid; idx < kSimtRows * DD; idx += 256) {
        const int rr = idx / DD, c = idx % DD;
        if (a.qd) {  // direct variant (Sec. 5): the row's own d_down query, at the global scale
            Qt[rr * LDD + c] = (i0 + rr < N)
                ? to_f32(static_cast<const T *>(a.qd)[(((size_t)b * a.Hq + h) * N + i0 + rr) * DD + c]) *
                      a.qd_ratio * a.qscale
                : 0.f;
            continue;
        }
        float acc = 0.f;
        for (int t = 0; t < kHeadDim; ++t)
            acc = fmaf(Qs[rr * kSimtLd + t], Uk[c * kHeadDim + t], acc);
        Qt[rr * LDD + c] = acc;
    }
    __syncthreads();

    float m = -INFINITY, l = 0.f;
    float ol[16], og[OG];
#pragma unroll
    for (int e = 0; e < 16; ++e)
        ol[e] = 0.f;
#pragma unroll
    for (int e = 0; e < OG; ++e)
        og[e] = 0.f;

    const int imax = min(N, i0 + kSimtRows) - 1;
    for (int j0 = 0; j0 <= imax; j0 += kSimtKeys) {
        const bool all_global = (i0 - (j0 + kSimtKeys - 1)) >= w;
        const bool all_local = (i0 + kSimtRows - 1 - j0) < w;
        if (!all_global) {
            for (int idx = tid; idx < kSimtKeys * kHeadDim; idx += 256) {
                const int jj = idx / kHeadDim, t = idx % kHeadDim, j = j0 + jj;
                Ks[jj * kSimtLd + t] = j < N ? to_f32(k[(size_t)j * kHeadDim + t]) : 0.f;
                Vs[jj * kSimtLd + t] = j < N ? to_f32(v[(size_t)j * kHeadDim + t]) : 0.f;
            }
        }
        if (!all_local) {
            for (int idx = tid; idx < kSimtKeys * DD; idx += 256) {
                const int jj = idx / DD, c = idx % DD, j = j0 + jj;
                KDs[jj * LDD + c] = j < N ? to_f32(kd[(size_t)j * DD + c]) : 0.f;
                VDs[jj * LDD + c] = j < N ? to_f32(vd[(size_t)j * DD + c]) : 0.f;
            }
        }
        __syncthreads();

        float s[16];
        float mx = -INFINITY;
#pragma unroll
        for (int jj = 0; jj < 16; ++jj) {
            const int jl = qd + 4 * jj, j = j0 + jl;
            float val = -INFINITY;
            if (i < N && j <= i) {
                float acc = 0.f;
                if (i - j < w) {
#pragma unroll 16
                    for (int t = 0; t < kHeadDim; ++t)
                        acc = fmaf(Qs[r * kSimtLd + t], Ks[jl * kSimtLd + t], acc);
                } else {
#pragma unroll
                    for (int c = 0; c < DD; ++c)
                        acc = fmaf(Qt[r * LDD + c], KDs[jl * LDD + c], acc);
                }
                val = acc;
            }
            s[jj] = val;
            mx = fmaxf(mx, val);
        }
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
        const float mnew = fmaxf(m, mx);
        const float alpha = (m == -INFINITY) ? 0.f : exp2f(m - mnew);
        float psum = 0.f;
#pragma unroll
        for (int jj = 0; jj < 16; ++jj) {
            const int jl = qd + 4 * jj, j = j0 + jl;
            const float p = (s[jj] == -INFINITY) ? 0.f : exp2f(s[jj] - mnew);
            const bool loc = (i - j) < w;
            Ps[r * kSimtLd + jl] = loc ? p : 0.f;
            Pg[r * kSimtLd + jl] = loc ? 0.f : p;
            psum += p;
        }
        psum += __shfl_xor_sync(0xffffffffu, psum, 1);
        psum += __shfl_xor_sync(0xffffffffu, psum, 2);
        l = l * alpha + psum;
        m = mnew;
#pragma unroll
        for (int e = 0; e < 16; ++e)
            ol[e] *= alpha;
#pragma unroll
        for (int e = 0; e < OG; ++e)
            og[e] *= alpha;
        __syncthreads();

        if (!all_global) {
            for (int jl = 0; jl < kSimtKeys; ++jl) {
                const float p = Ps[r * kSimtLd + jl];
#pragma unroll
                for (int e = 0; e < 16; ++e)
                    ol[e] = fmaf(p, Vs[jl * kSimtLd + qd * 16 + e], ol[e]);
            }
        }
        if (!all_local) {
            for (int jl = 0; jl < kSimtKeys; ++jl) {
                const float p = Pg[r * kSimtLd + jl];
#pragma unroll
                for (int e = 0; e < OG; ++e)
                    og[e] = fmaf(p, VDs[jl * LDD + qd * OG + e], og[e]);
            }
        }
        __syncthreads();
    }

    // epilogue: o = (o_loc + o_glob Uv) / l
#pragma unroll
    for (int e = 0; e < OG; ++e)
        Qt[r * LDD + qd * OG + e] = og[e];
    __syncthreads();
    if (i < N) {
        const float inv = 1.f / l;
        T *o = static_cast<T *>(a.out) + (((size_t)b * a.Hq + h) * N + i) * kHeadDim;
#pragma unroll
        for (int e = 0; e < 16; ++e) {
            const int dim = qd * 16 + e;
            float acc = ol[e];
            for (int c = 0; c < DD; ++c)
                acc = fmaf(Qt[r * LDD + c], Uv[c * kHeadDim + dim], acc);
            o[dim] = from_f32<T>(acc * inv);
        }
    }
}

template <typename T, int DD>
static cudaError_t simt_t(const PrefillArgs &a, cudaStream_t s)
{
    auto kern = prefill_simt_kernel<T, DD>;
    const size_t smem = simt_smem_floats<DD>() * sizeof(float);
    static PerDeviceOnce once;  // attribute set-up per instantiation and device
    const cudaError_t e = per_device_once(once, [&](int) {
        return cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    });
    if (e != cudaSuccess)
        return e;
    dim3 grid((a.N + kSimtRows - 1) / kSimtRows, a.B * a.Hq);
    kern<<<grid, 256, smem, s>>>(a);
    return cudaGetLastError();
}

template <typename T>
static cudaError_t simt_type(int dd, const PrefillArgs &a, cudaStream_t s)
{
    switch (dd) {
    case 8: return simt_t<T, 8>(a, s);
    case 16: return simt_t<T, 16>(a, s);
    case 32: return simt_t<T, 32>(a, s);
    case 64: return simt_t<T, 64>(a, s);
    default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_prefill_simt(dar_dtype dt, int dd, const PrefillArgs &a, cudaStream_t s)
{
    if (a.B == 0 || a.N == 0)
        return cudaSuccess;
    return dt == DAR_F32 ? simt_type<float>(dd, a, s) : simt_type<bf16>(dd, a, s);
}

}  // namespace dar
