// dar_append.cu -- Eq. 1 (bottleneck down-projection) as a bulk kernel and as
// the window-exit migration of the mixed-dimension cache.
//
// Every bottleneck element is ONE fp32 fused-multiply-add chain over
// t = 0..63 starting from +0.0f, rounded once to the storage type, so a
// token's cached vector is bit-identical whichever kernel produced it.
#include "dar_common.cuh"
#include "dar_launch.h"

namespace dar {

// ---------------------------------------------------------------- bulk Eq. 1
// grid (ceil(n / 128), B * Hkv), 128 threads; one thread per token row.
template <typename T, int DD>
__global__ void __launch_bounds__(128) down_project_kernel(const T *__restrict__ x,
                                                           const float *__restrict__ W,
                                                           T *__restrict__ out, int Hkv, int n,
                                                           int ostride)
{
    __shared__ float Ws[kHeadDim * DD];
    const int bg = blockIdx.y;
    const int g = bg % Hkv;
    for (int i = threadIdx.x; i < kHeadDim * DD; i += blockDim.x)
        Ws[i] = W[(size_t)g * kHeadDim * DD + i];
    __syncthreads();

    const int j = blockIdx.x * blockDim.x + threadIdx.x;
    if (j >= n)
        return;
    constexpr int E = Granule<T>::kElems;
    const T *row = x + ((size_t)bg * n + j) * kHeadDim;
    float xv[kHeadDim];
#pragma unroll
    for (int q = 0; q < kHeadDim / E; ++q) {
        uint4 r = *reinterpret_cast<const uint4 *>(row + q * E);
        float f[E];
        unpack(r, f, T());
#pragma unroll
        for (int e = 0; e < E; ++e)
            xv[q * E + e] = f[e];
    }
    float acc[DD];
#pragma unroll
    for (int c = 0; c < DD; ++c)
        acc[c] = 0.0f;
#pragma unroll
    for (int t = 0; t < kHeadDim; ++t)
#pragma unroll
        for (int c = 0; c < DD; ++c)
            acc[c] = __fmaf_rn(xv[t], Ws[t * DD + c], acc[c]);
    T *o = out + ((size_t)bg * n + j) * ostride;
#pragma unroll
    for (int c = 0; c < DD; ++c)
        o[c] = from_f32<T>(acc[c]);
    for (int c = DD; c < ostride; ++c)
        o[c] = from_f32<T>(0.f);
}

// ------------------------------------------------------------ cache append

// Eq. 1 for one row, computed by a warp: lane j holds x[2j], x[2j+1] and lane
// c (and c + 32) runs the fixed-order chain for output c, reading x[t] by
// shuffle and its column of W from registers loaded in one batch.
template <typename T, int DD>
__device__ __forceinline__ void project_row_warp(const T *x, const float *W, T *out, int lane)
{
    constexpr int CPL = (DD + 31) / 32;
    const float x0 = to_f32(x[2 * lane]), x1 = to_f32(x[2 * lane + 1]);
    float wcol[CPL][kHeadDim];
#pragma unroll
    for (int i = 0; i < CPL; ++i) {
        const int c = lane + 32 * i;
#pragma unroll
        for (int t = 0; t < kHeadDim; ++t)
            wcol[i][t] = c < DD ? __ldg(W + t * DD + c) : 0.f;
    }
    float acc[CPL];
#pragma unroll
    for (int i = 0; i < CPL; ++i)
        acc[i] = 0.0f;
#pragma unroll
    for (int t = 0; t < kHeadDim; ++t) {
        const float xt = __shfl_sync(0xffffffffu, (t & 1) ? x1 : x0, t >> 1);
#pragma unroll
        for (int i = 0; i < CPL; ++i)
            acc[i] = __fmaf_rn(xt, wcol[i][t], acc[i]);
    }
#pragma unroll
    for (int i = 0; i < CPL; ++i) {
        const int c = lane + 32 * i;
        if (c < DD)
            out[c] = from_f32<T>(acc[i]);
    }
}

// Copy one 64-element row with the warp (2 elements per lane).
template <typename T>
__device__ __forceinline__ void copy_row_warp(const T *src, T *dst, int lane)
{
    if constexpr (sizeof(T) == 2) {
        reinterpret_cast<uint32_t *>(dst)[lane] = reinterpret_cast<const uint32_t *>(src)[lane];
    } else {
        reinterpret_cast<uint2 *>(dst)[lane] = reinterpret_cast<const uint2 *>(src)[lane];
    }
}

// Row of the bottleneck pool for position p of sequence b, KV head g, or
// nullptr (status set) when its block-table entry is not a valid page.
template <typename T, int DD>
__device__ __forceinline__ T *pool_row(const AppendArgs &a, T *pool, int b, int g, int p)
{
    const int lp = p / kPage;
    const int id = lp < a.maxp ? a.block_table[(size_t)b * a.maxp + lp] : -1;
    if (id < 0 || id >= a.num_pages) {
        report(a.status, DAR_ERR_CAPACITY);
        return nullptr;
    }
    return pool + (((size_t)id * a.Hkv + g) * kPage + (p % kPage)) * DD;
}

// grid B (one CTA per sequence, so its length can be updated at the end),
// up to 1024 threads.  Sequence b appends nb = n_per_seq[b] (or n) tokens; k_new
// rows are strided by n.  Work unit = (KV head g, slot touched by this call): the slot's
// old occupant migrates to its page, then the new positions of that slot are
// processed in order (all but the last migrate straight from k_new; the last
// is written into the ring).
template <typename T, int DD>
__global__ void __launch_bounds__(1024) cache_append_kernel(AppendArgs a)
{
    const int b = blockIdx.x;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
    __shared__ int s_L, s_nb, s_ok;
    if (threadIdx.x == 0) {
        const int L = a.seq_lens[b];
        const int nb = a.n_per_seq ? a.n_per_seq[b] : a.n;
        const long long Lnew = (long long)L + nb;
        int ok = 1;
        if (L < 0 || nb < 0 || nb > a.n) {
            report(a.status, DAR_ERR_INVALID_ARG);
            ok = 0;
        } else if (Lnew - a.w > (long long)a.maxp * kPage || Lnew > 0x7fffffffLL) {
            report(a.status, DAR_ERR_CAPACITY);
            ok = 0;
        }
        s_L = L;
        s_nb = nb;
        s_ok = ok;
    }
    __syncthreads();
    if (!s_ok || s_nb == 0)
        return;
    const int L = s_L, n = a.n, nb = s_nb, w = a.w, Lnew = L + nb;
    const int touched = min(nb, w);
    const T *knew = static_cast<const T *>(a.k_new);
    const T *vnew = static_cast<const T *>(a.v_new);
    T *wk = static_cast<T *>(a.win_k);
    T *wv = static_cast<T *>(a.win_v);
    T *pk = static_cast<T *>(a.pool_kd);
    T *pv = static_cast<T *>(a.pool_vd);

    for (int u = warp; u < a.Hkv * touched; u += nwarps) {
        const int g = u / touched;
        const int first = L + u % touched;  // first new position landing in this slot
        const int slot = first % w;
        const size_t ring = ((size_t)(b * a.Hkv + g) * w + slot) * kHeadDim;
        const float *Dk = a.Dk + (size_t)g * kHeadDim * DD;
        const float *Dv = a.Dv + (size_t)g * kHeadDim * DD;
        const int old = first - w;
        if (old >= 0) {  // the slot's occupant leaves the window
            T *rk = pool_row<T, DD>(a, pk, b, g, old);
            T *rv = pool_row<T, DD>(a, pv, b, g, old);
            if (rk)
                project_row_warp<T, DD>(wk + ring, Dk, rk, lane);
            if (rv)
                project_row_warp<T, DD>(wv + ring, Dv, rv, lane);
        }
        __syncwarp();
        for (int p = first; p < Lnew; p += w) {
            const size_t src = ((size_t)(b * a.Hkv + g) * n + (p - L)) * kHeadDim;
            if (p + w < Lnew) {  // leaves the window within this call
                T *rk = pool_row<T, DD>(a, pk, b, g, p);
                T *rv = pool_row<T, DD>(a, pv, b, g, p);
                if (rk)
                    project_row_warp<T, DD>(knew + src, Dk, rk, lane);
                if (rv)
                    project_row_warp<T, DD>(vnew + src, Dv, rv, lane);
            } else {
                copy_row_warp(knew + src, wk + ring, lane);
                copy_row_warp(vnew + src, wv + ring, lane);
            }
            __syncwarp();
        }
    }
    __syncthreads();
    if (threadIdx.x == 0)
        a.seq_lens[b] = Lnew;
}

// ----------------------------------------------------------------- launchers

template <typename T>
static cudaError_t down_project_t(int dd, const void *x, const float *W, void *out, int B,
                                  int Hkv, int n, int os, cudaStream_t s)
{
    dim3 grid((n + 127) / 128, B * Hkv);
    const T *xi = static_cast<const T *>(x);
    T *o = static_cast<T *>(out);
    switch (dd) {
    case 8: down_project_kernel<T, 8><<<grid, 128, 0, s>>>(xi, W, o, Hkv, n, os); break;
    case 16: down_project_kernel<T, 16><<<grid, 128, 0, s>>>(xi, W, o, Hkv, n, os); break;
    case 32: down_project_kernel<T, 32><<<grid, 128, 0, s>>>(xi, W, o, Hkv, n, os); break;
    case 64: down_project_kernel<T, 64><<<grid, 128, 0, s>>>(xi, W, o, Hkv, n, os); break;
    default: return cudaErrorInvalidValue;
    }
    return cudaGetLastError();
}

cudaError_t launch_down_project(dar_dtype dt, int dd, const void *x, const float *W, void *out,
                                int B, int Hkv, int n, int ostride, cudaStream_t s)
{
    if (n == 0 || B == 0)
        return cudaSuccess;
    return dt == DAR_F32 ? down_project_t<float>(dd, x, W, out, B, Hkv, n, ostride, s)
                         : down_project_t<bf16>(dd, x, W, out, B, Hkv, n, ostride, s);
}

template <typename T>
static cudaError_t cache_append_t(int dd, const AppendArgs &a, cudaStream_t s)
{
    // one warp per (KV head, touched slot) unit, up to 32 warps per sequence
    const long long units = (long long)a.Hkv * (a.n < a.w ? a.n : a.w);
    const int threads = 32 * (int)(units < 1 ? 1 : units > 32 ? 32 : units);
    switch (dd) {
    case 8: cache_append_kernel<T, 8><<<a.B, threads, 0, s>>>(a); break;
    case 16: cache_append_kernel<T, 16><<<a.B, threads, 0, s>>>(a); break;
    case 32: cache_append_kernel<T, 32><<<a.B, threads, 0, s>>>(a); break;
    case 64: cache_append_kernel<T, 64><<<a.B, threads, 0, s>>>(a); break;
    default: return cudaErrorInvalidValue;
    }
    return cudaGetLastError();
}

cudaError_t launch_cache_append(dar_dtype dt, int dd, const AppendArgs &a, cudaStream_t s)
{
    if (a.B == 0)
        return cudaSuccess;
    return dt == DAR_F32 ? cache_append_t<float>(dd, a, s) : cache_append_t<bf16>(dd, a, s);
}

}  // namespace dar
