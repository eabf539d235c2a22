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
                                                           T *__restrict__ out, int Hkv, int n)
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
    T *o = out + ((size_t)bg * n + j) * DD;
#pragma unroll
    for (int c = 0; c < DD; ++c)
        o[c] = from_f32<T>(acc[c]);
}

// ------------------------------------------------------------ cache append

// Eq. 1 for one row, computed by a warp: lane c (and c + 32) owns output c.
template <typename T, int DD>
__device__ __forceinline__ void project_row_warp(const T *x, const float *W, T *out, int lane)
{
    constexpr int CPL = (DD + 31) / 32;
    float acc[CPL];
#pragma unroll
    for (int i = 0; i < CPL; ++i)
        acc[i] = 0.0f;
#pragma unroll 8
    for (int t = 0; t < kHeadDim; ++t) {
        const float xv = to_f32(x[t]);
#pragma unroll
        for (int i = 0; i < CPL; ++i) {
            const int c = lane + 32 * i;
            if (c < DD)
                acc[i] = __fmaf_rn(xv, W[t * DD + c], acc[i]);
        }
    }
#pragma unroll
    for (int i = 0; i < CPL; ++i) {
        const int c = lane + 32 * i;
        if (c < DD)
            out[c] = from_f32<T>(acc[i]);
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
// 256 threads.  Sequence b appends nb = n_per_seq[b] (or n) tokens; k_new
// rows are strided by n.  Work unit = (KV head g, slot touched by this call): the slot's
// old occupant migrates to its page, then the new positions of that slot are
// processed in order (all but the last migrate straight from k_new; the last
// is written into the ring).
template <typename T, int DD>
__global__ void __launch_bounds__(256) cache_append_kernel(AppendArgs a)
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
                wk[ring + lane] = knew[src + lane];
                wk[ring + lane + 32] = knew[src + lane + 32];
                wv[ring + lane] = vnew[src + lane];
                wv[ring + lane + 32] = vnew[src + lane + 32];
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
                                  int Hkv, int n, cudaStream_t s)
{
    dim3 grid((n + 127) / 128, B * Hkv);
    const T *xi = static_cast<const T *>(x);
    T *o = static_cast<T *>(out);
    switch (dd) {
    case 8: down_project_kernel<T, 8><<<grid, 128, 0, s>>>(xi, W, o, Hkv, n); break;
    case 16: down_project_kernel<T, 16><<<grid, 128, 0, s>>>(xi, W, o, Hkv, n); break;
    case 32: down_project_kernel<T, 32><<<grid, 128, 0, s>>>(xi, W, o, Hkv, n); break;
    case 64: down_project_kernel<T, 64><<<grid, 128, 0, s>>>(xi, W, o, Hkv, n); break;
    default: return cudaErrorInvalidValue;
    }
    return cudaGetLastError();
}

cudaError_t launch_down_project(dar_dtype dt, int dd, const void *x, const float *W, void *out,
                                int B, int Hkv, int n, cudaStream_t s)
{
    if (n == 0 || B == 0)
        return cudaSuccess;
    return dt == DAR_F32 ? down_project_t<float>(dd, x, W, out, B, Hkv, n, s)
                         : down_project_t<bf16>(dd, x, W, out, B, Hkv, n, s);
}

template <typename T>
static cudaError_t cache_append_t(int dd, const AppendArgs &a, cudaStream_t s)
{
    switch (dd) {
    case 8: cache_append_kernel<T, 8><<<a.B, 256, 0, s>>>(a); break;
    case 16: cache_append_kernel<T, 16><<<a.B, 256, 0, s>>>(a); break;
    case 32: cache_append_kernel<T, 32><<<a.B, 256, 0, s>>>(a); break;
    case 64: cache_append_kernel<T, 64><<<a.B, 256, 0, s>>>(a); break;
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
