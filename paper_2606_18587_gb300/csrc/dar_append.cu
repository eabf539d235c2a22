// dar_append.cu -- Eq. 1 (bottleneck down-projection) as a bulk kernel and as
// the window-exit migration of the mixed-dimension cache.
//
// Every bottleneck element is ONE fp32 fused-multiply-add chain over
// t = 0..63 starting from +0.0f, rounded once to the storage type, so a
// token's cached vector is bit-identical whichever kernel produced it.
#include "dar_common.cuh"
#include "dar_launch.h"
#include "dar_sm100.cuh"

namespace dar {

// ---------------------------------------------------------------- bulk Eq. 1
//
// A block stages kStageBytesBulk of contiguous token rows in shared memory
// with coalesced 16-byte loads (chunk c of row r stored at chunk c ^ (r & 7),
// so a warp reading one chunk of 32 different rows touches every bank group
// once); then each thread runs the chains of RPT rows at once, so that every
// W[t][c] read from shared memory feeds RPT rows.  Two chains advance per
// instruction (fma.rn.f32x2: outputs c and c + 1 share x_t); each element is
// still the exact fp32 chain acc = fma(x_t, W[t][c], acc), t = 0..63.
// blockIdx.z selects the tensor: 0 = (x0, W0, out0), 1 = (x1, W1, out1).
constexpr int kStageBytesBulk = 32 << 10;

template <typename T>
__host__ __device__ constexpr int rows_bulk()
{
    return kStageBytesBulk / (kHeadDim * (int)sizeof(T));
}
template <int DD>
__host__ __device__ constexpr int rows_per_thread()
{
    return DD <= 16 ? 4 : DD == 32 ? 2 : 1;
}
template <typename T, int DD>
__host__ __device__ constexpr int threads_bulk()
{
    return rows_bulk<T>() / rows_per_thread<DD>();
}

struct BulkArgs {
    const void *x[2];
    const float *W[2];
    void *out[2];
    int Hkv, n;
    int ostride[2];   // output row stride of each tensor (columns dd.. are padding)
    int ones_col[2];  // first of 16 padding columns set to 1 (-1: all padding is 0)
};

template <typename T, int DD>
__global__ void __launch_bounds__(threads_bulk<T, DD>()) down_project_kernel(BulkArgs a)
{
    constexpr int R = rows_bulk<T>();
    constexpr int RPT = rows_per_thread<DD>();
    constexpr int NT = threads_bulk<T, DD>();
    constexpr int E = Granule<T>::kElems;
    constexpr int CPR = kHeadDim / E;  // 16-byte chunks per row (8 for bf16, 16 for fp32)
    __shared__ __align__(16) unsigned char rows[kStageBytesBulk];
    __shared__ __align__(16) float Ws[kHeadDim * DD];
    const bool z = blockIdx.z != 0;  // (selects, not indexes: the arguments stay in parameter space)
    const T *x = static_cast<const T *>(z ? a.x[1] : a.x[0]);
    const int bg = blockIdx.y, g = bg % a.Hkv;
    const int j0 = blockIdx.x * R;
    const int nr = min(R, a.n - j0);
    const float *W = (z ? a.W[1] : a.W[0]) + (size_t)g * kHeadDim * DD;
    for (int i = threadIdx.x; i < kHeadDim * DD / 4; i += NT)
        reinterpret_cast<float4 *>(Ws)[i] = __ldg(reinterpret_cast<const float4 *>(W) + i);
    const uint4 *src = reinterpret_cast<const uint4 *>(x + ((size_t)bg * a.n + j0) * kHeadDim);
    for (int i = threadIdx.x; i < nr * CPR; i += NT) {
        const int r = i / CPR, c = i % CPR;
        reinterpret_cast<uint4 *>(rows)[r * CPR + (c ^ (r & 7))] = ld_stream_v4(src + i);
    }
    __syncthreads();
    // this thread's rows: threadIdx.x + k * NT, k < RPT (rows past nr compute on
    // stale staging bytes and are not stored)
    float acc[RPT][DD];
#pragma unroll
    for (int k = 0; k < RPT; ++k)
#pragma unroll
        for (int c = 0; c < DD; ++c)
            acc[k][c] = 0.0f;
#pragma unroll 1
    for (int q = 0; q < CPR; ++q) {
        float xf[RPT][E];
#pragma unroll
        for (int k = 0; k < RPT; ++k) {
            const int r = threadIdx.x + k * NT;
            unpack(reinterpret_cast<const uint4 *>(rows)[r * CPR + (q ^ (r & 7))], xf[k], T());
        }
#pragma unroll
        for (int e = 0; e < E; ++e) {
            const int t = q * E + e;
#pragma unroll
            for (int c = 0; c < DD; c += 4) {
                const float4 w4 = *reinterpret_cast<const float4 *>(Ws + t * DD + c);
#pragma unroll
                for (int k = 0; k < RPT; ++k) {
                    sm100::ffma2(acc[k][c], acc[k][c + 1], xf[k][e], xf[k][e], w4.x, w4.y, acc[k][c], acc[k][c + 1]);
                    sm100::ffma2(acc[k][c + 2], acc[k][c + 3], xf[k][e], xf[k][e], w4.z, w4.w, acc[k][c + 2],
                                 acc[k][c + 3]);
                }
            }
        }
    }
    const int ostride = z ? a.ostride[1] : a.ostride[0];
    const int ones_col = z ? a.ones_col[1] : a.ones_col[0];
#pragma unroll
    for (int k = 0; k < RPT; ++k) {
        const int r = threadIdx.x + k * NT;
        if (r >= nr)
            continue;
        T *o = static_cast<T *>(z ? a.out[1] : a.out[0]) + ((size_t)bg * a.n + j0 + r) * ostride;
        if (ostride == DD && (DD * sizeof(T)) % 16 == 0) {
            constexpr int OE = 16 / sizeof(T);
#pragma unroll
            for (int c = 0; c < DD; c += OE) {
                uint32_t u[4];
                if constexpr (sizeof(T) == 2) {
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        __nv_bfloat162 v = __floats2bfloat162_rn(acc[k][c + 2 * i], acc[k][c + 2 * i + 1]);
                        u[i] = *reinterpret_cast<uint32_t *>(&v);
                    }
                } else {
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        u[i] = __float_as_uint(acc[k][c + i]);
                }
                *reinterpret_cast<uint4 *>(o + c) = make_uint4(u[0], u[1], u[2], u[3]);
            }
        } else if ((ostride * sizeof(T)) % 16 == 0 && ostride <= kHeadDim) {
            // padded rows (values, then zeros or a block of 16 ones), 16 bytes at a time
            constexpr int OE = 16 / sizeof(T);
#pragma unroll
            for (int c0 = 0; c0 < kHeadDim; c0 += OE) {
                if (c0 >= ostride)
                    break;
                float v[OE];
#pragma unroll
                for (int e = 0; e < OE; ++e) {
                    const int c = c0 + e;
                    v[e] = c < DD ? acc[k][c < DD ? c : 0]
                                  : (ones_col >= 0 && c >= ones_col && c < ones_col + 16 ? 1.f : 0.f);
                }
                uint32_t u[4];
                if constexpr (sizeof(T) == 2) {
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        __nv_bfloat162 b2 = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]);
                        u[i] = *reinterpret_cast<uint32_t *>(&b2);
                    }
                } else {
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        u[i] = __float_as_uint(v[i]);
                }
                *reinterpret_cast<uint4 *>(o + c0) = make_uint4(u[0], u[1], u[2], u[3]);
            }
        } else {
#pragma unroll
            for (int c = 0; c < DD; ++c)
                o[c] = from_f32<T>(acc[k][c]);
            for (int c = DD; c < ostride; ++c)
                o[c] = from_f32<T>(c >= ones_col && c < ones_col + 16 && ones_col >= 0 ? 1.f : 0.f);
        }
    }
}

// ------------------------------------------------------------ cache append
//
// One CTA per sequence (so its length can be updated at the end).  Thread ch
// owns the Eq. 1 chains (kv, g, c) -- output c of KV head g of the keys
// (kv = 0) or values (kv = 1) -- and keeps that column of W in registers.
// Positions that leave the window in this call are staged up to kAppRows at a
// time in shared memory (from the ring for old occupants, from k_new/v_new for
// new tokens that leave at once); every chain thread runs its fixed-order
// chains over the staged rows and writes the pages.  After all ring reads, the
// new tokens that stay in the window are copied into their ring slots, then
// the length is updated.  Loads that do not depend on the length (W columns,
// the last new rows) are issued at entry, so a one-token step costs about two
// round trips to memory.
constexpr int kAppThreads = 512;
constexpr int kAppRows = 8;  // rows staged per round (fewer for many heads)
constexpr int kAppStageBytes = 96 << 10;

template <typename T>
__host__ __device__ inline int app_rows(int Hkv)
{
    const int per_row = 2 * Hkv * kHeadDim * (int)sizeof(T);
    const int r = kAppStageBytes / per_row;
    return r < 1 ? 1 : r > kAppRows ? kAppRows : r;
}

template <typename T, int DD>
__global__ void __launch_bounds__(kAppThreads) cache_append_kernel(AppendArgs a)
{
    constexpr int E = Granule<T>::kElems;
    constexpr int GPR = kHeadDim / E;  // 16-byte granules per 64-element row
    extern __shared__ __align__(16) unsigned char app_smem[];
    T *s_x = reinterpret_cast<T *>(app_smem);  // [rows][kv][Hkv][64]
    __shared__ int s_L, s_nb, s_ok;
    __shared__ int s_pid[kAppRows];  // page of each staged row (-1: invalid)

    // a decode launched after this kernel may start its query-only work now
    sm100::grid_dep_launch();
    const int b = blockIdx.x, tid = threadIdx.x;
    const int Hkv = a.Hkv, n = a.n, w = a.w;
    const int nchains = 2 * Hkv * DD;
    const int R = app_rows<T>(Hkv);
    const T *knew = static_cast<const T *>(a.k_new);
    const T *vnew = static_cast<const T *>(a.v_new);
    T *wk = static_cast<T *>(a.win_k);
    T *wv = static_cast<T *>(a.win_v);
    T *pk = static_cast<T *>(a.pool_kd);
    T *pv = static_cast<T *>(a.pool_vd);

    // ---- issued at entry: the length, this thread's first W column and one
    // granule of the last min(n, w) new rows (those land in the ring when the
    // sequence appends all n)
    if (tid == 0) {
        s_L = a.seq_lens[b];
        s_nb = a.n_per_seq ? a.n_per_seq[b] : n;
    }
    float wc[kHeadDim];
    auto load_w = [&](int ch) {
        const int kv = ch / (Hkv * DD), g = (ch / DD) % Hkv, c = ch % DD;
        const float *W = (kv ? a.Dv : a.Dk) + (size_t)g * kHeadDim * DD + c;
#pragma unroll
        for (int t = 0; t < kHeadDim; ++t)
            wc[t] = __ldg(W + (size_t)t * DD);
    };
    if (tid < nchains)
        load_w(tid);
    // granule i of the rows j0, j0 + 1, ... of k_new / v_new (i runs over
    // [row][kv][g][granule])
    auto new_granule = [&](int i, int j0) {
        const int q = i % GPR, rest = i / GPR;
        const int g = rest % Hkv, kv = (rest / Hkv) & 1, j = j0 + rest / (2 * Hkv);
        return (kv ? vnew : knew) + (((size_t)b * Hkv + g) * n + j) * kHeadDim + q * E;
    };
    const int pre_rows = min(n, w);
    uint4 pre = make_uint4(0u, 0u, 0u, 0u);
    if (tid < 2 * Hkv * pre_rows * GPR)
        pre = *reinterpret_cast<const uint4 *>(new_granule(tid, n - pre_rows));
    __syncthreads();
    if (tid == 0) {
        const int L = s_L, nb = s_nb;
        const long long Lnew = (long long)L + nb;
        int ok = 1;
        if (L < 0 || nb < 0 || nb > n) {
            report(a.status, DAR_ERR_INVALID_ARG);
            ok = 0;
        } else if (Lnew - w > (long long)a.maxp * kPage || Lnew > 0x7fffffffLL) {
            report(a.status, DAR_ERR_CAPACITY);
            ok = 0;
        }
        s_ok = ok;
    }
    __syncthreads();
    if (!s_ok || s_nb == 0)
        return;
    const int L = s_L, nb = s_nb, Lnew = L + nb;

    // ---- positions leaving the window: [p_lo, p_hi)
    const int p_lo = max(0, L - w), p_hi = max(0, Lnew - w);
    for (int m0 = p_lo; m0 < p_hi; m0 += R) {
        const int nr = min(R, p_hi - m0);
        for (int i = tid; i < nr * 2 * Hkv * GPR; i += blockDim.x) {  // stage [row][kv][g][64]
            const int q = i % GPR, rest = i / GPR;
            const int g = rest % Hkv, kv = (rest / Hkv) & 1, r = rest / (2 * Hkv);
            const int p = m0 + r;
            const T *src = p < L ? (kv ? wv : wk) + (((size_t)b * Hkv + g) * w + p % w) * kHeadDim
                                 : (kv ? vnew : knew) + (((size_t)b * Hkv + g) * n + (p - L)) * kHeadDim;
            reinterpret_cast<uint4 *>(s_x)[i] = *reinterpret_cast<const uint4 *>(src + q * E);
        }
        if (tid < nr) {
            const int lp = (m0 + tid) / kPage;
            const int id = lp < a.maxp ? a.block_table[(size_t)b * a.maxp + lp] : -1;
            const bool valid = id >= 0 && id < a.num_pages;
            if (!valid)
                report(a.status, DAR_ERR_CAPACITY);
            s_pid[tid] = valid ? id : -1;
        }
        __syncthreads();
        for (int ch0 = 0; ch0 < nchains; ch0 += blockDim.x) {
            const int ch = ch0 + tid;
            if (ch >= nchains)
                break;
            if (ch0 > 0)
                load_w(ch);
            const int kv = ch / (Hkv * DD), g = (ch / DD) % Hkv, c = ch % DD;
            T *pool = kv ? pv : pk;
            for (int r = 0; r < nr; ++r) {
                const uint4 *x4 = reinterpret_cast<const uint4 *>(s_x + ((size_t)(r * 2 + kv) * Hkv + g) * kHeadDim);
                float acc = 0.0f;  // Eq. 1: one fp32 FMA chain over t = 0..63
#pragma unroll
                for (int q = 0; q < GPR; ++q) {
                    float xf[E];
                    unpack(x4[q], xf, T());
#pragma unroll
                    for (int e = 0; e < E; ++e)
                        acc = __fmaf_rn(xf[e], wc[q * E + e], acc);
                }
                const int id = s_pid[r], p = m0 + r;
                if (id >= 0)
                    pool[(((size_t)id * Hkv + g) * kPage + p % kPage) * DD + c] = from_f32<T>(acc);
            }
        }
        // the first chain group's W columns are needed again in the next round
        if (nchains > (int)blockDim.x && m0 + R < p_hi && tid < nchains)
            load_w(tid);
        __syncthreads();
    }

    // ---- new tokens that stay in the window: rows j_lo .. nb-1 (positions
    // L + j); every ring read above is complete
    const int j_lo = max(0, nb - w);
    const int granules = 2 * Hkv * (nb - j_lo) * GPR;
    const bool use_pre = nb == n;  // then the prefetched granules are exactly these
    for (int i = tid; i < granules; i += blockDim.x) {
        const int q = i % GPR, rest = i / GPR;
        const int g = rest % Hkv, kv = (rest / Hkv) & 1, j = j_lo + rest / (2 * Hkv);
        const uint4 v = (use_pre && i == tid) ? pre : *reinterpret_cast<const uint4 *>(new_granule(i, j_lo));
        T *dst = (kv ? wv : wk) + (((size_t)b * Hkv + g) * w + (L + j) % w) * kHeadDim + q * E;
        *reinterpret_cast<uint4 *>(dst) = v;
    }
    __syncthreads();
    if (tid == 0)
        a.seq_lens[b] = Lnew;
}

// ----------------------------------------------------------------- launchers

template <typename T>
static cudaError_t down_project_t(int dd, const BulkArgs &a, int B, int nz, cudaStream_t s)
{
    constexpr int R = rows_bulk<T>();
    dim3 grid((a.n + R - 1) / R, B * a.Hkv, nz);
    switch (dd) {
    case 8: down_project_kernel<T, 8><<<grid, threads_bulk<T, 8>(), 0, s>>>(a); break;
    case 16: down_project_kernel<T, 16><<<grid, threads_bulk<T, 16>(), 0, s>>>(a); break;
    case 32: down_project_kernel<T, 32><<<grid, threads_bulk<T, 32>(), 0, s>>>(a); break;
    case 64: down_project_kernel<T, 64><<<grid, threads_bulk<T, 64>(), 0, s>>>(a); break;
    default: return cudaErrorInvalidValue;
    }
    return cudaGetLastError();
}

static cudaError_t down_project_any(dar_dtype dt, int dd, const BulkArgs &a, int B, int nz, cudaStream_t s)
{
    if (a.n == 0 || B == 0)
        return cudaSuccess;
    return dt == DAR_F32 ? down_project_t<float>(dd, a, B, nz, s) : down_project_t<bf16>(dd, a, B, nz, s);
}

cudaError_t launch_down_project(dar_dtype dt, int dd, const void *x, const float *W, void *out,
                                int B, int Hkv, int n, int ostride, cudaStream_t s)
{
    BulkArgs a = {{x, x}, {W, W}, {out, out}, Hkv, n, {ostride, ostride}, {-1, -1}};
    return down_project_any(dt, dd, a, B, 1, s);
}

cudaError_t launch_down_project_kv(dar_dtype dt, int dd, const void *k, const void *v, const float *Dk,
                                   const float *Dv, void *kd, void *vd, int B, int Hkv, int n, int kstride,
                                   int vstride, int v_ones_col, cudaStream_t s)
{
    BulkArgs a = {{k, v}, {Dk, Dv}, {kd, vd}, Hkv, n, {kstride, vstride}, {-1, v_ones_col}};
    return down_project_any(dt, dd, a, B, 2, s);
}

template <typename T>
static cudaError_t cache_append_t(int dd, const AppendArgs &a, cudaStream_t s)
{
    const size_t smem = (size_t)app_rows<T>(a.Hkv) * 2 * a.Hkv * kHeadDim * sizeof(T);
    static PerDeviceOnce once;  // opt-in to more than 48 KB of shared memory, once per device
    const cudaError_t e = per_device_once(once, [](int) {
        for (auto k : {cache_append_kernel<T, 8>, cache_append_kernel<T, 16>, cache_append_kernel<T, 32>,
                       cache_append_kernel<T, 64>}) {
            const cudaError_t e2 = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, kAppStageBytes);
            if (e2 != cudaSuccess)
                return e2;
        }
        return cudaSuccess;
    });
    if (e != cudaSuccess)
        return e;
    switch (dd) {
    case 8: cache_append_kernel<T, 8><<<a.B, kAppThreads, smem, s>>>(a); break;
    case 16: cache_append_kernel<T, 16><<<a.B, kAppThreads, smem, s>>>(a); break;
    case 32: cache_append_kernel<T, 32><<<a.B, kAppThreads, smem, s>>>(a); break;
    case 64: cache_append_kernel<T, 64><<<a.B, kAppThreads, smem, s>>>(a); break;
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
