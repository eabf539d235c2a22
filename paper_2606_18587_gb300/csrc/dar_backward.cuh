// dar_backward.cuh -- gradients of the causal DAR attention forward (the
// training mode of Sec. 2.3: backpropagation reaches W_down and W_up through
// every position that attends to a token via the global path).
//
// Forward being differentiated (per query head h, KV head g, row i, j <= i):
//   s_ij = scale * q_i . k_j            (local, i - j < w; Eq. 3)
//   s_ij = scale * q~_i . k^D_j         (global; q~ = q Uk^T absorbs Eq. 2)
//   p_i = softmax_j(s_ij)               (one softmax over both, Eq. 4)
//   o_i = sum_local p_ij v_j + (sum_global p_ij v^D_j) Uv
// with k^D = k Dk, v^D = v Dv (Eq. 1, stored rounded to T; the rounding is
// not differentiated).  With dO the output gradient, D_i = dO_i . o_i and
// dO~_i = dO_i Uv^T:
//   dP_ij = dO_i . v_j  |  dO~_i . v^D_j ;   dS_ij = p_ij (dP_ij - D_i)
//   dq_i  = scale (sum_local dS_ij k_j + (sum_global dS_ij k^D_j) Uk)
//   dk_j  = scale sum_local dS_ij q_i + dk^D_j Dk^T,  dk^D_j = scale sum_global dS_ij q~_i
//   dv_j  = sum_local p_ij dO_i + dv^D_j Dv^T,        dv^D_j = sum_global p_ij dO~_i
//   dDk = sum_j k_j^T dk^D_j, dDv = sum_j v_j^T dv^D_j,
//   dUk = sum_i dq~_i^T q_i (dq~_i = scale sum_global dS_ij k^D_j),
//   dUv = sum_i O^D_i^T dO_i (O^D_i = sum_global p_ij v^D_j).
//
// Kernels (fp32 arithmetic on the CUDA cores; used for fp32 storage and for
// bf16 with d_down = 8 -- other bf16 shapes run steps 2 and 3 on the tensor
// cores, dar_backward_tc.cu, and share steps 1 and 4):
//  1. bwd_rows: per row, q~, dO~ and D (one warp per row, Uk and Uv staged
//     in shared memory per KV head).
//  2. bwd_dq: per 64-row query tile, the row log-sum-exp (first pass over the
//     keys) and then dq, dq~ and O^D (second pass).
//  3. bwd_dkv: per 64-key tile of a KV head, over the query heads of the
//     group and the query tiles that see it: dk, dv, dk^D, dv^D.
//  4. bwd_wpart / bwd_wsum: the four projection gradients as sums of outer
//     products, in fixed row chunks and then summed in chunk order (the
//     result does not depend on scheduling).
#pragma once

#include "dar_common.cuh"
#include "dar_launch.h"

namespace dar {
namespace bwd {

constexpr int kRows = 64, kKeys = 64, kLd = 65, kThreads = 256;
constexpr int kChunks = 64;  // row chunks of the projection gradients
constexpr float kLog2e = 1.4426950408889634f;

struct Args {
    const void *q, *k, *v, *out, *dout;  // [B][Hq|Hkv][N][64] T
    const void *kd, *vd;                 // [B][Hkv][N][DD] T (Eq. 1, as stored)
    const float *Dk, *Uk, *Dv, *Uv;
    void *dq, *dk, *dv;                  // T
    float *dDk, *dUk, *dDv, *dUv;        // [Hkv][64][DD], [Hkv][DD][64]
    float *qt, *dot;                     // [B][Hq][N][DD]: q~, dO~
    float *drow, *lse;                   // [B][Hq][N]: D, log2-sum-exp2 of the scaled scores
    float *dqt, *od;                     // [B][Hq][N][DD]: dq~ (scaled), O^D
    float *dkd, *dvd;                    // [B][Hkv][N][DD]: dk^D (scaled), dv^D
    bf16 *qtb, *dotb;                    // [B][Hq][N][DD]: q~, dO~ rounded to bf16 (tensor-core operands)
    float *part;                         // [kChunks][4][Hkv][64 * DD]
    int B, Hq, Hkv, G, N, w;
    float scale, c2;                     // scale, scale * log2(e)
};

// ---------------------------------------------------------------- 1. rows

// Block (g, row range): Uk^g and Uv^g staged transposed ([t][c]) in shared
// memory; one warp per row of KV head g's query heads: D = dO . o by a warp
// reduction, q~ = q Uk^T and dO~ = dO Uv^T with lanes over c (the row's q and
// dO broadcast from shared memory).
template <typename T, int DD>
__global__ void __launch_bounds__(256) bwd_rows_kernel(Args a)
{
    __shared__ float ukt[64 * DD], uvt[64 * DD];
    __shared__ float xs[8][2][64];
    const int g = blockIdx.x, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int i = threadIdx.x; i < DD * 64; i += blockDim.x) {
        const int c = i / 64, t = i % 64;
        ukt[t * DD + c] = a.Uk[((size_t)g * DD + c) * kHeadDim + t];
        uvt[t * DD + c] = a.Uv[((size_t)g * DD + c) * kHeadDim + t];
    }
    __syncthreads();
    const long nrows = (long)a.B * a.G * a.N;  // rows of KV head g's query heads
    for (long r = (long)blockIdx.y * 8 + warp; r < nrows; r += (long)gridDim.y * 8) {
        const long bq = r / a.N;
        const int i = (int)(r % a.N), b = (int)(bq / a.G), hh = (int)(bq % a.G);
        const long row = ((long)b * a.Hq + g * a.G + hh) * a.N + i;
        const T *qr = static_cast<const T *>(a.q) + row * kHeadDim;
        const T *dr = static_cast<const T *>(a.dout) + row * kHeadDim;
        const T *orow = static_cast<const T *>(a.out) + row * kHeadDim;
        const float q0 = to_f32(qr[lane]), q1 = to_f32(qr[lane + 32]);
        const float d0 = to_f32(dr[lane]), d1 = to_f32(dr[lane + 32]);
        float D = d0 * to_f32(orow[lane]) + d1 * to_f32(orow[lane + 32]);
#pragma unroll
        for (int o = 16; o; o >>= 1)
            D += __shfl_xor_sync(0xffffffffu, D, o);
        if (lane == 0)
            a.drow[row] = D;
        xs[warp][0][lane] = q0;
        xs[warp][0][lane + 32] = q1;
        xs[warp][1][lane] = d0;
        xs[warp][1][lane + 32] = d1;
        __syncwarp();
        for (int c = lane; c < DD; c += 32) {
            float sq = 0.f, sd = 0.f;
#pragma unroll 16
            for (int t = 0; t < kHeadDim; ++t) {
                sq = fmaf(xs[warp][0][t], ukt[t * DD + c], sq);
                sd = fmaf(xs[warp][1][t], uvt[t * DD + c], sd);
            }
            a.qt[row * DD + c] = sq;
            a.dot[row * DD + c] = sd;
            if (a.qtb) {
                a.qtb[row * DD + c] = __float2bfloat16_rn(sq);
                a.dotb[row * DD + c] = __float2bfloat16_rn(sd);
            }
        }
        __syncwarp();
    }
}

// Grid of the row kernel: one column of blocks per KV head.
inline dim3 rows_grid(const Args &a)
{
    const long per_g = (long)a.B * a.G * a.N;
    const long by = (per_g + 7) / 8, cap = 2432 / a.Hkv > 0 ? 2432 / a.Hkv : 1;
    return dim3(a.Hkv, (unsigned)(by < cap ? by : cap));
}

// Shared helpers for the two attention kernels.
template <typename T>
__device__ __forceinline__ void load_rows64(float *dst, const T *src, int n_valid, int tid)
{
    for (int idx = tid; idx < 64 * kHeadDim; idx += kThreads) {
        const int r = idx / kHeadDim, t = idx % kHeadDim;
        dst[r * kLd + t] = r < n_valid ? to_f32(src[(size_t)r * kHeadDim + t]) : 0.f;
    }
}
template <typename T, int DD>
__device__ __forceinline__ void load_rows_dd(float *dst, const T *src, int n_valid, int tid)
{
    for (int idx = tid; idx < 64 * DD; idx += kThreads) {
        const int r = idx / DD, c = idx % DD;
        dst[r * (DD + 1) + c] = r < n_valid ? to_f32(src[(size_t)r * DD + c]) : 0.f;
    }
}

template <int DD>
constexpr size_t dq_smem_floats()
{
    return 7 * 64 * kLd + 4 * 64 * (DD + 1) + 64;
}

// ---------------------------------------------------------------- 2. dq

template <typename T, int DD>
__global__ void __launch_bounds__(kThreads) bwd_dq_kernel(Args a)
{
    constexpr int LDD = DD + 1, OG = DD / 4;
    extern __shared__ float sm[];
    float *Qs = sm;                    // [64][65] q
    float *dOs = Qs + 64 * kLd;        // [64][65] dO
    float *Ks = dOs + 64 * kLd;        // [64][65]
    float *Vs = Ks + 64 * kLd;         // [64][65]
    float *S1 = Vs + 64 * kLd;         // [row][key] dS of local pairs
    float *S2 = S1 + 64 * kLd;         // dS of global pairs
    float *S3 = S2 + 64 * kLd;         // p of global pairs
    float *Qt = S3 + 64 * kLd;         // [64][DD+1] q~
    float *dOt = Qt + 64 * LDD;        // dO~
    float *KDs = dOt + 64 * LDD;
    float *VDs = KDs + 64 * LDD;

    const int N = a.N, w = a.w;
    const int bh = blockIdx.y, b = bh / a.Hq, h = bh % a.Hq, g = h / a.G;
    const int i0 = blockIdx.x * kRows;
    const int tid = threadIdx.x, r = tid >> 2, qd = tid & 3;
    const int i = i0 + r;
    const int nv = min(kRows, N - i0);
    const size_t rowbase = ((size_t)b * a.Hq + h) * N + i0;
    const size_t kvbase = ((size_t)b * a.Hkv + g) * N;
    load_rows64(Qs, static_cast<const T *>(a.q) + rowbase * kHeadDim, nv, tid);
    load_rows64(dOs, static_cast<const T *>(a.dout) + rowbase * kHeadDim, nv, tid);
    for (int idx = tid; idx < 64 * DD; idx += kThreads) {
        const int rr = idx / DD, c = idx % DD;
        Qt[rr * LDD + c] = rr < nv ? a.qt[(rowbase + rr) * DD + c] : 0.f;
        dOt[rr * LDD + c] = rr < nv ? a.dot[(rowbase + rr) * DD + c] : 0.f;
    }
    const float Di = i < N ? a.drow[rowbase + r] : 0.f;
    const T *k = static_cast<const T *>(a.k) + kvbase * kHeadDim;
    const T *v = static_cast<const T *>(a.v) + kvbase * kHeadDim;
    const T *kd = static_cast<const T *>(a.kd) + kvbase * DD;
    const T *vd = static_cast<const T *>(a.vd) + kvbase * DD;
    const int imax = min(N, i0 + kRows) - 1;

    // scores of this thread's 16 keys of a tile (log2 units), -inf where masked
    auto scores = [&](int j0, bool all_global, bool all_local, float (&x)[16]) {
#pragma unroll
        for (int jj = 0; jj < 16; ++jj) {
            const int jl = qd + 4 * jj, j = j0 + jl;
            float val = -INFINITY;
            if (i < N && j <= i) {
                float acc = 0.f;
                if (i - j < w) {
#pragma unroll 8
                    for (int t = 0; t < kHeadDim; ++t)
                        acc = fmaf(Qs[r * kLd + t], Ks[jl * kLd + t], acc);
                } else {
#pragma unroll
                    for (int c = 0; c < DD; ++c)
                        acc = fmaf(Qt[r * LDD + c], KDs[jl * LDD + c], acc);
                }
                val = acc * a.c2;
            }
            x[jj] = val;
        }
    };
    auto load_keys = [&](int j0, bool all_global, bool all_local) {
        const int nk = min(kKeys, N - j0);
        if (!all_global) {
            load_rows64(Ks, k + (size_t)j0 * kHeadDim, nk, tid);
            load_rows64(Vs, v + (size_t)j0 * kHeadDim, nk, tid);
        }
        if (!all_local) {
            load_rows_dd<T, DD>(KDs, kd + (size_t)j0 * DD, nk, tid);
            load_rows_dd<T, DD>(VDs, vd + (size_t)j0 * DD, nk, tid);
        }
    };

    // pass 1: the row's log-sum-exp (log2 units)
    float m = -INFINITY, l = 0.f;
    for (int j0 = 0; j0 <= imax; j0 += kKeys) {
        const bool all_global = (i0 - (j0 + kKeys - 1)) >= w;
        const bool all_local = (i0 + kRows - 1 - j0) < w;
        __syncthreads();
        load_keys(j0, all_global, all_local);
        __syncthreads();
        float x[16];
        scores(j0, all_global, all_local, x);
        float mx = -INFINITY;
#pragma unroll
        for (int jj = 0; jj < 16; ++jj)
            mx = fmaxf(mx, x[jj]);
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
        const float mnew = fmaxf(m, mx);  // the same for the row's four threads
        float ps = 0.f;
#pragma unroll
        for (int jj = 0; jj < 16; ++jj)
            ps += x[jj] == -INFINITY ? 0.f : exp2f(x[jj] - mnew);
        ps += __shfl_xor_sync(0xffffffffu, ps, 1);
        ps += __shfl_xor_sync(0xffffffffu, ps, 2);
        if (mnew != -INFINITY) {  // rows that have seen no key yet keep m = -inf, l = 0
            l = (m == -INFINITY ? 0.f : l * exp2f(m - mnew)) + ps;
            m = mnew;
        }
    }
    const float lse = m + log2f(l);
    if (i < N && qd == 0)
        a.lse[rowbase + r] = lse;

    // pass 2: dS, then dq (local keys), dq~ and O^D (global keys)
    float acc_q[16], acc_t[OG], acc_o[OG];
#pragma unroll
    for (int e = 0; e < 16; ++e)
        acc_q[e] = 0.f;
#pragma unroll
    for (int e = 0; e < OG; ++e)
        acc_t[e] = acc_o[e] = 0.f;
    for (int j0 = 0; j0 <= imax; j0 += kKeys) {
        const bool all_global = (i0 - (j0 + kKeys - 1)) >= w;
        const bool all_local = (i0 + kRows - 1 - j0) < w;
        __syncthreads();
        load_keys(j0, all_global, all_local);
        __syncthreads();
        float x[16];
        scores(j0, all_global, all_local, x);
#pragma unroll
        for (int jj = 0; jj < 16; ++jj) {
            const int jl = qd + 4 * jj, j = j0 + jl;
            float ds = 0.f, p = 0.f;
            const bool loc = i - j < w;
            if (x[jj] != -INFINITY) {
                p = exp2f(x[jj] - lse);
                float dp = 0.f;
                if (loc) {
#pragma unroll 8
                    for (int t = 0; t < kHeadDim; ++t)
                        dp = fmaf(dOs[r * kLd + t], Vs[jl * kLd + t], dp);
                } else {
#pragma unroll
                    for (int c = 0; c < DD; ++c)
                        dp = fmaf(dOt[r * LDD + c], VDs[jl * LDD + c], dp);
                }
                ds = p * (dp - Di);
            }
            S1[r * kLd + jl] = loc ? ds : 0.f;
            S2[r * kLd + jl] = loc ? 0.f : ds;
            S3[r * kLd + jl] = loc ? 0.f : p;
        }
        __syncthreads();
        if (!all_global) {
            for (int jl = 0; jl < kKeys; ++jl) {
                const float ds = S1[r * kLd + jl];
#pragma unroll
                for (int e = 0; e < 16; ++e)
                    acc_q[e] = fmaf(ds, Ks[jl * kLd + qd * 16 + e], acc_q[e]);
            }
        }
        if (!all_local) {
            for (int jl = 0; jl < kKeys; ++jl) {
                const float ds = S2[r * kLd + jl], p = S3[r * kLd + jl];
#pragma unroll
                for (int e = 0; e < OG; ++e) {
                    acc_t[e] = fmaf(ds, KDs[jl * LDD + qd * OG + e], acc_t[e]);
                    acc_o[e] = fmaf(p, VDs[jl * LDD + qd * OG + e], acc_o[e]);
                }
            }
        }
    }

    // epilogue: dq = scale (dq_loc + dq~ Uk); keep dq~ (scaled) and O^D
    __syncthreads();
#pragma unroll
    for (int e = 0; e < OG; ++e)
        Qt[r * LDD + qd * OG + e] = acc_t[e] * a.scale;
    __syncthreads();
    if (i < N) {
        const float *Uk = a.Uk + (size_t)g * DD * kHeadDim;
        T *dq = static_cast<T *>(a.dq) + (rowbase + r) * kHeadDim;
#pragma unroll
        for (int e = 0; e < 16; ++e) {
            const int t = qd * 16 + e;
            float acc = acc_q[e] * a.scale;
            for (int c = 0; c < DD; ++c)
                acc = fmaf(Qt[r * LDD + c], Uk[c * kHeadDim + t], acc);
            dq[t] = from_f32<T>(acc);
        }
#pragma unroll
        for (int e = 0; e < OG; ++e) {
            a.dqt[(rowbase + r) * DD + qd * OG + e] = acc_t[e] * a.scale;
            a.od[(rowbase + r) * DD + qd * OG + e] = acc_o[e];
        }
    }
}

// ---------------------------------------------------------------- 3. dk, dv

template <int DD>
constexpr size_t dkv_smem_floats()
{
    return 8 * 64 * kLd + 4 * 64 * (DD + 1) + 2 * 64;
}

template <typename T, int DD>
__global__ void __launch_bounds__(kThreads) bwd_dkv_kernel(Args a)
{
    constexpr int LDD = DD + 1, OG = DD / 4;
    extern __shared__ float sm[];
    float *Ks = sm;                    // [64][65] this tile's keys
    float *Vs = Ks + 64 * kLd;
    float *Qs = Vs + 64 * kLd;         // [64][65] a query tile
    float *dOs = Qs + 64 * kLd;
    float *T1 = dOs + 64 * kLd;        // [key][row] dS local
    float *T2 = T1 + 64 * kLd;         // p local
    float *T3 = T2 + 64 * kLd;         // dS global
    float *T4 = T3 + 64 * kLd;         // p global
    float *KDs = T4 + 64 * kLd;        // [64][DD+1]
    float *VDs = KDs + 64 * LDD;
    float *Qt = VDs + 64 * LDD;
    float *dOt = Qt + 64 * LDD;
    float *sL = dOt + 64 * LDD;        // [64] lse of the query tile
    float *sD = sL + 64;               // [64] D of the query tile

    const int N = a.N, w = a.w;
    const int bg = blockIdx.y, b = bg / a.Hkv, g = bg % a.Hkv;
    const int j0 = blockIdx.x * kKeys;
    const int tid = threadIdx.x, jl = tid >> 2, qd = tid & 3;
    const int j = j0 + jl;
    const int nk = min(kKeys, N - j0);
    const size_t kvbase = ((size_t)b * a.Hkv + g) * N + j0;
    load_rows64(Ks, static_cast<const T *>(a.k) + kvbase * kHeadDim, nk, tid);
    load_rows64(Vs, static_cast<const T *>(a.v) + kvbase * kHeadDim, nk, tid);
    load_rows_dd<T, DD>(KDs, static_cast<const T *>(a.kd) + kvbase * DD, nk, tid);
    load_rows_dd<T, DD>(VDs, static_cast<const T *>(a.vd) + kvbase * DD, nk, tid);

    float dk[16], dv[16], dkd[OG], dvd[OG];
#pragma unroll
    for (int e = 0; e < 16; ++e)
        dk[e] = dv[e] = 0.f;
#pragma unroll
    for (int e = 0; e < OG; ++e)
        dkd[e] = dvd[e] = 0.f;

    for (int hh = 0; hh < a.G; ++hh) {
        const int h = g * a.G + hh;
        for (int i0 = j0 / kRows * kRows; i0 < N; i0 += kRows) {
            const bool all_global = (i0 - (j0 + kKeys - 1)) >= w;
            const bool all_local = (i0 + kRows - 1 - j0) < w;
            const int nv = min(kRows, N - i0);
            const size_t rowbase = ((size_t)b * a.Hq + h) * N + i0;
            __syncthreads();
            if (!all_global) {
                load_rows64(Qs, static_cast<const T *>(a.q) + rowbase * kHeadDim, nv, tid);
                load_rows64(dOs, static_cast<const T *>(a.dout) + rowbase * kHeadDim, nv, tid);
            }
            if (!all_local) {
                for (int idx = tid; idx < 64 * DD; idx += kThreads) {
                    const int rr = idx / DD, c = idx % DD;
                    Qt[rr * LDD + c] = rr < nv ? a.qt[(rowbase + rr) * DD + c] : 0.f;
                    dOt[rr * LDD + c] = rr < nv ? a.dot[(rowbase + rr) * DD + c] : 0.f;
                }
            }
            if (tid < 64) {
                sL[tid] = tid < nv ? a.lse[rowbase + tid] : 0.f;
                sD[tid] = tid < nv ? a.drow[rowbase + tid] : 0.f;
            }
            __syncthreads();
#pragma unroll 1
            for (int mm = 0; mm < 16; ++mm) {
                const int ii = qd + 4 * mm, i = i0 + ii;
                float ds = 0.f, p = 0.f;
                const bool loc = i - j < w;
                if (j < N && i < N && j <= i) {
                    float s = 0.f, dp = 0.f;
                    if (loc) {
#pragma unroll 8
                        for (int t = 0; t < kHeadDim; ++t) {
                            s = fmaf(Qs[ii * kLd + t], Ks[jl * kLd + t], s);
                            dp = fmaf(dOs[ii * kLd + t], Vs[jl * kLd + t], dp);
                        }
                    } else {
#pragma unroll
                        for (int c = 0; c < DD; ++c) {
                            s = fmaf(Qt[ii * LDD + c], KDs[jl * LDD + c], s);
                            dp = fmaf(dOt[ii * LDD + c], VDs[jl * LDD + c], dp);
                        }
                    }
                    p = exp2f(s * a.c2 - sL[ii]);
                    ds = p * (dp - sD[ii]);
                }
                T1[jl * kLd + ii] = loc ? ds : 0.f;
                T2[jl * kLd + ii] = loc ? p : 0.f;
                T3[jl * kLd + ii] = loc ? 0.f : ds;
                T4[jl * kLd + ii] = loc ? 0.f : p;
            }
            __syncthreads();
            if (!all_global) {
                for (int ii = 0; ii < kRows; ++ii) {
                    const float ds = T1[jl * kLd + ii], p = T2[jl * kLd + ii];
#pragma unroll
                    for (int e = 0; e < 16; ++e) {
                        dk[e] = fmaf(ds, Qs[ii * kLd + qd * 16 + e], dk[e]);
                        dv[e] = fmaf(p, dOs[ii * kLd + qd * 16 + e], dv[e]);
                    }
                }
            }
            if (!all_local) {
                for (int ii = 0; ii < kRows; ++ii) {
                    const float ds = T3[jl * kLd + ii], p = T4[jl * kLd + ii];
#pragma unroll
                    for (int e = 0; e < OG; ++e) {
                        dkd[e] = fmaf(ds, Qt[ii * LDD + qd * OG + e], dkd[e]);
                        dvd[e] = fmaf(p, dOt[ii * LDD + qd * OG + e], dvd[e]);
                    }
                }
            }
        }
    }

    // epilogue: dk = scale dk_loc + dk^D Dk^T, dv = dv_loc + dv^D Dv^T
    __syncthreads();
#pragma unroll
    for (int e = 0; e < OG; ++e) {
        Qt[jl * LDD + qd * OG + e] = dkd[e] * a.scale;
        dOt[jl * LDD + qd * OG + e] = dvd[e];
    }
    __syncthreads();
    if (j < N) {
        const float *Dk = a.Dk + (size_t)g * kHeadDim * DD, *Dv = a.Dv + (size_t)g * kHeadDim * DD;
        T *dkr = static_cast<T *>(a.dk) + (kvbase + jl) * kHeadDim;
        T *dvr = static_cast<T *>(a.dv) + (kvbase + jl) * kHeadDim;
#pragma unroll
        for (int e = 0; e < 16; ++e) {
            const int t = qd * 16 + e;
            float ak = dk[e] * a.scale, av = dv[e];
            for (int c = 0; c < DD; ++c) {
                ak = fmaf(Qt[jl * LDD + c], Dk[t * DD + c], ak);
                av = fmaf(dOt[jl * LDD + c], Dv[t * DD + c], av);
            }
            dkr[t] = from_f32<T>(ak);
            dvr[t] = from_f32<T>(av);
        }
#pragma unroll
        for (int e = 0; e < OG; ++e) {
            a.dkd[(kvbase + jl) * DD + qd * OG + e] = dkd[e] * a.scale;
            a.dvd[(kvbase + jl) * DD + qd * OG + e] = dvd[e];
        }
    }
}

// ---------------------------------------------------------------- 4. projection gradients

// part[chunk][which][g][t * DD + c] = sum over the chunk's rows of X[t] Y[c]:
//   which 0: X = k, Y = dk^D (rows of (b, g))      -> dDk
//         1: X = q, Y = dq~  (rows of (b, h in g)) -> dUk (transposed at the end)
//         2: X = v, Y = dv^D                       -> dDv
//         3: X = dO, Y = O^D                       -> dUv (transposed)
template <typename T, int DD>
__global__ void __launch_bounds__(kThreads) bwd_wpart_kernel(Args a)
{
    constexpr int PER = 64 * DD / kThreads;  // outputs per thread
    constexpr int RS = 32;                   // rows staged at a time
    __shared__ float Xs[RS][kHeadDim + 1];
    __shared__ float Ys[RS][DD + 1];
    const int chunk = blockIdx.x, g = blockIdx.y, which = blockIdx.z;
    const bool per_kv = which == 0 || which == 2;
    const long nrows = per_kv ? (long)a.B * a.N : (long)a.B * a.G * a.N;
    const long r0 = nrows * chunk / kChunks, r1 = nrows * (chunk + 1) / kChunks;
    const T *X = static_cast<const T *>(which == 0 ? a.k : which == 1 ? a.q : which == 2 ? a.v : a.dout);
    const float *Y = which == 0 ? a.dkd : which == 1 ? a.dqt : which == 2 ? a.dvd : a.od;
    float acc[PER];
#pragma unroll
    for (int e = 0; e < PER; ++e)
        acc[e] = 0.f;
    for (long rb = r0; rb < r1; rb += RS) {
        const int n = (int)min((long)RS, r1 - rb);
        __syncthreads();
        for (int idx = threadIdx.x; idx < RS * kHeadDim; idx += kThreads) {
            const int rr = idx / kHeadDim, t = idx % kHeadDim;
            float xv = 0.f;
            if (rr < n) {
                const long u = rb + rr;  // per_kv: b * N + j; else (b * G + hh) * N + i
                long row;
                if (per_kv)
                    row = ((u / a.N) * a.Hkv + g) * a.N + u % a.N;
                else
                    row = (((u / a.N) / a.G) * a.Hq + g * a.G + (u / a.N) % a.G) * a.N + u % a.N;
                xv = to_f32(X[row * kHeadDim + t]);
                if (t < DD)
                    Ys[rr][t] = Y[row * DD + t];
            }
            Xs[rr][t] = xv;
        }
        __syncthreads();
        for (int rr = 0; rr < n; ++rr) {
#pragma unroll
            for (int e = 0; e < PER; ++e) {
                const int o = threadIdx.x + kThreads * e, t = o / DD, c = o % DD;
                acc[e] = fmaf(Xs[rr][t], Ys[rr][c], acc[e]);
            }
        }
    }
    float *dst = a.part + (((size_t)chunk * 4 + which) * a.Hkv + g) * 64 * DD;
#pragma unroll
    for (int e = 0; e < PER; ++e)
        dst[threadIdx.x + kThreads * e] = acc[e];
}

template <int DD>
__global__ void __launch_bounds__(kThreads) bwd_wsum_kernel(Args a)
{
    const int total = 4 * a.Hkv * 64 * DD;
    for (int idx = blockIdx.x * kThreads + threadIdx.x; idx < total; idx += gridDim.x * kThreads) {
        float s = 0.f;
        for (int ch = 0; ch < kChunks; ++ch)
            s += a.part[(size_t)ch * total + idx];
        const int which = idx / (a.Hkv * 64 * DD), rem = idx % (a.Hkv * 64 * DD);
        const int g = rem / (64 * DD), o = rem % (64 * DD), t = o / DD, c = o % DD;
        if (which == 0)
            a.dDk[rem] = s;
        else if (which == 2)
            a.dDv[rem] = s;
        else
            (which == 1 ? a.dUk : a.dUv)[((size_t)g * DD + c) * kHeadDim + t] = s;
    }
}

// ---------------------------------------------------------------- host side

// The projection gradients from the per-row and per-key intermediates.
template <typename T, int DD>
inline cudaError_t run_weights(const Args &a, cudaStream_t s)
{
    bwd_wpart_kernel<T, DD><<<dim3(kChunks, a.Hkv, 4), kThreads, 0, s>>>(a);
    bwd_wsum_kernel<DD><<<(4 * a.Hkv * 64 * DD + kThreads - 1) / kThreads, kThreads, 0, s>>>(a);
    return cudaGetLastError();
}

template <typename T, int DD>
inline cudaError_t run(const Args &a, cudaStream_t s)
{
    static PerDeviceOnce once;
    const size_t smq = dq_smem_floats<DD>() * sizeof(float), smk = dkv_smem_floats<DD>() * sizeof(float);
    cudaError_t e = per_device_once(once, [&](int) {
        cudaError_t e2 = cudaFuncSetAttribute(bwd_dq_kernel<T, DD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                              (int)smq);
        if (e2 == cudaSuccess)
            e2 = cudaFuncSetAttribute(bwd_dkv_kernel<T, DD>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smk);
        return e2;
    });
    if (e != cudaSuccess)
        return e;
    bwd_rows_kernel<T, DD><<<rows_grid(a), 256, 0, s>>>(a);
    const int tiles = (a.N + kRows - 1) / kRows;
    bwd_dq_kernel<T, DD><<<dim3(tiles, a.B * a.Hq), kThreads, smq, s>>>(a);
    bwd_dkv_kernel<T, DD><<<dim3(tiles, a.B * a.Hkv), kThreads, smk, s>>>(a);
    return run_weights<T, DD>(a, s);
}

template <typename T>
inline cudaError_t run_type(int dd, const Args &a, cudaStream_t s)
{
    switch (dd) {
    case 8: return run<T, 8>(a, s);
    case 16: return run<T, 16>(a, s);
    case 32: return run<T, 32>(a, s);
    case 64: return run<T, 64>(a, s);
    default: return cudaErrorInvalidValue;
    }
}

// The two storage types are compiled in separate translation units.
cudaError_t run_f32(int dd, const Args &a, cudaStream_t s);
cudaError_t run_bf16(int dd, const Args &a, cudaStream_t s);

}  // namespace bwd
}  // namespace dar
