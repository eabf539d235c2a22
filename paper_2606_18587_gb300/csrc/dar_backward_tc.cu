// dar_backward_tc.cu -- the backward pass for bf16 storage on the tensor
// cores (mma.sync m16n8k16: bf16 operands, fp32 accumulators), with the
// row kernel and the projection-gradient kernels of dar_backward.cuh.
//
// The same gradients as the CUDA-core kernels (dar_backward.cuh), arranged
// as FlashAttention-style recomputation in 16-key (or 16-query) steps held in
// registers:
//  - dq kernel, one CTA per 64 query rows of a head (four warps of 16 rows):
//    a first pass over the key tiles for the row log-sum-exp, a second for
//      P = 2^(s c2 - lse),  dP = dO v | dO~ v^D,  dS = P (dP - D),
//      dq += dS_loc K,  dq~ += dS_glob K^D,  O^D += P_glob V^D,
//    the score and dP fragments turned into A operands in registers;
//  - dkv kernel, one CTA per 64 keys of a KV head (four warps of 16 keys):
//    over the group's query heads and the query tiles that see the keys,
//    S^T and dP^T per 16-query step, then
//      dv += P_loc dO,  dk += dS_loc Q,  dv^D += P_glob dO~,  dk^D += dS_glob q~.
// Key / query tiles are staged with 16-byte cp.async copies into padded
// shared-memory rows (row stride a multiple of 16 bytes plus 16, so the eight
// rows of an ldmatrix fall in distinct banks), two stages deep; a tile whose
// pairs are all global skips the full-d rows and vice versa.
#include "dar_backward.cuh"
#include "dar_sm100.cuh"

namespace dar {
namespace bwd {

using sm100::cvt_bf16x2;
using sm100::ldsm_x4;
using sm100::ldsm_x4_t;
using sm100::mma_bf16_16816;
using sm100::smem_u32;

constexpr int kTc = 128;           // threads: four warps
constexpr int kLdW = 64 * 2 + 16;  // bytes per padded row of a 64-wide bf16 tile
template <int DD>
constexpr int ld_dd()
{
    return DD * 2 + 16;
}

__device__ __forceinline__ void cp16(uint32_t dst, const void *src)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp4(uint32_t dst, const void *src)
{
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_wait()
{
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// Rows [0, n) of a row-major [*][W] bf16 matrix into a padded tile of 64 rows
// (row stride LD bytes); rows n..63 are zero-filled.
template <int W, int LD>
__device__ __forceinline__ void stage_rows(uint32_t dst, unsigned char *dstp, const bf16 *src, int n, int tid)
{
    constexpr int CH = W / 8;
    for (int i = tid; i < 64 * CH; i += kTc) {
        const int r = i / CH, c = i % CH;
        if (r < n)
            cp16(dst + r * LD + c * 16, src + (size_t)r * W + c * 8);
        else
            *reinterpret_cast<uint4 *>(dstp + r * LD + c * 16) = make_uint4(0u, 0u, 0u, 0u);
    }
}

// 64 fp32 values (n valid, the rest zero).
__device__ __forceinline__ void stage_vec(uint32_t dst, float *dstp, const float *src, int n, int tid)
{
    if (tid < 64) {
        if (tid < n)
            cp4(dst + tid * 4, src + tid);
        else
            dstp[tid] = 0.f;
    }
}

// A fragment of a 16 x 16 k-step from two 16 x 8 accumulator fragments.
__device__ __forceinline__ void frag_a(uint32_t (&a)[4], const float (&c0)[4], const float (&c1)[4])
{
    a[0] = cvt_bf16x2(c0[0], c0[1]);
    a[1] = cvt_bf16x2(c0[2], c0[3]);
    a[2] = cvt_bf16x2(c1[0], c1[1]);
    a[3] = cvt_bf16x2(c1[2], c1[3]);
}

// Row address for ldmatrix (non-transposed, B operand of two n-tiles): the
// 16 rows r0.. of a tile with row stride LD, 16-element k-step kk.
template <int LD>
__device__ __forceinline__ uint32_t b_addr(uint32_t base, int r0, int kk, int lane)
{
    return base + (r0 + (lane & 7) + ((lane >> 4) << 3)) * LD + (2 * kk + ((lane >> 3) & 1)) * 16;
}
// Row address for ldmatrix.trans (B operand [k][n] of two n-tiles at column n0):
// k rows k0..k0+15.
template <int LD>
__device__ __forceinline__ uint32_t bt_addr(uint32_t base, int k0, int n0, int lane)
{
    return base + (k0 + (lane & 7) + (((lane >> 3) & 1) << 3)) * LD + ((n0 + ((lane >> 4) << 3)) / 8) * 16;
}
// Row address for ldmatrix of an A operand (16 rows r0.., k-step kk).
template <int LD>
__device__ __forceinline__ uint32_t a_addr(uint32_t base, int r0, int kk, int lane)
{
    return base + (r0 + (lane & 15)) * LD + (2 * kk + (lane >> 4)) * 16;
}

// ---------------------------------------------------------------- dq

template <int DD>
struct DqLayout {
    static constexpr int LD = ld_dd<DD>();
    static constexpr uint32_t Q = 0;                      // [64][kLdW] q rows
    static constexpr uint32_t DO = Q + 64 * kLdW;         // dO rows
    static constexpr uint32_t QT = DO + 64 * kLdW;        // [64][LD] q~ rows (bf16)
    static constexpr uint32_t DOT = QT + 64 * LD;         // dO~ rows (bf16)
    static constexpr uint32_t STG = DOT + 64 * LD;        // two stages of key-side tiles
    static constexpr uint32_t K_OFF = 0, V_OFF = 64 * kLdW, KD_OFF = 2 * 64 * kLdW, VD_OFF = KD_OFF + 64 * LD;
    static constexpr uint32_t STAGE = VD_OFF + 64 * LD;
    static constexpr uint32_t TOTAL = STG + 2 * STAGE;
    static_assert(64 * (DD + 1) * 4 <= 2 * STAGE, "the epilogue's lift rows fit in the stage area");
};

template <int DD>
__global__ void __launch_bounds__(kTc, DD <= 32 ? 3 : 1) bwd_dq_tc_kernel(Args a)
{
    using Ly = DqLayout<DD>;
    constexpr int LD = Ly::LD, KSD = DD / 16, NTD = DD / 8;
    extern __shared__ __align__(128) unsigned char tsm[];
    unsigned char *sm = tsm;
    const uint32_t sb = smem_u32(sm);
    const int N = a.N, w = a.w;
    const int bh = blockIdx.y, b = bh / a.Hq, h = bh % a.Hq, g = h / a.G;
    const int i0 = blockIdx.x * 64;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, grp = lane >> 2, tig = lane & 3;
    const int nv = min(64, N - i0);
    const size_t rowbase = ((size_t)b * a.Hq + h) * N + i0;
    const size_t kvbase = ((size_t)b * a.Hkv + g) * N;
    const bf16 *kp = static_cast<const bf16 *>(a.k) + kvbase * 64;
    const bf16 *vp = static_cast<const bf16 *>(a.v) + kvbase * 64;
    const bf16 *kdp = static_cast<const bf16 *>(a.kd) + kvbase * DD;
    const bf16 *vdp = static_cast<const bf16 *>(a.vd) + kvbase * DD;
    const int imax = min(N, i0 + 64) - 1;
    const int ntiles = imax / 64 + 1;
    const int wr0 = 16 * warp;  // this warp's first row in the tile

    stage_rows<64, kLdW>(sb + Ly::Q, sm + Ly::Q, static_cast<const bf16 *>(a.q) + rowbase * 64, nv, tid);
    stage_rows<64, kLdW>(sb + Ly::DO, sm + Ly::DO, static_cast<const bf16 *>(a.dout) + rowbase * 64, nv, tid);
    stage_rows<DD, LD>(sb + Ly::QT, sm + Ly::QT, a.qtb + rowbase * DD, nv, tid);
    stage_rows<DD, LD>(sb + Ly::DOT, sm + Ly::DOT, a.dotb + rowbase * DD, nv, tid);
    cp_commit();

    // virtual step v: pass v / ntiles (0: log-sum-exp, 1: gradients), key tile v % ntiles
    auto stage_keys = [&](int v, int st) {
        const int pass = v / ntiles, j0 = (v % ntiles) * 64, nk = min(64, N - j0);
        const bool all_global = (i0 - (j0 + 63)) >= w, all_local = (i0 + 63 - j0) < w;
        const uint32_t base = sb + Ly::STG + st * Ly::STAGE;
        unsigned char *bp = sm + Ly::STG + st * Ly::STAGE;
        if (!all_global) {
            stage_rows<64, kLdW>(base + Ly::K_OFF, bp + Ly::K_OFF, kp + (size_t)j0 * 64, nk, tid);
            if (pass)
                stage_rows<64, kLdW>(base + Ly::V_OFF, bp + Ly::V_OFF, vp + (size_t)j0 * 64, nk, tid);
        }
        if (!all_local) {
            stage_rows<DD, LD>(base + Ly::KD_OFF, bp + Ly::KD_OFF, kdp + (size_t)j0 * DD, nk, tid);
            if (pass)
                stage_rows<DD, LD>(base + Ly::VD_OFF, bp + Ly::VD_OFF, vdp + (size_t)j0 * DD, nk, tid);
        }
        cp_commit();
    };
    const int nvs = 2 * ntiles;
    stage_keys(0, 0);
    cp_wait<1>();  // the query-side rows (the first key stage may still be in flight)
    __syncthreads();

    // A fragments: the d_down-wide rows stay in registers (every global step
    // uses them); the 64-wide q and dO rows are read from shared memory by the
    // (rarer) steps with local pairs, which keeps registers for occupancy
    uint32_t qta[KSD][4], dota[KSD][4];
#pragma unroll
    for (int kk = 0; kk < KSD; ++kk) {
        ldsm_x4(a_addr<LD>(sb + Ly::QT, wr0, kk, lane), qta[kk]);
        ldsm_x4(a_addr<LD>(sb + Ly::DOT, wr0, kk, lane), dota[kk]);
    }
    const int ir0 = i0 + wr0 + grp;  // this thread's rows: ir0 and ir0 + 8
    float Dr[2], m[2] = {-INFINITY, -INFINITY}, l[2] = {0.f, 0.f}, lse[2] = {0.f, 0.f};
#pragma unroll
    for (int r = 0; r < 2; ++r)
        Dr[r] = ir0 + 8 * r < N ? a.drow[rowbase + wr0 + grp + 8 * r] : 0.f;
    float dq[8][4], dqt[NTD][4], od[NTD][4];
#pragma unroll
    for (int n = 0; n < 8; ++n)
        dq[n][0] = dq[n][1] = dq[n][2] = dq[n][3] = 0.f;
#pragma unroll
    for (int n = 0; n < NTD; ++n)
        dqt[n][0] = dqt[n][1] = dqt[n][2] = dqt[n][3] = od[n][0] = od[n][1] = od[n][2] = od[n][3] = 0.f;

    for (int v = 0; v < nvs; ++v) {
        const int pass = v / ntiles, st = v & 1;
        const int j0 = (v % ntiles) * 64;
        if (v + 1 < nvs) {
            stage_keys(v + 1, st ^ 1);
            cp_wait<1>();
        } else {
            cp_wait<0>();
        }
        __syncthreads();
        if (pass == 1 && v == ntiles) {
            // the rows' log-sum-exp: combine the four threads of each row
#pragma unroll
            for (int r = 0; r < 2; ++r) {
#pragma unroll
                for (int o = 1; o <= 2; o <<= 1) {
                    const float mo = __shfl_xor_sync(0xffffffffu, m[r], o), lo = __shfl_xor_sync(0xffffffffu, l[r], o);
                    const float mn = fmaxf(m[r], mo);
                    l[r] = (m[r] == -INFINITY ? 0.f : l[r] * exp2f(m[r] - mn)) +
                           (mo == -INFINITY ? 0.f : lo * exp2f(mo - mn));
                    m[r] = mn;
                }
                lse[r] = m[r] + log2f(l[r]);
                if (tig == 0 && ir0 + 8 * r < N)
                    a.lse[rowbase + wr0 + grp + 8 * r] = lse[r];
            }
        }
        const bool all_global = (i0 - (j0 + 63)) >= w, all_local = (i0 + 63 - j0) < w;
        // all pairs global, every key before every row, every row inside the sequence
        const bool interior = all_global && j0 + 63 <= i0 && i0 + 63 < N;
        const uint32_t stg = sb + Ly::STG + st * Ly::STAGE;
#pragma unroll 1
        for (int kc = 0; kc < 4; ++kc) {
            if (j0 + 16 * kc > i0 + wr0 + 15)
                break;  // every key of the step is after every row of this warp (causal)
            float sl[2][4] = {}, sg[2][4] = {};
            if (!all_global) {
#pragma unroll
                for (int kk = 0; kk < 4; ++kk) {
                    uint32_t bfr[4], afr[4];
                    ldsm_x4(a_addr<kLdW>(sb + Ly::Q, wr0, kk, lane), afr);
                    ldsm_x4(b_addr<kLdW>(stg + Ly::K_OFF, 16 * kc, kk, lane), bfr);
                    mma_bf16_16816(sl[0], afr, bfr[0], bfr[1]);
                    mma_bf16_16816(sl[1], afr, bfr[2], bfr[3]);
                }
            }
            if (!all_local) {
#pragma unroll
                for (int kk = 0; kk < KSD; ++kk) {
                    uint32_t bfr[4];
                    ldsm_x4(b_addr<LD>(stg + Ly::KD_OFF, 16 * kc, kk, lane), bfr);
                    mma_bf16_16816(sg[0], qta[kk], bfr[0], bfr[1]);
                    mma_bf16_16816(sg[1], qta[kk], bfr[2], bfr[3]);
                }
            }
            if (interior) {  // every pair of the step is valid and global: no masks, no local part
                if (pass == 0) {
#pragma unroll
                    for (int r = 0; r < 2; ++r) {
                        const float x0 = sg[0][2 * r] * a.c2, x1 = sg[0][2 * r + 1] * a.c2;
                        const float x2 = sg[1][2 * r] * a.c2, x3 = sg[1][2 * r + 1] * a.c2;
                        const float mn = fmaxf(m[r], fmaxf(fmaxf(x0, x1), fmaxf(x2, x3)));
                        l[r] = l[r] * sm100::ex2_approx(m[r] - mn) + (sm100::ex2_approx(x0 - mn) + sm100::ex2_approx(x1 - mn)) +
                               (sm100::ex2_approx(x2 - mn) + sm100::ex2_approx(x3 - mn));
                        m[r] = mn;
                    }
                    continue;
                }
                float dpg[2][4] = {};
#pragma unroll
                for (int kk = 0; kk < KSD; ++kk) {
                    uint32_t bfr[4];
                    ldsm_x4(b_addr<LD>(stg + Ly::VD_OFF, 16 * kc, kk, lane), bfr);
                    mma_bf16_16816(dpg[0], dota[kk], bfr[0], bfr[1]);
                    mma_bf16_16816(dpg[1], dota[kk], bfr[2], bfr[3]);
                }
                float pg[2][4], dsg[2][4];
#pragma unroll
                for (int nt = 0; nt < 2; ++nt)
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        pg[nt][e] = sm100::ex2_approx(fmaf(sg[nt][e], a.c2, -lse[e >> 1]));
                        dsg[nt][e] = pg[nt][e] * (dpg[nt][e] - Dr[e >> 1]);
                    }
                uint32_t ag[4], ap[4];
                frag_a(ag, dsg[0], dsg[1]);
                frag_a(ap, pg[0], pg[1]);
#pragma unroll
                for (int n0 = 0; n0 < DD; n0 += 16) {
                    uint32_t bfr[4];
                    ldsm_x4_t(bt_addr<LD>(stg + Ly::KD_OFF, 16 * kc, n0, lane), bfr);
                    mma_bf16_16816(dqt[n0 / 8], ag, bfr[0], bfr[1]);
                    mma_bf16_16816(dqt[n0 / 8 + 1], ag, bfr[2], bfr[3]);
                    ldsm_x4_t(bt_addr<LD>(stg + Ly::VD_OFF, 16 * kc, n0, lane), bfr);
                    mma_bf16_16816(od[n0 / 8], ap, bfr[0], bfr[1]);
                    mma_bf16_16816(od[n0 / 8 + 1], ap, bfr[2], bfr[3]);
                }
                continue;
            }
            float x[2][4];
            bool loc[2][4];
#pragma unroll
            for (int nt = 0; nt < 2; ++nt)
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int i = ir0 + 8 * (e >> 1), j = j0 + 16 * kc + 8 * nt + 2 * tig + (e & 1);
                    loc[nt][e] = i - j < w;
                    x[nt][e] = (i < N && j <= i) ? (loc[nt][e] ? sl[nt][e] : sg[nt][e]) * a.c2 : -INFINITY;
                }
            if (pass == 0) {
#pragma unroll
                for (int r = 0; r < 2; ++r) {
                    const float mx = fmaxf(fmaxf(x[0][2 * r], x[0][2 * r + 1]), fmaxf(x[1][2 * r], x[1][2 * r + 1]));
                    const float mn = fmaxf(m[r], mx);
                    if (mn == -INFINITY)
                        continue;
                    float ps = 0.f;
#pragma unroll
                    for (int nt = 0; nt < 2; ++nt)
#pragma unroll
                        for (int e = 0; e < 2; ++e)
                            ps += x[nt][2 * r + e] == -INFINITY ? 0.f : sm100::ex2_approx(x[nt][2 * r + e] - mn);
                    l[r] = (m[r] == -INFINITY ? 0.f : l[r] * sm100::ex2_approx(m[r] - mn)) + ps;
                    m[r] = mn;
                }
                continue;
            }
            float dpl[2][4] = {}, dpg[2][4] = {};
            if (!all_global) {
#pragma unroll
                for (int kk = 0; kk < 4; ++kk) {
                    uint32_t bfr[4], afr[4];
                    ldsm_x4(a_addr<kLdW>(sb + Ly::DO, wr0, kk, lane), afr);
                    ldsm_x4(b_addr<kLdW>(stg + Ly::V_OFF, 16 * kc, kk, lane), bfr);
                    mma_bf16_16816(dpl[0], afr, bfr[0], bfr[1]);
                    mma_bf16_16816(dpl[1], afr, bfr[2], bfr[3]);
                }
            }
            if (!all_local) {
#pragma unroll
                for (int kk = 0; kk < KSD; ++kk) {
                    uint32_t bfr[4];
                    ldsm_x4(b_addr<LD>(stg + Ly::VD_OFF, 16 * kc, kk, lane), bfr);
                    mma_bf16_16816(dpg[0], dota[kk], bfr[0], bfr[1]);
                    mma_bf16_16816(dpg[1], dota[kk], bfr[2], bfr[3]);
                }
            }
            float dsl[2][4], dsg[2][4], pgl[2][4];
#pragma unroll
            for (int nt = 0; nt < 2; ++nt)
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float p = x[nt][e] == -INFINITY ? 0.f : sm100::ex2_approx(x[nt][e] - lse[e >> 1]);
                    const float ds = p * ((loc[nt][e] ? dpl[nt][e] : dpg[nt][e]) - Dr[e >> 1]);
                    dsl[nt][e] = loc[nt][e] ? ds : 0.f;
                    dsg[nt][e] = loc[nt][e] ? 0.f : ds;
                    pgl[nt][e] = loc[nt][e] ? 0.f : p;
                }
            if (!all_global) {
                uint32_t af[4];
                frag_a(af, dsl[0], dsl[1]);
#pragma unroll
                for (int n0 = 0; n0 < 64; n0 += 16) {
                    uint32_t bfr[4];
                    ldsm_x4_t(bt_addr<kLdW>(stg + Ly::K_OFF, 16 * kc, n0, lane), bfr);
                    mma_bf16_16816(dq[n0 / 8], af, bfr[0], bfr[1]);
                    mma_bf16_16816(dq[n0 / 8 + 1], af, bfr[2], bfr[3]);
                }
            }
            if (!all_local) {
                uint32_t ag[4], ap[4];
                frag_a(ag, dsg[0], dsg[1]);
                frag_a(ap, pgl[0], pgl[1]);
#pragma unroll
                for (int n0 = 0; n0 < DD; n0 += 16) {
                    uint32_t bfr[4];
                    ldsm_x4_t(bt_addr<LD>(stg + Ly::KD_OFF, 16 * kc, n0, lane), bfr);
                    mma_bf16_16816(dqt[n0 / 8], ag, bfr[0], bfr[1]);
                    mma_bf16_16816(dqt[n0 / 8 + 1], ag, bfr[2], bfr[3]);
                    ldsm_x4_t(bt_addr<LD>(stg + Ly::VD_OFF, 16 * kc, n0, lane), bfr);
                    mma_bf16_16816(od[n0 / 8], ap, bfr[0], bfr[1]);
                    mma_bf16_16816(od[n0 / 8 + 1], ap, bfr[2], bfr[3]);
                }
            }
        }
        __syncthreads();  // stage st is free for the copy issued in the next step
    }

    // epilogue: dq = scale (dq_loc + dq~ Uk), dq~ (scaled) and O^D for the projection gradients
    float *lift = reinterpret_cast<float *>(sm + Ly::STG);  // [64][DD + 1], the idle stage area
#pragma unroll
    for (int n = 0; n < NTD; ++n)
#pragma unroll
        for (int e = 0; e < 4; ++e)
            lift[(wr0 + grp + 8 * (e >> 1)) * (DD + 1) + 8 * n + 2 * tig + (e & 1)] = dqt[n][e] * a.scale;
    __syncwarp();
    const float *Uk = a.Uk + (size_t)g * DD * 64;
#pragma unroll
    for (int r = 0; r < 2; ++r) {
        const int rr = wr0 + grp + 8 * r;
        if (i0 + rr >= N)
            continue;
        const size_t row = rowbase + rr;
        bf16 *dqr = static_cast<bf16 *>(a.dq) + row * 64;
#pragma unroll
        for (int n = 0; n < 8; ++n) {
            const int t = 8 * n + 2 * tig;
            float o0 = dq[n][2 * r] * a.scale, o1 = dq[n][2 * r + 1] * a.scale;
            for (int c = 0; c < DD; ++c) {
                const float x2 = lift[rr * (DD + 1) + c];
                o0 = fmaf(x2, __ldg(Uk + c * 64 + t), o0);
                o1 = fmaf(x2, __ldg(Uk + c * 64 + t + 1), o1);
            }
            *reinterpret_cast<uint32_t *>(dqr + t) = cvt_bf16x2(o0, o1);
        }
#pragma unroll
        for (int n = 0; n < NTD; ++n) {
            const int c = 8 * n + 2 * tig;
            *reinterpret_cast<float2 *>(a.dqt + row * DD + c) =
                make_float2(dqt[n][2 * r] * a.scale, dqt[n][2 * r + 1] * a.scale);
            *reinterpret_cast<float2 *>(a.od + row * DD + c) = make_float2(od[n][2 * r], od[n][2 * r + 1]);
        }
    }
}

// ---------------------------------------------------------------- dk, dv

template <int DD>
struct DkvLayout {
    static constexpr int LD = ld_dd<DD>();
    static constexpr uint32_t K = 0;                      // [64][kLdW] this CTA's keys
    static constexpr uint32_t V = K + 64 * kLdW;
    static constexpr uint32_t KD = V + 64 * kLdW;         // [64][LD]
    static constexpr uint32_t VD = KD + 64 * LD;
    static constexpr uint32_t STG = VD + 64 * LD;         // two stages of query-side tiles
    static constexpr uint32_t Q_OFF = 0, DO_OFF = 64 * kLdW, QT_OFF = 2 * 64 * kLdW, DOT_OFF = QT_OFF + 64 * LD;
    static constexpr uint32_t LSE_OFF = DOT_OFF + 64 * LD, DR_OFF = LSE_OFF + 256;
    static constexpr uint32_t STAGE = DR_OFF + 256;
    static constexpr uint32_t TOTAL = STG + 2 * STAGE;
    static_assert(2 * 64 * (DD + 1) * 4 <= 2 * STAGE, "the epilogue's lift rows fit in the stage area");
};

template <int DD>
__global__ void __launch_bounds__(kTc, DD <= 32 ? 3 : 1) bwd_dkv_tc_kernel(Args a)
{
    using Ly = DkvLayout<DD>;
    constexpr int LD = Ly::LD, KSD = DD / 16, NTD = DD / 8;
    extern __shared__ __align__(128) unsigned char tsm[];
    unsigned char *sm = tsm;
    const uint32_t sb = smem_u32(sm);
    const int N = a.N, w = a.w;
    const int bg = blockIdx.y, b = bg / a.Hkv, g = bg % a.Hkv;
    const int j0 = blockIdx.x * 64;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, grp = lane >> 2, tig = lane & 3;
    const int nk = min(64, N - j0);
    const size_t kvbase = ((size_t)b * a.Hkv + g) * N + j0;
    const int wk0 = 16 * warp;
    const int jr0 = j0 + wk0 + grp;  // this thread's keys: jr0 and jr0 + 8

    stage_rows<64, kLdW>(sb + Ly::K, sm + Ly::K, static_cast<const bf16 *>(a.k) + kvbase * 64, nk, tid);
    stage_rows<64, kLdW>(sb + Ly::V, sm + Ly::V, static_cast<const bf16 *>(a.v) + kvbase * 64, nk, tid);
    stage_rows<DD, LD>(sb + Ly::KD, sm + Ly::KD, static_cast<const bf16 *>(a.kd) + kvbase * DD, nk, tid);
    stage_rows<DD, LD>(sb + Ly::VD, sm + Ly::VD, static_cast<const bf16 *>(a.vd) + kvbase * DD, nk, tid);
    cp_commit();

    const int it0 = j0 / 64, ntq = (N + 63) / 64, per_head = ntq - it0, nvs = a.G * per_head;
    auto stage_q = [&](int v, int st) {
        const int h = g * a.G + v / per_head, i0 = (it0 + v % per_head) * 64, nv = min(64, N - i0);
        const bool all_global = (i0 - (j0 + 63)) >= w, all_local = (i0 + 63 - j0) < w;
        const size_t rowbase = ((size_t)b * a.Hq + h) * N + i0;
        const uint32_t base = sb + Ly::STG + st * Ly::STAGE;
        unsigned char *bp = sm + Ly::STG + st * Ly::STAGE;
        if (!all_global) {
            stage_rows<64, kLdW>(base + Ly::Q_OFF, bp + Ly::Q_OFF, static_cast<const bf16 *>(a.q) + rowbase * 64, nv,
                                 tid);
            stage_rows<64, kLdW>(base + Ly::DO_OFF, bp + Ly::DO_OFF, static_cast<const bf16 *>(a.dout) + rowbase * 64,
                                 nv, tid);
        }
        if (!all_local) {
            stage_rows<DD, LD>(base + Ly::QT_OFF, bp + Ly::QT_OFF, a.qtb + rowbase * DD, nv, tid);
            stage_rows<DD, LD>(base + Ly::DOT_OFF, bp + Ly::DOT_OFF, a.dotb + rowbase * DD, nv, tid);
        }
        stage_vec(base + Ly::LSE_OFF, reinterpret_cast<float *>(bp + Ly::LSE_OFF), a.lse + rowbase, nv, tid);
        stage_vec(base + Ly::DR_OFF, reinterpret_cast<float *>(bp + Ly::DR_OFF), a.drow + rowbase, nv, tid);
        cp_commit();
    };
    if (nvs > 0)
        stage_q(0, 0);
    cp_wait<1>();  // the key-side rows
    __syncthreads();

    // A fragments: the d_down-wide key rows stay in registers; the 64-wide k
    // and v rows are read from shared memory by the steps with local pairs
    uint32_t kda[KSD][4], vda[KSD][4];
#pragma unroll
    for (int kk = 0; kk < KSD; ++kk) {
        ldsm_x4(a_addr<LD>(sb + Ly::KD, wk0, kk, lane), kda[kk]);
        ldsm_x4(a_addr<LD>(sb + Ly::VD, wk0, kk, lane), vda[kk]);
    }
    float dk[8][4], dv[8][4], dkd[NTD][4], dvd[NTD][4];
#pragma unroll
    for (int n = 0; n < 8; ++n)
        dk[n][0] = dk[n][1] = dk[n][2] = dk[n][3] = dv[n][0] = dv[n][1] = dv[n][2] = dv[n][3] = 0.f;
#pragma unroll
    for (int n = 0; n < NTD; ++n)
        dkd[n][0] = dkd[n][1] = dkd[n][2] = dkd[n][3] = dvd[n][0] = dvd[n][1] = dvd[n][2] = dvd[n][3] = 0.f;

    for (int v = 0; v < nvs; ++v) {
        const int st = v & 1;
        const int i0 = (it0 + v % per_head) * 64;
        if (v + 1 < nvs) {
            stage_q(v + 1, st ^ 1);
            cp_wait<1>();
        } else {
            cp_wait<0>();
        }
        __syncthreads();
        const bool all_global = (i0 - (j0 + 63)) >= w, all_local = (i0 + 63 - j0) < w;
        // all pairs global, every key before every query, every key and query inside the sequence
        const bool interior = all_global && j0 + 63 <= i0 && i0 + 63 < N;
        const uint32_t stg = sb + Ly::STG + st * Ly::STAGE;
        const float *lse_s = reinterpret_cast<const float *>(sm + Ly::STG + st * Ly::STAGE + Ly::LSE_OFF);
        const float *dr_s = reinterpret_cast<const float *>(sm + Ly::STG + st * Ly::STAGE + Ly::DR_OFF);
#pragma unroll 1
        for (int qc = 0; qc < 4; ++qc) {
            if (i0 + 16 * qc + 15 < j0 + wk0)
                continue;  // every query of the step is before every key of this warp (causal)
            float sl[2][4] = {}, sg[2][4] = {};
            if (!all_global) {
#pragma unroll
                for (int kk = 0; kk < 4; ++kk) {
                    uint32_t bfr[4], afr[4];
                    ldsm_x4(a_addr<kLdW>(sb + Ly::K, wk0, kk, lane), afr);
                    ldsm_x4(b_addr<kLdW>(stg + Ly::Q_OFF, 16 * qc, kk, lane), bfr);
                    mma_bf16_16816(sl[0], afr, bfr[0], bfr[1]);
                    mma_bf16_16816(sl[1], afr, bfr[2], bfr[3]);
                }
            }
            if (!all_local) {
#pragma unroll
                for (int kk = 0; kk < KSD; ++kk) {
                    uint32_t bfr[4];
                    ldsm_x4(b_addr<LD>(stg + Ly::QT_OFF, 16 * qc, kk, lane), bfr);
                    mma_bf16_16816(sg[0], kda[kk], bfr[0], bfr[1]);
                    mma_bf16_16816(sg[1], kda[kk], bfr[2], bfr[3]);
                }
            }
            if (interior) {  // every pair of the step is valid and global: no masks, no local part
                float dpg[2][4] = {};
#pragma unroll
                for (int kk = 0; kk < KSD; ++kk) {
                    uint32_t bfr[4];
                    ldsm_x4(b_addr<LD>(stg + Ly::DOT_OFF, 16 * qc, kk, lane), bfr);
                    mma_bf16_16816(dpg[0], vda[kk], bfr[0], bfr[1]);
                    mma_bf16_16816(dpg[1], vda[kk], bfr[2], bfr[3]);
                }
                float pg[2][4], dsg[2][4];
#pragma unroll
                for (int nt = 0; nt < 2; ++nt)
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const int il = 16 * qc + 8 * nt + 2 * tig + (e & 1);
                        pg[nt][e] = sm100::ex2_approx(fmaf(sg[nt][e], a.c2, -lse_s[il]));
                        dsg[nt][e] = pg[nt][e] * (dpg[nt][e] - dr_s[il]);
                    }
                uint32_t ap[4], ad[4];
                frag_a(ap, pg[0], pg[1]);
                frag_a(ad, dsg[0], dsg[1]);
#pragma unroll
                for (int n0 = 0; n0 < DD; n0 += 16) {
                    uint32_t bfr[4];
                    ldsm_x4_t(bt_addr<LD>(stg + Ly::DOT_OFF, 16 * qc, n0, lane), bfr);
                    mma_bf16_16816(dvd[n0 / 8], ap, bfr[0], bfr[1]);
                    mma_bf16_16816(dvd[n0 / 8 + 1], ap, bfr[2], bfr[3]);
                    ldsm_x4_t(bt_addr<LD>(stg + Ly::QT_OFF, 16 * qc, n0, lane), bfr);
                    mma_bf16_16816(dkd[n0 / 8], ad, bfr[0], bfr[1]);
                    mma_bf16_16816(dkd[n0 / 8 + 1], ad, bfr[2], bfr[3]);
                }
                continue;
            }
            float dpl[2][4] = {}, dpg[2][4] = {};
            if (!all_global) {
#pragma unroll
                for (int kk = 0; kk < 4; ++kk) {
                    uint32_t bfr[4], afr[4];
                    ldsm_x4(a_addr<kLdW>(sb + Ly::V, wk0, kk, lane), afr);
                    ldsm_x4(b_addr<kLdW>(stg + Ly::DO_OFF, 16 * qc, kk, lane), bfr);
                    mma_bf16_16816(dpl[0], afr, bfr[0], bfr[1]);
                    mma_bf16_16816(dpl[1], afr, bfr[2], bfr[3]);
                }
            }
            if (!all_local) {
#pragma unroll
                for (int kk = 0; kk < KSD; ++kk) {
                    uint32_t bfr[4];
                    ldsm_x4(b_addr<LD>(stg + Ly::DOT_OFF, 16 * qc, kk, lane), bfr);
                    mma_bf16_16816(dpg[0], vda[kk], bfr[0], bfr[1]);
                    mma_bf16_16816(dpg[1], vda[kk], bfr[2], bfr[3]);
                }
            }
            float pl[2][4], dsl[2][4], pg[2][4], dsg[2][4];
#pragma unroll
            for (int nt = 0; nt < 2; ++nt)
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int j = jr0 + 8 * (e >> 1), il = 16 * qc + 8 * nt + 2 * tig + (e & 1), i = i0 + il;
                    const bool loc = i - j < w;
                    float p = 0.f, ds = 0.f;
                    if (j < N && i < N && j <= i) {
                        p = sm100::ex2_approx((loc ? sl[nt][e] : sg[nt][e]) * a.c2 - lse_s[il]);
                        ds = p * ((loc ? dpl[nt][e] : dpg[nt][e]) - dr_s[il]);
                    }
                    pl[nt][e] = loc ? p : 0.f;
                    dsl[nt][e] = loc ? ds : 0.f;
                    pg[nt][e] = loc ? 0.f : p;
                    dsg[nt][e] = loc ? 0.f : ds;
                }
            if (!all_global) {
                uint32_t ap[4], ad[4];
                frag_a(ap, pl[0], pl[1]);
                frag_a(ad, dsl[0], dsl[1]);
#pragma unroll
                for (int n0 = 0; n0 < 64; n0 += 16) {
                    uint32_t bfr[4];
                    ldsm_x4_t(bt_addr<kLdW>(stg + Ly::DO_OFF, 16 * qc, n0, lane), bfr);
                    mma_bf16_16816(dv[n0 / 8], ap, bfr[0], bfr[1]);
                    mma_bf16_16816(dv[n0 / 8 + 1], ap, bfr[2], bfr[3]);
                    ldsm_x4_t(bt_addr<kLdW>(stg + Ly::Q_OFF, 16 * qc, n0, lane), bfr);
                    mma_bf16_16816(dk[n0 / 8], ad, bfr[0], bfr[1]);
                    mma_bf16_16816(dk[n0 / 8 + 1], ad, bfr[2], bfr[3]);
                }
            }
            if (!all_local) {
                uint32_t ap[4], ad[4];
                frag_a(ap, pg[0], pg[1]);
                frag_a(ad, dsg[0], dsg[1]);
#pragma unroll
                for (int n0 = 0; n0 < DD; n0 += 16) {
                    uint32_t bfr[4];
                    ldsm_x4_t(bt_addr<LD>(stg + Ly::DOT_OFF, 16 * qc, n0, lane), bfr);
                    mma_bf16_16816(dvd[n0 / 8], ap, bfr[0], bfr[1]);
                    mma_bf16_16816(dvd[n0 / 8 + 1], ap, bfr[2], bfr[3]);
                    ldsm_x4_t(bt_addr<LD>(stg + Ly::QT_OFF, 16 * qc, n0, lane), bfr);
                    mma_bf16_16816(dkd[n0 / 8], ad, bfr[0], bfr[1]);
                    mma_bf16_16816(dkd[n0 / 8 + 1], ad, bfr[2], bfr[3]);
                }
            }
        }
        __syncthreads();  // stage st is free for the copy issued in the next step
    }
    cp_wait<0>();
    __syncthreads();

    // epilogue: dk = scale dk_loc + dk^D Dk^T (dk^D = scale sum dS q~), dv = dv_loc + dv^D Dv^T
    float *lk = reinterpret_cast<float *>(sm + Ly::STG);  // [64][DD + 1] dk^D, then dv^D
    float *lv = lk + 64 * (DD + 1);
#pragma unroll
    for (int n = 0; n < NTD; ++n)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const int idx = (wk0 + grp + 8 * (e >> 1)) * (DD + 1) + 8 * n + 2 * tig + (e & 1);
            lk[idx] = dkd[n][e] * a.scale;
            lv[idx] = dvd[n][e];
        }
    __syncwarp();
    const float *Dk = a.Dk + (size_t)g * 64 * DD, *Dv = a.Dv + (size_t)g * 64 * DD;
#pragma unroll
    for (int r = 0; r < 2; ++r) {
        const int kr = wk0 + grp + 8 * r;
        if (j0 + kr >= N)
            continue;
        const size_t row = kvbase + kr;
        bf16 *dkr = static_cast<bf16 *>(a.dk) + row * 64;
        bf16 *dvr = static_cast<bf16 *>(a.dv) + row * 64;
#pragma unroll
        for (int n = 0; n < 8; ++n) {
            const int t = 8 * n + 2 * tig;
            float k0 = dk[n][2 * r] * a.scale, k1 = dk[n][2 * r + 1] * a.scale;
            float v0 = dv[n][2 * r], v1 = dv[n][2 * r + 1];
            for (int c = 0; c < DD; ++c) {
                const float xk = lk[kr * (DD + 1) + c], xv = lv[kr * (DD + 1) + c];
                k0 = fmaf(xk, __ldg(Dk + t * DD + c), k0);
                k1 = fmaf(xk, __ldg(Dk + (t + 1) * DD + c), k1);
                v0 = fmaf(xv, __ldg(Dv + t * DD + c), v0);
                v1 = fmaf(xv, __ldg(Dv + (t + 1) * DD + c), v1);
            }
            *reinterpret_cast<uint32_t *>(dkr + t) = cvt_bf16x2(k0, k1);
            *reinterpret_cast<uint32_t *>(dvr + t) = cvt_bf16x2(v0, v1);
        }
#pragma unroll
        for (int n = 0; n < NTD; ++n) {
            const int c = 8 * n + 2 * tig;
            *reinterpret_cast<float2 *>(a.dkd + row * DD + c) =
                make_float2(dkd[n][2 * r] * a.scale, dkd[n][2 * r + 1] * a.scale);
            *reinterpret_cast<float2 *>(a.dvd + row * DD + c) = make_float2(dvd[n][2 * r], dvd[n][2 * r + 1]);
        }
    }
}

// ---------------------------------------------------------------- host side

template <int DD>
static cudaError_t run_tc(const Args &a, cudaStream_t s)
{
    const size_t smq = DqLayout<DD>::TOTAL, smk = DkvLayout<DD>::TOTAL;
    static PerDeviceOnce once;
    cudaError_t e = per_device_once(once, [&](int) {
        cudaError_t e2 = cudaFuncSetAttribute(bwd_dq_tc_kernel<DD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                              (int)smq);
        if (e2 == cudaSuccess)
            e2 = cudaFuncSetAttribute(bwd_dkv_tc_kernel<DD>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smk);
        return e2;
    });
    if (e != cudaSuccess)
        return e;
    bwd_rows_kernel<bf16, DD><<<rows_grid(a), 256, 0, s>>>(a);
    const int tiles = (a.N + 63) / 64;
    bwd_dq_tc_kernel<DD><<<dim3(tiles, a.B * a.Hq), kTc, smq, s>>>(a);
    bwd_dkv_tc_kernel<DD><<<dim3(tiles, a.B * a.Hkv), kTc, smk, s>>>(a);
    return run_weights<bf16, DD>(a, s);
}

// bf16 storage: the tensor-core kernels for d_down >= 16 (whole 16-wide
// k-steps); d_down = 8 keeps the CUDA-core kernels.
cudaError_t run_bf16(int dd, const Args &a, cudaStream_t s)
{
    switch (dd) {
    case 8: return run<bf16, 8>(a, s);
    case 16: return run_tc<16>(a, s);
    case 32: return run_tc<32>(a, s);
    case 64: return run_tc<64>(a, s);
    default: return cudaErrorInvalidValue;
    }
}

}  // namespace bwd
}  // namespace dar
