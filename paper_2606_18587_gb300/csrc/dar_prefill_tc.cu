// dar_prefill_tc.cu -- causal DAR attention forward (bf16) on the 5th-generation
// tensor cores: tcgen05.mma with operands staged by TMA in shared memory (or,
// for P, held in tensor memory) and fp32 accumulators in tensor memory (TMEM).
//
// One CTA = 128 query rows of one head; key tiles of 64, visited from the
// diagonal down to key 0.  Per key tile (Eq. 3: local iff i - j < w):
//   local part   S_loc  = Q  K^T       (M128 N64 K64)   O_loc  += P_loc  V    (N64)
//   global part  S_glob = Q~ (K^D)^T   (M128 N64 Kdd)   O_glob += P_glob V^D  (Ndd)
// with q~ = q Uk^T (W_up absorbed into the query, exact by linearity of
// Eq. 2).  A tile that holds both kinds (the window edge crosses it) is run
// as two virtual tiles, each with the other kind masked out.  One online
// softmax over every virtual tile (Eq. 4), with the running max raised lazily
// (only when it grows by more than 2^8), and the epilogue lifts the global
// part once:  o = (O_loc + O_glob Uv) / l.
//
// Warp roles (192 threads): warp 0 issues TMA loads, warp 1 allocates TMEM and
// issues the MMAs (one thread), warps 2-5 own one query row per thread
// (TMEM lane = row) for the softmax and the epilogue.  q~ is computed by a
// pre-pass into the first d_down entries of each output row and loaded with Q.  The softmax writes
// P (bf16) into TMEM with tcgen05.st and the PV products take it from there
// as their A operand, so P never touches shared memory.  Two S buffers (when
// d_down <= 32) let S run two virtual tiles ahead of the softmax.  256 TMEM
// columns and ~80 KB of shared memory per CTA let two CTAs share an SM, so
// one CTA's softmax overlaps the other's MMA and load waits.  Every wait is
// bounded; on a timeout the CTA flags *status and exits.
#include <cuda.h>

#include "dar_common.cuh"
#include "dar_launch.h"
#include "dar_sm100.cuh"

namespace dar {
namespace tcp {

using namespace sm100;

constexpr int BM = 128, BN = 64;
constexpr int kThreads = 192;
constexpr uint32_t kTmemCols = 256;
constexpr float kRescaleThreshold = 8.0f;  // log2 units: p stays below 2^8 between rescales

constexpr uint32_t align_up(uint32_t x, uint32_t a) { return (x + a - 1) / a * a; }

// Tensor-memory columns of one CTA (256 of the SM's 512, two CTAs per SM):
// S buffers (fp32, BN columns each; two when they fit, so S runs two virtual
// tiles ahead of the softmax), O_loc (64), O_glob (DP) and P (bf16 pairs,
// BN / 2 columns; the A operand of the PV products).
template <int DP>
struct Tmem {
    static constexpr int NSB = DP <= 32 ? 2 : 1;
    static constexpr uint32_t S = 0;  // buffer b at S + b * BN
    static constexpr uint32_t OL = NSB * BN;
    static constexpr uint32_t OG = OL + 64;
    static constexpr uint32_t P = kTmemCols - BN / 2;
    static_assert(OG + DP <= P, "tensor-memory columns overlap");
};

// Shared-memory layout (offsets from a 1024-byte aligned base).  A stage holds
// the operands of one virtual tile: K and V (local) or K^D and V^D (global).
template <int DP>
struct Layout {
    static constexpr int NS = 3;                          // K/V stages
    static constexpr uint32_t Q = 0;                      // [128][64] bf16, 128B swizzle
    static constexpr uint32_t QT = BM * 64 * 2;           // [128][DP] bf16 (q~, loaded by TMA)
    static constexpr uint32_t STG = align_up(QT + BM * DP * 2, 1024);
    static constexpr uint32_t K_OFF = 0;                  // [64][64]
    static constexpr uint32_t V_OFF = BN * 64 * 2;        // [64][64]
    static constexpr uint32_t KD_OFF = 0;                 // [64][DP]
    static constexpr uint32_t VD_OFF = align_up(BN * DP * 2, 1024);
    static constexpr uint32_t STAGE = align_up(2 * BN * 64 * 2, 1024);
    static constexpr uint32_t UV = STG + NS * STAGE;      // fp32 [DP][64]
    static constexpr uint32_t BAR = UV + DP * 64 * 4;
    static constexpr uint32_t TOTAL = BAR + 256;
    static_assert(STAGE % 1024 == 0 && STG % 1024 == 0, "operand tiles must stay 1024-byte aligned");
    static_assert(VD_OFF + BN * DP * 2 <= STAGE, "a stage holds either part");
};

template <int DP>
__host__ __device__ constexpr Swizzle dp_swizzle()
{
    return DP == 16 ? kSw32 : DP == 32 ? kSw64 : kSw128;
}

struct TileKind {
    bool loc, glob;
};

__device__ __forceinline__ TileKind tile_kind(int i0, int i_last, int j0, int w)
{
    const int min_d = i0 - (j0 + BN - 1), max_d = i_last - j0;
    TileKind k;
    k.glob = max_d >= w;
    k.loc = max(min_d, 0) <= min(max_d, w - 1);
    return k;
}

template <int N>
__device__ __forceinline__ float tree_max(const float (&v)[N])
{
    float t[N / 2];
#pragma unroll
    for (int e = 0; e < N / 2; ++e)
        t[e] = fmaxf(v[2 * e], v[2 * e + 1]);
#pragma unroll
    for (int n = N / 4; n >= 1; n /= 2)
#pragma unroll
        for (int e = 0; e < n; ++e)
            t[e] = fmaxf(t[e], t[e + n]);
    return t[0];
}

__device__ __forceinline__ float max3(float a, float b, float c)
{
    float d;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}

// Maximum of N values with the 3-input max.f32: four independent running
// maxima, two new values per step each.
template <int N>
__device__ __forceinline__ float tree_max3(const float (&v)[N])
{
    float m[4] = {v[0], v[1], v[2], v[3]};
#pragma unroll
    for (int e = 4; e + 8 <= N; e += 8)
#pragma unroll
        for (int k = 0; k < 4; ++k)
            m[k] = max3(m[k], v[e + 2 * k], v[e + 2 * k + 1]);
    constexpr int R = 4 + (N - 4) / 8 * 8;
#pragma unroll
    for (int e = R; e < N; ++e)
        m[e & 3] = fmaxf(m[e & 3], v[e]);
    return max3(m[0], m[1], fmaxf(m[2], m[3]));
}

template <int N>
__device__ __forceinline__ float tree_sum(const float (&v)[N])
{
    float t[N / 2];
#pragma unroll
    for (int e = 0; e < N / 2; ++e)
        t[e] = v[2 * e] + v[2 * e + 1];
#pragma unroll
    for (int n = N / 4; n >= 1; n /= 2)
#pragma unroll
        for (int e = 0; e < n; ++e)
            t[e] = t[e] + t[e + n];
    return t[0];
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi)
{
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t *>(&v);
}

// Write 8 bf16 values (one 16-byte chunk, logical chunk c) of row r of a
// K-major operand whose rows are RB bytes, with the matching TMA/MMA swizzle.
template <int RB>
__device__ __forceinline__ void st_swz(unsigned char *base, int r, int c, uint4 v)
{
    constexpr int mask = RB / 16 - 1;
    const int phys = c ^ ((r * RB >> 7) & mask);
    *reinterpret_cast<uint4 *>(base + (size_t)r * RB + phys * 16) = v;
}

template <int RB>
__device__ __forceinline__ uint4 ld_swz(const unsigned char *base, int r, int c)
{
    constexpr int mask = RB / 16 - 1;
    const int phys = c ^ ((r * RB >> 7) & mask);
    return *reinterpret_cast<const uint4 *>(base + (size_t)r * RB + phys * 16);
}

// Virtual tiles: a key tile whose pairs are all local or all global is one
// virtual tile; a band tile (the window edge crosses it) is two, its local
// part then its global part, each with the other part masked out.  All roles
// walk the same sequence, from the diagonal down to key 0.
struct VTile {
    int kt;    // key tile index (keys kt*BN .. kt*BN+BN-1)
    bool loc;  // local part (Q K^T, V) or global part (Q~ K^D^T, V^D)
    bool band; // the key tile also has the other part
};

__device__ __forceinline__ VTile vt_first(int i0, int i_last, int w)
{
    const int kt = i_last / BN;
    const TileKind k = tile_kind(i0, i_last, kt * BN, w);
    return VTile{kt, k.loc, k.loc && k.glob};
}

__device__ __forceinline__ VTile vt_next(VTile v, int i0, int i_last, int w)
{
    if (v.band && v.loc)
        return VTile{v.kt, false, true};
    const int kt = v.kt - 1;
    if (kt < 0)
        return VTile{-1, false, false};
    const TileKind k = tile_kind(i0, i_last, kt * BN, w);
    return VTile{kt, k.loc, k.loc && k.glob};
}

__device__ __forceinline__ int vt_count(int i0, int i_last, int w)
{
    int n = 0;
    for (VTile v = vt_first(i0, i_last, w); v.kt >= 0; v = vt_next(v, i0, i_last, w))
        ++n;
    return n;
}

template <int DP>
__global__ void __launch_bounds__(kThreads, 2)
    prefill_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmQT,
                      const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                      const __grid_constant__ CUtensorMap tmKD, const __grid_constant__ CUtensorMap tmVD,
                      PrefillArgs a)
{
    using Ly = Layout<DP>;
    using Tm = Tmem<DP>;
    constexpr int NS = Ly::NS;
    constexpr int NSB = Tm::NSB;
    extern __shared__ unsigned char smem_raw[];
    unsigned char *sm = reinterpret_cast<unsigned char *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t *bars = reinterpret_cast<uint64_t *>(sm + Ly::BAR);
    uint64_t *full = bars;                 // [NS] TMA -> MMA
    uint64_t *empty = bars + NS;           // [NS] MMA -> TMA
    uint64_t *s_full = bars + 2 * NS;      // [NSB] S of a virtual tile computed
    uint64_t *q_full = s_full + NSB;       // Q and q~ landed
    uint64_t *qt_ready = q_full + 1;       // O zeroed (128 arrivals)
    uint64_t *p_full = q_full + 2;         // P written to TMEM (128 arrivals)
    uint64_t *pv_done = q_full + 3;        // PV of a virtual tile finished
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(q_full + 4);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int N = a.N, w = a.w;
    const int nqt = (N + BM - 1) / BM;
    const int qt = nqt - 1 - (int)blockIdx.y;  // longest rows first
    const int bh = blockIdx.x, b = bh / a.Hq, h = bh % a.Hq, g = h / (a.Hq / a.Hkv);
    const int i0 = qt * BM, i_last = min(i0 + BM, N) - 1;
    const int VT = vt_count(i0, i_last, w);

    if (threadIdx.x == 0) {
        for (int s = 0; s < NS; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int b2 = 0; b2 < NSB; ++b2)
            mbar_init(&s_full[b2], 1);
        mbar_init(q_full, 1);
        mbar_init(qt_ready, 128);
        mbar_init(p_full, 128);
        mbar_init(pv_done, 1);
        *abort_flag = 0;
        mbar_init_fence();
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            prefetch_tensormap(&tmQ);
            prefetch_tensormap(&tmQT);
            prefetch_tensormap(&tmK);
            prefetch_tensormap(&tmV);
            prefetch_tensormap(&tmKD);
            prefetch_tensormap(&tmVD);
            mbar_expect_tx(q_full, BM * 64 * 2 + BM * DP * 2);
            tma_load_2d(sm + Ly::Q, &tmQ, 0, (b * a.Hq + h) * N + i0, q_full);
            tma_load_2d(sm + Ly::QT, &tmQT, 0, (b * a.Hq + h) * N + i0, q_full);
            VTile vt = vt_first(i0, i_last, w);
            for (int t = 0; t < VT; ++t, vt = vt_next(vt, i0, i_last, w)) {
                const int s = t % NS;
                if (t >= NS && !mbar_wait(&empty[s], ((t / NS) - 1) & 1, abort_flag))
                    break;
                unsigned char *st = sm + Ly::STG + s * Ly::STAGE;
                const int krow = (b * a.Hkv + g) * N + vt.kt * BN;
                if (vt.loc) {
                    mbar_expect_tx(&full[s], 2 * BN * 64 * 2);
                    tma_load_2d(st + Ly::K_OFF, &tmK, 0, krow, &full[s]);
                    tma_load_2d(st + Ly::V_OFF, &tmV, 0, krow, &full[s]);
                } else {
                    mbar_expect_tx(&full[s], 2 * BN * DP * 2);
                    tma_load_2d(st + Ly::KD_OFF, &tmKD, 0, krow, &full[s]);
                    tma_load_2d(st + Ly::VD_OFF, &tmVD, 0, krow, &full[s]);
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t idS = idesc_bf16(BM, BN, false);
            constexpr uint32_t idPV = idesc_bf16(BM, 64, true);
            constexpr uint32_t idPVg = idesc_bf16(BM, DP, true);
            const uint32_t sQ = smem_u32(sm + Ly::Q), sQT = smem_u32(sm + Ly::QT);
            bool ok = mbar_wait(qt_ready, 0, abort_flag);
            tc_fence_after();
            auto issue_S = [&](int t, VTile vt) -> bool {
                const int s = t % NS, sb = t % NSB;
                if (!mbar_wait(&full[s], (t / NS) & 1, abort_flag))
                    return false;
                tc_fence_after();
                const uint32_t st = smem_u32(sm + Ly::STG + s * Ly::STAGE);
                const uint32_t dS = tmem + Tm::S + sb * BN;
                if (vt.loc)
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk)
                        mma_f16_ss(dS, smem_desc(sQ + kk * 32, 16, 1024, kSw128),
                                   smem_desc(st + Ly::K_OFF + kk * 32, 16, 1024, kSw128), idS, kk > 0);
                else
#pragma unroll
                    for (int kk = 0; kk < DP / 16; ++kk)
                        mma_f16_ss(dS, smem_desc(sQT + kk * 32, 16, 8 * DP * 2, dp_swizzle<DP>()),
                                   smem_desc(st + Ly::KD_OFF + kk * 32, 16, 8 * DP * 2, dp_swizzle<DP>()), idS,
                                   kk > 0);
                mma_commit(&s_full[sb]);
                return true;
            };
            auto issue_PV = [&](int t, VTile vt) -> bool {
                const int s = t % NS;
                if (!mbar_wait(p_full, t & 1, abort_flag))
                    return false;
                tc_fence_after();
                const uint32_t st = smem_u32(sm + Ly::STG + s * Ly::STAGE);
                const uint32_t P = tmem + Tm::P;
#pragma unroll
                for (int kk = 0; kk < BN / 16; ++kk) {  // P (TMEM, 8 columns per 16 keys) times V / V^D
                    const uint32_t aP = P + kk * 8;
                    if (vt.loc)
                        mma_f16_ts(tmem + Tm::OL, aP, smem_desc(st + Ly::V_OFF + kk * 16 * 128, 16, 1024, kSw128),
                                   idPV, true);
                    else
                        mma_f16_ts(tmem + Tm::OG, aP,
                                   smem_desc(st + Ly::VD_OFF + kk * 16 * DP * 2, 16, 8 * DP * 2, dp_swizzle<DP>()),
                                   idPVg, true);
                }
                mma_commit(pv_done);
                mma_commit(&empty[s]);
                return true;
            };
            // S runs NSB virtual tiles ahead: S(t + NSB) reuses the buffer of S(t),
            // which P(t) being written proves the softmax has read
            VTile vs = vt_first(i0, i_last, w), vp = vs;
            for (int t = 0; ok && t < NSB && t < VT; ++t) {
                ok = issue_S(t, vs);
                vs = vt_next(vs, i0, i_last, w);
            }
            for (int t = 0; ok && t < VT; ++t) {
                ok = issue_PV(t, vp);
                vp = vt_next(vp, i0, i_last, w);
                if (ok && t + NSB < VT) {
                    ok = issue_S(t + NSB, vs);
                    vs = vt_next(vs, i0, i_last, w);
                }
            }
        }
    } else {
        // ------------------------------------------------------------ softmax warps
        const int quad = warp & 3;
        const int row = 32 * quad + lane;
        const int i = i0 + row;
        const uint32_t tl = tmem + ((uint32_t)(32 * quad) << 16);
        const int stid = threadIdx.x - 64;  // 0..127
        float *sUv = reinterpret_cast<float *>(sm + Ly::UV);
        for (int idx = stid; idx < DP * 64; idx += 128) {
            const int c = idx / 64, t = idx % 64;
            sUv[idx] = c < a.dd ? a.Uv[((size_t)g * a.dd + c) * 64 + t] : 0.f;
        }
        asm volatile("bar.sync 1, 128;" ::: "memory");
        // tcgen05.ld/st are warp-collective: every branch around them is warp-uniform
        auto wait_uniform = [&](uint64_t *bar, unsigned parity) {
            const bool r = mbar_wait(bar, parity, abort_flag);
            return __all_sync(0xffffffffu, r) != 0;
        };
        bool ok = wait_uniform(q_full, 0);
        {  // zero the accumulators
            uint32_t z[16];
#pragma unroll
            for (int e = 0; e < 16; ++e)
                z[e] = 0u;
#pragma unroll
            for (int c = 0; c < 64; c += 16)
                tmem_st16(tl + Tm::OL + c, z);
#pragma unroll
            for (int c = 0; c < DP; c += 16)
                tmem_st16(tl + Tm::OG + c, z);
            tmem_wait_st();
        }
        tc_fence_before();
        mbar_arrive(qt_ready);

        const float c2 = a.qscale;  // softmax scale * log2(e)
        float m_used = -INFINITY, l = 0.f;
        int pv_waited = -1;  // highest virtual tile whose PV completion has been observed
        VTile vt = vt_first(i0, i_last, w);
        for (int t = 0; ok && t < VT; ++t, vt = vt_next(vt, i0, i_last, w)) {
            const int j0 = vt.kt * BN;
            const int sb = t % NSB;
            if (!wait_uniform(&s_full[sb], (t / NSB) & 1)) {
                ok = false;
                break;
            }
            tc_fence_after();
            float s[BN];
            {
                uint32_t r[BN];  // both halves in flight, one wait
                tmem_ld32_nowait(tl + Tm::S + sb * BN, *reinterpret_cast<uint32_t(*)[32]>(&r[0]));
                tmem_ld32_nowait(tl + Tm::S + sb * BN + 32, *reinterpret_cast<uint32_t(*)[32]>(&r[32]));
                tmem_wait_ld_regs(r);
#pragma unroll
                for (int e = 0; e < BN; ++e)
                    s[e] = __uint_as_float(r[e]);
            }
            // masks: causal (tiles reaching past row i0), the other part of a
            // band tile, rows past the end
            if (j0 + BN - 1 > i0 || vt.band || i >= N) {
#pragma unroll
                for (int e = 0; e < BN; ++e) {
                    const int j = j0 + e;
                    const bool keep = j <= i && i < N && (!vt.band || ((i - j < w) == vt.loc));
                    s[e] = keep ? s[e] : -INFINITY;
                }
            }
            const float mt = tree_max3(s) * c2;
            // raise the running max only when it grows by more than the threshold
            const bool raise = mt > m_used + kRescaleThreshold;
            const bool scale_o = raise && m_used != -INFINITY;
            const float alpha = scale_o ? ex2_approx(m_used - mt) : 1.f;
            if (__any_sync(0xffffffffu, scale_o)) {
                // every earlier PV must have landed before O is rescaled
                if (pv_waited < t - 1) {
                    if (!wait_uniform(pv_done, (t - 1) & 1)) {
                        ok = false;
                        break;
                    }
                    pv_waited = t - 1;
                    tc_fence_after();
                }
#pragma unroll
                for (int c = 0; c < 64; c += 16) {
                    uint32_t r[16];
                    tmem_ld16(tl + Tm::OL + c, r);
#pragma unroll
                    for (int e = 0; e < 16; ++e)
                        r[e] = __float_as_uint(__uint_as_float(r[e]) * alpha);
                    tmem_st16(tl + Tm::OL + c, r);
                }
#pragma unroll
                for (int c = 0; c < DP; c += 16) {
                    uint32_t r[16];
                    tmem_ld16(tl + Tm::OG + c, r);
#pragma unroll
                    for (int e = 0; e < 16; ++e)
                        r[e] = __float_as_uint(__uint_as_float(r[e]) * alpha);
                    tmem_st16(tl + Tm::OG + c, r);
                }
            }
            l *= alpha;
            if (raise)
                m_used = mt;
            // P = 2^(s * c2 - m) (masked entries give 0); the PV of the previous
            // virtual tile must be done reading the P columns
            const float mneg = m_used == -INFINITY ? 0.f : -m_used;
            uint32_t pk[BN / 2];
            float ls = 0.f;
#pragma unroll
            for (int e = 0; e < BN; e += 2) {
                const float p0 = ex2_approx(fmaf(s[e], c2, mneg));
                const float p1 = ex2_approx(fmaf(s[e + 1], c2, mneg));
                ls += p0 + p1;
                pk[e / 2] = pack_bf16(p0, p1);
            }
            l += ls;
            if (t > 0 && pv_waited < t - 1) {
                if (!wait_uniform(pv_done, (t - 1) & 1)) {
                    ok = false;
                    break;
                }
                pv_waited = t - 1;
                tc_fence_after();
            }
            tmem_st16(tl + Tm::P, *reinterpret_cast<const uint32_t(*)[16]>(&pk[0]));
            tmem_st16(tl + Tm::P + 16, *reinterpret_cast<const uint32_t(*)[16]>(&pk[16]));
            tmem_wait_st();
            tc_fence_before();
            mbar_arrive(p_full);
        }

        // ---- epilogue: o = (O_loc + O_glob Uv) / l
        // every PV before the last has been waited for (before writing P)
        if (ok && wait_uniform(pv_done, (VT - 1) & 1)) {
            tc_fence_after();
            float og[DP];
#pragma unroll
            for (int c = 0; c < DP; c += 16) {
                uint32_t r[16];
                tmem_ld16(tl + Tm::OG + c, r);
#pragma unroll
                for (int e = 0; e < 16; ++e)
                    og[c + e] = __uint_as_float(r[e]);
            }
            const float inv = l > 0.f ? 1.f / l : 0.f;
            bf16 *orow = static_cast<bf16 *>(a.out) + (((size_t)b * a.Hq + h) * N + i) * 64;
#pragma unroll
            for (int c = 0; c < 64; c += 16) {
                uint32_t r[16];
                tmem_ld16(tl + Tm::OL + c, r);
                float o[16];
#pragma unroll
                for (int e = 0; e < 16; ++e)
                    o[e] = __uint_as_float(r[e]);
#pragma unroll
                for (int kk = 0; kk < DP; ++kk) {
                    const float4 *u4 = reinterpret_cast<const float4 *>(sUv + kk * 64 + c);
#pragma unroll
                    for (int e4 = 0; e4 < 4; ++e4) {
                        const float4 u = u4[e4];
                        o[4 * e4 + 0] = fmaf(og[kk], u.x, o[4 * e4 + 0]);
                        o[4 * e4 + 1] = fmaf(og[kk], u.y, o[4 * e4 + 1]);
                        o[4 * e4 + 2] = fmaf(og[kk], u.z, o[4 * e4 + 2]);
                        o[4 * e4 + 3] = fmaf(og[kk], u.w, o[4 * e4 + 3]);
                    }
                }
#pragma unroll
                for (int e = 0; e < 16; ++e)
                    o[e] *= inv;
                if (i < N) {
                    uint4 *dst = reinterpret_cast<uint4 *>(orow + c);
                    dst[0] = make_uint4(pack_bf16(o[0], o[1]), pack_bf16(o[2], o[3]), pack_bf16(o[4], o[5]),
                                        pack_bf16(o[6], o[7]));
                    dst[1] = make_uint4(pack_bf16(o[8], o[9]), pack_bf16(o[10], o[11]), pack_bf16(o[12], o[13]),
                                        pack_bf16(o[14], o[15]));
                }
            }
        } else {
            ok = false;
        }
        if (!ok)
            *abort_flag = 1;
    }

    // ---- teardown
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (threadIdx.x == 0 && *abort_flag)
        report(a.status, DAR_ERR_DEVICE);
    if (warp == 1)
        tmem_dealloc(tmem, kTmemCols);
}

// ---------------------------------------------------------------- host side

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn()
{
    static EncodeTiledFn fn = nullptr;
    if (!fn) {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    }
    return fn;
}

// 2-D bf16 tensor [rows][cols] with a row pitch of `pitch` elements (0: cols),
// box [box_rows][cols].
static bool make_map(CUtensorMap *m, const void *base, unsigned long long rows, int cols, int box_rows,
                     CUtensorMapSwizzle sw, int pitch = 0)
{
    EncodeTiledFn fn = encode_fn();
    if (!fn)
        return false;
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)(pitch > 0 ? pitch : cols) * 2};
    cuuint32_t box[2] = {(cuuint32_t)cols, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int DP>
static cudaError_t launch_dp(const PrefillArgs &a, cudaStream_t s)
{
    CUtensorMap mq, mqt, mk, mv, mkd, mvd;
    const CUtensorMapSwizzle swd = DP == 16 ? CU_TENSOR_MAP_SWIZZLE_32B
                                   : DP == 32 ? CU_TENSOR_MAP_SWIZZLE_64B
                                              : CU_TENSOR_MAP_SWIZZLE_128B;
    const unsigned long long rq = (unsigned long long)a.B * a.Hq * a.N, rk = (unsigned long long)a.B * a.Hkv * a.N;
    // q~ sits in the first DP entries of each output row (written by the pre-pass)
    if (!make_map(&mq, a.q, rq, 64, BM, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&mqt, a.out, rq, DP, BM, swd, 64) ||
        !make_map(&mk, a.k, rk, 64, BN, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&mv, a.v, rk, 64, BN, CU_TENSOR_MAP_SWIZZLE_128B) || !make_map(&mkd, a.kd, rk, DP, BN, swd) ||
        !make_map(&mvd, a.vd, rk, DP, BN, swd))
        return cudaErrorInvalidValue;
    auto kern = prefill_tc_kernel<DP>;
    const size_t smem = Layout<DP>::TOTAL + 1024;
    static PerDeviceOnce once;
    cudaError_t e = per_device_once(once, [&](int) {
        return cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    });
    if (e != cudaSuccess)
        return e;
    dim3 grid(a.B * a.Hq, (a.N + BM - 1) / BM);
    kern<<<grid, kThreads, smem, s>>>(mq, mqt, mk, mv, mkd, mvd, a);
    return cudaGetLastError();
}

// ---------------------------------------------------------------- q~ pre-pass

// q~ = q Uk^T for every query row (fp32 chains, rounded once to bf16), written
// into the first DP entries of the row's output slot (entries dd..DP-1 zero):
// the CTA that owns a row reads its q~ before it writes the row's output.
// grid (ceil(N / 128), B * Hq), 128 threads, one row per thread.
template <int DP>
__global__ void __launch_bounds__(128) qtilde_kernel(const bf16 *__restrict__ q, const float *__restrict__ Uk,
                                                     bf16 *__restrict__ out, int Hq, int G, int dd, int N)
{
    __shared__ __align__(16) float sUk[DP * 64];
    const int bh = blockIdx.y, g = (bh % Hq) / G;
    for (int i = threadIdx.x; i < DP * 64; i += blockDim.x)
        sUk[i] = i / 64 < dd ? Uk[((size_t)g * dd + i / 64) * 64 + i % 64] : 0.f;
    __syncthreads();
    const int j = blockIdx.x * blockDim.x + threadIdx.x;
    if (j >= N)
        return;
    const size_t row = (size_t)bh * N + j;
    float x[64];
    const uint4 *q4 = reinterpret_cast<const uint4 *>(q + row * 64);
#pragma unroll
    for (int c = 0; c < 8; ++c) {
        const uint4 v = q4[c];
        x[8 * c + 0] = bf16lo(v.x);
        x[8 * c + 1] = bf16hi(v.x);
        x[8 * c + 2] = bf16lo(v.y);
        x[8 * c + 3] = bf16hi(v.y);
        x[8 * c + 4] = bf16lo(v.z);
        x[8 * c + 5] = bf16hi(v.z);
        x[8 * c + 6] = bf16lo(v.w);
        x[8 * c + 7] = bf16hi(v.w);
    }
    uint4 *o4 = reinterpret_cast<uint4 *>(out + row * 64);
#pragma unroll 1
    for (int c8 = 0; c8 < DP / 8; ++c8) {
        float o[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const float4 *u4 = reinterpret_cast<const float4 *>(sUk + (c8 * 8 + e) * 64);
            float a0 = 0.f, a1 = 0.f;
#pragma unroll
            for (int t4 = 0; t4 < 16; ++t4) {
                const float4 u = u4[t4];
                a0 = fmaf(x[4 * t4 + 0], u.x, a0);
                a1 = fmaf(x[4 * t4 + 1], u.y, a1);
                a0 = fmaf(x[4 * t4 + 2], u.z, a0);
                a1 = fmaf(x[4 * t4 + 3], u.w, a1);
            }
            o[e] = a0 + a1;
        }
        o4[c8] = make_uint4(pack_bf16(o[0], o[1]), pack_bf16(o[2], o[3]), pack_bf16(o[4], o[5]),
                            pack_bf16(o[6], o[7]));
    }
}

template <int DP>
static cudaError_t launch_qtilde(const PrefillArgs &a, cudaStream_t s)
{
    dim3 grid((a.N + 127) / 128, a.B * a.Hq);
    qtilde_kernel<DP><<<grid, 128, 0, s>>>(static_cast<const bf16 *>(a.q), a.Uk, static_cast<bf16 *>(a.out), a.Hq,
                                           a.Hq / a.Hkv, a.dd, a.N);
    return cudaGetLastError();
}

}  // namespace tcp

bool make_tma_2d_bf16(CUtensorMap *map, const void *base, unsigned long long rows, int cols, int box_rows)
{
    const CUtensorMapSwizzle sw = cols == 8    ? CU_TENSOR_MAP_SWIZZLE_NONE
                                  : cols == 16 ? CU_TENSOR_MAP_SWIZZLE_32B
                                  : cols == 32 ? CU_TENSOR_MAP_SWIZZLE_64B
                                               : CU_TENSOR_MAP_SWIZZLE_128B;
    return tcp::make_map(map, base, rows, cols, box_rows, sw);
}

cudaError_t launch_prefill_tc(int dd, const PrefillArgs &a, cudaStream_t s)
{
    if (a.B == 0 || a.N == 0)
        return cudaSuccess;
    cudaError_t e;
    switch (a.kd_stride) {
    case 16: e = tcp::launch_qtilde<16>(a, s); return e != cudaSuccess ? e : tcp::launch_dp<16>(a, s);
    case 32: e = tcp::launch_qtilde<32>(a, s); return e != cudaSuccess ? e : tcp::launch_dp<32>(a, s);
    case 64: e = tcp::launch_qtilde<64>(a, s); return e != cudaSuccess ? e : tcp::launch_dp<64>(a, s);
    default: return cudaErrorInvalidValue;
    }
}

}  // namespace dar
