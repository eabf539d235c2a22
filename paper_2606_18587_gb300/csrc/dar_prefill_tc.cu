// dar_prefill_tc.cu -- causal DAR attention forward (bf16) on the 5th-generation
// tensor cores: tcgen05.mma with operands in shared memory (staged by TMA) and
// fp32 accumulators in tensor memory (TMEM).
//
// One CTA = 128 query rows of one head; key tiles of 64, visited from the
// diagonal down to key 0.  Per key tile (Eq. 3: local iff i - j < w):
//   local part   S_loc  = Q  K^T       (M128 N64 K64)   O_loc  += P_loc  V    (N64)
//   global part  S_glob = Q~ (K^D)^T   (M128 N64 Kdd)   O_glob += P_glob V^D  (Ndd)
// with q~ = q Uk^T (W_up absorbed into the query, exact by linearity of
// Eq. 2).  A tile issues only the parts it needs; a band tile (both kinds)
// selects per element.  One online softmax over both parts (Eq. 4), with the
// running max raised lazily (only when it grows by more than 2^8), and the
// epilogue lifts the global part once:  o = (O_loc + O_glob Uv) / l.
//
// Warp roles (192 threads): warp 0 issues TMA loads, warp 1 allocates TMEM and
// issues the MMAs (one thread), warps 2-5 own one query row per thread
// (TMEM lane = row) for q~, the softmax and the epilogue.  256 TMEM columns
// and ~100 KB of shared memory per CTA let two CTAs share an SM, so one CTA's
// softmax overlaps the other's MMA and load waits.  Every wait is bounded; on
// a timeout the CTA flags *status and exits.
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
constexpr uint32_t COL_SL = 0, COL_SG = 64, COL_OL = 128, COL_OG = 192;
constexpr float kRescaleThreshold = 8.0f;  // log2 units: p stays below 2^8 between rescales

constexpr uint32_t align_up(uint32_t x, uint32_t a) { return (x + a - 1) / a * a; }

// Shared-memory layout (offsets from a 1024-byte aligned base).
template <int DP>
struct Layout {
    static constexpr int NS = 2;                          // K/V stages
    static constexpr uint32_t Q = 0;                      // [128][64] bf16, 128B swizzle
    static constexpr uint32_t QT = BM * 64 * 2;           // [128][DP] bf16
    static constexpr uint32_t STG = align_up(QT + BM * DP * 2, 1024);
    static constexpr uint32_t K_OFF = 0;                  // [64][64]
    static constexpr uint32_t V_OFF = BN * 64 * 2;        // [64][64]
    static constexpr uint32_t KD_OFF = 2 * BN * 64 * 2;   // [64][DP]
    static constexpr uint32_t VD_OFF = KD_OFF + BN * DP * 2;
    static constexpr uint32_t STAGE = align_up(VD_OFF + BN * DP * 2, 1024);
    static constexpr uint32_t PL = STG + NS * STAGE;      // P_loc  [128][64] bf16 (one 128B-swizzle atom wide)
    static constexpr uint32_t PG = PL + BM * BN * 2;      // P_glob
    static constexpr uint32_t UK = PG + BM * BN * 2;      // fp32 [DP][64]
    static constexpr uint32_t UV = UK + DP * 64 * 4;
    static constexpr uint32_t BAR = UV + DP * 64 * 4;
    static constexpr uint32_t TOTAL = BAR + 256;
    static_assert(STAGE % 1024 == 0 && STG % 1024 == 0, "operand tiles must stay 1024-byte aligned");
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

template <int DP>
__global__ void __launch_bounds__(kThreads, 2)
    prefill_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                      const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmKD,
                      const __grid_constant__ CUtensorMap tmVD, PrefillArgs a)
{
    using Ly = Layout<DP>;
    constexpr int NS = Ly::NS;
    extern __shared__ unsigned char smem_raw[];
    unsigned char *sm = reinterpret_cast<unsigned char *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t *bars = reinterpret_cast<uint64_t *>(sm + Ly::BAR);
    uint64_t *full = bars;            // [NS] TMA -> MMA
    uint64_t *empty = bars + NS;      // [NS] MMA -> TMA
    uint64_t *q_full = bars + 2 * NS; // Q landed
    uint64_t *qt_ready = q_full + 1;  // q~ written, O zeroed (128 arrivals)
    uint64_t *s_full = q_full + 2;    // S of a tile computed
    uint64_t *s_free = q_full + 3;    // S read into registers (128 arrivals)
    uint64_t *p_full = q_full + 4;    // P written (128 arrivals)
    uint64_t *pv_done = q_full + 5;   // PV of a tile finished
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(q_full + 6);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int N = a.N, w = a.w;
    const int nqt = (N + BM - 1) / BM;
    const int qt = nqt - 1 - (int)blockIdx.y;  // longest rows first
    const int bh = blockIdx.x, b = bh / a.Hq, h = bh % a.Hq, g = h / (a.Hq / a.Hkv);
    const int i0 = qt * BM, i_last = min(i0 + BM, N) - 1;
    const int T = i_last / BN + 1;  // key tiles kt = T-1-t, t = 0..T-1

    if (threadIdx.x == 0) {
        for (int s = 0; s < NS; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_init(q_full, 1);
        mbar_init(qt_ready, 128);
        mbar_init(s_full, 1);
        mbar_init(s_free, 128);
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
            prefetch_tensormap(&tmK);
            prefetch_tensormap(&tmV);
            prefetch_tensormap(&tmKD);
            prefetch_tensormap(&tmVD);
            mbar_expect_tx(q_full, BM * 64 * 2);
            tma_load_2d(sm + Ly::Q, &tmQ, 0, (b * a.Hq + h) * N + i0, q_full);
            for (int t = 0; t < T; ++t) {
                const int s = t % NS;
                if (t >= NS && !mbar_wait(&empty[s], ((t / NS) - 1) & 1, abort_flag))
                    break;
                const int j0 = (T - 1 - t) * BN;
                const TileKind k = tile_kind(i0, i_last, j0, w);
                const unsigned bytes = (k.loc ? 2 * BN * 64 * 2 : 0) + (k.glob ? 2 * BN * DP * 2 : 0);
                unsigned char *st = sm + Ly::STG + s * Ly::STAGE;
                const int krow = (b * a.Hkv + g) * N + j0;
                mbar_expect_tx(&full[s], bytes);
                if (k.loc) {
                    tma_load_2d(st + Ly::K_OFF, &tmK, 0, krow, &full[s]);
                    tma_load_2d(st + Ly::V_OFF, &tmV, 0, krow, &full[s]);
                }
                if (k.glob) {
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
            const uint32_t sPL = smem_u32(sm + Ly::PL), sPG = smem_u32(sm + Ly::PG);
            bool ok = mbar_wait(qt_ready, 0, abort_flag);
            tc_fence_after();
            auto issue_S = [&](int t) -> bool {
                const int s = t % NS;
                if (!mbar_wait(&full[s], (t / NS) & 1, abort_flag))
                    return false;
                if (t > 0 && !mbar_wait(s_free, (t - 1) & 1, abort_flag))
                    return false;
                tc_fence_after();
                const TileKind k = tile_kind(i0, i_last, (T - 1 - t) * BN, w);
                const uint32_t st = smem_u32(sm + Ly::STG + s * Ly::STAGE);
                if (k.loc)
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk)
                        mma_f16_ss(tmem + COL_SL, smem_desc(sQ + kk * 32, 16, 1024, kSw128),
                                   smem_desc(st + Ly::K_OFF + kk * 32, 16, 1024, kSw128), idS, kk > 0);
                if (k.glob)
#pragma unroll
                    for (int kk = 0; kk < DP / 16; ++kk)
                        mma_f16_ss(tmem + COL_SG, smem_desc(sQT + kk * 32, 16, 8 * DP * 2, dp_swizzle<DP>()),
                                   smem_desc(st + Ly::KD_OFF + kk * 32, 16, 8 * DP * 2, dp_swizzle<DP>()), idS,
                                   kk > 0);
                mma_commit(s_full);
                return true;
            };
            auto issue_PV = [&](int t) -> bool {
                const int s = t % NS;
                if (!mbar_wait(p_full, t & 1, abort_flag))
                    return false;
                tc_fence_after();
                const TileKind k = tile_kind(i0, i_last, (T - 1 - t) * BN, w);
                const uint32_t st = smem_u32(sm + Ly::STG + s * Ly::STAGE);
#pragma unroll
                for (int kk = 0; kk < BN / 16; ++kk) {
                    const uint32_t aoff = kk * 32;
                    if (k.loc)
                        mma_f16_ss(tmem + COL_OL, smem_desc(sPL + aoff, 16, 1024, kSw128),
                                   smem_desc(st + Ly::V_OFF + kk * 16 * 128, 16, 1024, kSw128), idPV, true);
                    if (k.glob)
                        mma_f16_ss(tmem + COL_OG, smem_desc(sPG + aoff, 16, 1024, kSw128),
                                   smem_desc(st + Ly::VD_OFF + kk * 16 * DP * 2, 16, 8 * DP * 2,
                                             dp_swizzle<DP>()),
                                   idPVg, true);
                }
                mma_commit(pv_done);
                mma_commit(&empty[s]);
                return true;
            };
            // S(t) is issued as soon as the softmax has read S(t-1), so it
            // overlaps the softmax of tile t-1; PV(t-1) follows once P(t-1) is written
            for (int t = 0; ok && t <= T; ++t) {
                if (t < T)
                    ok = issue_S(t);
                if (ok && t > 0)
                    ok = issue_PV(t - 1);
            }
        }
    } else {
        // ------------------------------------------------------------ softmax warps
        const int quad = warp & 3;
        const int row = 32 * quad + lane;
        const int i = i0 + row;
        const uint32_t tl = tmem + ((uint32_t)(32 * quad) << 16);
        const int stid = threadIdx.x - 64;  // 0..127
        float *sUk = reinterpret_cast<float *>(sm + Ly::UK);
        float *sUv = reinterpret_cast<float *>(sm + Ly::UV);
        for (int idx = stid; idx < DP * 64; idx += 128) {
            const int c = idx / 64, t = idx % 64;
            const bool in = c < a.dd;
            sUk[idx] = in ? a.Uk[((size_t)g * a.dd + c) * 64 + t] : 0.f;
            sUv[idx] = in ? a.Uv[((size_t)g * a.dd + c) * 64 + t] : 0.f;
        }
        asm volatile("bar.sync 1, 128;" ::: "memory");
        // tcgen05.ld/st are warp-collective: every branch around them is warp-uniform
        auto wait_uniform = [&](uint64_t *bar, unsigned parity) {
            const bool r = mbar_wait(bar, parity, abort_flag);
            return __all_sync(0xffffffffu, r) != 0;
        };
        bool ok = wait_uniform(q_full, 0);

        // q~ row = q Uk^T  (fp32, rounded once to bf16 for the MMA)
        {
            float q[64];
#pragma unroll
            for (int c = 0; c < 8; ++c) {
                const uint4 v = ld_swz<128>(sm + Ly::Q, row, c);
                q[8 * c + 0] = bf16lo(v.x);
                q[8 * c + 1] = bf16hi(v.x);
                q[8 * c + 2] = bf16lo(v.y);
                q[8 * c + 3] = bf16hi(v.y);
                q[8 * c + 4] = bf16lo(v.z);
                q[8 * c + 5] = bf16hi(v.z);
                q[8 * c + 6] = bf16lo(v.w);
                q[8 * c + 7] = bf16hi(v.w);
            }
#pragma unroll 1
            for (int c8 = 0; c8 < DP / 8; ++c8) {
                float o[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const float *u = sUk + (c8 * 8 + e) * 64;
                    float a0 = 0.f, a1 = 0.f;
#pragma unroll
                    for (int t = 0; t < 64; t += 2) {
                        a0 = fmaf(q[t], u[t], a0);
                        a1 = fmaf(q[t + 1], u[t + 1], a1);
                    }
                    o[e] = a0 + a1;
                }
                st_swz<DP * 2>(sm + Ly::QT, row, c8,
                               make_uint4(pack_bf16(o[0], o[1]), pack_bf16(o[2], o[3]), pack_bf16(o[4], o[5]),
                                          pack_bf16(o[6], o[7])));
            }
        }
        {  // zero the accumulators
            uint32_t z[16];
#pragma unroll
            for (int e = 0; e < 16; ++e)
                z[e] = 0u;
#pragma unroll
            for (int c = 0; c < 64 + DP; c += 16)
                tmem_st16(tl + COL_OL + c, z);
            tmem_wait_st();
        }
        fence_proxy_async_smem();
        tc_fence_before();
        mbar_arrive(qt_ready);

        const float c2 = a.qscale;  // softmax scale * log2(e)
        float m_used = -INFINITY, l = 0.f;
        int pv_waited = -1;  // highest tile whose PV completion has been observed
        for (int t = 0; ok && t < T; ++t) {
            const int j0 = (T - 1 - t) * BN;
            const TileKind k = tile_kind(i0, i_last, j0, w);
            const bool band = k.loc && k.glob;
            if (!wait_uniform(s_full, t & 1)) {
                ok = false;
                break;
            }
            tc_fence_after();
            float s[BN];
#pragma unroll
            for (int c = 0; c < BN; c += 32) {
                uint32_t r[32];
                tmem_ld32(tl + (k.loc ? COL_SL : COL_SG) + c, r);
                if (band) {
                    uint32_t r2[32];
                    tmem_ld32(tl + COL_SG + c, r2);
#pragma unroll
                    for (int e = 0; e < 32; ++e)
                        s[c + e] = (i - (j0 + c + e) < w) ? __uint_as_float(r[e]) : __uint_as_float(r2[e]);
                } else {
#pragma unroll
                    for (int e = 0; e < 32; ++e)
                        s[c + e] = __uint_as_float(r[e]);
                }
            }
            tc_fence_before();
            mbar_arrive(s_free);
            // causal mask (tiles reaching past row i0) and rows past the end
            if (j0 + BN - 1 > i0 || i >= N) {
#pragma unroll
                for (int e = 0; e < BN; ++e)
                    if (j0 + e > i || i >= N)
                        s[e] = -INFINITY;
            }
            const float mt = tree_max(s) * c2;
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
                for (int c = 0; c < 64 + DP; c += 16) {
                    uint32_t r[16];
                    tmem_ld16(tl + COL_OL + c, r);
#pragma unroll
                    for (int e = 0; e < 16; ++e)
                        r[e] = __float_as_uint(__uint_as_float(r[e]) * alpha);
                    tmem_st16(tl + COL_OL + c, r);
                }
                tmem_wait_st();
            }
            l *= alpha;
            if (raise)
                m_used = mt;
            // P = 2^(s * c2 - m); masked entries (s = -inf) give 0
            const float mneg = m_used == -INFINITY ? 0.f : -m_used;
#pragma unroll
            for (int e = 0; e < BN; ++e)
                s[e] = ex2_approx(fmaf(s[e], c2, mneg));
            l += tree_sum(s);
            // the PV of the previous tile must be done reading the P buffers
            if (t > 0 && pv_waited < t - 1) {
                if (!wait_uniform(pv_done, (t - 1) & 1)) {
                    ok = false;
                    break;
                }
                pv_waited = t - 1;
                tc_fence_after();
            }
#pragma unroll
            for (int c = 0; c < BN / 8; ++c) {
                float vl[8], vg[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const int j = j0 + 8 * c + e;
                    const bool is_loc = band ? (i - j < w) : k.loc;
                    vl[e] = is_loc ? s[8 * c + e] : 0.f;
                    vg[e] = is_loc ? 0.f : s[8 * c + e];
                }
                if (k.loc)
                    st_swz<128>(sm + Ly::PL, row, c,
                                make_uint4(pack_bf16(vl[0], vl[1]), pack_bf16(vl[2], vl[3]),
                                           pack_bf16(vl[4], vl[5]), pack_bf16(vl[6], vl[7])));
                if (k.glob)
                    st_swz<128>(sm + Ly::PG, row, c,
                                make_uint4(pack_bf16(vg[0], vg[1]), pack_bf16(vg[2], vg[3]),
                                           pack_bf16(vg[4], vg[5]), pack_bf16(vg[6], vg[7])));
            }
            fence_proxy_async_smem();
            tc_fence_before();
            mbar_arrive(p_full);
        }

        // ---- epilogue: o = (O_loc + O_glob Uv) / l
        if (ok && wait_uniform(pv_done, (T - 1) & 1)) {
            tc_fence_after();
            float og[DP];
#pragma unroll
            for (int c = 0; c < DP; c += 16) {
                uint32_t r[16];
                tmem_ld16(tl + COL_OG + c, r);
                tmem_wait_ld();
#pragma unroll
                for (int e = 0; e < 16; ++e)
                    og[c + e] = __uint_as_float(r[e]);
            }
            const float inv = l > 0.f ? 1.f / l : 0.f;
            bf16 *orow = static_cast<bf16 *>(a.out) + (((size_t)b * a.Hq + h) * N + i) * 64;
#pragma unroll
            for (int c = 0; c < 64; c += 16) {
                uint32_t r[16];
                tmem_ld16(tl + COL_OL + c, r);
                tmem_wait_ld();
                float o[16];
#pragma unroll
                for (int e = 0; e < 16; ++e) {
                    float acc = __uint_as_float(r[e]);
#pragma unroll
                    for (int kk = 0; kk < DP; ++kk)
                        acc = fmaf(og[kk], sUv[kk * 64 + c + e], acc);
                    o[e] = acc * inv;
                }
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
        report(a.status, DAR_ERR_CUDA);
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

// 2-D bf16 tensor [rows][cols] (row pitch = cols), box [box_rows][cols].
static bool make_map(CUtensorMap *m, const void *base, unsigned long long rows, int cols, int box_rows,
                     CUtensorMapSwizzle sw)
{
    EncodeTiledFn fn = encode_fn();
    if (!fn)
        return false;
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
    cuuint32_t box[2] = {(cuuint32_t)cols, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int DP>
static cudaError_t launch_dp(const PrefillArgs &a, cudaStream_t s)
{
    CUtensorMap mq, mk, mv, mkd, mvd;
    const CUtensorMapSwizzle swd = DP == 16 ? CU_TENSOR_MAP_SWIZZLE_32B
                                   : DP == 32 ? CU_TENSOR_MAP_SWIZZLE_64B
                                              : CU_TENSOR_MAP_SWIZZLE_128B;
    const unsigned long long rq = (unsigned long long)a.B * a.Hq * a.N, rk = (unsigned long long)a.B * a.Hkv * a.N;
    if (!make_map(&mq, a.q, rq, 64, BM, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&mk, a.k, rk, 64, BN, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&mv, a.v, rk, 64, BN, CU_TENSOR_MAP_SWIZZLE_128B) || !make_map(&mkd, a.kd, rk, DP, BN, swd) ||
        !make_map(&mvd, a.vd, rk, DP, BN, swd))
        return cudaErrorInvalidValue;
    auto kern = prefill_tc_kernel<DP>;
    const size_t smem = Layout<DP>::TOTAL + 1024;
    static bool configured = false;
    if (!configured) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess)
            return e;
        configured = true;
    }
    dim3 grid(a.B * a.Hq, (a.N + BM - 1) / BM);
    kern<<<grid, kThreads, smem, s>>>(mq, mk, mv, mkd, mvd, a);
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
    switch (a.kd_stride) {
    case 16: return tcp::launch_dp<16>(a, s);
    case 32: return tcp::launch_dp<32>(a, s);
    case 64: return tcp::launch_dp<64>(a, s);
    default: return cudaErrorInvalidValue;
    }
}

}  // namespace dar
