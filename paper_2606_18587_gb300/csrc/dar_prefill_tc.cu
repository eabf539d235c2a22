// dar_prefill_tc.cu -- causal DAR attention forward (bf16) on the 5th-generation
// tensor cores: tcgen05.mma with operands staged by TMA in shared memory (or,
// for P, held in tensor memory) and fp32 accumulators in tensor memory (TMEM).
//
// One CTA = 128 query rows of one head; key tiles of 64, visited from the
// diagonal down to key 0.  Per key tile (Eq. 3: local iff i - j < w):
//   local part   S_loc  = Q  K^T       (M128 N64 K64)   O_loc  += P_loc  V    (N64)
//   global part  S_glob = Q~ (K^D)^T   (M128 N64 Kdd)   O_glob += P_glob V^D  (Ndd)
// with q~ = q Uk^T (W_up absorbed into the query, exact by linearity of
// Eq. 2), computed at the start of the CTA by one more tensor-core product
// (Q times Uk^T, M128 N(dd) K64) and kept in shared memory as a bf16 operand.
// A tile that holds both kinds (the window edge crosses it) is run as two
// virtual tiles, each with the other kind masked out.  One online softmax over
// every virtual tile (Eq. 4), with the running max raised lazily (only when it
// grows by more than 2^8), and the epilogue lifts the global part once:
//   o = (O_loc + O_glob Uv) / l.
// The softmax denominator l is summed by the tensor core as well: each P also
// multiplies a block of ones into 16 extra accumulator columns, so l adds up
// exactly the bf16 weights the numerators use and is rescaled with them.  For
// the global part the ones ride in the v^D rows of the workspace (16 columns
// after the d_down values), so one product of N = d_down + 16 gives both.
//
// Softmax arithmetic per score (the kernel is bound by the exponentials: one
// per causal pair, 32 per clock per SM on the multi-function unit): a 3-input
// max for the tile maximum, then per pair of scores one fp32x2 FMA
// (x = s * scale * log2(e) - m), one conversion of the pair to bf16x2 and one
// bf16x2 exp2, whose result is the packed bf16 P the PV product reads.
//
// Warp roles (352 threads): warp 0 issues TMA loads, warp 10 the S products
// (and q~), warp 1 allocates TMEM and issues the PV products (each issuing
// warp runs its loop together; one elected lane issues), warps 2-9 run the
// softmax and the epilogue, four threads per query row (TMEM lanes through
// the 16-lane load/store shapes; a row's maximum is combined with shuffles).
// For d_down <= 32 the softmax writes P into TMEM over the S it came from
// (two S buffers), where the PV products take it as their A operand, so the S
// products run a tile ahead of the softmax and only wait for the PV that last
// read a buffer; d_down = 64 keeps one S buffer and P in columns of its own.
// Two CTAs share an SM (256 TMEM columns each), so one CTA's softmax overlaps
// the other's waits.  Every wait is bounded; on a timeout the CTA flags
// *status and exits.
#include <cuda.h>

#include "dar_common.cuh"
#include "dar_launch.h"
#include "dar_sm100.cuh"

namespace dar {
namespace tcp {

using namespace sm100;

constexpr int BM = 128, BN = 64;
constexpr int kSoftmaxWarps = 8, kSoftmaxThreads = 32 * kSoftmaxWarps;  // four threads per query row, two rows each
constexpr int kThreads = 32 * (3 + kSoftmaxWarps);
constexpr int kWarpPV = 1, kWarpS = 2 + kSoftmaxWarps;  // MMA issuers (warp 0: TMA, warps 2-9: softmax)
constexpr uint32_t kTmemCols = 256;
constexpr float kRescaleThreshold = 8.0f;  // log2 units: p stays below 2^8 between rescales
constexpr uint32_t kOnesBf16x2 = 0x3F803F80u;

constexpr uint32_t align_up(uint32_t x, uint32_t a) { return (x + a - 1) / a * a; }

template <int DP>
__host__ __device__ constexpr Swizzle dp_swizzle()
{
    return DP == 16 ? kSw32 : DP == 32 ? kSw64 : kSw128;
}

// Elements per v^D row in the workspace: the DP values, then (DP < 64) 16
// ones and zero padding to a swizzle width, so the global PV product with
// N = DP + 16 also sums P into the row-sum columns that follow O_glob.
template <int DP>
__host__ __device__ constexpr int vd_row()
{
    return DP == 16 ? 32 : 64;
}
template <int DP>
__host__ __device__ constexpr bool vd_has_ones()
{
    return vd_row<DP>() > DP;
}
template <int DP>
__host__ __device__ constexpr Swizzle vd_swizzle()
{
    return vd_row<DP>() == 32 ? kSw64 : kSw128;
}

// Tensor-memory columns of one CTA (256 of the SM's 512, two CTAs per SM):
// S buffers (fp32, BN columns each), O_loc (64), O_glob (DP) and the row sum
// (16 identical columns).
//  - d_down <= 32: two S buffers.  The softmax writes P(t) (bf16 pairs, BN / 2
//    columns; the A operand of the PV products) over the first half of the S
//    buffer it came from, and S(t + 2) goes into that buffer once PV(t) has
//    read P(t), so the S products run a tile ahead of the softmax.
//  - d_down = 64: one S buffer, released as soon as the softmax has loaded it,
//    and P in 32 columns of its own.
// q~ passes through the O_loc columns before the accumulators are cleared.
template <int DP>
struct Tmem {
    static constexpr bool kAlias = 2 * BN + 64 + DP + 16 <= (int)kTmemCols;
    static constexpr uint32_t S = 0;                      // buffer b at S + b * BN
    static constexpr uint32_t OL = kAlias ? 2 * BN : BN;
    static constexpr uint32_t OG = OL + 64;
    static constexpr uint32_t SUM = OG + DP;
    static constexpr uint32_t P = kAlias ? S : SUM + 16;  // alias: P of buffer b at S + b * BN
    static_assert(SUM + 16 <= kTmemCols && (kAlias || P + BN / 2 <= kTmemCols), "tensor-memory columns overflow");
};

// Shared-memory layout (offsets from a 1024-byte aligned base).  A stage holds
// the operands of one virtual tile: K and V (local) or K^D and V^D (global).
template <int DP>
struct Layout {
    static constexpr int NS = DP == 16 ? 5 : DP == 32 ? 4 : 3;  // K/V stages (two CTAs per SM)
    static constexpr uint32_t Q = 0;                      // [128][64] bf16, 128B swizzle
    static constexpr uint32_t QT = BM * 64 * 2;           // [128][DP] bf16 q~ (written by the softmax warps)
    static constexpr uint32_t UKB = align_up(QT + BM * DP * 2, 1024);  // [DP][64] bf16 Uk, 128B swizzle
    static constexpr uint32_t ONES = align_up(UKB + DP * 64 * 2, 1024);  // 1 KB of bf16 ones
    static constexpr uint32_t STG = ONES + 1024;
    static constexpr uint32_t K_OFF = 0;                  // [64][64]
    static constexpr uint32_t V_OFF = BN * 64 * 2;        // [64][64]
    static constexpr uint32_t KD_OFF = 0;                 // [64][DP]
    static constexpr uint32_t VD_OFF = align_up(BN * DP * 2, 1024);  // [64][vd_row] (values, ones)
    static constexpr uint32_t STAGE = align_up(2 * BN * 64 * 2, 1024);
    static constexpr uint32_t UV = STG + NS * STAGE;      // fp32 [DP][64]
    static constexpr uint32_t BAR = UV + DP * 64 * 4;
    static constexpr uint32_t TOTAL = BAR + 256;
    static_assert(STAGE % 1024 == 0 && STG % 1024 == 0, "operand tiles must stay 1024-byte aligned");
    static_assert(VD_OFF + BN * vd_row<DP>() * 2 <= STAGE, "a stage holds either part");
};

__device__ __forceinline__ float max3(float a, float b, float c)
{
    float d;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
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

// Write one 32-bit word (bf16 pair) at word q of 16-byte chunk c of row r of a
// K-major operand whose rows are RB bytes, with the matching swizzle.
template <int RB>
__device__ __forceinline__ void st_swz4(unsigned char *base, int r, int c, int q, uint32_t v)
{
    constexpr int mask = RB / 16 - 1;
    const int phys = c ^ ((r * RB >> 7) & mask);
    *reinterpret_cast<uint32_t *>(base + (size_t)r * RB + phys * 16 + q * 4) = v;
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

// The sequence of query rows i0 .. i_last in closed form (Eq. 3: pair (i, j)
// is local iff i - j < w).  Key tile kt has local pairs iff kt >= kt_l (none
// when w = 0) and global pairs iff kt <= kt_g, so going down from
// kt_hi = i_last / BN: nL local-only tiles, nB band tiles (two virtual tiles
// each), then the global-only tiles.  at(t) depends on t alone, so a loop
// computes it without a chain through the previous tile.
struct TileMap {
    int kt_hi, kt_b, kt_go, nL, nLB, VT;
    __device__ __forceinline__ TileMap(int i0, int i_last, int w)
    {
        kt_hi = i_last / BN;
        const int kt_g = i_last >= w ? (i_last - w) / BN : -1;
        int kt_l = kt_hi + 1;  // no local pairs (w = 0)
        if (w > 0) {
            const int a = i0 - BN + 2 - w;  // local iff kt * BN >= a
            kt_l = a > 0 ? (a + BN - 1) / BN : 0;
        }
        nL = kt_hi - max(kt_g, kt_l - 1);
        kt_b = min(kt_hi, kt_g);
        nLB = nL + 2 * max(0, kt_b - kt_l + 1);
        kt_go = min(kt_g, kt_l - 1);
        VT = nLB + max(0, kt_go + 1);
    }
    __device__ __forceinline__ VTile at(int t) const
    {
        if (t < nL)
            return VTile{kt_hi - t, true, false};
        if (t < nLB)
            return VTile{kt_b - ((t - nL) >> 1), ((t - nL) & 1) == 0, true};
        return VTile{kt_go - (t - nLB), false, false};
    }
};

// S buffer b of virtual tile t and u = the number of earlier tiles that used
// it (the phase of that buffer's barriers).
template <bool ALIAS>
__device__ __forceinline__ void buf_of(int t, int &b, int &u)
{
    b = ALIAS ? t & 1 : 0;
    u = ALIAS ? t >> 1 : t;
}

// CH = false: the causal forward over positions 0..N-1 of q, k, v.  CH = true:
// chunked prefill over a cache (positions pos0[b] .. pos0[b] + n - 1; local
// keys from the window buffer, global keys from whole pages (tmPK, tmPV)
// or the tail buffer; v^D rows without ones, so every row sum takes a
// product of its own).
template <int DP, bool CH>
__global__ void __launch_bounds__(kThreads, 2)
    prefill_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                      const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmKD,
                      const __grid_constant__ CUtensorMap tmVD, const __grid_constant__ CUtensorMap tmPK,
                      const __grid_constant__ CUtensorMap tmPV, PrefillArgs a)
{
    using Ly = Layout<DP>;
    using Tm = Tmem<DP>;
    constexpr bool ALIAS = Tm::kAlias;
    constexpr int NS = Ly::NS;
    constexpr int NB = ALIAS ? 2 : 1;  // S buffers
    extern __shared__ unsigned char smem_raw[];
    unsigned char *sm = reinterpret_cast<unsigned char *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t *bars = reinterpret_cast<uint64_t *>(sm + Ly::BAR);
    uint64_t *full = bars;              // [NS] TMA -> MMA
    uint64_t *empty = bars + NS;        // [NS] last reader (the PV product) -> TMA
    uint64_t *s_full = bars + 2 * NS;   // [NB] S computed into buffer b
    uint64_t *p_full = s_full + NB;     // [NB] P of buffer b written (one arrival per softmax warp)
    uint64_t *pv_done = p_full + NB;    // [NB] PV reading P of buffer b finished
    uint64_t *s_free = pv_done + NB;    // single buffer: S loaded by the softmax (one arrival per softmax warp)
    uint64_t *q_full = s_free + 1;      // Q landed
    uint64_t *ukb_ready = q_full + 1;   // Uk (bf16) and the ones block written (every softmax thread)
    uint64_t *qt_mma = q_full + 2;      // q~ = Q Uk^T computed into TMEM
    uint64_t *qt_ready = q_full + 3;    // q~ in shared memory, accumulators zeroed (every softmax thread)
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(q_full + 4);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

    // global pv rows carry the ones of the row sums (plain rows in chunk mode)
    constexpr bool kOnes = !CH && vd_has_ones<DP>();
    constexpr int VR = kOnes ? vd_row<DP>() : DP;  // elements per v^D row in a stage
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int w = a.w;
    const bool direct = a.qd != nullptr;  // Sec. 5 direct variant: q~ given, not absorbed
    const int bh = blockIdx.x, b = bh / a.Hq, h = bh % a.Hq, g = h / (a.Hq / a.Hkv);
    const int L0 = CH ? __ldg(a.pos0 + b) : 0;  // position of query row 0
    const int nrows = CH ? a.n : a.N;            // query rows per (b, h)
    const int N = L0 + nrows;                    // end of the query positions
    const int nqt = (nrows + BM - 1) / BM;
    const int qt = nqt - 1 - (int)blockIdx.y;  // longest rows first
    const int i0 = L0 + qt * BM, i_last = min(i0 + BM, N) - 1;
    const TileMap tiles(i0, i_last, w);
    const int VT = tiles.VT;
    // chunk mode: first positions of the window and tail buffers
    const int kb0 = CH ? max(0, L0 - w + 1) / BN * BN : 0;
    const int kt0 = CH ? max(0, L0 - w) / BN * BN : 0;

    if (threadIdx.x == 0) {
        for (int s = 0; s < NS; ++s) {
            mbar_init(&full[s], 1);
            // released by the PV commit alone: PV(t) follows P(t), which follows
            // the completion of S(t), so K and V have both been read by then
            mbar_init(&empty[s], 1);
        }
        for (int b2 = 0; b2 < NB; ++b2) {
            mbar_init(&s_full[b2], 1);
            mbar_init(&p_full[b2], kSoftmaxWarps);
            mbar_init(&pv_done[b2], 1);
        }
        mbar_init(s_free, kSoftmaxWarps);
        mbar_init(q_full, 1);
        mbar_init(ukb_ready, kSoftmaxThreads);
        mbar_init(qt_mma, 1);
        mbar_init(qt_ready, kSoftmaxThreads);
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
            if constexpr (CH) {
                prefetch_tensormap(&tmPK);
                prefetch_tensormap(&tmPV);
            }
            mbar_expect_tx(q_full, BM * 64 * 2);
            tma_load_2d(sm + Ly::Q, &tmQ, 0, (b * a.Hq + h) * nrows + qt * BM, q_full);
            for (int t = 0; t < VT; ++t) {
                const VTile vt = tiles.at(t);
                const int s = t % NS;
                if (t >= NS && !mbar_wait(&empty[s], ((t / NS) - 1) & 1, abort_flag))
                    break;
                unsigned char *st = sm + Ly::STG + s * Ly::STAGE;
                const int j0 = vt.kt * BN;
                if (vt.loc) {
                    const int krow = CH ? (b * a.Hkv + g) * a.NW + (j0 - kb0) : (b * a.Hkv + g) * a.N + j0;
                    mbar_expect_tx(&full[s], 2 * BN * 64 * 2);
                    tma_load_2d(st + Ly::K_OFF, &tmK, 0, krow, &full[s]);
                    tma_load_2d(st + Ly::V_OFF, &tmV, 0, krow, &full[s]);
                } else {
                    mbar_expect_tx(&full[s], BN * DP * 2 + BN * VR * 2);
                    if (CH && j0 + BN <= kt0) {  // a whole page migrated before this call
                        int pid = a.block_table[(size_t)b * a.maxp + vt.kt];
                        if (pid < 0 || pid >= a.num_pages) {
                            report(a.status, DAR_ERR_CAPACITY);
                            pid = 0;
                        }
                        const int prow = (pid * a.Hkv + g) * BN;
                        tma_load_2d(st + Ly::KD_OFF, &tmPK, 0, prow, &full[s]);
                        tma_load_2d(st + Ly::VD_OFF, &tmPV, 0, prow, &full[s]);
                    } else {
                        const int krow = CH ? (b * a.Hkv + g) * a.NT + (j0 - kt0) : (b * a.Hkv + g) * a.N + j0;
                        tma_load_2d(st + Ly::KD_OFF, &tmKD, 0, krow, &full[s]);
                        tma_load_2d(st + Ly::VD_OFF, &tmVD, 0, krow, &full[s]);
                    }
                }
            }
        }
    } else if (warp == kWarpS || warp == kWarpPV) {
        // ------------------------------------------------------------ MMA issuers
        // Two warps: S products (and q~) from one, PV products from the other.
        // Each warp runs its loop together and one elected lane issues the
        // products and their commits, so descriptors and TMEM addresses stay
        // warp-uniform.  They write disjoint TMEM columns; each commit covers
        // the products of its tile, and the PV commit also frees the tile's
        // stage.
        constexpr uint64_t kStageStep = Ly::STAGE >> 4;
        const uint64_t dStg = smem_desc(smem_u32(sm + Ly::STG), 16, 1024, kSw128);  // stage 0, K / V tile
        auto wait_all = [&](uint64_t *bar, unsigned parity) {
            const bool r = mbar_wait(bar, parity, abort_flag);
            return __all_sync(0xffffffffu, r) != 0;
        };
        bool ok = true;
        if (warp == kWarpS) {
            constexpr uint32_t idS = idesc_bf16(BM, BN, false);
            constexpr uint32_t idQT = idesc_bf16(BM, DP, false);
            // Shared-memory descriptors, built once: a k-step of 16 elements adds
            // 32 bytes along a K-major row (2 in the address field).
            const uint64_t dQ = smem_desc(smem_u32(sm + Ly::Q), 16, 1024, kSw128);
            const uint64_t dQT = smem_desc(smem_u32(sm + Ly::QT), 16, 8 * DP * 2, dp_swizzle<DP>());
            const uint64_t dUKB = smem_desc(smem_u32(sm + Ly::UKB), 16, 1024, kSw128);
            const uint64_t dStgD = smem_desc(smem_u32(sm + Ly::STG), 16, 8 * DP * 2, dp_swizzle<DP>());
            const uint32_t tS = tmem + Tm::S, tOL = tmem + Tm::OL;
            // q~ = Q Uk^T into the O_loc columns (the direct variant reads its
            // d_down queries from memory instead)
            ok = wait_all(q_full, 0) && wait_all(ukb_ready, 0);
            if (ok) {
                tc_fence_after();
                if (!direct) {
                    if (elect_one()) {
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk)
                            mma_f16_ss(tOL, dQ + 2 * kk, dUKB + 2 * kk, idQT, kk > 0);
                        mma_commit(qt_mma);
                    }
                    __syncwarp();
                }
                ok = wait_all(qt_ready, 0);
                tc_fence_after();
            }
            // S(t) into buffer b once that buffer is free: PV(t - 2) has read the
            // P written over it (two buffers), or the softmax has loaded S(t - 1)
            // (one buffer)
            int s = 0, sph = 0;
            for (int t = 0; ok && t < VT; ++t) {
                const VTile vt = tiles.at(t);
                int sb, u;
                buf_of<ALIAS>(t, sb, u);
                bool fine = wait_all(&full[s], sph);
                if (fine && u > 0)
                    fine = wait_all(ALIAS ? &pv_done[sb] : s_free, (u - 1) & 1);
                if (!fine) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t tSb = tS + sb * BN;
                if (elect_one()) {
                    if (vt.loc) {
                        const uint64_t dK = dStg + s * kStageStep;
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk)
                            mma_f16_ss(tSb, dQ + 2 * kk, dK + 2 * kk, idS, kk > 0);
                    } else {
                        const uint64_t dKD = dStgD + s * kStageStep;
#pragma unroll
                        for (int kk = 0; kk < DP / 16; ++kk)
                            mma_f16_ss(tSb, dQT + 2 * kk, dKD + 2 * kk, idS, kk > 0);
                    }
                    mma_commit(&s_full[sb]);
                }
                __syncwarp();
                if (++s == NS) {
                    s = 0;
                    sph ^= 1;
                }
            }
        } else {
            constexpr uint32_t idPV = idesc_bf16(BM, 64, true);
            // global PV: N = DP + 16 when v^D rows carry the ones (O_glob, then the row sums)
            constexpr uint32_t idPVg = idesc_bf16(BM, kOnes ? DP + 16 : DP, true);
            constexpr uint32_t idSum = idesc_bf16(BM, 16, false);
            // a k-step of 16 keys adds 16 rows (16 * row bytes) along an MN-major operand
            const uint64_t dStgVD = smem_desc(smem_u32(sm + Ly::STG), 16, 8 * VR * 2,
                                              kOnes ? vd_swizzle<DP>() : dp_swizzle<DP>());
            constexpr uint64_t kVOff = Ly::V_OFF >> 4, kVDOff = Ly::VD_OFF >> 4;
            constexpr uint64_t kVStep = (16 * 128) >> 4, kVDStep = (16 * VR * 2) >> 4;
            // all-ones B operand (16 columns x 16 keys per k-step; every byte pair is 1.0)
            const uint64_t ones_desc = smem_desc(smem_u32(sm + Ly::ONES), 128, 256, kSwNone);
            const uint32_t tOL = tmem + Tm::OL, tOG = tmem + Tm::OG, tSum = tmem + Tm::SUM;
            int s = 0;
            for (int t = 0; ok && t < VT; ++t) {
                const VTile vt = tiles.at(t);
                int pb, u;
                buf_of<ALIAS>(t, pb, u);
                if (!wait_all(&p_full[pb], u & 1)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t aP = tmem + Tm::P + (ALIAS ? pb * BN : 0);
                if (elect_one()) {
                    if (vt.loc) {
                        const uint64_t dV = dStg + s * kStageStep + kVOff;
#pragma unroll
                        for (int kk = 0; kk < BN / 16; ++kk) {  // P (TMEM, 8 columns per 16 keys) times V
                            mma_f16_ts(tOL, aP + kk * 8, dV + kk * kVStep, idPV, true);
                            mma_f16_ts(tSum, aP + kk * 8, ones_desc, idSum, true);  // row sums of P
                        }
                    } else {
                        const uint64_t dVD = dStgVD + s * kStageStep + kVDOff;
#pragma unroll
                        for (int kk = 0; kk < BN / 16; ++kk) {  // P times [V^D | ones]
                            mma_f16_ts(tOG, aP + kk * 8, dVD + kk * kVDStep, idPVg, true);
                            if constexpr (!kOnes)
                                mma_f16_ts(tSum, aP + kk * 8, ones_desc, idSum, true);
                        }
                    }
                    mma_commit(&pv_done[pb]);
                    mma_commit(&empty[s]);
                }
                __syncwarp();
                if (++s == NS)
                    s = 0;
            }
        }
        if (!ok)
            *abort_flag = 1;
    } else {  // warps 2 .. 2 + kSoftmaxWarps - 1
        // ------------------------------------------------------------ softmax warps
        // Warp w covers TMEM lanes 32 (w % 4) + 16 h .. + 15 (h = 0 for warps
        // 2-5, 1 for warps 6-9) with the 16-lane load/store shapes: four
        // threads per query row, each thread two rows (ra, ra + 8) and 16 of a
        // tile's 64 columns, 8k + 2 q4 + {0, 1} (k = 0 .. 7, q4 = lane % 4).  A
        // row's maximum is combined across its four threads with shuffles.
        const int quad = warp & 3;
        const int half = (warp - 2) >> 2;
        const int q4 = lane & 3;
        const int ra = 32 * quad + 16 * half + (lane >> 2);  // rows ra and ra + 8 of the 128
        const int iA = i0 + ra, iB = iA + 8;
        const uint32_t tl = tmem + ((uint32_t)(32 * quad + 16 * half) << 16);
        const int stid = threadIdx.x - 64;  // 0 .. kSoftmaxThreads - 1
        // ---- set-up: Uk as a bf16 operand, the ones block, Uv for the epilogue
        {
            const float *Ukg = a.Uk + (size_t)g * a.dd * 64;
            for (int idx = direct ? DP * 8 : stid; idx < DP * 8; idx += kSoftmaxThreads) {  // row c, chunk ch of 8 values
                const int c = idx / 8, ch = idx % 8;
                uint4 v = make_uint4(0u, 0u, 0u, 0u);
                if (c < a.dd) {
                    const float4 u0 = *reinterpret_cast<const float4 *>(Ukg + c * 64 + ch * 8);
                    const float4 u1 = *reinterpret_cast<const float4 *>(Ukg + c * 64 + ch * 8 + 4);
                    v = make_uint4(pack_bf16(u0.x, u0.y), pack_bf16(u0.z, u0.w), pack_bf16(u1.x, u1.y),
                                   pack_bf16(u1.z, u1.w));
                }
                st_swz<128>(sm + Ly::UKB, c, ch, v);
            }
            if (stid < 64)
                reinterpret_cast<uint4 *>(sm + Ly::ONES)[stid] =
                    make_uint4(kOnesBf16x2, kOnesBf16x2, kOnesBf16x2, kOnesBf16x2);
            fence_proxy_async_smem();
            mbar_arrive(ukb_ready);
            float *sUv = reinterpret_cast<float *>(sm + Ly::UV);
            for (int idx = stid; idx < DP * 64; idx += kSoftmaxThreads) {
                const int c = idx / 64, t = idx % 64;
                sUv[idx] = c < a.dd ? a.Uv[((size_t)g * a.dd + c) * 64 + t] : 0.f;
            }
        }
        // tcgen05.ld/st are warp-collective: every branch around them is warp-uniform
        auto wait_uniform = [&](uint64_t *bar, unsigned parity) {
            const bool r = mbar_wait(bar, parity, abort_flag);
            return __all_sync(0xffffffffu, r) != 0;
        };
        bool ok = direct || wait_uniform(qt_mma, 0);
        if (ok && direct) {
            // the direct variant's d_down queries, times scale_down / scale, as
            // bf16 operand rows (zero past the end and past d_down)
            unsigned char *qrow = sm + Ly::QT;
            const bf16 *qdh = static_cast<const bf16 *>(a.qd) + ((size_t)b * a.Hq + h) * nrows * a.dd;
            auto pair = [&](int i, int e) -> uint32_t {
                if (i >= N || e >= a.dd)
                    return 0u;
                const bf16 *p = qdh + (size_t)(i - L0) * a.dd + e;
                return pack_bf16(__bfloat162float(p[0]) * a.qd_ratio, __bfloat162float(p[1]) * a.qd_ratio);
            };
#pragma unroll
            for (int ch = 0; ch < DP / 8; ++ch) {
                st_swz4<DP * 2>(qrow, ra, ch, q4, pair(iA, 8 * ch + 2 * q4));
                st_swz4<DP * 2>(qrow, ra + 8, ch, q4, pair(iB, 8 * ch + 2 * q4));
            }
        }
        if (ok) {
            tc_fence_after();
            // q~ (fp32, TMEM) -> bf16 operand rows in shared memory; then clear the accumulators
            unsigned char *qrow = sm + Ly::QT;
            if (!direct) {
#pragma unroll
                for (int c = 0; c < DP; c += 16) {
                    uint32_t r[8];
                    tmem_ld_16x256b_x2(tl + Tm::OL + c, r);
#pragma unroll
                    for (int k = 0; k < 2; ++k) {
                        st_swz4<DP * 2>(qrow, ra, c / 8 + k, q4,
                                        pack_bf16(__uint_as_float(r[4 * k]), __uint_as_float(r[4 * k + 1])));
                        st_swz4<DP * 2>(qrow, ra + 8, c / 8 + k, q4,
                                        pack_bf16(__uint_as_float(r[4 * k + 2]), __uint_as_float(r[4 * k + 3])));
                    }
                }
            }
            uint32_t z[8];
#pragma unroll
            for (int e = 0; e < 8; ++e)
                z[e] = 0u;
#pragma unroll
            for (int c = 0; c < 64; c += 16)
                tmem_st_16x256b_x2(tl + Tm::OL + c, z);
#pragma unroll
            for (int c = 0; c < DP + 16; c += 16)  // O_glob and the row-sum columns
                tmem_st_16x256b_x2(tl + Tm::OG + c, z);
            tmem_wait_st();
            fence_proxy_async_smem();
        }
        asm volatile("bar.sync 1, %0;" ::"n"(kSoftmaxThreads) : "memory");  // Uv staged by all softmax threads
        tc_fence_before();
        mbar_arrive(qt_ready);

        const float c2 = a.qscale;  // softmax scale * log2(e)
        float mA = -INFINITY, mB = -INFINITY;  // running maxima (log2 units) of rows ra, ra + 8
        // last tile whose PV this thread has seen complete, per S buffer
        int pv_seen0 = -1, pv_seen1 = -1;
        // wait until PV(v) (its own products) has completed
        auto wait_pv = [&](int v) -> bool {
            if (v < 0)
                return true;
            int pb, u;
            buf_of<ALIAS>(v, pb, u);
            const int seen = pb == 0 ? pv_seen0 : pv_seen1;
            if (seen >= v)
                return true;
            if (!wait_uniform(&pv_done[pb], u & 1))
                return false;
            if (pb == 0)
                pv_seen0 = v;
            else
                pv_seen1 = v;
            tc_fence_after();
            return true;
        };
        // scale 16 columns of both rows' accumulators
        auto rescale16 = [&](uint32_t col, float alA, float alB) {
            uint32_t r[8];
            tmem_ld_16x256b_x2(tl + col, r);
#pragma unroll
            for (int k = 0; k < 2; ++k) {
                r[4 * k + 0] = __float_as_uint(__uint_as_float(r[4 * k + 0]) * alA);
                r[4 * k + 1] = __float_as_uint(__uint_as_float(r[4 * k + 1]) * alA);
                r[4 * k + 2] = __float_as_uint(__uint_as_float(r[4 * k + 2]) * alB);
                r[4 * k + 3] = __float_as_uint(__uint_as_float(r[4 * k + 3]) * alB);
            }
            tmem_st_16x256b_x2(tl + col, r);
        };
        for (int t = 0; ok && t < VT; ++t) {
            const VTile vt = tiles.at(t);
            int sb, u;
            buf_of<ALIAS>(t, sb, u);
            const int j0 = vt.kt * BN;
            if (!wait_uniform(&s_full[sb], u & 1)) {
                ok = false;
                break;
            }
            tc_fence_after();
            // row ra: sa[2k + j], row ra + 8: sv[2k + j] = score column 8k + 2 q4 + j
            float sa[16], sv[16];
            {
                uint32_t r[32];
                tmem_ld_16x256b_x8(tl + Tm::S + sb * BN, r);
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    sa[2 * k] = __uint_as_float(r[4 * k]);
                    sa[2 * k + 1] = __uint_as_float(r[4 * k + 1]);
                    sv[2 * k] = __uint_as_float(r[4 * k + 2]);
                    sv[2 * k + 1] = __uint_as_float(r[4 * k + 3]);
                }
            }
            if constexpr (!ALIAS) {  // the S buffer may be overwritten now (S(t + 1))
                tc_fence_before();
                __syncwarp();
                if (lane == 0)
                    mbar_arrive(s_free);
            }

            // masks: causal (tiles reaching past row i0), the other part of a
            // band tile, rows past the end; the kept columns of a row form one
            // range, here relative to this thread's column offset 2 q4
            if (__builtin_expect(j0 + BN - 1 > i0 || vt.band || i0 + BM > N, 0)) {
                int hiA = iA < N ? iA - j0 : -1, hiB = iB < N ? iB - j0 : -1, loA = 0, loB = 0;
                if (vt.band) {
                    if (vt.loc) {
                        loA = iA - w - j0 + 1;
                        loB = iB - w - j0 + 1;
                    } else {
                        hiA = min(hiA, iA - w - j0);
                        hiB = min(hiB, iB - w - j0);
                    }
                }
                loA -= 2 * q4;
                loB -= 2 * q4;
                hiA -= 2 * q4;
                hiB -= 2 * q4;
                // one bound at a time, each only where some row of the warp needs it
                if (__any_sync(0xffffffffu, loA > -2 * q4 || loB > -2 * q4)) {
#pragma unroll
                    for (int e = 0; e < 16; ++e) {
                        const int col = 8 * (e >> 1) + (e & 1);
                        sa[e] = col >= loA ? sa[e] : -INFINITY;
                        sv[e] = col >= loB ? sv[e] : -INFINITY;
                    }
                }
                if (__any_sync(0xffffffffu, hiA + 2 * q4 < BN - 1 || hiB + 2 * q4 < BN - 1)) {
#pragma unroll
                    for (int e = 0; e < 16; ++e) {
                        const int col = 8 * (e >> 1) + (e & 1);
                        sa[e] = col <= hiA ? sa[e] : -INFINITY;
                        sv[e] = col <= hiB ? sv[e] : -INFINITY;
                    }
                }
            }
            // row maxima: this thread's 16 columns, then across the row's four threads
            float xA = max3(max3(sa[0], sa[1], sa[2]), max3(sa[3], sa[4], sa[5]), max3(sa[6], sa[7], sa[8]));
            float xB = max3(max3(sv[0], sv[1], sv[2]), max3(sv[3], sv[4], sv[5]), max3(sv[6], sv[7], sv[8]));
            xA = max3(xA, max3(sa[9], sa[10], sa[11]), max3(sa[12], sa[13], fmaxf(sa[14], sa[15])));
            xB = max3(xB, max3(sv[9], sv[10], sv[11]), max3(sv[12], sv[13], fmaxf(sv[14], sv[15])));
            xA = fmaxf(xA, __shfl_xor_sync(0xffffffffu, xA, 1));
            xB = fmaxf(xB, __shfl_xor_sync(0xffffffffu, xB, 1));
            xA = fmaxf(xA, __shfl_xor_sync(0xffffffffu, xA, 2)) * c2;
            xB = fmaxf(xB, __shfl_xor_sync(0xffffffffu, xB, 2)) * c2;
            // raise a running max only when it grows by more than the threshold
            const bool raiseA = xA > mA + kRescaleThreshold, raiseB = xB > mB + kRescaleThreshold;
            const bool scaleA = raiseA && mA != -INFINITY, scaleB = raiseB && mB != -INFINITY;
            // O's scale factors when a running max is raised (applied below, once P is computed)
            const float alA = scaleA ? ex2_approx(mA - xA) : 1.f, alB = scaleB ? ex2_approx(mB - xB) : 1.f;
            if (raiseA)
                mA = xA;
            if (raiseB)
                mB = xB;
            // P = 2^(s * c2 - m) in bf16 pairs (masked entries give 0): pw[2k] row
            // ra, pw[2k + 1] row ra + 8, P column 4k + q4 (keys 8k + 2 q4, + 1)
            const float nA = mA == -INFINITY ? 0.f : -mA, nB = mB == -INFINITY ? 0.f : -mB;
            uint32_t pw[16];
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                float x0, x1, y0, y1;
                ffma2(x0, x1, sa[2 * k], sa[2 * k + 1], c2, c2, nA, nA);
                ffma2(y0, y1, sv[2 * k], sv[2 * k + 1], c2, c2, nB, nB);
                pw[2 * k] = ex2_bf16x2(cvt_bf16x2(x0, x1));
                pw[2 * k + 1] = ex2_bf16x2(cvt_bf16x2(y0, y1));
            }
            if (__builtin_expect(__any_sync(0xffffffffu, scaleA || scaleB), 0)) {
                // every earlier PV must have landed before O is rescaled (PV(t),
                // which needs P(t), cannot start before it is)
                if (!wait_pv(t - 1) || !wait_pv(t - 2)) {
                    ok = false;
                    break;
                }
#pragma unroll
                for (int c = 0; c < 64; c += 16)
                    rescale16(Tm::OL + c, alA, alB);
#pragma unroll
                for (int c = 0; c < DP + 16; c += 16)  // O_glob and the row sums
                    rescale16(Tm::OG + c, alA, alB);
            }
            // one buffer: PV(t - 1) must be done with the P buffer (two buffers:
            // P goes over S(t), whose buffer was free before S(t) was computed)
            if (!ALIAS && !wait_pv(t - 1)) {
                ok = false;
                break;
            }
            tmem_st_16x128b_x8(tl + Tm::P + (ALIAS ? sb * BN : 0), pw);
            tmem_wait_st();
            tc_fence_before();
            __syncwarp();
            if (lane == 0)
                mbar_arrive(&p_full[sb]);
        }

        // ---- epilogue: o = (O_loc + O_glob Uv) / l (the last products may
        // still be running on either buffer).  O_glob rows go through shared
        // memory (the stage area, idle by now), so each thread can take the
        // whole d_down vector of its two rows.
        if (ok && wait_pv(VT - 1) && wait_pv(VT - 2)) {
            const float *sUv = reinterpret_cast<const float *>(sm + Ly::UV);
            constexpr int OGS = DP + 1;  // padded row stride (floats)
            float *sOG = reinterpret_cast<float *>(sm + Ly::STG);
#pragma unroll
            for (int c = 0; c < DP; c += 16) {
                uint32_t r[8];
                tmem_ld_16x256b_x2(tl + Tm::OG + c, r);
#pragma unroll
                for (int k = 0; k < 2; ++k)
#pragma unroll
                    for (int j = 0; j < 2; ++j) {
                        sOG[ra * OGS + c + 8 * k + 2 * q4 + j] = __uint_as_float(r[4 * k + j]);
                        sOG[(ra + 8) * OGS + c + 8 * k + 2 * q4 + j] = __uint_as_float(r[4 * k + 2 + j]);
                    }
            }
            float lA, lB;
            {
                uint32_t r[8];
                tmem_ld_16x256b_x2(tl + Tm::SUM, r);  // 16 identical columns
                lA = __uint_as_float(r[0]);
                lB = __uint_as_float(r[2]);
            }
            // O_loc: oa[2k + j] row ra, ov[2k + j] row ra + 8, output column 8k + 2 q4 + j
            float oa[16], ov[16];
            {
                uint32_t r[32];
                tmem_ld_16x256b_x8(tl + Tm::OL, r);
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    oa[2 * k] = __uint_as_float(r[4 * k]);
                    oa[2 * k + 1] = __uint_as_float(r[4 * k + 1]);
                    ov[2 * k] = __uint_as_float(r[4 * k + 2]);
                    ov[2 * k + 1] = __uint_as_float(r[4 * k + 3]);
                }
            }
            __syncwarp();
#pragma unroll 4
            for (int kk = 0; kk < DP; ++kk) {
                const float gA = sOG[ra * OGS + kk], gB = sOG[(ra + 8) * OGS + kk];
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    const float2 uu = *reinterpret_cast<const float2 *>(sUv + kk * 64 + 8 * k + 2 * q4);
                    oa[2 * k] = fmaf(gA, uu.x, oa[2 * k]);
                    oa[2 * k + 1] = fmaf(gA, uu.y, oa[2 * k + 1]);
                    ov[2 * k] = fmaf(gB, uu.x, ov[2 * k]);
                    ov[2 * k + 1] = fmaf(gB, uu.y, ov[2 * k + 1]);
                }
            }
            const float invA = lA > 0.f ? 1.f / lA : 0.f, invB = lB > 0.f ? 1.f / lB : 0.f;
            bf16 *orowA = static_cast<bf16 *>(a.out) + (((size_t)b * a.Hq + h) * nrows + (iA - L0)) * 64 + 2 * q4;
            bf16 *orowB = orowA + 8 * 64;
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                if (iA < N)
                    *reinterpret_cast<uint32_t *>(orowA + 8 * k) = pack_bf16(oa[2 * k] * invA, oa[2 * k + 1] * invA);
                if (iB < N)
                    *reinterpret_cast<uint32_t *>(orowB + 8 * k) = pack_bf16(ov[2 * k] * invB, ov[2 * k + 1] * invB);
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
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    });
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

constexpr CUtensorMapSwizzle dp_map_swizzle(int DP)
{
    return DP == 16 ? CU_TENSOR_MAP_SWIZZLE_32B : DP == 32 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_128B;
}

// One-time attribute set-up per device and instantiation, then the launch.
template <int DP, bool CH>
static cudaError_t launch_kernel(const CUtensorMap (&m)[7], const PrefillArgs &a, int nrows, cudaStream_t s)
{
    auto kern = prefill_tc_kernel<DP, CH>;
    const size_t smem = Layout<DP>::TOTAL + 1024;
    static PerDeviceOnce once;
    cudaError_t e = per_device_once(once, [&](int) {
        // two CTAs per SM need the largest shared-memory carve-out of the unified L1
        cudaError_t e2 = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e2 == cudaSuccess)
            e2 = cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout,
                                      (int)cudaSharedmemCarveoutMaxShared);
        return e2;
    });
    if (e != cudaSuccess)
        return e;
    dim3 grid(a.B * a.Hq, (nrows + BM - 1) / BM);
    kern<<<grid, kThreads, smem, s>>>(m[0], m[1], m[2], m[3], m[4], m[5], m[6], a);
    return cudaGetLastError();
}

template <int DP>
static cudaError_t launch_dp(const PrefillArgs &a, cudaStream_t s)
{
    CUtensorMap m[7];
    const unsigned long long rq = (unsigned long long)a.B * a.Hq * a.N, rk = (unsigned long long)a.B * a.Hkv * a.N;
    if (!make_map(&m[0], a.q, rq, 64, BM, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&m[1], a.k, rk, 64, BN, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&m[2], a.v, rk, 64, BN, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&m[3], a.kd, rk, DP, BN, dp_map_swizzle(DP)) ||
        !make_map(&m[4], a.vd, rk, vd_row<DP>(), BN,
                  vd_row<DP>() == 32 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_128B))
        return cudaErrorInvalidValue;
    if (a.vd_stride != vd_row<DP>())
        return cudaErrorInvalidValue;
    m[5] = m[3];  // no pages in this mode
    m[6] = m[4];
    return launch_kernel<DP, false>(m, a, a.N, s);
}

// ---------------------------------------------------------------- chunked prefill: gather

// For sequence b (L0 = its length before the chunk) and KV head g:
//  window buffer rows r < NW hold the full-d key / value of position kb0 + r
//    when it can be local to a chunk query (kb0 + r in [L0 - w + 1, L0 + n)):
//    from the ring for positions < L0, from k_new / v_new after; zero otherwise.
//  tail buffer rows r < NT hold k^D / v^D of position kt0 + r when it is
//    global to some chunk query (< L0 + n - w): copied from its page when it
//    migrated before this call (< L0 - w), else Eq. 1 of its full-d row with
//    the same fp32 chain as the cache append; zero otherwise.
// grid (B, Hkv), 256 threads.  Block (b, 0) records L0 in pos0[b].
template <int DD>
__global__ void __launch_bounds__(256) chunk_gather_kernel(ChunkArgs c)
{
    const AppendArgs &ap = c.app;
    const int b = blockIdx.x, g = blockIdx.y, tid = threadIdx.x;
    const int w = ap.w, n = ap.n, Hkv = ap.Hkv;
    const int NW = c.pf.NW, NT = c.pf.NT;
    int L0 = __ldcg(ap.seq_lens + b);
    if (L0 < 0 || (long long)L0 + n - w > (long long)ap.maxp * kPage) {
        if (tid == 0 && g == 0)
            report(ap.status, DAR_ERR_CAPACITY);
        L0 = max(0, min(L0, ap.maxp * kPage + w - n));
    }
    if (g == 0 && tid == 0)
        c.pos0[b] = L0;
    const int kb0 = max(0, L0 - w + 1) / BN * BN, kt0 = max(0, L0 - w) / BN * BN;
    const int loc_lo = max(0, L0 - w + 1);
    const size_t bg = (size_t)b * Hkv + g;
    const bf16 *ring_k = static_cast<const bf16 *>(c.win_k) + bg * w * 64;
    const bf16 *ring_v = static_cast<const bf16 *>(c.win_v) + bg * w * 64;
    const bf16 *new_k = static_cast<const bf16 *>(ap.k_new) + bg * n * 64;
    const bf16 *new_v = static_cast<const bf16 *>(ap.v_new) + bg * n * 64;
    // full-d row of position p (ring or chunk); nullptr when neither holds it
    auto row_of = [&](int p, bool v) -> const bf16 * {
        if (p >= max(0, L0 - w) && p < L0)
            return (v ? ring_v : ring_k) + (size_t)(p % w) * 64;
        if (p >= L0 && p < L0 + n)
            return (v ? new_v : new_k) + (size_t)(p - L0) * 64;
        return nullptr;
    };
    // ---- window rows, 16 bytes at a time
    uint4 *kw = reinterpret_cast<uint4 *>(static_cast<bf16 *>(c.kw) + bg * NW * 64);
    uint4 *vw = reinterpret_cast<uint4 *>(static_cast<bf16 *>(c.vw) + bg * NW * 64);
    for (int i = tid; i < NW * 8; i += blockDim.x) {
        const int p = kb0 + i / 8, ch = i % 8;
        uint4 k4 = make_uint4(0u, 0u, 0u, 0u), v4 = k4;
        if (p >= loc_lo && p < L0 + n) {
            k4 = reinterpret_cast<const uint4 *>(row_of(p, false))[ch];
            v4 = reinterpret_cast<const uint4 *>(row_of(p, true))[ch];
        }
        kw[i] = k4;
        vw[i] = v4;
    }
    // ---- tail rows, one element per thread and tensor
    bf16 *kdt = static_cast<bf16 *>(c.kdt) + bg * NT * DD;
    bf16 *vdt = static_cast<bf16 *>(c.vdt) + bg * NT * DD;
    const bf16 *pk = static_cast<const bf16 *>(ap.pool_kd);
    const bf16 *pv = static_cast<const bf16 *>(ap.pool_vd);
    for (int i = tid; i < NT * DD; i += blockDim.x) {
        const int r = i / DD, col = i % DD, p = kt0 + r;
        bf16 kx = __float2bfloat16_rn(0.f), vx = kx;
        if (p < L0 - w) {  // migrated before this call: its page
            int pid = ap.block_table[(size_t)b * ap.maxp + p / kPage];
            if (pid >= 0 && pid < ap.num_pages) {
                const size_t off = (((size_t)pid * Hkv + g) * kPage + p % kPage) * DD + col;
                kx = pk[off];
                vx = pv[off];
            } else {
                report(ap.status, DAR_ERR_CAPACITY);
            }
        } else if (p < L0 + n - w) {  // leaves the window in this chunk: Eq. 1
            const bf16 *xk = row_of(p, false), *xv = row_of(p, true);
            const float *Wk = ap.Dk + (size_t)g * 64 * DD + col, *Wv = ap.Dv + (size_t)g * 64 * DD + col;
            float ak = 0.0f, av = 0.0f;  // the fp32 chain over t = 0..63 of the cache append
            for (int t = 0; t < 64; ++t) {
                ak = __fmaf_rn(__bfloat162float(xk[t]), __ldg(Wk + (size_t)t * DD), ak);
                av = __fmaf_rn(__bfloat162float(xv[t]), __ldg(Wv + (size_t)t * DD), av);
            }
            kx = __float2bfloat16_rn(ak);
            vx = __float2bfloat16_rn(av);
        }
        kdt[i] = kx;
        vdt[i] = vx;
    }
}

template <int DP>
static cudaError_t launch_chunk_dp(const ChunkArgs &c, cudaStream_t s)
{
    const PrefillArgs &a = c.pf;
    chunk_gather_kernel<DP><<<dim3(a.B, a.Hkv), 256, 0, s>>>(c);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess)
        return e;
    CUtensorMap m[7];
    const unsigned long long rq = (unsigned long long)a.B * a.Hq * a.n;
    const unsigned long long rw = (unsigned long long)a.B * a.Hkv * a.NW, rt = (unsigned long long)a.B * a.Hkv * a.NT;
    const unsigned long long rp = (unsigned long long)(a.num_pages > 0 ? a.num_pages : 1) * a.Hkv * kPage;
    if (!make_map(&m[0], a.q, rq, 64, BM, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&m[1], c.kw, rw, 64, BN, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&m[2], c.vw, rw, 64, BN, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&m[3], c.kdt, rt, DP, BN, dp_map_swizzle(DP)) ||
        !make_map(&m[4], c.vdt, rt, DP, BN, dp_map_swizzle(DP)) ||
        !make_map(&m[5], a.pool_kd, rp, DP, BN, dp_map_swizzle(DP)) ||
        !make_map(&m[6], a.pool_vd, rp, DP, BN, dp_map_swizzle(DP)))
        return cudaErrorInvalidValue;
    e = launch_kernel<DP, true>(m, a, a.n, s);
    if (e != cudaSuccess)
        return e;
    // the chunk joins the cache last: its ring slots and migrated pages
    return launch_cache_append(DAR_BF16, DP, c.app, s);
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

cudaError_t launch_prefill_chunk(int dd, const ChunkArgs &c, cudaStream_t s)
{
    if (c.pf.B == 0 || c.pf.n == 0)
        return cudaSuccess;
    switch (dd) {
    case 16: return tcp::launch_chunk_dp<16>(c, s);
    case 32: return tcp::launch_chunk_dp<32>(c, s);
    case 64: return tcp::launch_chunk_dp<64>(c, s);
    default: return cudaErrorInvalidValue;
    }
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
