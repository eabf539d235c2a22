// dar_latent.cu -- DAR attention in the paper's own latent form (Sec. 2,
// Eq. 1-4 on hidden states, with the cache scheme of Sec. 5 "Compute and
// memory efficiency"): every token keeps ONE bottleneck c_j = h_j W_down,
// shared by all heads and by keys and values; a head g reaches a distant token
// through k'_j = (c_j W_up) W_K^g and v'_j = (c_j W_up) W_V^g.  With W_up
// absorbed (A_K^g = W_up W_K^g, A_V^g = W_up W_V^g, d_lat x d each):
//   global score   scale * q_i . k'_j = scale * (q_i A_K^gT) . c_j = scale * q~_i . c_j
//   global value   sum_j p_ij v'_j  = (sum_j p_ij c_j) A_V^g
// so a decode step streams each distant token's d_lat-vector once for all Hq
// heads (an MLA-like contraction: heads x d_lat against tokens x d_lat),
// while the last w tokens keep full keys and values per KV head.
//
// Kernels:
//  - latent_append: Eq. 1 (c = h W_down, one fp32 FMA chain over the D
//    inputs per element, rounded once to bf16) into the page of every new
//    token; new keys/values into the ring; then the lengths.
//  - latent_absorb: A_K, A_V (fp32 chains over D).
//  - decode: prep (q~ = q A_K^T, bf16), main (a persistent kernel: work
//    items are latent splits of four pages and windows of one KV head; a
//    producer warp streams their 64-token tiles through a TMA ring, four
//    consumer warps compute S = A B^T and O += P V on mma.sync tensor cores
//    with one online softmax per head and write one partial record per item),
//    merge (exact log-sum-exp combination of the partial records, then
//    o = (O_loc + O_lat A_V) / l).
#include <cuda.h>

#include <mutex>

#include "dar_common.cuh"
#include "dar_launch.h"
#include "dar_sm100.cuh"

namespace dar {
namespace lat {

using namespace sm100;

constexpr int kTok = DAR_PAGE_SIZE;  // tokens per page
constexpr int kPagesPerSplit = 4;
constexpr int kSplitTok = kTok * kPagesPerSplit;

struct Args {
    const void *q;  // [B][Hq][64]
    void *out;      // [B][Hq][64]
    const void *win_k, *win_v;
    const int32_t *block_table, *seq_lens;
    int32_t *status;
    const float *Ak, *Av;  // [Hkv][64][DL] (transposed), [Hkv][DL][64]
    bf16 *qt;              // [B][Hq][DL]
    float *rec_lat;        // [B][Hq][nspl][DL + 2]
    float *rec_win;        // [B][Hq][66]
    int B, Hq, Hkv, G, w, maxp, num_pages, nspl;
    float c2;  // scale * log2(e)
};

// ---------------------------------------------------------------- append

struct AppendArgs {
    const void *h;  // [B][n][D]
    const void *k_new, *v_new;  // [B][Hkv][n][64]
    const float *Wdown;         // [D][DL]
    void *win_k, *win_v, *pool_c;
    const int32_t *block_table, *n_per_seq;
    int32_t *seq_lens, *status;
    int B, Hkv, n, D, DL, w, maxp, num_pages;
};

constexpr int kAppTok = 4;  // tokens per block

// Block (token group, b): c = round_bf16(chain_e h[e] Wdown[e][a]) for the
// group's tokens, written to their pages; ring rows of the tokens that stay in
// the window.  The lengths are read here and advanced by latent_lens_kernel.
__global__ void __launch_bounds__(256) latent_append_kernel(AppendArgs a)
{
    extern __shared__ float hs[];  // [kAppTok][D]
    const int b = blockIdx.y, r0 = blockIdx.x * kAppTok;
    const int nb = a.n_per_seq ? __ldg(a.n_per_seq + b) : a.n;
    if (nb < 0 || nb > a.n) {
        if (threadIdx.x == 0 && blockIdx.x == 0)
            report(a.status, DAR_ERR_INVALID_ARG);
        return;
    }
    if (r0 >= nb)
        return;
    const int L = __ldg(a.seq_lens + b);
    const int Lnew = L + nb;
    if (Lnew > a.maxp * kTok) {
        if (threadIdx.x == 0)
            report(a.status, DAR_ERR_CAPACITY);
        return;
    }
    const int nt = min(kAppTok, nb - r0);
    const bf16 *h = static_cast<const bf16 *>(a.h) + ((size_t)b * a.n + r0) * a.D;
    for (int i = threadIdx.x; i < nt * a.D; i += blockDim.x)
        hs[i] = __bfloat162float(h[i]);
    // ring rows of the tokens that are still inside the window after the append
    for (int i = threadIdx.x; i < nt * a.Hkv * 8; i += blockDim.x) {  // 16-byte chunks of 64-wide rows
        const int t = i / (a.Hkv * 8), g = (i / 8) % a.Hkv, ch = i % 8;
        const int p = L + r0 + t;
        if (p < Lnew - a.w)
            continue;
        const size_t src = (((size_t)b * a.Hkv + g) * a.n + r0 + t) * 64 + ch * 8;
        const size_t dst = (((size_t)b * a.Hkv + g) * a.w + p % a.w) * 64 + ch * 8;
        reinterpret_cast<uint4 *>(a.win_k)[dst / 8] = reinterpret_cast<const uint4 *>(a.k_new)[src / 8];
        reinterpret_cast<uint4 *>(a.win_v)[dst / 8] = reinterpret_cast<const uint4 *>(a.v_new)[src / 8];
    }
    __syncthreads();
    for (int i = threadIdx.x; i < nt * a.DL; i += blockDim.x) {
        const int t = i / a.DL, c = i % a.DL;
        const int p = L + r0 + t;
        const int pid = __ldg(a.block_table + (size_t)b * a.maxp + p / kTok);
        if (pid < 0 || pid >= a.num_pages) {
            report(a.status, DAR_ERR_CAPACITY);
            continue;
        }
        float acc = 0.f;  // Eq. 1: one fp32 chain over e = 0..D-1 from +0
        for (int e = 0; e < a.D; ++e)
            acc = fmaf(hs[t * a.D + e], __ldg(a.Wdown + (size_t)e * a.DL + c), acc);
        static_cast<bf16 *>(a.pool_c)[((size_t)pid * kTok + p % kTok) * a.DL + c] = __float2bfloat16_rn(acc);
    }
}

__global__ void latent_lens_kernel(AppendArgs a)
{
    const int b = blockIdx.x * blockDim.x + threadIdx.x;
    if (b >= a.B)
        return;
    const int nb = a.n_per_seq ? a.n_per_seq[b] : a.n;
    if (nb < 0 || nb > a.n)
        return;
    if (a.seq_lens[b] + nb <= a.maxp * kTok)
        a.seq_lens[b] += nb;
}

// A[g][c][t] = chain_e Wup[c][e] W[g][e][t] (fp32), for A_K (stored as
// [g][t][c]) and A_V (stored as [g][c][t]).
__global__ void latent_absorb_kernel(const float *Wup, const float *WK, const float *WV, float *Ak, float *Av, int D,
                                     int DL)
{
    const int g = blockIdx.y, c = blockIdx.x, t = threadIdx.x;  // 64 threads
    const float *wk = WK + (size_t)g * D * 64, *wv = WV + (size_t)g * D * 64;
    float ak = 0.f, av = 0.f;
    for (int e = 0; e < D; ++e) {
        const float u = __ldg(Wup + (size_t)c * D + e);
        ak = fmaf(u, __ldg(wk + (size_t)e * 64 + t), ak);
        av = fmaf(u, __ldg(wv + (size_t)e * 64 + t), av);
    }
    Ak[((size_t)g * 64 + t) * DL + c] = ak;  // [Hkv][d][d_lat]: the prep kernel reads rows of d_lat
    Av[((size_t)g * DL + c) * 64 + t] = av;  // [Hkv][d_lat][d]: the merge reads rows of d
}

// ---------------------------------------------------------------- decode: prep

// q~[b][h][c] = sum_t q[b][h][t] A_K[g][t][c] (fp32, stored as bf16).  Block
// (g, 4 rows of KV head g): A_K^g staged in shared memory by one bulk copy,
// then one warp per row, lanes over c.  It starts the main kernel's launch at once: that
// kernel stages its first pages before it waits for q~.
constexpr int kRowsPerBlock = 4;  // rows (one per warp) of one KV head per block

// One bulk asynchronous copy of `bytes` (a multiple of 16) from global to
// shared memory, waited for by the whole block (bounded; on a timeout the
// status is flagged and false returned).
__device__ __forceinline__ bool stage_matrix(void *dst, const void *src, unsigned bytes, uint64_t *bar,
                                             int32_t *status)
{
    if (threadIdx.x == 0) {
        mbar_init(bar, 1);
        mbar_init_fence();
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        mbar_expect_tx(bar, bytes);
        for (unsigned off = 0; off < bytes; off += 16384u)  // in copies of at most 16 KB
            bulk_g2s(static_cast<char *>(dst) + off, static_cast<const char *>(src) + off,
                     bytes - off < 16384u ? bytes - off : 16384u, bar);
    }
    const bool ok = mbar_wait(bar, 0, nullptr);
    if (!ok && threadIdx.x == 0)
        report(status, DAR_ERR_DEVICE);
    return __syncthreads_and(ok) != 0;
}

template <int DL>
__global__ void __launch_bounds__(128) latent_prep_kernel(Args a)
{
    extern __shared__ __align__(16) float aks[];  // [64][DL], then the barrier
    grid_dep_launch();
    const int g = blockIdx.x, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (!stage_matrix(aks, a.Ak + (size_t)g * 64 * DL, 64 * DL * 4, reinterpret_cast<uint64_t *>(aks + 64 * DL),
                      a.status))
        return;
    const int nrows = a.B * a.G;
    for (int r = blockIdx.y * kRowsPerBlock + warp; r < min(nrows, (int)(blockIdx.y + 1) * kRowsPerBlock); r += 4) {
        const int row = (r / a.G) * a.Hq + g * a.G + r % a.G;
        const bf16 *qr = static_cast<const bf16 *>(a.q) + (size_t)row * 64;
        const float q0 = __bfloat162float(qr[lane]), q1 = __bfloat162float(qr[lane + 32]);
        float acc[DL / 32];
#pragma unroll
        for (int e = 0; e < DL / 32; ++e)
            acc[e] = 0.f;
#pragma unroll 8
        for (int t = 0; t < 64; ++t) {
            const float qv = __shfl_sync(0xffffffffu, t < 32 ? q0 : q1, t & 31);
#pragma unroll
            for (int e = 0; e < DL / 32; ++e)
                acc[e] = fmaf(qv, aks[t * DL + 32 * e + lane], acc[e]);
        }
#pragma unroll
        for (int e = 0; e < DL / 32; ++e)
            a.qt[(size_t)row * DL + 32 * e + lane] = __float2bfloat16_rn(acc[e]);
    }
}

// ---------------------------------------------------------------- decode: main

// Shared-memory tiles are rows of 128 bytes (64 bf16) with the 16-byte chunk
// index XOR (row % 8), the layout the 128-byte TMA swizzle writes; a W-wide
// row is W / 64 such blocks of rows.
__device__ __forceinline__ uint32_t swz(uint32_t base, int row, int chunk)
{
    return base + (uint32_t)(row * 128 + ((chunk ^ (row & 7)) << 4));
}

constexpr int kConsumerThreads = 128;                   // warps 0-3: tensor-core work
constexpr int kMainThreads2 = kConsumerThreads + 32;    // warp 4: TMA producer

// Persistent main kernel.  Work items, enumerated the same way by every
// thread: first the latent splits (sequence b, up to four 64-token pages of
// its distant part), then the windows (sequence b, KV head g: the last
// min(L_b, w) tokens' full keys and values, in 64-token tiles).  CTA c takes
// items c, c + gridDim.x, ...  Warp 4 streams the items' pages and tiles
// through a ring of NST stages with TMA; warps 0-3 run each stage on the
// tensor cores and release it.
template <int DL, int MT>
struct MainLayout {
    static constexpr uint32_t CST = DL >= 128 ? DL / 64 * 8192 : 16384;  // a latent page, or a window K + V tile
    static constexpr int NST = DL <= 128 ? 6 : DL == 192 ? 4 : 2;
    static constexpr uint32_t QA = 0;                                     // [DL/64][MT*16][128 B] A operand
    static constexpr uint32_t STG = (DL / 64 * MT * 16 * 128 + 1023) / 1024 * 1024;
    static constexpr uint32_t P = STG + NST * CST;                        // [MT*16][128 B]
    static constexpr uint32_t RED = P + MT * 16 * 128;                    // [4][MT*16] floats
    static constexpr uint32_t PREF = RED + 4 * MT * 16 * 4;               // [B + 1] ints (B <= 1024)
    static constexpr uint32_t BAR = PREF + (DAR_DECODE_MAX_BATCH + 1) * 4 + 4;
    static constexpr uint32_t TOTAL = (BAR + 16 * NST + 16 + 15) / 16 * 16;
};

struct Item {
    bool latent;
    int b, part;  // latent: split index; window: KV head
    int npg;      // pages / tiles
};

template <int MT>
__device__ __forceinline__ void consumer_sync()
{
    asm volatile("bar.sync 1, %0;" ::"n"(kConsumerThreads) : "memory");
}

// One stage on the tensor cores: S = A B^T over W-wide rows (A: the item's
// q~ / q rows, MTT m-tiles; B: the stage's key-side tile), masks past ntok,
// one online-softmax step per row (maxima exchanged through `red`), P into
// shared memory, O += P V (V: the stage's value-side tile, W-wide rows).
template <int W, int MTT, int MTR>
__device__ __forceinline__ void run_stage(uint32_t qa, uint32_t ktile, uint32_t vtile, unsigned char *sm_p,
                                          uint32_t pbase, float *red, int ntok, float c2, float (&o)[MTT][W / 32][4],
                                          float (&mrun)[MTT][2], float (&lpart)[MTT][2], int warp, int lane)
{
    constexpr int NT = W / 32;
    const int grp = lane >> 2, tig = lane & 3;
    float sc[MTT][2][4];
#pragma unroll
    for (int mt = 0; mt < MTT; ++mt)
#pragma unroll
        for (int nt = 0; nt < 2; ++nt)
            sc[mt][nt][0] = sc[mt][nt][1] = sc[mt][nt][2] = sc[mt][nt][3] = 0.f;
    {
        const int tok = 16 * warp + (lane & 7) + ((lane >> 4) << 3);
        const int khalf = (lane >> 3) & 1;
#pragma unroll
        for (int kk = 0; kk < W / 16; ++kk) {
            const int ch = 2 * kk + khalf;
            uint32_t bfr[4];
            ldsm_x4(swz(ktile + (ch / 8) * 8192, tok, ch % 8), bfr);
#pragma unroll
            for (int mt = 0; mt < MTT; ++mt) {
                const int row = mt * 16 + (lane & 15), ach = 2 * kk + (lane >> 4);
                uint32_t afr[4];
                ldsm_x4(swz(qa + (ach / 8) * (MTR * 16 * 128), row, ach % 8), afr);
                mma_bf16_16816(sc[mt][0], afr, bfr[0], bfr[1]);
                mma_bf16_16816(sc[mt][1], afr, bfr[2], bfr[3]);
            }
        }
    }
#pragma unroll
    for (int mt = 0; mt < MTT; ++mt) {
        float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
        for (int nt = 0; nt < 2; ++nt)
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                const int col = 16 * warp + 8 * nt + 2 * tig + e;
                if (col >= ntok)
                    sc[mt][nt][e] = sc[mt][nt][2 + e] = -INFINITY;
                mx0 = fmaxf(mx0, sc[mt][nt][e]);
                mx1 = fmaxf(mx1, sc[mt][nt][2 + e]);
            }
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
        if (tig == 0) {
            red[warp * MTT * 16 + mt * 16 + grp] = mx0;
            red[warp * MTT * 16 + mt * 16 + grp + 8] = mx1;
        }
    }
    consumer_sync<MTT>();
#pragma unroll
    for (int mt = 0; mt < MTT; ++mt)
#pragma unroll
        for (int hr = 0; hr < 2; ++hr) {
            const int row = mt * 16 + grp + 8 * hr;
            float tmax = red[row];
#pragma unroll
            for (int w2 = 1; w2 < 4; ++w2)
                tmax = fmaxf(tmax, red[w2 * MTT * 16 + row]);
            const float mnew = fmaxf(mrun[mt][hr], tmax * c2);
            const float alpha = mrun[mt][hr] == -INFINITY ? 0.f : ex2_approx(mrun[mt][hr] - mnew);
            mrun[mt][hr] = mnew;
            lpart[mt][hr] *= alpha;
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
                o[mt][nt][2 * hr] *= alpha;
                o[mt][nt][2 * hr + 1] *= alpha;
            }
#pragma unroll
            for (int nt = 0; nt < 2; ++nt) {
                const float x0 = sc[mt][nt][2 * hr], x1 = sc[mt][nt][2 * hr + 1];
                const float p0 = x0 == -INFINITY ? 0.f : ex2_approx(fmaf(x0, c2, -mnew));
                const float p1 = x1 == -INFINITY ? 0.f : ex2_approx(fmaf(x1, c2, -mnew));
                const uint32_t pk = cvt_bf16x2(p0, p1);
                lpart[mt][hr] += bf16lo(pk) + bf16hi(pk);  // the weights the PV product uses
                const int col = 16 * warp + 8 * nt + 2 * tig;
                *reinterpret_cast<uint32_t *>(sm_p + row * 128 + (((col >> 3) ^ (row & 7)) << 4) + 4 * tig) = pk;
            }
        }
    consumer_sync<MTT>();
#pragma unroll
    for (int kk = 0; kk < kTok / 16; ++kk) {
        uint32_t afr[MTT][4];
#pragma unroll
        for (int mt = 0; mt < MTT; ++mt)
            ldsm_x4(swz(pbase, mt * 16 + (lane & 15), 2 * kk + (lane >> 4)), afr[mt]);
        const int krow = 16 * kk + (lane & 7) + (((lane >> 3) & 1) << 3);
#pragma unroll
        for (int np = 0; np < NT / 2; ++np) {
            const int n0 = warp * (W / 4) + 16 * np + ((lane >> 4) << 3);
            uint32_t bfr[4];
            ldsm_x4_t(swz(vtile + (n0 / 64) * 8192, krow, (n0 % 64) / 8), bfr);
#pragma unroll
            for (int mt = 0; mt < MTT; ++mt) {
                mma_bf16_16816(o[mt][2 * np], afr[mt], bfr[0], bfr[1]);
                mma_bf16_16816(o[mt][2 * np + 1], afr[mt], bfr[2], bfr[3]);
            }
        }
    }
}

template <int DL, int MT>
__global__ void __launch_bounds__(kMainThreads2) latent_main_kernel(const __grid_constant__ CUtensorMap tmC,
                                                                    const __grid_constant__ CUtensorMap tmK,
                                                                    const __grid_constant__ CUtensorMap tmV, Args a)
{
    using Ly = MainLayout<DL, MT>;
    constexpr int NST = Ly::NST;
    extern __shared__ unsigned char smem_raw[];
    unsigned char *sm = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                          ~uintptr_t(1023));
    const uint32_t sbase = smem_u32(sm);
    uint64_t *full = reinterpret_cast<uint64_t *>(sm + Ly::BAR);
    uint64_t *empty = full + NST;
    volatile int *abort_flag = reinterpret_cast<volatile int *>(empty + NST);
    float *red = reinterpret_cast<float *>(sm + Ly::RED);
    int *pref = reinterpret_cast<int *>(sm + Ly::PREF);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    grid_dep_launch();  // the merge kernel may launch; it waits for this grid to finish

    // lengths -> latent splits per sequence, prefix sums (every CTA, the same)
    const int B = a.B, cap = a.maxp * kTok;
    auto len_of = [&](int b) {
        const int L = __ldg(a.seq_lens + b);
        return (L < 0 || L > cap) ? 0 : L;  // reported below; such a sequence gets no items
    };
    for (int b = tid; b < B; b += blockDim.x) {
        const int L = __ldg(a.seq_lens + b);
        if ((L < 0 || L > cap) && blockIdx.x == 0)
            report(a.status, DAR_ERR_CAPACITY);
        const int Lg = len_of(b) > a.w ? len_of(b) - a.w : 0;
        pref[b + 1] = (Lg + kSplitTok - 1) / kSplitTok;
    }
    __syncthreads();
    if (warp == 0) {
        int run = 0;
        for (int c0 = 0; c0 < B; c0 += 32) {
            int v = c0 + lane < B ? pref[c0 + lane + 1] : 0;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int u = __shfl_up_sync(0xffffffffu, v, o);
                if (lane >= o)
                    v += u;
            }
            if (c0 + lane < B)
                pref[c0 + lane + 1] = run + v;
            run += __shfl_sync(0xffffffffu, v, 31);
        }
        if (lane == 0)
            pref[0] = 0;
    }
    if (tid == 0) {
        for (int st = 0; st < NST; ++st) {
            mbar_init(&full[st], 1);
            mbar_init(&empty[st], 4);  // one arrival per consumer warp
        }
        *abort_flag = 0;
        mbar_init_fence();
    }
    __syncthreads();
    const int n_lat = pref[B], n_items = n_lat + B * a.Hkv;
    auto item_of = [&](int k) {
        Item it;
        if (k < n_lat) {
            int lo = 0, hi = B - 1;  // the last b with pref[b] <= k
            while (lo < hi) {
                const int mid = (lo + hi + 1) >> 1;
                if (pref[mid] <= k)
                    lo = mid;
                else
                    hi = mid - 1;
            }
            it.latent = true;
            it.b = lo;
            it.part = k - pref[lo];
            const int L = len_of(lo), Lg = L > a.w ? L - a.w : 0;
            const int t0 = it.part * kSplitTok, t1 = min(Lg, t0 + kSplitTok);
            it.npg = (t1 - t0 + kTok - 1) / kTok;
        } else {
            const int r = k - n_lat;
            it.latent = false;
            it.b = r / a.Hkv;
            it.part = r % a.Hkv;
            const int nwin = min(len_of(it.b), a.w);
            it.npg = (nwin + kTok - 1) / kTok;
        }
        return it;
    };

    if (warp == 4) {
        // ------------------------------------------------ producer
        if (lane == 0) {
            prefetch_tensormap(&tmC);
            prefetch_tensormap(&tmK);
            prefetch_tensormap(&tmV);
            int gp = 0;
            for (int k = blockIdx.x; k < n_items; k += gridDim.x) {
                const Item it = item_of(k);
                for (int p = 0; p < it.npg; ++p, ++gp) {
                    const int st = gp % NST;
                    if (gp >= NST && !mbar_wait(&empty[st], ((gp / NST) - 1) & 1, abort_flag))
                        goto done;
                    unsigned char *dst = sm + Ly::STG + st * Ly::CST;
                    if (it.latent) {
                        int pid = __ldg(a.block_table + (size_t)it.b * a.maxp + it.part * kPagesPerSplit + p);
                        if (pid < 0 || pid >= a.num_pages) {
                            report(a.status, DAR_ERR_CAPACITY);
                            pid = 0;
                        }
                        mbar_expect_tx(&full[st], kTok * DL * 2);
#pragma unroll
                        for (int cb = 0; cb < DL / 64; ++cb)
                            tma_load_2d(dst + cb * 8192, &tmC, cb * 64, pid * kTok, &full[st]);
                    } else {
                        const int row = (it.b * a.Hkv + it.part) * a.w + p * kTok;
                        mbar_expect_tx(&full[st], 2 * 8192);
                        tma_load_2d(dst, &tmK, 0, row, &full[st]);
                        tma_load_2d(dst + 8192, &tmV, 0, row, &full[st]);
                    }
                }
            }
        done:;
        }
        return;
    }

    // ---------------------------------------------------- consumers (warps 0-3)
    grid_dep_wait();  // q~ comes from the prep kernel
    const int grp = lane >> 2, tig = lane & 3;
    int gp = 0;
    bool ok = true;
    for (int k = blockIdx.x; k < n_items && ok; k += gridDim.x) {
        const Item it = item_of(k);
        if (it.npg == 0)
            continue;
        if (it.latent) {
            // q~ rows of every head (zero past Hq) into the A-operand tile
            for (int i = tid; i < MT * 16 * (DL / 8); i += kConsumerThreads) {
                const int r = i / (DL / 8), ch = i % (DL / 8);
                uint4 v = make_uint4(0u, 0u, 0u, 0u);
                if (r < a.Hq)
                    v = *reinterpret_cast<const uint4 *>(a.qt + ((size_t)it.b * a.Hq + r) * DL + ch * 8);
                *reinterpret_cast<uint4 *>(sm + Ly::QA + (ch / 8) * (MT * 16 * 128) + r * 128 +
                                           (((ch % 8) ^ (r & 7)) << 4)) = v;
            }
        } else {
            // q rows of KV head g's query heads (zero past G) into a 64-wide A tile
            for (int i = tid; i < 16 * 8; i += kConsumerThreads) {
                const int r = i / 8, ch = i % 8;
                uint4 v = make_uint4(0u, 0u, 0u, 0u);
                if (r < a.G)
                    v = *reinterpret_cast<const uint4 *>(static_cast<const bf16 *>(a.q) +
                                                         ((size_t)it.b * a.Hq + it.part * a.G + r) * 64 + ch * 8);
                *reinterpret_cast<uint4 *>(sm + Ly::QA + r * 128 + ((ch ^ (r & 7)) << 4)) = v;
            }
        }
        consumer_sync<MT>();
        const int L = len_of(it.b), Lg = L > a.w ? L - a.w : 0, nwin = min(L, a.w);
        // Wait for a stage, zero its rows past the item's last token (their P is
        // 0; 0 * NaN must not arise), then one barrier so every consumer thread
        // takes the same decision if any wait gave up (the flag is set first).
        auto stage_wait = [&](int st, int ntok, int rows_w) -> bool {
            const bool got = mbar_wait(&full[st], (gp / NST) & 1, abort_flag);
            if (got && ntok < kTok) {
                unsigned char *t = sm + Ly::STG + st * Ly::CST;
                for (int i = tid; i < (kTok - ntok) * (rows_w / 8); i += kConsumerThreads) {
                    const int r = ntok + i / (rows_w / 8), ch = i % (rows_w / 8);
                    *reinterpret_cast<uint4 *>(t + (ch / 8) * 8192 + r * 128 + (((ch % 8) ^ (r & 7)) << 4)) =
                        make_uint4(0u, 0u, 0u, 0u);
                }
                fence_proxy_async_smem();  // these writes precede the stage's next TMA fill
            }
            consumer_sync<MT>();
            return *abort_flag == 0;
        };
        auto release = [&](int st) {
            __syncwarp();
            if (lane == 0)
                mbar_arrive(&empty[st]);
        };
        if (it.latent) {
            float o[MT][DL / 32][4];
            float mrun[MT][2], lpart[MT][2];
#pragma unroll
            for (int mt = 0; mt < MT; ++mt) {
#pragma unroll
                for (int nt = 0; nt < DL / 32; ++nt)
                    o[mt][nt][0] = o[mt][nt][1] = o[mt][nt][2] = o[mt][nt][3] = 0.f;
                mrun[mt][0] = mrun[mt][1] = -INFINITY;
                lpart[mt][0] = lpart[mt][1] = 0.f;
            }
            const int t0 = it.part * kSplitTok, t1 = min(Lg, t0 + kSplitTok);
            for (int p = 0; p < it.npg; ++p, ++gp) {
                const int st = gp % NST, ntok = min(kTok, t1 - (t0 + p * kTok));
                if (!stage_wait(st, ntok, DL)) {
                    ok = false;
                    break;
                }
                const uint32_t t = sbase + Ly::STG + st * Ly::CST;
                run_stage<DL, MT, MT>(sbase + Ly::QA, t, t, sm + Ly::P, sbase + Ly::P, red, ntok, a.c2, o, mrun,
                                      lpart, warp, lane);
                release(st);
            }
            if (!ok)
                break;
            // record (O_lat, m, l) of every head: row sums across the quad, then the warps
#pragma unroll
            for (int mt = 0; mt < MT; ++mt)
#pragma unroll
                for (int hr = 0; hr < 2; ++hr) {
                    float ls = lpart[mt][hr];
                    ls += __shfl_xor_sync(0xffffffffu, ls, 1);
                    ls += __shfl_xor_sync(0xffffffffu, ls, 2);
                    lpart[mt][hr] = ls;
                }
            consumer_sync<MT>();
            if (tig == 0)
#pragma unroll
                for (int mt = 0; mt < MT; ++mt) {
                    red[warp * MT * 16 + mt * 16 + grp] = lpart[mt][0];
                    red[warp * MT * 16 + mt * 16 + grp + 8] = lpart[mt][1];
                }
            consumer_sync<MT>();
#pragma unroll
            for (int mt = 0; mt < MT; ++mt)
#pragma unroll
                for (int hr = 0; hr < 2; ++hr) {
                    const int row = mt * 16 + grp + 8 * hr;
                    if (row >= a.Hq)
                        continue;
                    // records of one (b, h) are consecutive over the splits
                    float *rec = a.rec_lat + (((size_t)it.b * a.Hq + row) * a.nspl + it.part) * (DL + 2);
#pragma unroll
                    for (int nt = 0; nt < DL / 32; ++nt) {
                        const int col = warp * (DL / 4) + 8 * nt + 2 * tig;
                        *reinterpret_cast<float2 *>(rec + col) =
                            make_float2(o[mt][nt][2 * hr], o[mt][nt][2 * hr + 1]);
                    }
                    if (warp == 0 && tig == 0) {
                        rec[DL] = mrun[mt][hr];
                        rec[DL + 1] =
                            red[row] + red[MT * 16 + row] + red[2 * MT * 16 + row] + red[3 * MT * 16 + row];
                    }
                }
        } else {
            float o[1][2][4];
            float mrun[1][2] = {{-INFINITY, -INFINITY}}, lpart[1][2] = {{0.f, 0.f}};
#pragma unroll
            for (int nt = 0; nt < 2; ++nt)
                o[0][nt][0] = o[0][nt][1] = o[0][nt][2] = o[0][nt][3] = 0.f;
            for (int p = 0; p < it.npg; ++p, ++gp) {
                const int st = gp % NST, ntok = min(kTok, nwin - p * kTok);
                // zero both tiles' rows past the window (K block at +0, V block at +8192)
                if (!stage_wait(st, ntok, 128)) {
                    ok = false;
                    break;
                }
                const uint32_t t = sbase + Ly::STG + st * Ly::CST;
                run_stage<64, 1, 1>(sbase + Ly::QA, t, t + 8192, sm + Ly::P, sbase + Ly::P, red, ntok, a.c2, o, mrun,
                                    lpart, warp, lane);
                release(st);
            }
            if (!ok)
                break;
#pragma unroll
            for (int hr = 0; hr < 2; ++hr) {
                float ls = lpart[0][hr];
                ls += __shfl_xor_sync(0xffffffffu, ls, 1);
                ls += __shfl_xor_sync(0xffffffffu, ls, 2);
                lpart[0][hr] = ls;
            }
            consumer_sync<MT>();
            if (tig == 0) {
                red[warp * 16 + grp] = lpart[0][0];
                red[warp * 16 + grp + 8] = lpart[0][1];
            }
            consumer_sync<MT>();
#pragma unroll
            for (int hr = 0; hr < 2; ++hr) {
                const int row = grp + 8 * hr;
                if (row >= a.G)
                    continue;
                float *rec = a.rec_win + ((size_t)it.b * a.Hq + it.part * a.G + row) * 66;
#pragma unroll
                for (int nt = 0; nt < 2; ++nt) {
                    const int col = warp * 16 + 8 * nt + 2 * tig;
                    *reinterpret_cast<float2 *>(rec + col) = make_float2(o[0][nt][2 * hr], o[0][nt][2 * hr + 1]);
                }
                if (warp == 0 && tig == 0) {
                    rec[64] = mrun[0][hr];
                    rec[65] = red[row] + red[16 + row] + red[32 + row] + red[48 + row];
                }
            }
        }
        consumer_sync<MT>();  // the A tile and `red` are reused by the next item
    }
    if (!ok && tid == 0)
        report(a.status, DAR_ERR_DEVICE);
}

// ---------------------------------------------------------------- decode: merge

// Block (g, 4 rows of KV head g): A_V^g staged in shared memory by one bulk
// copy (before the dependency wait: it does not come from the main kernel),
// then one warp per row: combine the window record and the sequence's latent splits
// (log-sum-exp, one split per lane), lift the latent sum with A_V, divide.
template <int DL>
__global__ void __launch_bounds__(128) latent_merge_kernel(Args a)
{
    extern __shared__ __align__(16) float msm[];
    float *avs = msm;                  // [DL][64]
    float *olat = avs + DL * 64;       // [4 warps][DL]
    float *fs = olat + 4 * DL;         // [4 warps][32]
    uint64_t *bar = reinterpret_cast<uint64_t *>(fs + 4 * 32);
    const int g = blockIdx.x, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (!stage_matrix(avs, a.Av + (size_t)g * DL * 64, DL * 64 * 4, bar, a.status))
        return;
    grid_dep_wait();  // the main kernel's records
    const int nrows = a.B * a.G;
    for (int r = blockIdx.y * kRowsPerBlock + warp; r < min(nrows, (int)(blockIdx.y + 1) * kRowsPerBlock); r += 4) {
        const int b = r / a.G, h = g * a.G + r % a.G, row = b * a.Hq + h;
        int L = __ldg(a.seq_lens + b);
        if (L < 0 || L > a.maxp * kTok)
            L = 0;  // reported by the main kernel; the output is undefined then
        const int Lg = L > a.w ? L - a.w : 0;
        const int ns = (Lg + kSplitTok - 1) / kSplitTok;
        const float *rw = a.rec_win + (size_t)row * 66;
        const float *rl0 = a.rec_lat + (size_t)row * a.nspl * (DL + 2);  // this row's splits, consecutive
        const float mw = L > 0 ? rw[64] : -INFINITY;
        // the splits' maxima and sums, one split per lane (32 at a time); the
        // weighted sum of their O in batches of 8 splits with every load issued
        // before it is used
        float M = mw;
        for (int s2 = lane; s2 < ns; s2 += 32)
            M = fmaxf(M, rl0[s2 * (DL + 2) + DL]);
#pragma unroll
        for (int o = 16; o; o >>= 1)
            M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
        float l = 0.f;
        float acc[DL / 32];
#pragma unroll
        for (int e = 0; e < DL / 32; ++e)
            acc[e] = 0.f;
        for (int s0 = 0; s0 < ns; s0 += 32) {
            float f = 0.f;
            if (s0 + lane < ns) {
                const float *rl = rl0 + (s0 + lane) * (DL + 2);
                f = ex2_approx(rl[DL] - M);
                l += f * rl[DL + 1];
            }
            fs[warp * 32 + lane] = f;
            __syncwarp();
            const int n = min(32, ns - s0);
            for (int j0 = 0; j0 < n; j0 += 8) {
                float x[8][DL / 32];
#pragma unroll
                for (int j = 0; j < 8; ++j)
#pragma unroll
                    for (int e = 0; e < DL / 32; ++e)
                        x[j][e] = j0 + j < n ? rl0[(s0 + j0 + j) * (DL + 2) + lane + 32 * e] : 0.f;
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    const float fj = j0 + j < n ? fs[warp * 32 + j0 + j] : 0.f;
#pragma unroll
                    for (int e = 0; e < DL / 32; ++e)
                        acc[e] = fmaf(fj, x[j][e], acc[e]);
                }
            }
            __syncwarp();
        }
#pragma unroll
        for (int o = 16; o; o >>= 1)
            l += __shfl_xor_sync(0xffffffffu, l, o);
        const float fw = L > 0 ? ex2_approx(mw - M) : 0.f;
        if (L > 0)
            l += fw * rw[65];
#pragma unroll
        for (int e = 0; e < DL / 32; ++e)
            olat[warp * DL + lane + 32 * e] = acc[e];
        __syncwarp();
        float o0 = L > 0 ? fw * rw[lane] : 0.f, o1 = L > 0 ? fw * rw[lane + 32] : 0.f;
#pragma unroll 16
        for (int c = 0; c < DL; ++c) {
            const float x = olat[warp * DL + c];
            o0 = fmaf(x, avs[c * 64 + lane], o0);
            o1 = fmaf(x, avs[c * 64 + lane + 32], o1);
        }
        const float inv = l > 0.f ? 1.f / l : 0.f;
        bf16 *out = static_cast<bf16 *>(a.out) + (size_t)row * 64;
        out[lane] = __float2bfloat16_rn(o0 * inv);
        out[lane + 32] = __float2bfloat16_rn(o1 * inv);
        __syncwarp();
    }
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

static bool encode_2d(CUtensorMap *tm, const void *base, unsigned long long rows, int cols)
{
    EncodeTiledFn enc = encode_fn();
    if (!enc)
        return false;
    const cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    const cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
    const cuuint32_t box[2] = {64, (cuuint32_t)kTok};
    const cuuint32_t estr[2] = {1, 1};
    return enc(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int DL, int MT>
static cudaError_t decode_t(const Args &a, const void *pool_c, const void *win_k, const void *win_v, cudaStream_t s)
{
    using Ly = MainLayout<DL, MT>;
    const size_t smem = 1024 + Ly::TOTAL;
    constexpr size_t prep_smem = (size_t)64 * DL * sizeof(float) + 16;
    constexpr size_t merge_smem = ((size_t)DL * 64 + 4 * DL + 4 * 32) * sizeof(float) + 16;
    static PerDeviceOnce once;  // records the SM count
    int sms = 0;
    cudaError_t e = per_device_once(
        once,
        [&](int dev) {
            cudaError_t e2 = cudaFuncSetAttribute(latent_main_kernel<DL, MT>,
                                                  cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            if (e2 == cudaSuccess)
                e2 = cudaFuncSetAttribute(latent_prep_kernel<DL>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                          (int)prep_smem);
            if (e2 == cudaSuccess)
                e2 = cudaFuncSetAttribute(latent_merge_kernel<DL>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                          (int)merge_smem);
            int n = 0;
            if (e2 == cudaSuccess)
                e2 = cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
            once.value[dev] = n;
            return e2;
        },
        &sms);
    if (e != cudaSuccess)
        return e;
    CUtensorMap tm[3];
    if (!encode_2d(&tm[0], pool_c, (unsigned long long)a.num_pages * kTok, DL) ||
        !encode_2d(&tm[1], win_k, (unsigned long long)a.B * a.Hkv * a.w, 64) ||
        !encode_2d(&tm[2], win_v, (unsigned long long)a.B * a.Hkv * a.w, 64))
        return cudaErrorInvalidValue;
    // prep starts after all earlier work on the stream; main and merge are
    // launched programmatically (each waits in-kernel for what it reads)
    const dim3 rgrid(a.Hkv, (a.B * a.G + kRowsPerBlock - 1) / kRowsPerBlock);
    latent_prep_kernel<DL><<<rgrid, 128, prep_smem, s>>>(a);
    cudaLaunchAttribute pdl[1];
    pdl[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    pdl[0].val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.stream = s;
    cfg.attrs = pdl;
    cfg.numAttrs = 1;
    cfg.gridDim = dim3(2 * (sms > 0 ? sms : 1));  // persistent: two CTAs per SM
    cfg.blockDim = dim3(kMainThreads2);
    cfg.dynamicSmemBytes = smem;
    e = cudaLaunchKernelEx(&cfg, latent_main_kernel<DL, MT>, tm[0], tm[1], tm[2], a);
    if (e != cudaSuccess)
        return e;
    cfg.gridDim = rgrid;
    cfg.blockDim = dim3(128);
    cfg.dynamicSmemBytes = merge_smem;
    e = cudaLaunchKernelEx(&cfg, latent_merge_kernel<DL>, a);
    if (e != cudaSuccess)
        return e;
    return cudaGetLastError();
}

template <int DL>
static cudaError_t decode_dl(const Args &a, const void *pool_c, const void *win_k, const void *win_v, cudaStream_t s)
{
    return a.Hq <= 16 ? decode_t<DL, 1>(a, pool_c, win_k, win_v, s) : decode_t<DL, 2>(a, pool_c, win_k, win_v, s);
}

}  // namespace lat

size_t latent_decode_workspace_bytes(int B, int Hq, int DL, int maxp)
{
    auto al = [](size_t x) { return (x + 255) & ~size_t(255); };
    const size_t nspl = (size_t)(maxp + lat::kPagesPerSplit - 1) / lat::kPagesPerSplit;
    return al((size_t)B * Hq * DL * 2) + al((size_t)B * nspl * Hq * (DL + 2) * 4) + al((size_t)B * Hq * 66 * 4);
}

cudaError_t launch_latent_decode(const LatentDecodeArgs &x, void *workspace, cudaStream_t s)
{
    if (x.B == 0)
        return cudaSuccess;
    auto al = [](size_t v) { return (v + 255) & ~size_t(255); };
    lat::Args a;
    a.q = x.q;
    a.out = x.out;
    a.win_k = x.win_k;
    a.win_v = x.win_v;
    a.block_table = x.block_table;
    a.seq_lens = x.seq_lens;
    a.status = x.status;
    a.Ak = x.Ak;
    a.Av = x.Av;
    a.B = x.B;
    a.Hq = x.Hq;
    a.Hkv = x.Hkv;
    a.G = x.Hq / x.Hkv;
    a.w = x.w;
    a.maxp = x.maxp;
    a.num_pages = x.num_pages;
    a.nspl = (x.maxp + lat::kPagesPerSplit - 1) / lat::kPagesPerSplit;
    a.c2 = x.scale * 1.4426950408889634f;
    char *p = static_cast<char *>(workspace);
    a.qt = reinterpret_cast<bf16 *>(p);
    p += al((size_t)x.B * x.Hq * x.DL * 2);
    a.rec_lat = reinterpret_cast<float *>(p);
    p += al((size_t)x.B * a.nspl * x.Hq * (x.DL + 2) * 4);
    a.rec_win = reinterpret_cast<float *>(p);
    switch (x.DL) {
    case 64: return lat::decode_dl<64>(a, x.pool_c, x.win_k, x.win_v, s);
    case 128: return lat::decode_dl<128>(a, x.pool_c, x.win_k, x.win_v, s);
    case 192: return lat::decode_dl<192>(a, x.pool_c, x.win_k, x.win_v, s);
    case 256: return lat::decode_dl<256>(a, x.pool_c, x.win_k, x.win_v, s);
    default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_latent_append(const LatentAppendArgs &x, cudaStream_t s)
{
    if (x.B == 0 || x.n == 0)
        return cudaSuccess;
    lat::AppendArgs a;
    a.h = x.h;
    a.k_new = x.k_new;
    a.v_new = x.v_new;
    a.Wdown = x.Wdown;
    a.win_k = x.win_k;
    a.win_v = x.win_v;
    a.pool_c = x.pool_c;
    a.block_table = x.block_table;
    a.n_per_seq = x.n_per_seq;
    a.seq_lens = x.seq_lens;
    a.status = x.status;
    a.B = x.B;
    a.Hkv = x.Hkv;
    a.n = x.n;
    a.D = x.D;
    a.DL = x.DL;
    a.w = x.w;
    a.maxp = x.maxp;
    a.num_pages = x.num_pages;
    const size_t smem = (size_t)lat::kAppTok * x.D * sizeof(float);
    static PerDeviceOnce once;
    cudaError_t e = per_device_once(once, [&](int) {
        return cudaFuncSetAttribute(lat::latent_append_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)(lat::kAppTok * 8192 * sizeof(float)));
    });
    if (e != cudaSuccess)
        return e;
    lat::latent_append_kernel<<<dim3((x.n + lat::kAppTok - 1) / lat::kAppTok, x.B), 256, smem, s>>>(a);
    lat::latent_lens_kernel<<<(x.B + 255) / 256, 256, 0, s>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_latent_absorb(const float *Wup, const float *WK, const float *WV, float *Ak, float *Av, int Hkv,
                                 int D, int DL, cudaStream_t s)
{
    lat::latent_absorb_kernel<<<dim3(DL, Hkv), 64, 0, s>>>(Wup, WK, WV, Ak, Av, D, DL);
    return cudaGetLastError();
}

}  // namespace dar
