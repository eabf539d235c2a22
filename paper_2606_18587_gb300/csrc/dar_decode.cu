// dar_decode.cu -- one decode step of DAR attention over the mixed-dimension
// cache (Eq. 3-4 for the query at position L_b - 1; cache scheme of Sec. 5).
//
// Work decomposition (split-K over the sequence):
//   item = (sequence b, KV head g, head slice hs, chunk c).  Chunks 0..nwc-1
//   cover the ring (full d = 64 keys/values, `cw` tokens each); the rest cover
//   the pages (d_down vectors, `cd` tokens each, page aligned).  Each launch
//   scales both chunk sizes so that there are a few items per warp; a warp
//   takes its first item statically and later ones from an atomic counter,
//   fetched one item ahead so the atomic's latency is never waited on.
//
// Streaming: every warp owns a ring of kStages shared-memory slots of
// kSlotBytes (keys in the first half, values in the second).  Lane 0 fills a
// slot with 1-D TMA bulk copies (cp.async.bulk, completion counted on the
// slot's mbarrier) and the warp consumes slots in order, refilling each one as
// soon as it has been read, across item boundaries; page ids are loaded one
// item ahead.  So every warp keeps up to kStages * kSlotBytes of cache in
// flight while it computes.
//
// Compute (bf16, d_down >= 16): the two small contractions of a stage run on
// the tensor cores with warp-level mma.sync m16n8k16 (bf16 in, fp32 out): the
// GH query heads of the slice are rows of A, 8 tokens a column block of B,
// fed by ldmatrix from swizzled 2-D TMA tiles; the scores stay in registers,
// become P (bf16) and multiply V (ldmatrix.trans).  Global tokens are scored
// against q~ = q Uk^T (W_up absorbed into the query, exact by linearity of
// Eq. 2) and their values are summed in d_down space.  Other cases (fp32
// storage, d_down = 8) use the CUDA cores: LPT lanes own one token row (one
// 16-byte granule each).  One online softmax (running max m, sum l, log2
// domain) covers an item.
//
// Combine: each item writes (m, l, acc) per head; the warp that arrives last
// for (b, g, hs) merges all chunks, lifts the global part once with Uv and
// writes o = (acc_local + acc_global Uv) / l.  No warp waits on another warp.
#include <type_traits>

#include "dar_common.cuh"
#include "dar_launch.h"
#include "dar_sm100.cuh"

namespace dar {

constexpr int kDecWarps = 8;
constexpr int kDecThreads = kDecWarps * 32;
constexpr int kStages = 3;
constexpr int kSlotBytes = 8192;
constexpr int kHalf = kSlotBytes / 2;
constexpr int kItemStages = 4;     // stages per minimum-size item
constexpr int kMaxChunkScale = 16;  // items grow to at most 16x the minimum (64 pages)
constexpr int kItemsPerWarp = 3;    // chunk sizes aim at about this many items per warp

// bf16 caches with d_down >= 16 use the tensor-core consumer (fed by 2-D TMA).
template <typename T, int DD>
__host__ __device__ constexpr bool decode_uses_mma()
{
    return sizeof(T) == 2 && DD >= 16;
}

// --------------------------------------------------------------------- PTX

using sm100::bulk_g2s;
using sm100::ldsm_x4;
using sm100::ldsm_x4_t;
using sm100::mma_bf16_16816;
using sm100::smem_u32;
using sm100::mbar_expect_tx;
using sm100::mbar_init;
using sm100::mbar_try_wait;

// Bounded wait (see sm100::mbar_wait); a warp that gives up reports to *status.
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, unsigned parity, int32_t *status)
{
    if (sm100::mbar_wait(bar, parity, nullptr))
        return true;
    report(status, DAR_ERR_CUDA);
    return false;
}

// --------------------------------------------------------------------- items

struct Item {
    int it;  // -1 = none
    int b, g, hs, c;
    bool window;
    int t0, t1;  // token range (ring slots, or distant positions)
    int nst;     // stages
    int nwc, nchunks;
};

struct SeqTables {
    const int *pre;  // [B + 1] exclusive prefix of chunk counts
    const int *len;  // [B] validated length (-1 invalid)
    int cw, cd;      // chunk sizes of this launch (multiples of the host's minimum sizes)
};

template <int TPS_W, int TPS_D>
__device__ __forceinline__ Item decode_item(int it, int items, const DecodeArgs &a, SeqTables st)
{
    Item I;
    I.it = it < items ? it : -1;
    I.b = I.g = I.hs = I.c = I.t0 = I.t1 = I.nst = I.nwc = I.nchunks = 0;
    I.window = false;
    if (I.it < 0)
        return I;
    const int per_chunk = a.Hkv * a.HS;
    const int u = it / per_chunk, rem = it % per_chunk;
    I.g = rem / a.HS;
    I.hs = rem % a.HS;
    int lo = 0, hi = a.B;  // largest b with pre[b] <= u
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (st.pre[mid] <= u)
            lo = mid;
        else
            hi = mid;
    }
    I.b = lo;
    I.c = u - st.pre[lo];
    const int L = st.len[lo];
    const int nwin = min(L, a.w), ndist = L - nwin;
    I.nwc = (nwin + st.cw - 1) / st.cw;
    I.nchunks = I.nwc + (ndist + st.cd - 1) / st.cd;
    I.window = I.c < I.nwc;
    if (I.window) {
        I.t0 = I.c * st.cw;
        I.t1 = min(nwin, I.t0 + st.cw);
        I.nst = (I.t1 - I.t0 + TPS_W - 1) / TPS_W;
    } else {
        I.t0 = (I.c - I.nwc) * st.cd;
        I.t1 = min(ndist, I.t0 + st.cd);
        I.nst = (I.t1 - I.t0 + TPS_D - 1) / TPS_D;
    }
    return I;
}

template <int GH>
struct WarpSmem {
    float q[GH][kHeadDim];   // scaled queries
    float qt[GH][kHeadDim];  // q~ (first dd entries); combine scratch
};

template <int GH>
constexpr size_t decode_smem_bytes(int B)
{
    return 1024 + (size_t)kDecWarps * kStages * kSlotBytes + (size_t)kDecWarps * kStages * (8 + 8) +
           (size_t)kDecWarps * sizeof(WarpSmem<GH>) + (size_t)(2 * B + 1) * sizeof(int);
}

// --------------------------------------------------------------------- kernel

// Tensor-core consumer for one stage of ROW-wide rows (64 = ring keys/values,
// d_down = pages), TPS tokens, rows swizzled as the 2-D TMA wrote them.
// q_a: A fragments (KS k-steps) of the GH query rows; o: output fragments
// (ROW/8 n-tiles); m, lpart: the row's running max and this lane's part of the
// running sum (quad-uniform m).
template <int ROW, int TPS, int GH>
__device__ __forceinline__ void mma_stage(uint32_t sK, uint32_t sV, int ntok, unsigned pmask,
                                          const uint32_t (&q_a)[(ROW >= 16 ? ROW / 16 : 1)][4],
                                          float (&o)[ROW / 8][4], float &m, float &lpart, float c2, int lane)
{
    constexpr int KS = ROW / 16;   // k-steps of the score product
    constexpr int ND = ROW / 8;    // n-tiles of the output
    constexpr int RB = ROW * 2;    // bytes per row
    constexpr int SWM = RB / 16 - 1;
    constexpr int TB = TPS < 64 ? TPS : 64;  // tokens per block of the online softmax
    constexpr int NT = TB / 8;
    const int g = lane >> 2, c = lane & 3;
    const int mi = lane >> 3, ri = lane & 7;
    auto swz = [](int t) { return ((t * RB) >> 7) & SWM; };
#pragma unroll 1
    for (int t0 = 0; t0 < TPS; t0 += TB) {
        // ---- scores S[g][token] = q . k  for TB tokens
        float sc[NT][4];
#pragma unroll
        for (int n = 0; n < NT; ++n)
            sc[n][0] = sc[n][1] = sc[n][2] = sc[n][3] = 0.f;
#pragma unroll
        for (int np = 0; np < NT / 2; ++np) {
#pragma unroll
            for (int ks = 0; ks < KS; ++ks) {
                const int tok = t0 + 8 * (2 * np + (mi >> 1)) + ri;
                const int ch = 2 * ks + (mi & 1);
                uint32_t r[4];
                ldsm_x4(sK + tok * RB + ((ch ^ swz(tok)) << 4), r);
                mma_bf16_16816(sc[2 * np], q_a[ks], r[0], r[1]);
                mma_bf16_16816(sc[2 * np + 1], q_a[ks], r[2], r[3]);
            }
        }
        // ---- online softmax on row g (columns 2c, 2c+1 of each n-tile)
        float mx = -INFINITY;
#pragma unroll
        for (int n = 0; n < NT; ++n) {
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                const int tl = t0 + 8 * n + 2 * c + e;
                const bool ok = tl < ntok && ((pmask >> (tl / kPage)) & 1u);
                sc[n][e] = ok ? sc[n][e] : -INFINITY;
                mx = fmaxf(mx, sc[n][e]);
            }
        }
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
        const float mnew = fmaxf(m, mx * c2);
        const float alpha = m == -INFINITY ? 0.f : sm100::ex2_approx(m - mnew);
        const float mneg = mnew == -INFINITY ? 0.f : -mnew;
        m = mnew;
        float ps = 0.f;
        uint32_t pk[NT];
#pragma unroll
        for (int n = 0; n < NT; ++n) {
            const float p0 = sm100::ex2_approx(fmaf(sc[n][0], c2, mneg));
            const float p1 = sm100::ex2_approx(fmaf(sc[n][1], c2, mneg));
            ps += p0 + p1;
            __nv_bfloat162 v = __floats2bfloat162_rn(p0, p1);
            pk[n] = *reinterpret_cast<uint32_t *>(&v);
        }
        lpart = lpart * alpha + ps;
#pragma unroll
        for (int d = 0; d < ND; ++d) {
            o[d][0] *= alpha;
            o[d][1] *= alpha;
        }
        // ---- O += P V  (P rows g as A; V^T tiles by ldmatrix.trans)
#pragma unroll
        for (int kt = 0; kt < TB / 16; ++kt) {
            const uint32_t pa[4] = {pk[2 * kt], 0u, pk[2 * kt + 1], 0u};
            const int tok = t0 + 16 * kt + 8 * (mi & 1) + ri;
#pragma unroll
            for (int dp = 0; dp < ND / 2; ++dp) {
                const int ch = 2 * dp + (mi >> 1);
                uint32_t r[4];
                ldsm_x4_t(sV + tok * RB + ((ch ^ swz(tok)) << 4), r);
                mma_bf16_16816(o[2 * dp], pa, r[0], r[1]);
                mma_bf16_16816(o[2 * dp + 1], pa, r[2], r[3]);
            }
        }
    }
}

template <typename T, int DD, int GH>
__global__ void __launch_bounds__(kDecThreads, 1)
    decode_kernel(const __grid_constant__ CUtensorMap tm_wk, const __grid_constant__ CUtensorMap tm_wv,
                  const __grid_constant__ CUtensorMap tm_pk, const __grid_constant__ CUtensorMap tm_pv,
                  DecodeArgs a)
{
    constexpr int E = Granule<T>::kElems;
    constexpr int ES = sizeof(T);
    constexpr bool kMma = decode_uses_mma<T, DD>();
    constexpr int TPS_W = kHalf / (kHeadDim * ES);           // tokens per ring stage
    constexpr int TPS_D = kHalf / (DD * ES);                 // tokens per page stage
    constexpr int PPS = TPS_D >= kPage ? TPS_D / kPage : 1;  // pages touched per stage
    static_assert(TPS_D % kPage == 0 || kPage % TPS_D == 0, "stages must tile pages");
    static_assert(PPS <= 8, "stage page mask holds 8 pages");

    extern __shared__ __align__(128) unsigned char smem_raw[];
    // swizzled TMA tiles need 1024-byte alignment (static shared data may precede this)
    unsigned char *slots = reinterpret_cast<unsigned char *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));  // [warps][stages][slot]
    uint64_t *bars = reinterpret_cast<uint64_t *>(slots + (size_t)kDecWarps * kStages * kSlotBytes);
    int *meta = reinterpret_cast<int *>(bars + kDecWarps * kStages);  // [warps][stages][2]
    WarpSmem<GH> *wsm = reinterpret_cast<WarpSmem<GH> *>(meta + kDecWarps * kStages * 2);
    int *s_pre = reinterpret_cast<int *>(wsm + kDecWarps);
    int *s_len = s_pre + a.B + 1;
    __shared__ int s_geo[2];  // chunk sizes of this launch

    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int B = a.B, w = a.w;

    if (threadIdx.x < kDecWarps * kStages)
        mbar_init(&bars[threadIdx.x], 1);
    if (blockIdx.x == 0) {  // warm L2 with the small tables every CTA reads first
        for (int i = threadIdx.x * 32; i < B; i += kDecThreads * 32)
            asm volatile("prefetch.global.L2 [%0];" ::"l"(a.seq_lens + i));
    }
    // ---- chunk sizes and counts (warp 0).  The host sized the workspace for the
    // minimum chunks (a.cw, a.cd); the launch scales both by one factor f so that
    // the number of items is about the number of warps (one long stream per
    // warp).  Larger chunks only lower the chunk count, so records still fit.
    if (warp == 0) {
        const int per = (B + 31) / 32;
        const int lo = min(B, lane * per), hi = min(B, lo + per);
        long long units = 0;
        for (int b = lo; b < hi; ++b) {
            int L = a.seq_lens[b];
            if (L < 0 || (long long)L - w > (long long)a.maxp * kPage)
                L = -1;
            s_len[b] = L;
            if (L > 0) {
                const int nwin = min(L, w), ndist = L - nwin;
                units += (nwin + a.cw - 1) / a.cw + (ndist + a.cd - 1) / a.cd;
            }
        }
#pragma unroll
        for (int off = 16; off; off >>= 1)
            units += __shfl_xor_sync(0xffffffffu, units, off);
        const long long target = (long long)gridDim.x * kDecWarps * kItemsPerWarp;
        long long f = (units * a.Hkv * a.HS + target - 1) / target;
        const long long fmax = (long long)(64 * kPage) / a.cd;  // an item spans at most 64 pages
        f = f > fmax ? fmax : f;
        f = f > kMaxChunkScale ? kMaxChunkScale : f;
        f = f < 1 ? 1 : f;
        const int cw = a.cw * (int)f, cd = a.cd * (int)f;
        int run = 0;
        for (int b = lo; b < hi; ++b) {
            const int L = s_len[b];
            int cnt = 0;
            if (L > 0) {
                const int nwin = min(L, w), ndist = L - nwin;
                cnt = (nwin + cw - 1) / cw + (ndist + cd - 1) / cd;
            }
            s_pre[b] = cnt;
            run += cnt;
        }
        int incl = run;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, incl, off);
            if (lane >= off)
                incl += y;
        }
        int base = incl - run;
        for (int b = lo; b < hi; ++b) {
            const int cnt = s_pre[b];
            s_pre[b] = base;
            base += cnt;
        }
        if (lane == 31) {
            s_pre[B] = incl;
            s_geo[0] = cw;
            s_geo[1] = cd;
        }
    }
    sm100::mbar_init_fence();
    __syncthreads();

    // sequences with nothing to attend to get a zero output
    if (blockIdx.x == 0) {
        T *out = static_cast<T *>(a.out);
        for (int b = warp; b < B; b += kDecWarps) {
            if (s_len[b] > 0)
                continue;
            if (s_len[b] < 0 && lane == 0)
                report(a.status, DAR_ERR_CAPACITY);
            for (int i = lane; i < a.Hq * kHeadDim; i += 32)
                out[(size_t)b * a.Hq * kHeadDim + i] = from_f32<T>(0.f);
        }
    }

    const SeqTables tabs{s_pre, s_len, s_geo[0], s_geo[1]};
    const int items = s_pre[B] * a.Hkv * a.HS;
    const int nwarps_total = gridDim.x * kDecWarps;
    unsigned char *my_slots = slots + (size_t)warp * kStages * kSlotBytes;
    uint64_t *my_bars = bars + warp * kStages;
    int *my_meta = meta + warp * kStages * 2;
    WarpSmem<GH> &sc = wsm[warp];
    const T *qg = static_cast<const T *>(a.q);
    const T *wk = static_cast<const T *>(a.win_k);
    const T *wv = static_cast<const T *>(a.win_v);
    const T *pk = static_cast<const T *>(a.pool_kd);
    const T *pv = static_cast<const T *>(a.pool_vd);
    bool alive = true;

    // ---- issue side.  Item indices come from the counter one item ahead; the
    // page ids of the item being copied in and of the next one are held in
    // registers (lane j: pages j and 32 + j of the item).
    const int gw = blockIdx.x + gridDim.x * warp;
    // The counter hands out items from 2 * nwarps on (the first two per warp are
    // static).  Lane 0 keeps the fetched index unread until the following item
    // switch, so the atomic's round trip overlaps a whole item.
    auto fetch_index = [&]() {
        int v = 0;
        if (lane == 0)
            v = atomicAdd(a.sched, 1) + 2 * nwarps_total;
        return v;
    };
    auto use_index = [&](int v) { return __shfl_sync(0xffffffffu, v, 0); };
    auto load_pages = [&](const Item &I) {
        int2 id = make_int2(-1, -1);
        if (I.it >= 0 && !I.window) {
            const int p0 = I.t0 / kPage, np = (I.t1 - 1) / kPage - p0 + 1;
            const int32_t *row = a.block_table + (size_t)I.b * a.maxp + p0;
            if (lane < np)
                id.x = row[lane];
            if (lane + 32 < np)
                id.y = row[lane + 32];
        }
        return id;
    };
    Item iss = decode_item<TPS_W, TPS_D>(gw, items, a, tabs);
    int2 iss_pid = load_pages(iss);
    Item nxt = decode_item<TPS_W, TPS_D>(gw + nwarps_total, items, a, tabs);
    int2 nxt_pid = load_pages(nxt);
    int pending_raw = nxt.it >= 0 ? fetch_index() : items;  // lane 0: the item after `nxt`
    int iss_s = 0;
    int issued = 0, consumed = 0;               // stages issued / consumed by this warp
    int iss_slot = 0, con_slot = 0;             // ring positions
    unsigned con_phase = 0;                     // parity of the consumer's current pass over the ring
    auto page_id = [&](int j) {  // page j (0..63) of the item being issued
        const int x = __shfl_sync(0xffffffffu, iss_pid.x, j & 31);
        const int y = __shfl_sync(0xffffffffu, iss_pid.y, j & 31);
        return j < 32 ? x : y;
    };

    auto issue_one = [&]() {  // copy the next stage of `iss` into its slot
        const int slot = iss_slot;
        iss_slot = iss_slot + 1 == kStages ? 0 : iss_slot + 1;
        unsigned char *dst = my_slots + (size_t)slot * kSlotBytes;
        uint64_t *bar = &my_bars[slot];
        const int s = iss_s;
        if (iss.window) {
            const int tb = iss.t0 + s * TPS_W, te = min(iss.t1, tb + TPS_W);
            if (lane == 0) {
                my_meta[slot * 2 + 0] = iss.it;
                my_meta[slot * 2 + 1] = (s << 8) | 0xff;
                if constexpr (kMma) {  // whole boxes of TPS_W rows, 128-byte swizzle
                    const int y = (iss.b * a.Hkv + iss.g) * w + tb;
                    mbar_expect_tx(bar, 2 * TPS_W * kHeadDim * ES);
                    sm100::tma_load_2d_u(smem_u32(dst), &tm_wk, 0, y, bar);
                    sm100::tma_load_2d_u(smem_u32(dst + kHalf), &tm_wv, 0, y, bar);
                } else {
                    const unsigned bytes = (unsigned)(te - tb) * kHeadDim * ES;
                    const size_t off = ((size_t)(iss.b * a.Hkv + iss.g) * w + tb) * kHeadDim;
                    mbar_expect_tx(bar, 2 * bytes);
                    bulk_g2s(dst, wk + off, bytes, bar);
                    bulk_g2s(dst + kHalf, wv + off, bytes, bar);
                }
            }
        } else {
            const int tb = iss.t0 + s * TPS_D, te = min(iss.t1, tb + TPS_D);
            const int pfirst = tb / kPage - iss.t0 / kPage;  // index within the item's pages
            unsigned mask = 0, total = 0;
#pragma unroll
            for (int j = 0; j < PPS; ++j) {
                const int id = page_id(pfirst + j);
                const int ptb = max(tb, (tb / kPage + j) * kPage);
                const int pte = min(te, (tb / kPage + j + 1) * kPage);
                if (pte > ptb) {
                    if (id >= 0 && id < a.num_pages) {
                        mask |= 1u << j;
                        // the 2-D path copies whole boxes of min(64, TPS_D) rows
                        total += (unsigned)(kMma ? (TPS_D < kPage ? TPS_D : kPage) : (pte - ptb)) * DD * ES;
                    } else if (lane == 0) {
                        report(a.status, DAR_ERR_CAPACITY);
                    }
                }
            }
            if (lane == 0) {
                my_meta[slot * 2 + 0] = iss.it;
                my_meta[slot * 2 + 1] = (s << 8) | (int)mask;
                mbar_expect_tx(bar, 2 * total);
            }
#pragma unroll
            for (int j = 0; j < PPS; ++j) {
                const int id = page_id(pfirst + j);
                const int ptb = max(tb, (tb / kPage + j) * kPage);
                const int pte = min(te, (tb / kPage + j + 1) * kPage);
                if (lane == 0 && ((mask >> j) & 1u)) {
                    const size_t doff = (size_t)(ptb - tb) * DD * ES;
                    if constexpr (kMma) {
                        const int y = (id * a.Hkv + iss.g) * kPage + (ptb % kPage);
                        sm100::tma_load_2d_u(smem_u32(dst + doff), &tm_pk, 0, y, bar);
                        sm100::tma_load_2d_u(smem_u32(dst + kHalf + doff), &tm_pv, 0, y, bar);
                    } else {
                        const unsigned bytes = (unsigned)(pte - ptb) * DD * ES;
                        const size_t src = (((size_t)id * a.Hkv + iss.g) * kPage + (ptb % kPage)) * DD;
                        bulk_g2s(dst + doff, pk + src, bytes, bar);
                        bulk_g2s(dst + kHalf + doff, pv + src, bytes, bar);
                    }
                }
            }
        }
        __syncwarp();
        ++issued;
        if (++iss_s == iss.nst) {  // move on to the next item
            iss = nxt;
            iss_pid = nxt_pid;
            iss_s = 0;
            if (iss.it >= 0) {
                nxt = decode_item<TPS_W, TPS_D>(use_index(pending_raw), items, a, tabs);
                nxt_pid = load_pages(nxt);
                pending_raw = nxt.it >= 0 ? fetch_index() : items;
            }
        }
    };
    // Start from zeroed slots: a stage whose copies do not cover the whole slot
    // (a short last page) leaves rows that are masked out but still enter the
    // tensor-core products, so they must hold finite values.
    {
        uint4 *z = reinterpret_cast<uint4 *>(my_slots);
        for (int i = lane; i < kStages * kSlotBytes / 16; i += 32)
            z[i] = make_uint4(0, 0, 0, 0);
        sm100::fence_proxy_async_smem();
        __syncwarp();
    }
    while (issued - consumed < kStages && iss.it >= 0)
        issue_one();

    // ---- consume side
    Item cur = decode_item<TPS_W, TPS_D>(-1, 0, a, tabs);
    // tensor-core consumer state: A fragments of q (ring) / q~ (pages), output
    // fragments of row g = lane / 4 (query head h0 + g when g < GH)
    constexpr int KSD = DD >= 16 ? DD / 16 : 1;
    uint32_t qa_w[4][4], qa_d[KSD][4];
    float ow[8][4], od[DD / 8 > 0 ? DD / 8 : 1][4];
    float mm = -INFINITY, lp = 0.f;
    float m[GH], l[GH], acc[GH][E], qr[GH][E];
#pragma unroll
    for (int k = 0; k < GH; ++k) {
        m[k] = -INFINITY;
        l[k] = 0.f;
#pragma unroll
        for (int e = 0; e < E; ++e)
            acc[k][e] = qr[k][e] = 0.f;
    }
    while (consumed < issued) {
        const int slot = con_slot;
        const unsigned parity = con_phase;
        if (!mbar_wait(&my_bars[slot], parity, a.status)) {
            alive = false;
            break;
        }
        __syncwarp();
        const int mit = my_meta[slot * 2 + 0];
        const int minfo = my_meta[slot * 2 + 1];
        const int s = minfo >> 8;
        const unsigned pmask = (unsigned)(minfo & 0xff);
        if (s == 0) {
            // ---- new item: stage the queries (and q~ for the pages)
            cur = decode_item<TPS_W, TPS_D>(mit, items, a, tabs);
            const int h0 = cur.g * a.G + cur.hs * GH;
            const bool pages = !cur.window;
            const float *Ukg = a.Uk + (size_t)cur.g * DD * kHeadDim;
            // issue this lane's first Uk row and the query rows together (one round trip)
            float4 ur[kHeadDim / 4];
            if (pages && lane < GH * DD) {
                const float4 *src4 = reinterpret_cast<const float4 *>(Ukg + (size_t)(lane % DD) * kHeadDim);
#pragma unroll
                for (int t4 = 0; t4 < kHeadDim / 4; ++t4)
                    ur[t4] = __ldg(src4 + t4);
            }
            const float qs = kMma ? 1.f : a.qscale;  // the tensor-core path scales the scores instead
#pragma unroll
            for (int k = 0; k < GH; ++k) {
                const T *qrow = qg + ((size_t)cur.b * a.Hq + h0 + k) * kHeadDim;
                sc.q[k][lane] = to_f32(qrow[lane]) * qs;
                sc.q[k][lane + 32] = to_f32(qrow[lane + 32]) * qs;
            }
            __syncwarp();
            if (pages) {
                // q~[k][c] = sum_t q[k][t] Uk[g][c][t]
                for (int o = lane; o < GH * DD; o += 32) {
                    const int k = o / DD, cc = o % DD;
                    if (o != lane) {
                        const float4 *src4 = reinterpret_cast<const float4 *>(Ukg + (size_t)cc * kHeadDim);
#pragma unroll
                        for (int t4 = 0; t4 < kHeadDim / 4; ++t4)
                            ur[t4] = __ldg(src4 + t4);
                    }
                    float p0 = 0.f, p1 = 0.f, p2 = 0.f, p3 = 0.f;
#pragma unroll
                    for (int t4 = 0; t4 < kHeadDim / 4; ++t4) {
                        p0 = fmaf(sc.q[k][4 * t4 + 0], ur[t4].x, p0);
                        p1 = fmaf(sc.q[k][4 * t4 + 1], ur[t4].y, p1);
                        p2 = fmaf(sc.q[k][4 * t4 + 2], ur[t4].z, p2);
                        p3 = fmaf(sc.q[k][4 * t4 + 3], ur[t4].w, p3);
                    }
                    sc.qt[k][cc] = (p0 + p1) + (p2 + p3);
                }
                __syncwarp();
            }
            if constexpr (kMma) {
                // A fragments: row g holds head h0 + g (rows >= GH are zero)
                const int g = lane >> 2, c = lane & 3;
                auto frag = [&](const float *row, int k0) -> uint32_t {
                    if (g >= GH)
                        return 0u;
                    __nv_bfloat162 v = __floats2bfloat162_rn(row[k0], row[k0 + 1]);
                    return *reinterpret_cast<uint32_t *>(&v);
                };
                const float *qrow = sc.q[g < GH ? g : 0];
                const float *qtrow = sc.qt[g < GH ? g : 0];
#pragma unroll
                for (int ks = 0; ks < 4; ++ks) {
                    qa_w[ks][0] = frag(qrow, 16 * ks + 2 * c);
                    qa_w[ks][2] = frag(qrow, 16 * ks + 2 * c + 8);
                    qa_w[ks][1] = qa_w[ks][3] = 0u;
                }
#pragma unroll
                for (int ks = 0; ks < KSD; ++ks) {
                    qa_d[ks][0] = frag(qtrow, 16 * ks + 2 * c);
                    qa_d[ks][2] = frag(qtrow, 16 * ks + 2 * c + 8);
                    qa_d[ks][1] = qa_d[ks][3] = 0u;
                }
#pragma unroll
                for (int d = 0; d < 8; ++d)
                    ow[d][0] = ow[d][1] = ow[d][2] = ow[d][3] = 0.f;
#pragma unroll
                for (int d = 0; d < (DD / 8 > 0 ? DD / 8 : 1); ++d)
                    od[d][0] = od[d][1] = od[d][2] = od[d][3] = 0.f;
                mm = -INFINITY;
                lp = 0.f;
            } else {
                const int ROWc = cur.window ? kHeadDim : DD;
                const int sub = lane % (ROWc / E);
#pragma unroll
                for (int k = 0; k < GH; ++k) {
#pragma unroll
                    for (int e = 0; e < E; ++e)
                        qr[k][e] = cur.window ? sc.q[k][sub * E + e] : sc.qt[k][sub * E + e];
                    m[k] = -INFINITY;
                    l[k] = 0.f;
#pragma unroll
                    for (int e = 0; e < E; ++e)
                        acc[k][e] = 0.f;
                }
            }
        }

        // ---- this stage's tokens
        const unsigned char *src = my_slots + (size_t)slot * kSlotBytes;
        auto run_stage = [&](auto row_tag) {
            constexpr int ROW = decltype(row_tag)::value;
            constexpr int LPT = ROW / E;
            constexpr int TPI = 32 / LPT;
            constexpr int TPS = kHalf / (ROW * ES);
            constexpr int NI = TPS / TPI;  // warp-wide 16-byte loads per half slot
            constexpr int U = NI < 4 ? NI : 4;
            const int grp = lane / LPT, sub = lane % LPT;
            const int tb = cur.t0 + s * TPS;
            const int ntok = min(cur.t1 - tb, TPS);
#pragma unroll
            for (int u0 = 0; u0 < NI; u0 += U) {
                float sk[GH][U];
                uint4 vr[U];
                bool valid[U];
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    const int tl = (u0 + u) * TPI + grp;
                    valid[u] = tl < ntok && (ROW == kHeadDim || ((pmask >> (tl / kPage)) & 1u));
                    const size_t eoff = ((size_t)tl * ROW + sub * E) * ES;
                    const uint4 kr = *reinterpret_cast<const uint4 *>(src + eoff);
                    // masked rows may hold stale or never-written bytes: never let them reach acc
                    vr[u] = valid[u] ? *reinterpret_cast<const uint4 *>(src + kHalf + eoff)
                                     : make_uint4(0, 0, 0, 0);
                    float kf[E];
                    unpack(kr, kf, T());
#pragma unroll
                    for (int k = 0; k < GH; ++k) {
                        float d0 = 0.f;
#pragma unroll
                        for (int e = 0; e < E; ++e)
                            d0 = fmaf(qr[k][e], kf[e], d0);
                        sk[k][u] = d0;
                    }
                }
#pragma unroll
                for (int off = 1; off < LPT; off <<= 1)
#pragma unroll
                    for (int k = 0; k < GH; ++k)
#pragma unroll
                        for (int u = 0; u < U; ++u)
                            sk[k][u] += __shfl_xor_sync(0xffffffffu, sk[k][u], off);
#pragma unroll
                for (int k = 0; k < GH; ++k) {
                    float mx = -INFINITY;
#pragma unroll
                    for (int u = 0; u < U; ++u)
                        if (valid[u])
                            mx = fmaxf(mx, sk[k][u]);
                    const float mnew = fmaxf(m[k], mx);
                    const float alpha = (m[k] == -INFINITY) ? 0.f : exp2f(m[k] - mnew);
                    float psum = 0.f;
#pragma unroll
                    for (int u = 0; u < U; ++u) {
                        sk[k][u] = valid[u] ? exp2f(sk[k][u] - mnew) : 0.f;
                        psum += sk[k][u];
                    }
                    l[k] = l[k] * alpha + psum;
                    m[k] = mnew;
#pragma unroll
                    for (int e = 0; e < E; ++e)
                        acc[k][e] *= alpha;
                }
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    float vf[E];
                    unpack(vr[u], vf, T());
#pragma unroll
                    for (int k = 0; k < GH; ++k)
#pragma unroll
                        for (int e = 0; e < E; ++e)
                            acc[k][e] = fmaf(sk[k][u], vf[e], acc[k][e]);
                }
            }
        };
        if constexpr (kMma) {
            const uint32_t sK = smem_u32(src), sV = smem_u32(src + kHalf);
            if (cur.window)
                mma_stage<kHeadDim, TPS_W, GH>(sK, sV, min(cur.t1 - (cur.t0 + s * TPS_W), TPS_W), 0xffu, qa_w, ow,
                                              mm, lp, a.qscale, lane);
            else
                mma_stage<DD, TPS_D, GH>(sK, sV, min(cur.t1 - (cur.t0 + s * TPS_D), TPS_D), pmask, qa_d, od, mm,
                                         lp, a.qscale, lane);
        } else {
            if (cur.window)
                run_stage(std::integral_constant<int, kHeadDim>());
            else
                run_stage(std::integral_constant<int, DD>());
        }
        __syncwarp();
        ++consumed;
        if (++con_slot == kStages) {
            con_slot = 0;
            con_phase ^= 1u;
        }
        if (iss.it >= 0)
            issue_one();  // refill the slot just read

        if (s + 1 < cur.nst)
            continue;

        // ---- item done: write the partial result (m, l, acc) of every head
        const int h0 = cur.g * a.G + cur.hs * GH;
        if constexpr (kMma) {
            lp += __shfl_xor_sync(0xffffffffu, lp, 1);
            lp += __shfl_xor_sync(0xffffffffu, lp, 2);
            const int g = lane >> 2, c = lane & 3;
            if (g < GH) {
                const size_t rec = ((size_t)cur.b * a.Hq + h0 + g) * a.maxc + cur.c;
                float *ra = a.rec_acc + rec * kHeadDim;
                if (cur.window) {
#pragma unroll
                    for (int d = 0; d < 8; ++d)
                        *reinterpret_cast<float2 *>(ra + 8 * d + 2 * c) = make_float2(ow[d][0], ow[d][1]);
                } else {
#pragma unroll
                    for (int d = 0; d < (DD / 8 > 0 ? DD / 8 : 1); ++d)
                        *reinterpret_cast<float2 *>(ra + 8 * d + 2 * c) = make_float2(od[d][0], od[d][1]);
                }
                if (c == 0) {
                    a.rec_m[rec] = mm;
                    a.rec_l[rec] = lp;
                }
            }
        } else {
        const int LPTc = (cur.window ? kHeadDim : DD) / E;
        for (int off = LPTc; off < 32; off <<= 1) {
#pragma unroll
            for (int k = 0; k < GH; ++k) {
                const float mo = __shfl_xor_sync(0xffffffffu, m[k], off);
                const float lo = __shfl_xor_sync(0xffffffffu, l[k], off);
                const float mn = fmaxf(m[k], mo);
                const float fa = (m[k] == -INFINITY) ? 0.f : exp2f(m[k] - mn);
                const float fb = (mo == -INFINITY) ? 0.f : exp2f(mo - mn);
                l[k] = l[k] * fa + lo * fb;
#pragma unroll
                for (int e = 0; e < E; ++e) {
                    const float ao = __shfl_xor_sync(0xffffffffu, acc[k][e], off);
                    acc[k][e] = acc[k][e] * fa + ao * fb;
                }
                m[k] = mn;
            }
        }
#pragma unroll
        for (int k = 0; k < GH; ++k) {
            const size_t rec = ((size_t)cur.b * a.Hq + h0 + k) * a.maxc + cur.c;
            if (lane < LPTc) {
                float4 *dstv = reinterpret_cast<float4 *>(a.rec_acc + rec * kHeadDim + lane * E);
#pragma unroll
                for (int e4 = 0; e4 < E / 4; ++e4)
                    dstv[e4] = make_float4(acc[k][4 * e4], acc[k][4 * e4 + 1], acc[k][4 * e4 + 2],
                                           acc[k][4 * e4 + 3]);
            }
            if (lane == 0) {
                a.rec_m[rec] = m[k];
                a.rec_l[rec] = l[k];
            }
        }
        }
        // publish the record, then count the arrival (acquire-release at GPU scope)
        asm volatile("fence.acq_rel.gpu;" ::: "memory");
        __syncwarp();
        int arrived = 0;
        int32_t *cnt = a.counters + ((size_t)cur.b * a.Hkv + cur.g) * a.HS + cur.hs;
        if (lane == 0)
            asm volatile("atom.add.acq_rel.gpu.global.s32 %0, [%1], 1;" : "=r"(arrived) : "l"(cnt) : "memory");
        arrived = __shfl_sync(0xffffffffu, arrived, 0);
        if (arrived != cur.nchunks - 1)
            continue;

        // ---- last arrival for (b, g, hs): merge every chunk
        asm volatile("fence.acq_rel.gpu;" ::: "memory");
        const int nch = cur.nchunks, nwc = cur.nwc;
        const float *Uv = a.Uv + (size_t)cur.g * DD * kHeadDim;
        T *out = static_cast<T *>(a.out);
#pragma unroll 1
        for (int k = 0; k < GH; ++k) {
            const size_t rec0 = ((size_t)cur.b * a.Hq + h0 + k) * a.maxc;
            float M = -INFINITY;
            for (int c0 = 0; c0 < nch; c0 += 32)
                if (c0 + lane < nch)
                    M = fmaxf(M, __ldcg(a.rec_m + rec0 + c0 + lane));
#pragma unroll
            for (int off = 16; off; off >>= 1)
                M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
            float lsum = 0.f, o0 = 0.f, o1 = 0.f, gd0 = 0.f, gd1 = 0.f;
            for (int c0 = 0; c0 < nch; c0 += 32) {
                float f = 0.f;
                if (c0 + lane < nch) {
                    f = exp2f(__ldcg(a.rec_m + rec0 + c0 + lane) - M);
                    lsum = fmaf(f, __ldcg(a.rec_l + rec0 + c0 + lane), lsum);
                }
                const int jn = min(32, nch - c0);
#pragma unroll 4
                for (int j = 0; j < jn; ++j) {
                    const float fj = __shfl_sync(0xffffffffu, f, j);
                    const int cc = c0 + j;
                    const float *ra = a.rec_acc + (rec0 + cc) * kHeadDim;
                    if (cc < nwc) {
                        const float2 v = __ldcg(reinterpret_cast<const float2 *>(ra) + lane);
                        o0 = fmaf(fj, v.x, o0);
                        o1 = fmaf(fj, v.y, o1);
                    } else {
                        if (lane < DD)
                            gd0 = fmaf(fj, __ldcg(ra + lane), gd0);
                        if (lane + 32 < DD)
                            gd1 = fmaf(fj, __ldcg(ra + lane + 32), gd1);
                    }
                }
            }
#pragma unroll
            for (int off = 16; off; off >>= 1)
                lsum += __shfl_xor_sync(0xffffffffu, lsum, off);
            if (lane < DD)
                sc.qt[0][lane] = gd0;
            if (lane + 32 < DD)
                sc.qt[0][lane + 32] = gd1;
            __syncwarp();
#pragma unroll 4
            for (int cc = 0; cc < DD; ++cc) {
                const float gv = sc.qt[0][cc];
                const float2 u2 = __ldg(reinterpret_cast<const float2 *>(Uv + (size_t)cc * kHeadDim) + lane);
                o0 = fmaf(gv, u2.x, o0);
                o1 = fmaf(gv, u2.y, o1);
            }
            __syncwarp();
            const float inv = 1.f / lsum;
            T *orow = out + ((size_t)cur.b * a.Hq + h0 + k) * kHeadDim;
            orow[2 * lane] = from_f32<T>(o0 * inv);
            orow[2 * lane + 1] = from_f32<T>(o1 * inv);
        }
        if (lane == 0)
            *cnt = 0;  // ready for the next call
    }

    if (!alive) {
        // a wait gave up: let this warp's copies still in flight land (bounded) before leaving
        for (int r = consumed + 1; r < issued; ++r)
            mbar_wait(&my_bars[r % kStages], (unsigned)((r / kStages) & 1), a.status);
    }
    // the last warp to leave resets the item counter for the next call
    if (lane == 0) {
        if (atomicAdd(a.sched + 1, 1) == nwarps_total - 1) {
            a.sched[0] = 0;
            a.sched[1] = 0;
        }
    }
}

// --------------------------------------------------------------------- launch

DecodeGeometry decode_geometry(dar_dtype dt, int Hq, int Hkv, int dd, int w, int maxp)
{
    DecodeGeometry gm;
    const int esz = dt == DAR_F32 ? 4 : 2;
    gm.cw = kItemStages * (kHalf / (kHeadDim * esz));
    gm.cd = kItemStages * (kHalf / (dd * esz));
    gm.maxc = (w + gm.cw - 1) / gm.cw + (maxp * kPage + gm.cd - 1) / gm.cd;
    const int G = Hq / Hkv;
    gm.GH = (G % 4 == 0) ? 4 : (G % 2 == 0) ? 2 : 1;
    gm.HS = G / gm.GH;
    return gm;
}

template <typename T, int DD, int GH>
static cudaError_t decode_t(const DecodeArgs &a, cudaStream_t s)
{
    auto kern = decode_kernel<T, DD, GH>;
    CUtensorMap m_wk{}, m_wv{}, m_pk{}, m_pv{};
    if (decode_uses_mma<T, DD>()) {
        constexpr int tps_w = kHalf / (kHeadDim * 2), tps_d = kHalf / (DD * 2);
        const int pr = tps_d < kPage ? tps_d : kPage;
        const unsigned long long ring_rows = (unsigned long long)a.B * a.Hkv * a.w;
        const unsigned long long pool_rows = (unsigned long long)(a.num_pages > 0 ? a.num_pages : 1) * a.Hkv * kPage;
        if (!make_tma_2d_bf16(&m_wk, a.win_k, ring_rows, kHeadDim, tps_w) ||
            !make_tma_2d_bf16(&m_wv, a.win_v, ring_rows, kHeadDim, tps_w) ||
            !make_tma_2d_bf16(&m_pk, a.pool_kd, pool_rows, DD, pr) ||
            !make_tma_2d_bf16(&m_pv, a.pool_vd, pool_rows, DD, pr))
            return cudaErrorInvalidValue;
    }
    // one-time set-up per instantiation (kept out of the launch path so launches
    // stay cheap and can be captured in a CUDA graph)
    static int sms = 0;
    if (sms == 0) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)decode_smem_bytes<GH>(DAR_DECODE_MAX_BATCH));
        if (e != cudaSuccess)
            return e;
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    }
    kern<<<sms, kDecThreads, decode_smem_bytes<GH>(a.B), s>>>(m_wk, m_wv, m_pk, m_pv, a);
    return cudaGetLastError();
}

template <typename T, int DD>
static cudaError_t decode_dd(const DecodeArgs &a, cudaStream_t s)
{
    switch (a.GH) {
    case 4: return decode_t<T, DD, 4>(a, s);
    case 2: return decode_t<T, DD, 2>(a, s);
    default: return decode_t<T, DD, 1>(a, s);
    }
}

template <typename T>
static cudaError_t decode_type(int dd, const DecodeArgs &a, cudaStream_t s)
{
    switch (dd) {
    case 8: return decode_dd<T, 8>(a, s);
    case 16: return decode_dd<T, 16>(a, s);
    case 32: return decode_dd<T, 32>(a, s);
    case 64: return decode_dd<T, 64>(a, s);
    default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_decode(dar_dtype dt, int dd, const DecodeArgs &a, cudaStream_t s)
{
    if (a.B == 0)
        return cudaSuccess;
    return dt == DAR_F32 ? decode_type<float>(dd, a, s) : decode_type<bf16>(dd, a, s);
}

}  // namespace dar
