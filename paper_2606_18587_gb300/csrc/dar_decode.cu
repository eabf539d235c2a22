// dar_decode.cu -- one decode step of DAR attention over the mixed-dimension
// cache (Eq. 3-4 for the query at position L_b - 1; cache scheme of Sec. 5).
//
// Work decomposition (split-K over the sequence):
//   item = (sequence b, KV head g, head slice hs, chunk c).  Chunks 0..nwc-1
//   cover the ring (full d = 64 keys/values, `cw` tokens each); the rest cover
//   the pages (d_down vectors, `cd` tokens each, page aligned).  A warp takes
//   its first item statically and later ones from an atomic counter.
//
// Streaming: every warp owns a ring of kStages shared-memory slots of
// kSlotBytes (keys in the first half, values in the second).  Lane 0 fills a
// slot with 1-D TMA bulk copies (cp.async.bulk, completion counted on the
// slot's mbarrier) and the warp consumes slots in order, refilling each one as
// soon as it has been read, across item boundaries; page ids are loaded one
// item ahead.  So every warp keeps up to kStages * kSlotBytes of cache in
// flight while it computes.
//
// Compute: LPT lanes own one token row (one 16-byte granule each), the GH
// query heads of the slice share every row.  Global tokens are scored against
// q~ = q Uk^T (W_up absorbed into the query, exact by linearity of Eq. 2) and
// their values are summed in d_down space.  One online softmax (running max
// m, sum l, log2 domain) covers the item.
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
constexpr int kItemStages = 4;  // stages per full item

// --------------------------------------------------------------------- PTX

using sm100::bulk_g2s;
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
    I.nwc = (nwin + a.cw - 1) / a.cw;
    I.nchunks = I.nwc + (ndist + a.cd - 1) / a.cd;
    I.window = I.c < I.nwc;
    if (I.window) {
        I.t0 = I.c * a.cw;
        I.t1 = min(nwin, I.t0 + a.cw);
        I.nst = (I.t1 - I.t0 + TPS_W - 1) / TPS_W;
    } else {
        I.t0 = (I.c - I.nwc) * a.cd;
        I.t1 = min(ndist, I.t0 + a.cd);
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
    return (size_t)kDecWarps * kStages * kSlotBytes + (size_t)kDecWarps * kStages * (8 + 8) +
           (size_t)kDecWarps * sizeof(WarpSmem<GH>) + (size_t)(2 * B + 1) * sizeof(int);
}

// --------------------------------------------------------------------- kernel

template <typename T, int DD, int GH>
__global__ void __launch_bounds__(kDecThreads, 1) decode_kernel(DecodeArgs a)
{
    constexpr int E = Granule<T>::kElems;
    constexpr int ES = sizeof(T);
    constexpr int TPS_W = kHalf / (kHeadDim * ES);           // tokens per ring stage
    constexpr int TPS_D = kHalf / (DD * ES);                 // tokens per page stage
    constexpr int PPS = TPS_D >= kPage ? TPS_D / kPage : 1;  // pages touched per stage
    static_assert(TPS_D % kPage == 0 || kPage % TPS_D == 0, "stages must tile pages");
    static_assert(PPS <= 8, "stage page mask holds 8 pages");

    extern __shared__ __align__(128) unsigned char smem_raw[];
    unsigned char *slots = smem_raw;  // [warps][stages][slot]
    uint64_t *bars = reinterpret_cast<uint64_t *>(slots + (size_t)kDecWarps * kStages * kSlotBytes);
    int *meta = reinterpret_cast<int *>(bars + kDecWarps * kStages);  // [warps][stages][2]
    WarpSmem<GH> *wsm = reinterpret_cast<WarpSmem<GH> *>(meta + kDecWarps * kStages * 2);
    int *s_pre = reinterpret_cast<int *>(wsm + kDecWarps);
    int *s_len = s_pre + a.B + 1;

    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int B = a.B, w = a.w;

    if (threadIdx.x < kDecWarps * kStages)
        mbar_init(&bars[threadIdx.x], 1);
    // ---- chunk counts and their prefix (warp 0)
    if (warp == 0) {
        const int per = (B + 31) / 32;
        const int lo = min(B, lane * per), hi = min(B, lo + per);
        int run = 0;
        for (int b = lo; b < hi; ++b) {
            int L = a.seq_lens[b];
            if (L < 0 || (long long)L - w > (long long)a.maxp * kPage)
                L = -1;
            s_len[b] = L;
            int cnt = 0;
            if (L > 0) {
                const int nwin = min(L, w), ndist = L - nwin;
                cnt = (nwin + a.cw - 1) / a.cw + (ndist + a.cd - 1) / a.cd;
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
        if (lane == 31)
            s_pre[B] = incl;
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

    const SeqTables tabs{s_pre, s_len};
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

    // ---- issue side: the item being copied in and the next one (page ids prefetched)
    auto next_index = [&]() {
        int v = 0;
        if (lane == 0)
            v = atomicAdd(a.sched, 1) + nwarps_total;
        return __shfl_sync(0xffffffffu, v, 0);
    };
    auto load_pages = [&](const Item &I) {  // lane j: page id of the item's j-th page
        int id = -1;
        if (I.it >= 0 && !I.window) {
            const int p0 = I.t0 / kPage, np = (I.t1 - 1) / kPage - p0 + 1;
            if (lane < np)
                id = a.block_table[(size_t)I.b * a.maxp + p0 + lane];
        }
        return id;
    };
    Item iss = decode_item<TPS_W, TPS_D>(blockIdx.x + gridDim.x * warp, items, a, tabs);
    int iss_pid = load_pages(iss);
    int nxt_it = iss.it >= 0 ? next_index() : items;
    Item nxt = decode_item<TPS_W, TPS_D>(nxt_it, items, a, tabs);
    int nxt_pid = load_pages(nxt);
    int iss_s = 0;
    long long issued = 0, consumed = 0;

    auto issue_one = [&]() {  // copy the next stage of `iss` into its slot
        const int slot = (int)(issued % kStages);
        unsigned char *dst = my_slots + (size_t)slot * kSlotBytes;
        uint64_t *bar = &my_bars[slot];
        const int s = iss_s;
        if (iss.window) {
            const int tb = iss.t0 + s * TPS_W, te = min(iss.t1, tb + TPS_W);
            const unsigned bytes = (unsigned)(te - tb) * kHeadDim * ES;
            const size_t off = ((size_t)(iss.b * a.Hkv + iss.g) * w + tb) * kHeadDim;
            if (lane == 0) {
                my_meta[slot * 2 + 0] = iss.it;
                my_meta[slot * 2 + 1] = (s << 8) | 0xff;
                mbar_expect_tx(bar, 2 * bytes);
                bulk_g2s(dst, wk + off, bytes, bar);
                bulk_g2s(dst + kHalf, wv + off, bytes, bar);
            }
        } else {
            const int tb = iss.t0 + s * TPS_D, te = min(iss.t1, tb + TPS_D);
            const int pfirst = tb / kPage - iss.t0 / kPage;  // index within the item's pages
            unsigned mask = 0, total = 0;
#pragma unroll
            for (int j = 0; j < PPS; ++j) {
                const int id = __shfl_sync(0xffffffffu, iss_pid, (pfirst + j) & 31);
                const int ptb = max(tb, (tb / kPage + j) * kPage);
                const int pte = min(te, (tb / kPage + j + 1) * kPage);
                if (pte > ptb) {
                    if (id >= 0 && id < a.num_pages) {
                        mask |= 1u << j;
                        total += (unsigned)(pte - ptb) * DD * ES;
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
                const int id = __shfl_sync(0xffffffffu, iss_pid, (pfirst + j) & 31);
                const int ptb = max(tb, (tb / kPage + j) * kPage);
                const int pte = min(te, (tb / kPage + j + 1) * kPage);
                if (lane == 0 && ((mask >> j) & 1u)) {
                    const unsigned bytes = (unsigned)(pte - ptb) * DD * ES;
                    const size_t src = (((size_t)id * a.Hkv + iss.g) * kPage + (ptb % kPage)) * DD;
                    const size_t doff = (size_t)(ptb - tb) * DD * ES;
                    bulk_g2s(dst + doff, pk + src, bytes, bar);
                    bulk_g2s(dst + kHalf + doff, pv + src, bytes, bar);
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
                nxt_it = next_index();
                nxt = decode_item<TPS_W, TPS_D>(nxt_it, items, a, tabs);
                nxt_pid = load_pages(nxt);
            }
        }
    };
    while (issued - consumed < kStages && iss.it >= 0)
        issue_one();

    // ---- consume side
    Item cur = decode_item<TPS_W, TPS_D>(-1, 0, a, tabs);
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
        const int slot = (int)(consumed % kStages);
        const unsigned parity = (unsigned)((consumed / kStages) & 1);
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
#pragma unroll
            for (int k = 0; k < GH; ++k) {
                const T *qrow = qg + ((size_t)cur.b * a.Hq + h0 + k) * kHeadDim;
                sc.q[k][lane] = to_f32(qrow[lane]) * a.qscale;
                sc.q[k][lane + 32] = to_f32(qrow[lane + 32]) * a.qscale;
            }
            __syncwarp();
            if (!cur.window) {
                const float *Uk = a.Uk + (size_t)cur.g * DD * kHeadDim;
                for (int o = lane; o < GH * DD; o += 32) {
                    const int k = o / DD, cc = o % DD;
                    const float4 *ur = reinterpret_cast<const float4 *>(Uk + (size_t)cc * kHeadDim);
                    float p0 = 0.f, p1 = 0.f, p2 = 0.f, p3 = 0.f;
#pragma unroll
                    for (int t4 = 0; t4 < kHeadDim / 4; ++t4) {
                        const float4 u4 = __ldg(ur + t4);
                        p0 = fmaf(sc.q[k][4 * t4 + 0], u4.x, p0);
                        p1 = fmaf(sc.q[k][4 * t4 + 1], u4.y, p1);
                        p2 = fmaf(sc.q[k][4 * t4 + 2], u4.z, p2);
                        p3 = fmaf(sc.q[k][4 * t4 + 3], u4.w, p3);
                    }
                    sc.qt[k][cc] = (p0 + p1) + (p2 + p3);
                }
                __syncwarp();
            }
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
        if (cur.window)
            run_stage(std::integral_constant<int, kHeadDim>());
        else
            run_stage(std::integral_constant<int, DD>());
        __syncwarp();
        ++consumed;
        if (iss.it >= 0)
            issue_one();  // refill the slot just read

        if (s + 1 < cur.nst)
            continue;

        // ---- item done: merge lane groups, write the partial result
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
        const int h0 = cur.g * a.G + cur.hs * GH;
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
        __threadfence();
        __syncwarp();
        int arrived = 0;
        int32_t *cnt = a.counters + ((size_t)cur.b * a.Hkv + cur.g) * a.HS + cur.hs;
        if (lane == 0)
            arrived = atomicAdd(cnt, 1);
        arrived = __shfl_sync(0xffffffffu, arrived, 0);
        if (arrived != cur.nchunks - 1)
            continue;

        // ---- last arrival for (b, g, hs): merge every chunk
        __threadfence();
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
        for (long long r = consumed + 1; r < issued; ++r)
            mbar_wait(&my_bars[r % kStages], (unsigned)((r / kStages) & 1), a.status);
    }
    // the last warp to leave resets the scheduler for the next call
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
    kern<<<sms, kDecThreads, decode_smem_bytes<GH>(a.B), s>>>(a);
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
