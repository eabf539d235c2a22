// dar_decode.cu -- one decode step of DAR attention over the mixed-dimension
// cache (Eq. 3-4 for the query at position L_b - 1; cache scheme of Sec. 5).
//
// Work decomposition (split-K over the sequence):
//   item = (sequence b, KV head g, head slice hs, chunk c).  Chunks 0..nwc-1
//   cover the ring (full d = 64 keys/values, `cw` tokens each); the rest cover
//   the pages (d_down vectors, `cd` tokens each, page aligned).  Items are
//   taken by warps: the first one statically, the rest from an atomic counter.
//
// Inside an item a warp streams its tokens with 16-byte loads: LPT lanes own
// one token row (one 16-byte granule each), so every warp-wide load covers a
// contiguous 512-byte run.  The GH query heads of the slice share each load.
// Global tokens are scored against q~ = q Uk^T (W_up absorbed into the query,
// exact by linearity of Eq. 2) and their values are summed in d_down space.
// One online softmax (running max m, sum l, log2 domain) covers the item.
//
// Combine: each item writes (m, l, acc) per head; the warp that arrives last
// for (b, g, hs) merges all chunks, lifts the global part once with Uv and
// writes o = (acc_local + acc_global Uv) / l.  No warp ever waits on another.
#include <float.h>

#include "dar_common.cuh"
#include "dar_launch.h"

namespace dar {

constexpr int kDecWarps = 8;
constexpr int kDecThreads = kDecWarps * 32;

template <int GH>
struct WarpScratch {
    float q[GH][kHeadDim];   // scaled query of each head of the slice
    float qt[GH][kHeadDim];  // q~ (first dd entries); reused for the combine
};

// Online-softmax state of one lane for GH heads over a granule of E values.
template <int GH, int E>
struct SoftmaxState {
    float m[GH], l[GH], acc[GH][E];
    __device__ __forceinline__ void init()
    {
#pragma unroll
        for (int k = 0; k < GH; ++k) {
            m[k] = -INFINITY;
            l[k] = 0.f;
#pragma unroll
            for (int e = 0; e < E; ++e)
                acc[k][e] = 0.f;
        }
    }
};

// Stream tokens [t0, t1) of one segment.  ROW = elements per token row (64 for
// the ring, dd for the pages).  addr(t) returns the element offset of token
// t's row, or a negative value for a token that must be skipped (its page is
// not valid); tokens of one batch never straddle a page (batches divide 64 and
// segments start page aligned).
template <typename T, int ROW, int GH, typename AddrFn>
__device__ __forceinline__ void stream_segment(const T *__restrict__ Kbase,
                                               const T *__restrict__ Vbase, AddrFn addr, int t0,
                                               int t1, const float (&qsrc)[GH][kHeadDim],
                                               SoftmaxState<GH, Granule<T>::kElems> &st, int lane)
{
    constexpr int E = Granule<T>::kElems;
    constexpr int LPT = ROW / E;  // lanes per token row
    constexpr int TPI = 32 / LPT; // tokens per warp-wide load
    constexpr int U = (64 / TPI) < 4 ? (64 / TPI) : 4;
    constexpr int BT = U * TPI;   // tokens per batch
    static_assert(LPT >= 1 && LPT <= 32 && (32 % LPT) == 0, "row must be 16..512 bytes");
    const int grp = lane / LPT, sub = lane % LPT;

    float qr[GH][E];
#pragma unroll
    for (int k = 0; k < GH; ++k)
#pragma unroll
        for (int e = 0; e < E; ++e)
            qr[k][e] = qsrc[k][sub * E + e];

    uint4 kc[U], vc[U];
    bool okc[U];
    auto load = [&](int tb, uint4 (&kr)[U], uint4 (&vr)[U], bool (&ok)[U]) {
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int t = tb + u * TPI + grp;
            const long long row = t < t1 ? addr(t) : -1;
            ok[u] = row >= 0;
            if (ok[u]) {
                const size_t off = (size_t)row + (size_t)sub * E;
                kr[u] = ld_stream_v4(Kbase + off);
                vr[u] = ld_stream_v4(Vbase + off);
            } else {
                kr[u] = make_uint4(0, 0, 0, 0);
                vr[u] = make_uint4(0, 0, 0, 0);
            }
        }
    };
    load(t0, kc, vc, okc);
    for (int tb = t0; tb < t1; tb += BT) {
        uint4 kn[U], vn[U];
        bool okn[U];
        if (tb + BT < t1) {
            load(tb + BT, kn, vn, okn);
        } else {
#pragma unroll
            for (int u = 0; u < U; ++u)
                okn[u] = false;
        }
        float s[GH][U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            float kf[E];
            unpack(kc[u], kf, T());
#pragma unroll
            for (int k = 0; k < GH; ++k) {
                float acc = 0.f;
#pragma unroll
                for (int e = 0; e < E; ++e)
                    acc = fmaf(qr[k][e], kf[e], acc);
                s[k][u] = acc;
            }
        }
#pragma unroll
        for (int off = 1; off < LPT; off <<= 1)
#pragma unroll
            for (int k = 0; k < GH; ++k)
#pragma unroll
                for (int u = 0; u < U; ++u)
                    s[k][u] += __shfl_xor_sync(0xffffffffu, s[k][u], off);
        bool valid[U];
#pragma unroll
        for (int u = 0; u < U; ++u)
            valid[u] = okc[u];
#pragma unroll
        for (int k = 0; k < GH; ++k) {
            float mx = -INFINITY;
#pragma unroll
            for (int u = 0; u < U; ++u)
                if (valid[u])
                    mx = fmaxf(mx, s[k][u]);
            const float mnew = fmaxf(st.m[k], mx);
            const float alpha = (st.m[k] == -INFINITY) ? 0.f : exp2f(st.m[k] - mnew);
            float psum = 0.f;
#pragma unroll
            for (int u = 0; u < U; ++u) {
                s[k][u] = valid[u] ? exp2f(s[k][u] - mnew) : 0.f;  // score -> weight
                psum += s[k][u];
            }
            st.l[k] = st.l[k] * alpha + psum;
            st.m[k] = mnew;
#pragma unroll
            for (int e = 0; e < E; ++e)
                st.acc[k][e] *= alpha;
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            float vf[E];
            unpack(vc[u], vf, T());
#pragma unroll
            for (int k = 0; k < GH; ++k)
#pragma unroll
                for (int e = 0; e < E; ++e)
                    st.acc[k][e] = fmaf(s[k][u], vf[e], st.acc[k][e]);
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            kc[u] = kn[u];
            vc[u] = vn[u];
            okc[u] = okn[u];
        }
    }

    // merge the lane groups (lanes with the same granule index)
#pragma unroll
    for (int off = LPT; off < 32; off <<= 1) {
#pragma unroll
        for (int k = 0; k < GH; ++k) {
            const float mo = __shfl_xor_sync(0xffffffffu, st.m[k], off);
            const float lo = __shfl_xor_sync(0xffffffffu, st.l[k], off);
            const float mn = fmaxf(st.m[k], mo);
            const float a = (st.m[k] == -INFINITY) ? 0.f : exp2f(st.m[k] - mn);
            const float bo = (mo == -INFINITY) ? 0.f : exp2f(mo - mn);
            st.l[k] = st.l[k] * a + lo * bo;
#pragma unroll
            for (int e = 0; e < E; ++e) {
                const float ao = __shfl_xor_sync(0xffffffffu, st.acc[k][e], off);
                st.acc[k][e] = st.acc[k][e] * a + ao * bo;
            }
            st.m[k] = mn;
        }
    }
}

template <typename T, int DD, int GH>
__global__ void __launch_bounds__(kDecThreads, GH == 1 ? 2 : 1) decode_kernel(DecodeArgs a)
{
    constexpr int E = Granule<T>::kElems;
    extern __shared__ int s_dyn[];
    int *s_pre = s_dyn;            // [B + 1] exclusive prefix of chunk counts
    int *s_len = s_dyn + a.B + 1;  // [B] validated lengths (-1 = invalid)
    __shared__ WarpScratch<GH> scratch[kDecWarps];

    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int B = a.B, w = a.w;

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

    const int total_chunks = s_pre[B];
    const int per_chunk = a.Hkv * a.HS;
    const int items = total_chunks * per_chunk;
    const int nwarps_total = gridDim.x * kDecWarps;
    WarpScratch<GH> &sc = scratch[warp];
    const T *qg = static_cast<const T *>(a.q);

    int it = blockIdx.x + gridDim.x * warp;
    while (it < items) {
        // ---- decode the item index
        const int u = it / per_chunk, rem = it % per_chunk;
        const int g = rem / a.HS, hs = rem % a.HS;
        int lo = 0, hi = B;  // largest b with s_pre[b] <= u
        while (hi - lo > 1) {
            const int mid = (lo + hi) >> 1;
            if (s_pre[mid] <= u)
                lo = mid;
            else
                hi = mid;
        }
        const int b = lo, c = u - s_pre[b];
        const int L = s_len[b];
        const int nwin = min(L, w), ndist = L - nwin;
        const int nwc = (nwin + a.cw - 1) / a.cw;
        const int nchunks = nwc + (ndist + a.cd - 1) / a.cd;
        const int h0 = g * a.G + hs * GH;

        // ---- stage the scaled queries
#pragma unroll
        for (int k = 0; k < GH; ++k) {
            const T *qrow = qg + ((size_t)b * a.Hq + h0 + k) * kHeadDim;
            sc.q[k][lane] = to_f32(qrow[lane]) * a.qscale;
            sc.q[k][lane + 32] = to_f32(qrow[lane + 32]) * a.qscale;
        }
        __syncwarp();

        SoftmaxState<GH, E> st;
        st.init();
        int width;  // entries of acc this record carries
        if (c < nwc) {
            const int t0 = c * a.cw, t1 = min(nwin, t0 + a.cw);
            const size_t base = (size_t)(b * a.Hkv + g) * w * kHeadDim;
            const T *Kb = static_cast<const T *>(a.win_k) + base;
            const T *Vb = static_cast<const T *>(a.win_v) + base;
            stream_segment<T, kHeadDim, GH>(
                Kb, Vb, [](int t) { return (long long)t * kHeadDim; }, t0, t1, sc.q, st, lane);
            width = kHeadDim;
        } else {
            // q~[k][c] = sum_t q[k][t] Uk[g][c][t]
            const float *Uk = a.Uk + (size_t)g * DD * kHeadDim;
            for (int o = lane; o < GH * DD; o += 32) {
                const int k = o / DD, cc = o % DD;
                const float4 *ur = reinterpret_cast<const float4 *>(Uk + (size_t)cc * kHeadDim);
                float acc = 0.f;
#pragma unroll
                for (int t4 = 0; t4 < kHeadDim / 4; ++t4) {
                    const float4 u4 = __ldg(ur + t4);
                    acc = fmaf(sc.q[k][4 * t4 + 0], u4.x, acc);
                    acc = fmaf(sc.q[k][4 * t4 + 1], u4.y, acc);
                    acc = fmaf(sc.q[k][4 * t4 + 2], u4.z, acc);
                    acc = fmaf(sc.q[k][4 * t4 + 3], u4.w, acc);
                }
                sc.qt[k][cc] = acc;
            }
            __syncwarp();
            const int t0 = (c - nwc) * a.cd, t1 = min(ndist, t0 + a.cd);
            const int32_t *bt = a.block_table + (size_t)b * a.maxp;
            const int Hkv = a.Hkv, npages = a.num_pages;
            int32_t *status = a.status;
            // element offset of distant token t; a token whose page is not valid is
            // skipped (masked out) and flagged
            auto addr = [=](int t) -> long long {
                const int id = bt[t / kPage];
                if (id < 0 || id >= npages) {
                    report(status, DAR_ERR_CAPACITY);
                    return -1;
                }
                return (((long long)id * Hkv + g) * kPage + (t % kPage)) * DD;
            };
            stream_segment<T, DD, GH>(static_cast<const T *>(a.pool_kd),
                                      static_cast<const T *>(a.pool_vd), addr, t0, t1, sc.qt, st,
                                      lane);
            width = DD;
        }

        // ---- write this item's partial result
        const int LPTw = width / E;
#pragma unroll
        for (int k = 0; k < GH; ++k) {
            const size_t rec = ((size_t)b * a.Hq + h0 + k) * a.maxc + c;
            if (lane < LPTw) {
#pragma unroll
                for (int e = 0; e < E; ++e)
                    a.rec_acc[rec * kHeadDim + lane * E + e] = st.acc[k][e];
            }
            if (lane == 0) {
                a.rec_m[rec] = st.m[k];
                a.rec_l[rec] = st.l[k];
            }
        }
        __threadfence();
        __syncwarp();
        int arrived = 0;
        int32_t *cnt = a.counters + ((size_t)b * a.Hkv + g) * a.HS + hs;
        if (lane == 0)
            arrived = atomicAdd(cnt, 1);
        arrived = __shfl_sync(0xffffffffu, arrived, 0);

        if (arrived == nchunks - 1) {
            // ---- last arrival: merge every chunk of (b, g, hs)
            __threadfence();
            const float *Uv = a.Uv + (size_t)g * DD * kHeadDim;
            T *out = static_cast<T *>(a.out);
#pragma unroll 1
            for (int k = 0; k < GH; ++k) {
                const size_t rec0 = ((size_t)b * a.Hq + h0 + k) * a.maxc;
                float M = -INFINITY;
                for (int cc = lane; cc < nchunks; cc += 32)
                    M = fmaxf(M, __ldcg(a.rec_m + rec0 + cc));
#pragma unroll
                for (int off = 16; off; off >>= 1)
                    M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
                float lsum = 0.f;
                for (int cc = lane; cc < nchunks; cc += 32)
                    lsum += exp2f(__ldcg(a.rec_m + rec0 + cc) - M) * __ldcg(a.rec_l + rec0 + cc);
#pragma unroll
                for (int off = 16; off; off >>= 1)
                    lsum += __shfl_xor_sync(0xffffffffu, lsum, off);
                float o0 = 0.f, o1 = 0.f;  // local part, entries 2*lane, 2*lane+1
                for (int cc = 0; cc < nwc; ++cc) {
                    const float f = exp2f(__ldcg(a.rec_m + rec0 + cc) - M);
                    const float2 v = __ldcg(
                        reinterpret_cast<const float2 *>(a.rec_acc + (rec0 + cc) * kHeadDim) + lane);
                    o0 = fmaf(f, v.x, o0);
                    o1 = fmaf(f, v.y, o1);
                }
                float gd0 = 0.f, gd1 = 0.f;  // global part in d_down space
                for (int cc = nwc; cc < nchunks; ++cc) {
                    const float f = exp2f(__ldcg(a.rec_m + rec0 + cc) - M);
                    const float *ra = a.rec_acc + (rec0 + cc) * kHeadDim;
                    if (lane < DD)
                        gd0 = fmaf(f, __ldcg(ra + lane), gd0);
                    if (lane + 32 < DD)
                        gd1 = fmaf(f, __ldcg(ra + lane + 32), gd1);
                }
                if (lane < DD)
                    sc.qt[0][lane] = gd0;
                if (lane + 32 < DD)
                    sc.qt[0][lane + 32] = gd1;
                __syncwarp();
#pragma unroll 4
                for (int cc = 0; cc < DD; ++cc) {
                    const float gv = sc.qt[0][cc];
                    const float2 u2 =
                        __ldg(reinterpret_cast<const float2 *>(Uv + (size_t)cc * kHeadDim) + lane);
                    o0 = fmaf(gv, u2.x, o0);
                    o1 = fmaf(gv, u2.y, o1);
                }
                __syncwarp();
                const float inv = 1.f / lsum;
                T *orow = out + ((size_t)b * a.Hq + h0 + k) * kHeadDim;
                orow[2 * lane] = from_f32<T>(o0 * inv);
                orow[2 * lane + 1] = from_f32<T>(o1 * inv);
            }
            if (lane == 0)
                *cnt = 0;  // ready for the next call
        }

        // ---- next item
        int nxt = 0;
        if (lane == 0)
            nxt = atomicAdd(a.sched, 1) + nwarps_total;
        it = __shfl_sync(0xffffffffu, nxt, 0);
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
    const int item_bytes = 16384;  // K + V bytes streamed per item
    gm.cw = item_bytes / (2 * kHeadDim * esz);
    if (gm.cw < 16)
        gm.cw = 16;
    int pages = item_bytes / (2 * kPage * dd * esz);
    gm.cd = (pages < 1 ? 1 : pages) * kPage;
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
    const size_t dyn = (size_t)(2 * a.B + 1) * sizeof(int);
    if (dyn > 32768) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
        if (e != cudaSuccess)
            return e;
    }
    int dev = 0, sms = 0, per_sm = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kDecThreads, dyn);
    if (per_sm < 1)
        per_sm = 1;
    kern<<<sms * per_sm, kDecThreads, dyn, s>>>(a);
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
