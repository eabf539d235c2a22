// dar_decode.cu -- one decode step of DAR attention over the mixed-dimension
// cache (Eq. 3-4 for the query at position L_b - 1; cache scheme of Sec. 5).
//
// Two kernels on the caller's stream:
//
//  prep     q~ = q Uk^T for every query row (W_up absorbed into the query,
//           exact by linearity of Eq. 2) and zeroed group counters.  Neither
//           needs the cache, so when the kernel before it is this library's
//           cache append (dar_decode_step) prep is launched with programmatic
//           stream serialisation and overlaps it; it waits for that kernel
//           before exiting.  Otherwise it starts after all earlier work.
//           The stream kernel is always launched programmatically after prep.
//  stream   split-K over the sequence, balanced per warp (stream-K).  The
//           work of a group (sequence b, KV head g, head slice hs) is a run
//           of stages -- the ring's tokens (full d = 64 keys/values) in
//           stages of TPS_W tokens, then the pages' tokens (d_down vectors,
//           page aligned) in stages of TPS_D tokens -- and the groups are laid
//           end to end, ordered by sequence then group.  Every CTA builds the
//           per-sequence stage counts and their prefix sums in shared memory.
//           The S stages are split evenly over the NW warps of the grid (warp
//           k owns [Ss k / NW, Ss (k + 1) / NW), Ss = S); with a non-zero
//           kDecodePoolPercent the last share of the stages instead forms a
//           pool of small chunks that warps claim with an atomic counter once
//           their own range is done (off: its per-chunk costs outweighed the
//           balance it bought).  A range cuts groups into parts; within a
//           part, the ring stages and the page stages each leave one partial
//           result per head (running max m, sum l, unnormalised acc) in the
//           range's record slots.  When a part ends, a group that lies inside
//           the range is merged at once; a group spread over several ranges
//           is merged by the warp whose atomic completes its stage count.
//           The merge is one softmax over all parts (Eq. 4) with the global
//           part lifted once by Uv: o = (acc_local + acc_global Uv) / l.
//
// Streaming: every warp owns a ring of kStages shared-memory slots of
// kSlotBytes (keys in the first half, values in the second) plus a small
// header per slot.  Lane 0 fills a slot with TMA copies (2-D tensor copies of
// 128-byte lines into 128-byte-swizzled tiles for the tensor-core consumer --
// pages of d_down < 64 are viewed as lines holding 64 / d_down tokens, since
// boxes of short rows stream markedly slower -- and 1-D bulk copies otherwise;
// completion counted on the slot's mbarrier) and, with the first stage of a
// segment, copies the segment's query rows (q for the ring, q~ for the pages)
// into the slot's header.  The warp consumes slots in order and refills each
// one as soon as it has been read, across segment boundaries, so it keeps up
// to kStages * kSlotBytes of cache in flight while it computes.  Cache bytes
// are loaded with an evict-first L2 policy: they are read once per call.
//
// Compute (bf16, d_down >= 16): the two small contractions of a stage run on
// the tensor cores with warp-level mma.sync m16n8k16 (bf16 in, fp32 out): the
// GH query heads of the slice are rows of A, 8 tokens a column block of B,
// fed by ldmatrix from the swizzled tiles; the scores stay in registers,
// become P (bf16) and multiply V (ldmatrix.trans).  Global tokens are scored
// against q~ and their values are summed in d_down space.  When a KV head
// serves a single query head, page stages instead give each lane whole tokens
// on the CUDA cores (the tensor-core tile would be 15/16 idle).  Other cases
// (fp32 storage, d_down = 8) use the CUDA cores with LPT lanes per token row.
// One online softmax (log2 domain) covers a segment.
#include <type_traits>

#include "dar_common.cuh"
#include "dar_launch.h"
#include "dar_sm100.cuh"

namespace dar {

constexpr int kDecWarps = kDecodeWarpsPerCta;
constexpr int kDecThreads = kDecWarps * 32;
constexpr int kStages = 3;
constexpr int kSlotBytes = 8192;
constexpr int kHalf = kSlotBytes / 2;
constexpr int kHdrBytes = 1024;     // per slot: up to 4 query rows of 64 fp32
constexpr int kPrepThreads = 256;   // prep block size

static_assert(DAR_DECODE_MAX_BATCH % kDecThreads == 0, "stream threads hold whole groups of sequences");

// bf16 caches with d_down >= 16 use the tensor-core consumer (fed by 2-D TMA).
template <typename T, int DD>
__host__ __device__ constexpr bool decode_uses_mma()
{
    return sizeof(T) == 2 && DD >= 16;
}

// Tokens per stage: ring rows of 64 elements, page rows of DD elements.
template <typename T>
__host__ __device__ constexpr int tps_ring()
{
    return kHalf / (kHeadDim * (int)sizeof(T));
}
template <typename T, int DD>
__host__ __device__ constexpr int tps_page()
{
    return kHalf / (DD * (int)sizeof(T));
}

// --------------------------------------------------------------------- PTX

using sm100::bulk_g2s;
using sm100::ldsm_x4;
using sm100::ldsm_x4_t;
using sm100::mbar_expect_tx;
using sm100::mbar_init;
using sm100::mma_bf16_16816;
using sm100::smem_u32;

// Bounded wait (see sm100::mbar_wait); a warp that gives up reports to *status.
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, unsigned parity, int32_t *status)
{
    if (sm100::mbar_wait(bar, parity, nullptr))
        return true;
    report(status, DAR_ERR_DEVICE);
    return false;
}

// Stage metadata a slot carries from the issuing lane to the consumer:
//   x: group index (b * Hkv * HS + g * HS + hs); y: flags | page mask << 24;
//   z: valid tokens in the stage.
constexpr int kMetaRing = 1 << 16;      // a ring stage (else a page stage)
constexpr int kMetaSegStart = 1 << 17;  // first stage of a segment: query rows in the header
constexpr int kMetaSegEnd = 1 << 18;    // last stage of a segment: write its records
constexpr int kMetaPartEnd = 1 << 19;   // last stage of the warp's part of the group
constexpr int kMetaShared = 1 << 20;    // the group has parts in other warps
constexpr int kMetaSlot1 = 1 << 21;     // record slot 1 (else 0)

// Stages of one group of a sequence of validated length L (-1 or 0: none).
struct SeqStages {
    int nwin, ndist;  // ring tokens, page tokens
    int r, n;         // ring stages, all stages
};
template <int TPS_W, int TPS_D>
__device__ __forceinline__ SeqStages seq_stages(int L, int w)
{
    SeqStages q;
    q.nwin = L > 0 ? min(L, w) : 0;
    q.ndist = L > 0 ? L - q.nwin : 0;
    q.r = (q.nwin + TPS_W - 1) / TPS_W;
    q.n = q.r + (q.ndist + TPS_D - 1) / TPS_D;
    return q;
}

// Partial results: record (range, slot, type, head) at
// rec + (((range * 2 + slot) * 2 + type) * GH + head) * kRecFloats, holding
// acc[64] (type 0, ring) or acc[d_down] (type 1, pages), then m and l.
// Slot 0 belongs to a part whose group began before the range, slot 1 to any
// other part (a group that lies inside the range is merged at once and reuses
// slot 1 before the range's last part writes it).
__device__ __forceinline__ float *rec_ptr(float *rec, int range, int slot, int type, int k, int GH)
{
    return rec + (size_t)(((range * 2 + slot) * 2 + type) * GH + k) * kRecFloats;
}

// Dynamic shared memory of the stream kernel for a batch of B sequences:
// alignment slack, slots, headers, barriers, stage metadata, the tables.
constexpr size_t decode_smem_bytes(int B)
{
    return 1024 + (size_t)kDecWarps * kStages * (kSlotBytes + kHdrBytes + sizeof(uint64_t) + sizeof(int4)) +
           (size_t)(2 * B + 1) * sizeof(int);
}

// --------------------------------------------------------------------- prep

// q~ = q Uk^T for every (b, h) row, one row per warp (fp32, four partial sums
// over t mod 4), and zeroed group counters.  In the direct variant of Sec. 5
// (a.qd set) q~ is the row's own d_down query times scale_down / scale, so the
// stream kernel's global scores scale * q~ . k^D are scale_down * q^D . k^D.  Neither depends on the cache, so
// when launched programmatically after the cache append (which writes neither
// q nor Uk) this kernel runs while the append finishes; it waits for the
// kernel before it before exiting, so the stream kernel, which waits for this
// one, sees the finished cache.
template <typename T, int DD>
__global__ void __launch_bounds__(kPrepThreads) decode_prep_kernel(DecodeArgs a)
{
    constexpr int QR = DD > 32 ? 2 : 1;  // q~ entries per lane
    constexpr int kWarps = kPrepThreads / 32;
    sm100::grid_dep_launch();  // the stream kernel may start its set-up now
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int rows = a.B * a.Hq;
    for (int row = blockIdx.x * kWarps + warp; row < rows; row += gridDim.x * kWarps) {
        if (a.qd) {  // direct variant: the row's own d_down query, rescaled to the local scale
            for (int c = lane; c < DD; c += 32)
                a.qt[(size_t)row * DD + c] = to_f32(static_cast<const T *>(a.qd)[(size_t)row * DD + c]) * a.qd_ratio;
            continue;
        }
        const T *qrow = static_cast<const T *>(a.q) + (size_t)row * kHeadDim;
        const float q0 = to_f32(qrow[lane]), q1 = to_f32(qrow[lane + 32]);
        const int g = (row % a.Hq) / a.G;
#pragma unroll
        for (int rr = 0; rr < QR; ++rr) {
            const int c = lane + 32 * rr;
            const float4 *u4 = reinterpret_cast<const float4 *>(a.Uk + ((size_t)g * DD + (c < DD ? c : 0)) * kHeadDim);
            float4 uk[kHeadDim / 4];
#pragma unroll
            for (int t4 = 0; t4 < kHeadDim / 4; ++t4)
                uk[t4] = c < DD ? __ldg(u4 + t4) : make_float4(0.f, 0.f, 0.f, 0.f);
            float p[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
            for (int t4 = 0; t4 < kHeadDim / 4; ++t4) {
                const float uu[4] = {uk[t4].x, uk[t4].y, uk[t4].z, uk[t4].w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int t = 4 * t4 + e;
                    const float qv = __shfl_sync(0xffffffffu, t < 32 ? q0 : q1, t & 31);
                    p[e] = fmaf(qv, uu[e], p[e]);
                }
            }
            if (c < DD)
                a.qt[(size_t)row * DD + c] = (p[0] + p[1]) + (p[2] + p[3]);
        }
    }
    const int ngroups = a.B * a.Hkv * a.HS;  // group counters, then the pool's claim counter
    for (int i = blockIdx.x * kPrepThreads + threadIdx.x; i <= ngroups; i += gridDim.x * kPrepThreads)
        a.counters[i] = 0;
    sm100::grid_dep_wait();
}

// --------------------------------------------------------------------- stream

// Byte offset of 16-byte chunk `ch` of token t in a stage tile of ROW-element
// bf16 rows as the 2-D TMA wrote it: the tile is viewed as 128-byte lines
// (64 / ROW tokens per line) with the 128-byte swizzle, i.e. the chunk index
// within a line XOR (line % 8).  Eight consecutive tokens of one chunk column
// then fall in eight different bank groups (conflict-free ldmatrix).
template <int ROW>
__device__ __forceinline__ uint32_t tile_off(int t, int ch)
{
    constexpr int TR = kHeadDim / ROW;  // tokens per 128-byte line
    const int line = t / TR;
    const int c = (t % TR) * (ROW / 8) + ch;
    return (uint32_t)(line * 128 + ((c ^ (line & 7)) << 4));
}

// Zero the value rows of a stage that the softmax masks out (tokens past the
// stage's end, pages not copied): their P entries are zero, but stale or
// never-written bytes there could be Inf/NaN and 0 * NaN would reach acc.
// The fence orders these generic writes before the TMA that refills the slot.
template <int ROW, int TPS>
__device__ __forceinline__ void zero_masked_rows(unsigned char *v, int ntok, unsigned pmask, int lane)
{
    constexpr int CH = ROW / 8;  // 16-byte chunks per token
#pragma unroll 4
    for (int i = lane; i < TPS * CH; i += 32) {
        const int t = i / CH;
        if (!(t < ntok && ((pmask >> (t / kPage)) & 1u)))
            *reinterpret_cast<uint4 *>(v + tile_off<ROW>(t, i % CH)) = make_uint4(0u, 0u, 0u, 0u);
    }
    sm100::fence_proxy_async_smem();
    __syncwarp();
}

// Tensor-core consumer for one stage of ROW-wide rows (64 = ring keys/values,
// d_down = pages), TPS tokens, laid out as tile_off<ROW> describes.
// q_a: A fragments (KS k-steps) of the GH query rows; o: output fragments
// (ROW/8 n-tiles); m, lpart: the row's running max and this lane's part of the
// running sum (quad-uniform m).  kMasked: some tokens of the stage are invalid.
template <int ROW, int TPS, int GH, bool kMasked>
__device__ __forceinline__ void mma_stage(uint32_t sK, uint32_t sV, int ntok, unsigned pmask,
                                          const uint32_t (&q_a)[(ROW >= 16 ? ROW / 16 : 1)][4],
                                          float (&o)[ROW / 8][4], float &m, float &lpart, float c2, int lane)
{
    constexpr int KS = ROW / 16;  // k-steps of the score product
    constexpr int ND = ROW / 8;   // n-tiles of the output
    constexpr int TB = TPS < 64 ? TPS : 64;  // tokens per block of the online softmax
    constexpr int NT = TB / 8;
    const int c = lane & 3;
    const int mi = lane >> 3, ri = lane & 7;
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
                ldsm_x4(sK + tile_off<ROW>(tok, ch), r);
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
                if constexpr (kMasked) {
                    const int tl = t0 + 8 * n + 2 * c + e;
                    const bool ok = tl < ntok && ((pmask >> (tl / kPage)) & 1u);
                    sc[n][e] = ok ? sc[n][e] : -INFINITY;
                }
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
                ldsm_x4_t(sV + tile_off<ROW>(tok, ch), r);
                mma_bf16_16816(o[2 * dp], pa, r[0], r[1]);
                mma_bf16_16816(o[2 * dp + 1], pa, r[2], r[3]);
            }
        }
    }
}

// CUDA-core consumer for one page stage when a KV head serves one query head
// (the tensor-core tile would carry 15 idle rows): lane l owns tokens
// l, l + 32, ...; qd is q~ scaled to the log2 domain; m is the warp's running
// max, l and o this lane's parts of the running sum and value accumulator.
// Masked tokens never touch o, so their rows may hold anything.
template <int DD, int TPS>
__device__ __forceinline__ void lane_stage(uint32_t sK, uint32_t sV, int ntok, unsigned pmask, const float (&qd)[DD],
                                           float (&o)[DD], float &m, float &l, int lane)
{
    constexpr int TPL = TPS / 32;  // tokens per lane
    constexpr int CH = DD / 8;     // 16-byte chunks per row
    static_assert(TPS % 32 == 0, "whole tokens per lane");
    float sc[TPL];
    bool ok[TPL];
    float mx = -INFINITY;
#pragma unroll
    for (int i = 0; i < TPL; ++i) {
        const int t = lane + 32 * i;
        ok[i] = t < ntok && ((pmask >> (t / kPage)) & 1u);
        float acc = 0.f;
#pragma unroll
        for (int ch = 0; ch < CH; ++ch) {
            uint4 k4;
            asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];"
                         : "=r"(k4.x), "=r"(k4.y), "=r"(k4.z), "=r"(k4.w)
                         : "r"(sK + tile_off<DD>(t, ch)));
            float kf[8];
            unpack(k4, kf, bf16());
#pragma unroll
            for (int e = 0; e < 8; ++e)
                acc = fmaf(qd[8 * ch + e], kf[e], acc);
        }
        sc[i] = ok[i] ? acc : -INFINITY;
        mx = fmaxf(mx, sc[i]);
    }
#pragma unroll
    for (int off = 16; off; off >>= 1)
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
    if (mx > m) {  // warp-uniform: rescale only when the running max grows
        const float alpha = m == -INFINITY ? 0.f : sm100::ex2_approx(m - mx);
        l *= alpha;
#pragma unroll
        for (int c = 0; c < DD; ++c)
            o[c] *= alpha;
        m = mx;
    }
#pragma unroll
    for (int i = 0; i < TPL; ++i) {
        if (!ok[i])
            continue;
        const int t = lane + 32 * i;
        const float p = sm100::ex2_approx(sc[i] - m);
        l += p;
#pragma unroll
        for (int ch = 0; ch < CH; ++ch) {
            uint4 v4;
            asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];"
                         : "=r"(v4.x), "=r"(v4.y), "=r"(v4.z), "=r"(v4.w)
                         : "r"(sV + tile_off<DD>(t, ch)));
            float vf[8];
            unpack(v4, vf, bf16());
#pragma unroll
            for (int e = 0; e < 8; ++e)
                o[8 * ch + e] = fmaf(p, vf[e], o[8 * ch + e]);
        }
    }
}

// One halving step of a warp reduce-scatter: lanes with `mask` set keep the
// upper half of their values, the others the lower half, each adding its
// partner's copy of the half it keeps.
template <int N>
__device__ __forceinline__ void rs_step(const float (&in)[N], float (&out)[N / 2], int mask, int lane)
{
    const bool upper = (lane & mask) != 0;
#pragma unroll
    for (int j = 0; j < N / 2; ++j) {
        const float send = upper ? in[j] : in[j + N / 2];
        const float keep = upper ? in[j + N / 2] : in[j];
        out[j] = keep + __shfl_xor_sync(0xffffffffu, send, mask);
    }
}

// Warp sum of o[0..DD) (DD = 16 or 32): returns the total of entry
// lane / (32 / DD), held by 32 / DD lanes each.
template <int DD>
__device__ __forceinline__ float reduce_scatter(const float (&o)[DD], int lane)
{
    float a16[16], a8[8], a4[4], a2[2], a1[1];
    if constexpr (DD == 32) {
        rs_step<32>(o, a16, 16, lane);
        rs_step<16>(a16, a8, 8, lane);
        rs_step<8>(a8, a4, 4, lane);
        rs_step<4>(a4, a2, 2, lane);
        rs_step<2>(a2, a1, 1, lane);
        return a1[0];
    } else {
        static_assert(DD == 16, "reduce_scatter handles 16 or 32 values");
        rs_step<16>(o, a8, 16, lane);
        rs_step<8>(a8, a4, 8, lane);
        rs_step<4>(a4, a2, 4, lane);
        rs_step<2>(a2, a1, 2, lane);
        return a1[0] + __shfl_xor_sync(0xffffffffu, a1[0], 1);
    }
}

// Per-sequence tables of one decode call, built by every CTA of the stream
// kernel into its shared memory: s_len[b] = validated length (-1 if beyond
// the cache's capacity) and s_pre[b] = stages per group of the sequences
// before b (s_pre[B] = all).  validated_length reads a length from L2 (an L1
// copy could predate the append); scan_tables is warp 0's prefix sum over
// contiguous runs of sequences per lane.
__device__ __forceinline__ int validated_length(const DecodeArgs &a, int b)
{
    const int L = __ldcg(a.seq_lens + b);
    return (L < 0 || (long long)L - a.w > (long long)a.maxp * kPage) ? -1 : L;
}
template <int TPS_W, int TPS_D>
__device__ __forceinline__ void scan_tables(const DecodeArgs &a, int *s_pre, const int *s_len)
{
    const int lane = threadIdx.x & 31;
    const int B = a.B, w = a.w;
    const int per = (B + 31) / 32;
    const int b0 = min(B, lane * per), b1 = min(B, b0 + per);
    int mine = 0;
    for (int b = b0; b < b1; ++b)
        mine += seq_stages<TPS_W, TPS_D>(s_len[b], w).n;
    int incl = mine;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, off);
        if (lane >= off)
            incl += y;
    }
    int run = incl - mine;
    for (int b = b0; b < b1; ++b) {
        s_pre[b] = run;
        run += seq_stages<TPS_W, TPS_D>(s_len[b], w).n;
    }
    if (lane == 31)
        s_pre[B] = incl;
}

// The split of the S stages into ranges.  The first Ss stages are divided
// evenly over the NW warps of the grid (range k < NW = [lo(k), lo(k + 1)),
// lo(k) = floor(Ss k / NW)); the rest form a pool of NC chunks of C stages
// (range NW + u = chunk u), which warps that have finished their own range
// claim one at a time, so that SMs served faster by the memory system take
// more of them.  Range ids index the record slots.
struct Split {
    int S, Ss, NW, C, NC;
    int q0, r0;         // Ss = q0 NW + r0, so that floor(Ss k / NW) = q0 k + floor(r0 k / NW) in 32 bits
    float inv_nw, rate;  // 1 / NW and NW / Ss, for quotient estimates
    // floor(x / NW) for 0 <= x < 2^24: a float estimate off by at most one, corrected
    __device__ __forceinline__ int div_nw(int x) const
    {
        int q = (int)((float)x * inv_nw);
        q += (q + 1) * NW <= x;
        q -= q * NW > x;
        return q;
    }
    __device__ __forceinline__ int lo(int k) const
    {
        return k <= NW ? q0 * k + div_nw(r0 * k) : min(S, Ss + (k - NW) * C);
    }
    __device__ __forceinline__ int owner(int t) const  // the range holding stage t
    {
        if (t >= Ss)
            return NW + (t - Ss) / C;
        // the last k with lo(k) <= t: a float estimate, then exact steps
        int k = min(NW - 1, (int)((float)t * rate));
        while (k > 0 && lo(k) > t)
            --k;
        while (k + 1 < NW && lo(k + 1) <= t)
            ++k;
        return k;
    }
};
constexpr int kPoolPercent = kDecodePoolPercent;        // share of the stages in the pool
constexpr int kMaxPoolChunks = kMaxDecodeCtas * kDecWarps * 2;  // pool chunks the records hold
static_assert(kMaxPoolChunks == kDecodePoolChunks, "record slots of the pool");

__device__ __forceinline__ Split make_split(int S, int NW)
{
    Split sp;
    sp.S = S;
    sp.NW = NW;
    const int P = (int)((long long)S * kPoolPercent / 100);
    sp.C = max(1, (P + kMaxPoolChunks - 1) / kMaxPoolChunks);
    sp.NC = (P + sp.C - 1) / sp.C;
    sp.Ss = S - P;
    sp.q0 = sp.Ss / NW;
    sp.r0 = sp.Ss - sp.q0 * NW;
    sp.inv_nw = 1.f / (float)NW;
    sp.rate = sp.Ss > 0 ? (float)NW / (float)sp.Ss : 0.f;
    return sp;
}

// Merge of group `gid` from the records of all its parts, by one warp: one
// softmax over all parts (Eq. 4), o = (sum_p f_p acc_p[ring] + (sum_p f_p
// acc_p[pages]) Uv) / sum_p f_p l_p, f_p = 2^(m_p - max m).  With `rows` (the
// warp's idle slots, at the end of its streaming) lane i stages record i of a
// round of 32 in shared memory, all loads in flight at once; without it (a
// group that lies inside one range: two records at most) they are read in
// place.  Lane j holds entries 2j, 2j + 1 of the output row.
template <typename T, int DD, int GH, int TPS_W, int TPS_D>
__device__ __noinline__ void combine_group(const DecodeArgs &a, const int *s_pre, const int *s_len, int gid,
                                           Split sp, int lane, float *rows)
{
    const int per_chunk = a.Hkv * a.HS;
    const int b = gid / per_chunk, gh = gid - b * per_chunk;
    const int g = gh / a.HS, h0 = g * a.G + (gh - g * a.HS) * GH;
    const SeqStages sq = seq_stages<TPS_W, TPS_D>(s_len[b], a.w);
    const int G0 = s_pre[b] * per_chunk + gh * sq.n, G1 = G0 + sq.n, GR = G0 + sq.r;
    const int wa = sp.owner(G0);
    const int ncand = 2 * (sp.owner(G1 - 1) - wa + 1);
    // Uv rows in flight with the records (small d_down only: registers)
    constexpr int UVP = DD <= 32 ? DD : 1;
    const float *Uv = a.Uv + (size_t)g * DD * kHeadDim;
    float2 uv[UVP];
#pragma unroll
    for (int cc = 0; cc < UVP; ++cc)
        uv[cc] = __ldg(reinterpret_cast<const float2 *>(Uv + (size_t)cc * kHeadDim) + lane);
    // records in shared memory are final once the barrier completes; in place,
    // they are read from L2 (another SM's L1 copy could be stale)
    auto ld2 = [&](const float *p) {
        return rows ? *reinterpret_cast<const float2 *>(p) : __ldcg(reinterpret_cast<const float2 *>(p));
    };
    for (int k = 0; k < GH; ++k) {
        float M = -INFINITY, lsum = 0.f, o0 = 0.f, o1 = 0.f, gd0 = 0.f, gd1 = 0.f;
        // rounds of 32 candidates: candidate c0 + lane is (range wa + (c0 + lane) / 2,
        // type lane % 2); one online softmax runs over the rounds
        for (int c0 = 0; c0 < ncand; c0 += 32) {
            int r = -1;
            if (c0 + lane < ncand) {
                const int wk = wa + ((c0 + lane) >> 1);
                const int rlo = sp.lo(wk);
                const int lo = max(rlo, G0), hi = min(sp.lo(wk + 1), G1);
                if ((lane & 1) == 0 ? lo < min(hi, GR) : max(lo, GR) < hi)
                    r = ((wk * 2 + (G0 < rlo ? 0 : 1)) * 2 + (lane & 1)) * GH + k;
            }
            const unsigned live = __ballot_sync(0xffffffffu, r >= 0);
            // this lane's record: staged in shared memory (every lane's loads in
            // flight at once), or read where it is
            const float *mine = a.rec + (size_t)(r >= 0 ? r : 0) * kRecFloats;
            if (rows) {
                if (r >= 0) {  // 16-byte asynchronous copies through L2, no registers
                    const uint32_t dst = smem_u32(rows + lane * kRecFloats);
#pragma unroll
                    for (int i = 0; i < kRecFloats / 4; ++i)
                        asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst + 16 * i), "l"(mine + 4 * i)
                                     : "memory");
                }
                asm volatile("cp.async.wait_all;" ::: "memory");
                __syncwarp();
                mine = rows + lane * kRecFloats;
            }
            float mr = -INFINITY, lr = 0.f;
            if (r >= 0) {
                const float2 ml = ld2(mine + kHeadDim);
                mr = ml.x;
                lr = ml.y;
            }
            float mx = mr;
#pragma unroll
            for (int off = 16; off; off >>= 1)
                mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
            const float Mn = fmaxf(M, mx);
            const float sc = M == -INFINITY ? 0.f : exp2f(M - Mn);
            lsum *= sc;
            o0 *= sc;
            o1 *= sc;
            gd0 *= sc;
            gd1 *= sc;
            M = Mn;
            const float f = r >= 0 ? exp2f(mr - M) : 0.f;
            lsum = fmaf(f, lr, lsum);
            if (rows) {  // every candidate row up to the last live one; absent rows hold garbage
                const int jn = 32 - __clz(live);
#pragma unroll 8
                for (int j = 0; j < jn; ++j) {
                    const float fj = __shfl_sync(0xffffffffu, f, j);
                    const float2 x = *reinterpret_cast<const float2 *>(rows + j * kRecFloats + 2 * lane);
                    if ((live >> j) & 1u) {
                        if ((j & 1) == 0) {  // ring: acc[64]
                            o0 = fmaf(fj, x.x, o0);
                            o1 = fmaf(fj, x.y, o1);
                        } else if (2 * lane < DD) {  // pages: acc[DD]
                            gd0 = fmaf(fj, x.x, gd0);
                            gd1 = fmaf(fj, x.y, gd1);
                        }
                    }
                }
            } else {
                for (unsigned lv = live; lv; lv &= lv - 1) {
                    const int j = __ffs(lv) - 1;
                    const float fj = __shfl_sync(0xffffffffu, f, j);
                    const float *row = a.rec + (size_t)__shfl_sync(0xffffffffu, r, j) * kRecFloats;
                    if ((j & 1) == 0) {  // ring: acc[64]
                        const float2 x = ld2(row + 2 * lane);
                        o0 = fmaf(fj, x.x, o0);
                        o1 = fmaf(fj, x.y, o1);
                    } else if (2 * lane < DD) {  // pages: acc[DD]
                        const float2 x = ld2(row + 2 * lane);
                        gd0 = fmaf(fj, x.x, gd0);
                        gd1 = fmaf(fj, x.y, gd1);
                    }
                }
            }
            __syncwarp();  // the rows are read before the next round refills them
        }
#pragma unroll
        for (int off = 16; off; off >>= 1)
            lsum += __shfl_xor_sync(0xffffffffu, lsum, off);
        // lift the global part once: o += gd Uv[g]   (gd[c] sits in lane c / 2)
#pragma unroll
        for (int cc = 0; cc < DD; ++cc) {
            const float gv = __shfl_sync(0xffffffffu, (cc & 1) ? gd1 : gd0, cc >> 1);
            const float2 u2 = UVP == DD ? uv[cc < UVP ? cc : 0]
                                        : __ldg(reinterpret_cast<const float2 *>(Uv + (size_t)cc * kHeadDim) + lane);
            o0 = fmaf(gv, u2.x, o0);
            o1 = fmaf(gv, u2.y, o1);
        }
        const float inv = 1.f / lsum;
        T *orow = static_cast<T *>(a.out) + ((size_t)b * a.Hq + h0 + k) * kHeadDim;
        orow[2 * lane] = from_f32<T>(o0 * inv);
        orow[2 * lane + 1] = from_f32<T>(o1 * inv);
    }
}

template <typename T, int DD, int GH>
__global__ void __launch_bounds__(kDecThreads, 1)
    decode_kernel(const __grid_constant__ CUtensorMap tm_wk, const __grid_constant__ CUtensorMap tm_wv,
                  const __grid_constant__ CUtensorMap tm_pk, const __grid_constant__ CUtensorMap tm_pv,
                  const __grid_constant__ DecodeArgs a)
{
    constexpr int E = Granule<T>::kElems;
    constexpr int ES = sizeof(T);
    constexpr bool kMma = decode_uses_mma<T, DD>();
    constexpr int TPS_W = tps_ring<T>();
    constexpr int TPS_D = tps_page<T, DD>();
    constexpr int PPS = TPS_D >= kPage ? TPS_D / kPage : 1;  // pages touched per stage
    constexpr unsigned kFullPages = (1u << PPS) - 1u;
    static_assert(TPS_D % kPage == 0 || kPage % TPS_D == 0, "stages must tile pages");
    static_assert(PPS <= 8, "stage page mask holds 8 pages");
    static_assert(GH * kHeadDim * ES <= kHdrBytes && GH * DD * 4 <= kHdrBytes, "header holds the query rows");
    // one query head per KV head: page stages on the CUDA cores, one token per lane
    constexpr bool kLanePages = kMma && GH == 1 && DD == 16;

    extern __shared__ __align__(128) unsigned char smem_raw[];
    // swizzled TMA tiles need 1024-byte alignment (static shared data may precede this)
    unsigned char *slots = reinterpret_cast<unsigned char *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));  // [warps][stages][slot]
    unsigned char *hdrs = slots + (size_t)kDecWarps * kStages * kSlotBytes;  // [warps][stages][header]
    uint64_t *bars = reinterpret_cast<uint64_t *>(hdrs + (size_t)kDecWarps * kStages * kHdrBytes);
    int4 *meta = reinterpret_cast<int4 *>(bars + kDecWarps * kStages);
    int *s_pre = reinterpret_cast<int *>(meta + kDecWarps * kStages);  // [B + 1]
    int *s_len = s_pre + a.B + 1;                                      // [B]

    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    unsigned char *my_slots = slots + (size_t)warp * kStages * kSlotBytes;
    unsigned char *my_hdrs = hdrs + (size_t)warp * kStages * kHdrBytes;
    uint64_t *my_bars = bars + warp * kStages;
    int4 *my_meta = meta + warp * kStages;
    if (lane < kStages)
        mbar_init(&my_bars[lane], 1);
    sm100::mbar_init_fence();
    __syncthreads();
    if constexpr (kMma) {
        if (threadIdx.x == 0) {
            sm100::prefetch_tensormap(&tm_wk);
            sm100::prefetch_tensormap(&tm_wv);
            sm100::prefetch_tensormap(&tm_pk);
            sm100::prefetch_tensormap(&tm_pv);
        }
    }
    // The block table is not written by the cache append: warm L2 with this
    // CTA's share of it while the kernels before finish.
    {
        const size_t lines = ((size_t)a.B * a.maxp * sizeof(int32_t) + 127) / 128;
        const size_t l0 = lines * blockIdx.x / gridDim.x, l1 = lines * (blockIdx.x + 1) / gridDim.x;
        for (size_t i = l0 + threadIdx.x; i < l1; i += blockDim.x)
            asm volatile("prefetch.global.L2 [%0];" ::"l"(reinterpret_cast<const char *>(a.block_table) + i * 128));
    }
    // Tables from the lengths as they are now: the kernel before this one
    // (normally the cache append) may still be changing them, so they are a
    // guess, checked after the wait below.
    for (int b = threadIdx.x; b < a.B; b += blockDim.x)
        s_len[b] = validated_length(a, b);
    __syncthreads();
    if (warp == 0)
        scan_tables<TPS_W, TPS_D>(a, s_pre, s_len);
    __syncthreads();

    const int w = a.w;
    const T *qg = static_cast<const T *>(a.q);
    const T *wk = static_cast<const T *>(a.win_k);
    const T *wv = static_cast<const T *>(a.win_v);
    const T *pk = static_cast<const T *>(a.pool_kd);
    const T *pv = static_cast<const T *>(a.pool_vd);
    // cache pages are read once per call: first out of L2
    const uint64_t pol = sm100::l2_evict_first_policy();
    bool alive = true;

    // ---- the range being issued (first this warp's own, then pool chunks)
    // and the walk over it: sequence wb, group wgh of the sequence, stage wj
    // of the group (the ring's sq.r stages, then the pages')
    const int per_chunk = a.Hkv * a.HS;
    Split sp;
    int32_t *pool_next = a.counters + a.B * per_chunk;  // the pool's claim counter
    int rid = 0, lo = 0, hi = 0;
    int iss_s = 0;  // next stage to issue
    int wb = 0, wgh = 0, wj = 0;
    SeqStages sq = {0, 0, 0, 1};
    auto begin_range = [&]() {  // the walk's position at stage lo
        int lb = 0, hb = a.B;   // the last sequence whose first stage is <= lo
        while (hb - lb > 1) {
            const int mid = (lb + hb) >> 1;
            if (s_pre[mid] * per_chunk <= lo)
                lb = mid;
            else
                hb = mid;
        }
        wb = lb;
        sq = seq_stages<TPS_W, TPS_D>(s_len[wb], w);
        const int r0 = lo - s_pre[wb] * per_chunk;
        wgh = r0 / sq.n;
        wj = r0 - wgh * sq.n;
    };
    // block-table window: lane j holds the ids of pages pw0 + j and pw0 + 32 + j of sequence pwb
    int pwb = -1, pw0 = 0;
    int2 pid = make_int2(-1, -1);
    auto load_window = [&](int b, int p0) {
        pwb = b;
        pw0 = p0;
        const int32_t *bt = a.block_table + (size_t)b * a.maxp;
        pid.x = p0 + lane < a.maxp ? __ldg(bt + p0 + lane) : -1;
        pid.y = p0 + 32 + lane < a.maxp ? __ldg(bt + p0 + 32 + lane) : -1;
    };
    auto page_id = [&](int p) {  // page p of sequence pwb, inside the window
        const int j = p - pw0;
        const int x = __shfl_sync(0xffffffffu, pid.x, j & 31);
        const int y = __shfl_sync(0xffffffffu, pid.y, j & 31);
        return j < 32 ? x : y;
    };
    auto window_for_range = [&]() {  // a range that opens in a page run: fetch its ids now
        if (wj >= sq.r)
            load_window(wb, (wj - sq.r) * TPS_D / kPage);
    };
    // pool claims: lane 0 asks for the next chunk while issuing the last stages
    // of a range (two stages ahead), and the warp moves on to the claimed
    // chunk as soon as that range's last stage is issued
    int claim = 0;
    bool asked = false, pool_done = true;
    auto ask = [&]() {
        if (lane == 0)
            claim = atomicAdd(pool_next, 1);
        asked = true;
    };
    int ask_at = 0;
    auto next_range = [&]() {
        if (pool_done)
            return;
        if (!asked)
            ask();
        const int c = __shfl_sync(0xffffffffu, claim, 0);
        asked = false;
        if (c >= sp.NC) {
            pool_done = true;
            return;
        }
        rid = sp.NW + c;
        lo = sp.lo(rid);
        hi = sp.lo(rid + 1);
        iss_s = lo;
        ask_at = max(lo, hi - 2);
        begin_range();
        window_for_range();
    };
    // This warp's own range, the walk's start and its first block-table
    // window: they depend on the lengths only through the per-sequence stage
    // counts, so they are set up from the guessed tables before the wait and
    // kept if the counts hold.
#pragma unroll 1
    for (int pass = 0;; ++pass) {
        sp = make_split(s_pre[a.B] * per_chunk, gridDim.x * kDecWarps);
        rid = blockIdx.x * kDecWarps + warp;
        lo = sp.lo(rid);
        hi = sp.lo(rid + 1);
        iss_s = lo;
        ask_at = max(lo, hi - 2);
        pool_done = sp.NC == 0;
        if (lo < hi) {
            begin_range();
            window_for_range();
        }
        if (pass > 0)
            break;
        // everything below reads the cache and q~ (the prep kernel waited for
        // the kernel before it, so both are final)
        sm100::grid_dep_wait();
        // the final lengths: do their stage counts match the guess?
        int changed = 0;
        for (int b = threadIdx.x; b < a.B; b += blockDim.x) {
            const int L = validated_length(a, b);
            if (L < 0 && blockIdx.x == 0)
                report(a.status, DAR_ERR_CAPACITY);
            const SeqStages was = seq_stages<TPS_W, TPS_D>(s_len[b], w), now = seq_stages<TPS_W, TPS_D>(L, w);
            changed |= was.r != now.r || was.n != now.n;
            s_len[b] = L;
        }
        if (!__syncthreads_or(changed)) {
            if (lo < hi)
                sq = seq_stages<TPS_W, TPS_D>(s_len[wb], w);  // the walk's token bounds
            break;
        }
        if (warp == 0)  // counts changed: rebuild the prefix sums and set up again
            scan_tables<TPS_W, TPS_D>(a, s_pre, s_len);
        __syncthreads();
    }
    if (lo >= hi)
        next_range();  // no own stages (tiny workloads): straight to the pool
    if (blockIdx.x == 0) {  // sequences with nothing to attend to get a zero output
        T *out = static_cast<T *>(a.out);
        for (int b = warp; b < a.B; b += kDecWarps) {
            if (s_len[b] > 0)
                continue;
            for (int i = lane; i < a.Hq * kHeadDim; i += 32)
                out[(size_t)b * a.Hq * kHeadDim + i] = from_f32<T>(0.f);
        }
    }

    int issued = 0, consumed = 0;    // stages issued / consumed by this warp
    int iss_slot = 0, con_slot = 0;  // ring positions
    unsigned con_phase = 0;          // parity of the consumer's current pass over the ring

    auto issue_one = [&]() {  // copy stage iss_s into its slot
        const int slot = iss_slot;
        iss_slot = iss_slot + 1 == kStages ? 0 : iss_slot + 1;
        unsigned char *dst = my_slots + (size_t)slot * kSlotBytes;
        uint64_t *bar = &my_bars[slot];
        const bool ring = wj < sq.r;
        const int G0 = iss_s - wj, G1 = G0 + sq.n;
        const bool seg_start = iss_s == lo || wj == 0 || wj == sq.r;
        const bool seg_end = iss_s == hi - 1 || wj == sq.n - 1 || wj == sq.r - 1;
        const bool part_end = iss_s == hi - 1 || wj == sq.n - 1;
        int flags = (ring ? kMetaRing : 0) | (seg_start ? kMetaSegStart : 0) | (seg_end ? kMetaSegEnd : 0) |
                    (part_end ? kMetaPartEnd : 0) | (G0 < lo || G1 > hi ? kMetaShared : 0) |
                    (G0 < lo ? 0 : kMetaSlot1);
        const int g = wgh / a.HS;
        const int h0 = g * a.G + (wgh - g * a.HS) * GH;
        const int gid = wb * per_chunk + wgh;
        // a segment's query rows travel with its first stage
        unsigned hdr_bytes = 0;
        const void *hsrc = nullptr;
        if (seg_start) {
            if (ring) {
                hdr_bytes = GH * kHeadDim * ES;
                hsrc = qg + ((size_t)wb * a.Hq + h0) * kHeadDim;
            } else {
                hdr_bytes = GH * DD * 4;
                hsrc = a.qt + ((size_t)wb * a.Hq + h0) * DD;
            }
        }
        if (ring) {
            const int tb = wj * TPS_W, te = min(sq.nwin, tb + TPS_W);
            if (lane == 0) {
                my_meta[slot] = make_int4(gid, flags | (0xff << 24), te - tb, rid);
                const int y = (wb * a.Hkv + g) * w + tb;
                if constexpr (kMma) {  // whole boxes of TPS_W rows, 128-byte swizzle
                    mbar_expect_tx(bar, 2 * TPS_W * kHeadDim * ES + hdr_bytes);
                    sm100::tma_load_2d_hint(smem_u32(dst), &tm_wk, 0, y, bar, pol);
                    sm100::tma_load_2d_hint(smem_u32(dst + kHalf), &tm_wv, 0, y, bar, pol);
                } else {
                    const unsigned bytes = (unsigned)(te - tb) * kHeadDim * ES;
                    const size_t off = (size_t)y * kHeadDim;
                    mbar_expect_tx(bar, 2 * bytes + hdr_bytes);
                    sm100::bulk_g2s_hint(dst, wk + off, bytes, bar, pol);
                    sm100::bulk_g2s_hint(dst + kHalf, wv + off, bytes, bar, pol);
                }
                if (hdr_bytes)
                    bulk_g2s(my_hdrs + slot * kHdrBytes, hsrc, hdr_bytes, bar);
            }
        } else {
            const int tb = (wj - sq.r) * TPS_D, te = min(sq.ndist, tb + TPS_D);
            const int pfirst = tb / kPage;
            if (pwb != wb || pfirst < pw0 || pfirst + PPS > pw0 + 64)
                load_window(wb, pfirst);
            int id[PPS];
            unsigned mask = 0, total = 0;
#pragma unroll
            for (int j = 0; j < PPS; ++j) {
                id[j] = page_id(pfirst + j);
                const int ptb = max(tb, (pfirst + j) * kPage);
                const int pte = min(te, (pfirst + j + 1) * kPage);
                if (pte > ptb) {
                    if (id[j] >= 0 && id[j] < a.num_pages) {
                        mask |= 1u << j;
                        // the 2-D path copies whole boxes of min(64, TPS_D) rows
                        total += (unsigned)(kMma ? (TPS_D < kPage ? TPS_D : kPage) : (pte - ptb)) * DD * ES;
                    } else if (lane == 0) {
                        report(a.status, DAR_ERR_CAPACITY);
                    }
                }
            }
            if (lane == 0) {
                my_meta[slot] = make_int4(gid, flags | (int)(mask << 24), te - tb, rid);
                mbar_expect_tx(bar, 2 * total + hdr_bytes);
#pragma unroll
                for (int j = 0; j < PPS; ++j) {
                    if ((mask >> j) & 1u) {
                        const int ptb = max(tb, (pfirst + j) * kPage);
                        const int pte = min(te, (pfirst + j + 1) * kPage);
                        const size_t doff = (size_t)(ptb - tb) * DD * ES;
                        if constexpr (kMma) {  // page (id, g) = DD lines of 128 bytes
                            const int y = (id[j] * a.Hkv + g) * DD + (ptb % kPage) * DD / kHeadDim;
                            sm100::tma_load_2d_hint(smem_u32(dst + doff), &tm_pk, 0, y, bar, pol);
                            sm100::tma_load_2d_hint(smem_u32(dst + kHalf + doff), &tm_pv, 0, y, bar, pol);
                        } else {
                            const unsigned bytes = (unsigned)(pte - ptb) * DD * ES;
                            const size_t src = (((size_t)id[j] * a.Hkv + g) * kPage + (ptb % kPage)) * DD;
                            sm100::bulk_g2s_hint(dst + doff, pk + src, bytes, bar, pol);
                            sm100::bulk_g2s_hint(dst + kHalf + doff, pv + src, bytes, bar, pol);
                        }
                    }
                }
                if (hdr_bytes)
                    bulk_g2s(my_hdrs + slot * kHdrBytes, hsrc, hdr_bytes, bar);
            }
        }
        __syncwarp();
        ++issued;
        if (iss_s == ask_at && !pool_done && !asked)
            ask();  // the pool chunk after this range
        // step the walk to the next stage of the range, or to the next range
        if (++iss_s == hi) {
            next_range();
        } else if (++wj == sq.n) {
            wj = 0;
            if (++wgh == per_chunk) {
                wgh = 0;
                do {
                    ++wb;
                } while (s_pre[wb + 1] == s_pre[wb]);  // sequences without stages
                sq = seq_stages<TPS_W, TPS_D>(s_len[wb], w);
            }
        }
    };

    // ---- consume side
    // tensor-core consumer state: A fragments of q (ring) or q~ (pages), output
    // fragments of row g = lane / 4 (query head h0 + g when g < GH)
    constexpr int KSD = DD >= 16 ? DD / 16 : 1;
    constexpr int NDD = DD / 8 > 0 ? DD / 8 : 1;
    uint32_t qa_w[4][4], qa_d[KSD][4];
    float ow[8][4], od[NDD][4];
    float mm = -INFINITY, lp = 0.f;
    // lane-per-token page consumer state (kLanePages)
    float qd[kLanePages ? DD : 1], ol[kLanePages ? DD : 1];
    // CUDA-core consumer state (per head of the slice)
    float m[GH], l[GH], acc[GH][E], qr[GH][E];
#pragma unroll
    for (int k = 0; k < GH; ++k) {
        m[k] = -INFINITY;
        l[k] = 0.f;
#pragma unroll
        for (int e = 0; e < E; ++e)
            acc[k][e] = qr[k][e] = 0.f;
    }
    int4 pend = make_int4(0, 0, 0, 0);  // metadata of the last stage consumed, if it ends a segment
    // Shared parts finished by this warp: lane i holds the group and stage
    // count of the i-th.  Their counts are added together (after one fence)
    // when the warp runs out of work, so the streaming never waits on them; a
    // count that completes its group's stages makes this warp merge the group.
    int pg = 0, pp = 0, npend = 0;
    auto flush = [&]() {
        if (npend == 0)
            return;
        // each count is an acquire-release atomic: it publishes the warp's
        // records (ordered before it by the warp barrier) and, for the count
        // that completes a group, makes the other parts' records visible
        __syncwarp();
        bool fin = false;
        if (lane < npend) {
            int old;
            asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], %2;"
                         : "=r"(old)
                         : "l"(a.counters + pg), "r"(pp)
                         : "memory");
            fin = old + pp == seq_stages<TPS_W, TPS_D>(s_len[pg / per_chunk], w).n;
        }
        unsigned fm = __ballot_sync(0xffffffffu, fin);
        if (fm)
            __syncwarp();  // the acquiring lane's view, to the lanes that load
        // the slots are idle here only if every issued stage has been consumed
        float *rows = issued == consumed ? reinterpret_cast<float *>(my_slots) : nullptr;
        while (fm) {
            const int j = __ffs(fm) - 1;
            fm &= fm - 1;
            combine_group<T, DD, GH, TPS_W, TPS_D>(a, s_pre, s_len, __shfl_sync(0xffffffffu, pg, j), sp, lane,
                                                   rows);
        }
        npend = 0;
    };
    for (;;) {
        // refill first, so that the copies run while a finished segment is written.
        // The first fill stops one stage short: at the start every warp of the SM
        // issues at once, and the warp should not wait on the copy unit for its
        // last stage while its first one may already have landed.
        while (issued - consumed < (consumed > 0 ? kStages : kStages - 1) && iss_s < hi)
            issue_one();
        if (pend.y & kMetaSegEnd) {
            // ---- segment done: write the partial result (m, l, acc) of every head
            const bool win = (pend.y & kMetaRing) != 0;
            float *rec0 = rec_ptr(a.rec, pend.w, (pend.y & kMetaSlot1) ? 1 : 0, win ? 0 : 1, 0, GH);
            if (kLanePages && !win) {
                if constexpr (kLanePages) {
#pragma unroll
                    for (int off = 16; off; off >>= 1)
                        lp += __shfl_xor_sync(0xffffffffu, lp, off);
                    const float tot = reduce_scatter<DD>(ol, lane);
                    constexpr int LPE = 32 / DD;  // lanes holding each entry
                    if (lane % LPE == 0)
                        rec0[lane / LPE] = tot;
                    if (lane == 0)
                        *reinterpret_cast<float2 *>(rec0 + kHeadDim) = make_float2(mm, lp);
                }
            } else if constexpr (kMma) {
                lp += __shfl_xor_sync(0xffffffffu, lp, 1);
                lp += __shfl_xor_sync(0xffffffffu, lp, 2);
                const int g = lane >> 2, c = lane & 3;
                if (g < GH) {
                    float *ra = rec0 + (size_t)g * kRecFloats;
                    if (win) {
#pragma unroll
                        for (int d = 0; d < 8; ++d)
                            *reinterpret_cast<float2 *>(ra + 8 * d + 2 * c) = make_float2(ow[d][0], ow[d][1]);
                    } else {
#pragma unroll
                        for (int d = 0; d < NDD; ++d)
                            *reinterpret_cast<float2 *>(ra + 8 * d + 2 * c) = make_float2(od[d][0], od[d][1]);
                    }
                    if (c == 0)
                        *reinterpret_cast<float2 *>(ra + kHeadDim) = make_float2(mm, lp);
                }
            } else {
                const int LPTc = (win ? kHeadDim : DD) / E;
                for (int off = LPTc; off < 32; off <<= 1) {
#pragma unroll
                    for (int k = 0; k < GH; ++k) {
                        const float mo = __shfl_xor_sync(0xffffffffu, m[k], off);
                        const float lo2 = __shfl_xor_sync(0xffffffffu, l[k], off);
                        const float mn = fmaxf(m[k], mo);
                        const float fa = (m[k] == -INFINITY) ? 0.f : exp2f(m[k] - mn);
                        const float fb = (mo == -INFINITY) ? 0.f : exp2f(mo - mn);
                        l[k] = l[k] * fa + lo2 * fb;
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
                    float *ra = rec0 + (size_t)k * kRecFloats;
                    if (lane < LPTc) {
                        float4 *dstv = reinterpret_cast<float4 *>(ra + lane * E);
#pragma unroll
                        for (int e4 = 0; e4 < E / 4; ++e4)
                            dstv[e4] = make_float4(acc[k][4 * e4], acc[k][4 * e4 + 1], acc[k][4 * e4 + 2],
                                                   acc[k][4 * e4 + 3]);
                    }
                    if (lane == 0)
                        *reinterpret_cast<float2 *>(ra + kHeadDim) = make_float2(m[k], l[k]);
                }
            }
            if (pend.y & kMetaPartEnd) {
                // ---- the range's part of the group is done
                if (pend.y & kMetaShared) {  // counted later, with the warp's other shared parts
                    const int gid = pend.x;
                    const int b = gid / per_chunk, gh = gid - b * per_chunk;
                    const SeqStages gq = seq_stages<TPS_W, TPS_D>(s_len[b], w);
                    const int G0 = s_pre[b] * per_chunk + gh * gq.n;
                    if (lane == npend) {
                        pg = gid;
                        pp = min(sp.lo(pend.w + 1), G0 + gq.n) - max(sp.lo(pend.w), G0);
                    }
                    if (++npend == 32)
                        flush();
                } else {
                    __syncwarp();  // this warp's own records, read back by other lanes
                    combine_group<T, DD, GH, TPS_W, TPS_D>(a, s_pre, s_len, pend.x, sp, lane, nullptr);
                }
            }
        }
        pend.y = 0;
        if (consumed == issued)
            break;

        const int slot = con_slot;
        const unsigned parity = con_phase;
        if (!mbar_wait(&my_bars[slot], parity, a.status)) {
            alive = false;
            break;
        }
        __syncwarp();
        const int4 md = my_meta[slot];
        const bool win = (md.y & kMetaRing) != 0;
        const unsigned pmask = ((unsigned)md.y >> 24) & 0xffu;
        const int ntok = md.z;
        const unsigned char *hdr = my_hdrs + slot * kHdrBytes;
        if (md.y & kMetaSegStart) {
            // ---- new segment: its query rows arrived in this slot's header
            if constexpr (kMma) {
                const int g = lane >> 2, c = lane & 3;
                if (win) {
                    const uint32_t *hq = reinterpret_cast<const uint32_t *>(hdr) + (g < GH ? g : 0) * (kHeadDim / 2);
#pragma unroll
                    for (int ks = 0; ks < 4; ++ks) {
                        qa_w[ks][0] = g < GH ? hq[8 * ks + c] : 0u;
                        qa_w[ks][2] = g < GH ? hq[8 * ks + c + 4] : 0u;
                        qa_w[ks][1] = qa_w[ks][3] = 0u;
                    }
#pragma unroll
                    for (int d = 0; d < 8; ++d)
                        ow[d][0] = ow[d][1] = ow[d][2] = ow[d][3] = 0.f;
                } else if constexpr (kLanePages) {
                    const float *hqt = reinterpret_cast<const float *>(hdr);
#pragma unroll
                    for (int c = 0; c < DD; ++c) {
                        qd[c] = hqt[c] * a.qscale;
                        ol[c] = 0.f;
                    }
                } else {
                    const float *hqt = reinterpret_cast<const float *>(hdr) + (g < GH ? g : 0) * DD;
                    auto pack = [&](int k0) -> uint32_t {
                        if (g >= GH)
                            return 0u;
                        const float2 v2 = *reinterpret_cast<const float2 *>(hqt + k0);
                        __nv_bfloat162 v = __floats2bfloat162_rn(v2.x, v2.y);
                        return *reinterpret_cast<uint32_t *>(&v);
                    };
#pragma unroll
                    for (int ks = 0; ks < KSD; ++ks) {
                        qa_d[ks][0] = pack(16 * ks + 2 * c);
                        qa_d[ks][2] = pack(16 * ks + 2 * c + 8);
                        qa_d[ks][1] = qa_d[ks][3] = 0u;
                    }
#pragma unroll
                    for (int d = 0; d < NDD; ++d)
                        od[d][0] = od[d][1] = od[d][2] = od[d][3] = 0.f;
                }
                mm = -INFINITY;
                lp = 0.f;
            } else {
                const int ROWc = win ? kHeadDim : DD;
                const int sub = lane % (ROWc / E);
#pragma unroll
                for (int k = 0; k < GH; ++k) {
#pragma unroll
                    for (int e = 0; e < E; ++e)
                        qr[k][e] = (win ? to_f32(reinterpret_cast<const T *>(hdr)[k * kHeadDim + sub * E + e])
                                        : reinterpret_cast<const float *>(hdr)[k * DD + sub * E + e]) *
                                   a.qscale;
                    m[k] = -INFINITY;
                    l[k] = 0.f;
#pragma unroll
                    for (int e = 0; e < E; ++e)
                        acc[k][e] = 0.f;
                }
            }
        }

        // ---- this stage's tokens
        unsigned char *src = my_slots + (size_t)slot * kSlotBytes;
        auto run_stage = [&](auto row_tag) {
            constexpr int ROW = decltype(row_tag)::value;
            constexpr int LPT = ROW / E;
            constexpr int TPI = 32 / LPT;
            constexpr int TPS = kHalf / (ROW * ES);
            constexpr int NI = TPS / TPI;  // warp-wide 16-byte loads per half slot
            constexpr int U = NI < 4 ? NI : 4;
            const int grp = lane / LPT, sub = lane % LPT;
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
            const uint32_t sK = smem_u32(src), sV = sK + kHalf;
            if (win) {
                if (ntok == TPS_W) {
                    mma_stage<kHeadDim, TPS_W, GH, false>(sK, sV, ntok, 0xffu, qa_w, ow, mm, lp, a.qscale, lane);
                } else {
                    zero_masked_rows<kHeadDim, TPS_W>(src + kHalf, ntok, 0xffu, lane);
                    mma_stage<kHeadDim, TPS_W, GH, true>(sK, sV, ntok, 0xffu, qa_w, ow, mm, lp, a.qscale, lane);
                }
            } else if constexpr (kLanePages) {
                lane_stage<DD, TPS_D>(sK, sV, ntok, pmask, qd, ol, mm, lp, lane);
            } else {
                if (ntok == TPS_D && pmask == kFullPages) {
                    mma_stage<DD, TPS_D, GH, false>(sK, sV, ntok, pmask, qa_d, od, mm, lp, a.qscale, lane);
                } else {
                    zero_masked_rows<DD, TPS_D>(src + kHalf, ntok, pmask, lane);
                    mma_stage<DD, TPS_D, GH, true>(sK, sV, ntok, pmask, qa_d, od, mm, lp, a.qscale, lane);
                }
            }
        } else {
            if (win)
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
        pend = md;
    }

    if (alive)
        flush();
    if (!alive) {
        // a wait gave up: let this warp's copies still in flight land (bounded) before leaving
        for (int r = consumed + 1; r < issued; ++r)
            mbar_wait(&my_bars[r % kStages], (unsigned)((r / kStages) & 1), a.status);
    }
}


// --------------------------------------------------------------------- launch

DecodeGeometry decode_geometry(dar_dtype dt, int Hq, int Hkv, int dd, int w, int maxp)
{
    DecodeGeometry gm;
    const int esz = dt == DAR_F32 ? 4 : 2;
    const long long tw = kHalf / (kHeadDim * esz), td = kHalf / (dd * esz);
    gm.sph = (w + tw - 1) / tw + ((long long)maxp * kPage + td - 1) / td;
    const int G = Hq / Hkv;
    gm.GH = (G % 4 == 0) ? 4 : (G % 2 == 0) ? 2 : 1;
    gm.HS = G / gm.GH;
    return gm;
}

template <typename T, int DD, int GH>
static cudaError_t decode_t(const DecodeArgs &a, cudaStream_t s)
{
    auto kern = decode_kernel<T, DD, GH>;
    // The four tensor maps of the cache.  A serving loop decodes the same cache
    // call after call, so the maps last encoded on this thread are reused when
    // the buffers and their extents are unchanged (the encoding is a driver
    // call per map).
    struct MapCache {
        const void *base[4] = {nullptr, nullptr, nullptr, nullptr};
        unsigned long long ring_rows = 0, pool_lines = 0;
        CUtensorMap m[4];
    };
    static thread_local MapCache mc;
    CUtensorMap m_wk{}, m_wv{}, m_pk{}, m_pv{};
    if (decode_uses_mma<T, DD>()) {
        constexpr int tps_w = tps_ring<T>(), tps_d = tps_page<T, DD>();
        // one page box: min(64, tps_d) tokens = that many * DD / 64 lines of 128 bytes
        const int pr = (tps_d < kPage ? tps_d : kPage) * DD / kHeadDim;
        const unsigned long long ring_rows = (unsigned long long)a.B * a.Hkv * a.w;
        const unsigned long long pool_lines = (unsigned long long)(a.num_pages > 0 ? a.num_pages : 1) * a.Hkv * DD;
        if (mc.base[0] != a.win_k || mc.base[1] != a.win_v || mc.base[2] != a.pool_kd || mc.base[3] != a.pool_vd ||
            mc.ring_rows != ring_rows || mc.pool_lines != pool_lines) {
            mc.base[0] = nullptr;  // invalid until all four are encoded
            if (!make_tma_2d_bf16(&mc.m[0], a.win_k, ring_rows, kHeadDim, tps_w) ||
                !make_tma_2d_bf16(&mc.m[1], a.win_v, ring_rows, kHeadDim, tps_w) ||
                !make_tma_2d_bf16(&mc.m[2], a.pool_kd, pool_lines, kHeadDim, pr) ||
                !make_tma_2d_bf16(&mc.m[3], a.pool_vd, pool_lines, kHeadDim, pr))
                return cudaErrorInvalidValue;
            mc.base[0] = a.win_k;
            mc.base[1] = a.win_v;
            mc.base[2] = a.pool_kd;
            mc.base[3] = a.pool_vd;
            mc.ring_rows = ring_rows;
            mc.pool_lines = pool_lines;
        }
        m_wk = mc.m[0];
        m_wv = mc.m[1];
        m_pk = mc.m[2];
        m_pv = mc.m[3];
    }
    // one-time set-up per instantiation (kept out of the launch path so launches
    // stay cheap and can be captured in a CUDA graph)
    static PerDeviceOnce once;
    int ctas = 0;
    cudaError_t e = per_device_once(
        once,
        [&](int dev) {
            cudaError_t e2 = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                  (int)decode_smem_bytes(DAR_DECODE_MAX_BATCH));
            int n = 0;
            if (e2 == cudaSuccess)
                e2 = cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
            once.value[dev] = n < kMaxDecodeCtas ? n : kMaxDecodeCtas;  // the workspace holds records for this many
            return e2;
        },
        &ctas);
    if (e != cudaSuccess)
        return e;
    const int rows = a.B * a.Hq;
    const int prep_blocks = min(2 * ctas, max(1, (rows + kPrepThreads / 32 - 1) / (kPrepThreads / 32)));
    // The stream kernel always uses programmatic launch: it sets up while prep
    // drains (prep is this library's own kernel and writes nothing the set-up
    // reads).  prep itself reads q and Uk before its dependency wait, so it may
    // overlap the kernel before it only when the caller vouches that this
    // kernel writes neither (a.prep_overlaps_prev: this library's own cache
    // append, launched by dar_decode_step); otherwise it starts after all
    // earlier work on the stream has finished.
    cudaLaunchAttribute pdl[1];
    pdl[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    pdl[0].val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.stream = s;
    cfg.attrs = pdl;
    cfg.numAttrs = a.prep_overlaps_prev ? 1 : 0;
    cfg.gridDim = dim3(prep_blocks);
    cfg.blockDim = dim3(kPrepThreads);
    e = cudaLaunchKernelEx(&cfg, decode_prep_kernel<T, DD>, a);
    if (e != cudaSuccess)
        return e;
    // one CTA per SM (the records of the workspace are sized for kMaxDecodeCtas)
    cfg.numAttrs = 1;
    cfg.gridDim = dim3(ctas);
    cfg.blockDim = dim3(kDecThreads);
    cfg.dynamicSmemBytes = decode_smem_bytes(a.B);
    return cudaLaunchKernelEx(&cfg, kern, m_wk, m_wv, m_pk, m_pv, a);
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
