// dar_launch.h -- internal launchers behind the C ABI (host side).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include <mutex>

#include "dar.h"

namespace dar {

struct AppendArgs {
    const void *k_new, *v_new;  // [B][Hkv][n][64]
    const float *Dk, *Dv;       // [Hkv][64][dd]
    void *win_k, *win_v;        // [B][Hkv][w][64]
    void *pool_kd, *pool_vd;    // [num_pages][Hkv][64][dd]
    const int32_t *block_table; // [B][maxp]
    const int32_t *n_per_seq;   // [B] or nullptr (every sequence appends n)
    int32_t *seq_lens;
    int32_t *status;
    int B, Hkv, n, w, maxp, num_pages;
};

struct DecodeArgs {
    const void *q;  // [B][Hq][64]
    void *out;      // [B][Hq][64]
    const void *win_k, *win_v;
    const void *pool_kd, *pool_vd;
    const int32_t *block_table;
    const int32_t *seq_lens;
    int32_t *status;
    const float *Uk, *Uv;  // [Hkv][dd][64]
    float *rec;         // split-K partial results, kRecFloats per (warp, slot, type, head)
    float *qt;          // [B][Hq][dd] q~ = q Uk^T
    int32_t *counters;  // [B][Hkv][HS] finished stages per group, then the pool's claim counter
    int B, Hq, Hkv, G, GH, HS, w, maxp, num_pages;
    float qscale;  // scale * log2(e)
    // direct lower-dimensional global attention (Sec. 5): the d_down query of
    // each row [B][Hq][dd] T, used as q~ after multiplying by qd_ratio =
    // scale_down / scale (nullptr: q~ = q Uk^T)
    const void *qd = nullptr;
    float qd_ratio = 1.f;
    // the kernel before the decode on the stream is this library's cache
    // append (which writes neither q nor Uk): the decode's query-side set-up
    // may overlap it
    int prep_overlaps_prev;
};

struct PrefillArgs {
    const void *q, *k, *v;  // [B][Hq|Hkv][N][64]
    const void *kd, *vd;    // [B][Hkv][N][kd_stride], [B][Hkv][N][vd_stride] (Eq. 1 output, padded)
    const float *Uk, *Uv;   // [Hkv][dd][64]
    void *out;              // [B][Hq][N][64]
    int32_t *status;        // device error word or nullptr
    int B, Hq, Hkv, N, w, dd, kd_stride, vd_stride;
    float qscale;  // scale * log2(e)
    // direct lower-dimensional global attention (Sec. 5): the d_down query of
    // each row [B][Hq][N][dd] T, used as q~ after multiplying by qd_ratio =
    // scale_down / scale (nullptr: q~ = q Uk^T)
    const void *qd = nullptr;
    float qd_ratio = 1.f;
    // chunked prefill over a cache (dar_prefill_chunk): query b sits at
    // position pos0[b] + r, r < n; local keys come from a window buffer of NW
    // rows per (b, KV head), starting at the 64-aligned position below
    // pos0[b] - w + 1; global keys from whole pages through the block table,
    // and from a tail buffer of NT rows per (b, KV head) from the 64-aligned
    // position below pos0[b] - w on (k, v, kd, vd then point at the buffers)
    const int32_t *pos0 = nullptr;
    const int32_t *block_table = nullptr;
    const void *pool_kd = nullptr, *pool_vd = nullptr;
    int n = 0, NW = 0, NT = 0, maxp = 0, num_pages = 0;
};

// Row stride (elements) of the prefill bottleneck workspace: the tensor-core
// path needs rows of at least 16 bf16 (one MMA K step).
inline int prefill_kd_stride(dar_dtype dt, int dd) { return (dt == DAR_BF16 && dd < 16) ? 16 : dd; }
// Row stride of the prefill's v^D workspace.  The tensor-core path appends 16
// columns of ones after the kd_stride values (zero padding after them), so one
// PV product also sums P into the softmax denominator: 32 for d_down <= 16, 64
// for d_down = 32; d_down = 64 keeps plain rows (its sums take a product of
// their own).
inline int prefill_vd_stride(dar_dtype dt, int dd)
{
    if (dt != DAR_BF16)
        return dd;
    const int ks = prefill_kd_stride(dt, dd);
    return ks == 16 ? 32 : ks == 32 ? 64 : ks;
}
// First column of the ones block in a v^D row (-1: none).
inline int prefill_vd_ones_col(dar_dtype dt, int dd)
{
    const int ks = prefill_kd_stride(dt, dd);
    return prefill_vd_stride(dt, dd) > ks ? ks : -1;
}

// Each launcher returns cudaSuccess or the launch error.
// Eq. 1 into rows of `ostride` elements (entries dd..ostride-1 are zeroed).
cudaError_t launch_down_project(dar_dtype dt, int dd, const void *x, const float *W, void *out,
                                int B, int Hkv, int n, int ostride, cudaStream_t s);
// The same for keys and values in one launch: kd = k Dk (rows of kstride),
// vd = v Dv (rows of vstride, with 16 ones from column v_ones_col if >= 0).
cudaError_t launch_down_project_kv(dar_dtype dt, int dd, const void *k, const void *v, const float *Dk,
                                   const float *Dv, void *kd, void *vd, int B, int Hkv, int n, int kstride,
                                   int vstride, int v_ones_col, cudaStream_t s);
cudaError_t launch_cache_append(dar_dtype dt, int dd, const AppendArgs &a, cudaStream_t s);
cudaError_t launch_decode(dar_dtype dt, int dd, const DecodeArgs &a, cudaStream_t s);
cudaError_t launch_prefill_simt(dar_dtype dt, int dd, const PrefillArgs &a, cudaStream_t s);
cudaError_t launch_prefill_tc(int dd, const PrefillArgs &a, cudaStream_t s);

// Gradients of the causal forward (dar_backward.cu); the workspace holds the
// Eq. 1 vectors, per-row q~, dO~, D, log-sum-exp, dq~, O^D, per-key dk^D,
// dv^D and the projection gradients' partial sums.
struct BackwardArgs {
    const void *q, *k, *v, *out, *dout;
    const float *Dk, *Uk, *Dv, *Uv;
    void *dq, *dk, *dv;
    float *dDk, *dUk, *dDv, *dUv;
    int B, Hq, Hkv, N, w, dd;
    float scale;
};
size_t backward_workspace_bytes(dar_dtype dt, int B, int Hq, int Hkv, int N, int dd);
cudaError_t launch_backward(dar_dtype dt, const BackwardArgs &a, void *workspace, cudaStream_t s);

// The latent form (dar_latent.cu): one bottleneck per token shared by all heads.
struct LatentAppendArgs {
    const void *h, *k_new, *v_new;
    const float *Wdown;
    void *win_k, *win_v, *pool_c;
    const int32_t *block_table, *n_per_seq;
    int32_t *seq_lens, *status;
    int B, Hkv, n, D, DL, w, maxp, num_pages;
};
struct LatentDecodeArgs {
    const void *q;
    void *out;
    const void *win_k, *win_v, *pool_c;
    const int32_t *block_table, *seq_lens;
    int32_t *status;
    const float *Ak, *Av;
    int B, Hq, Hkv, DL, w, maxp, num_pages;
    float scale;
};
size_t latent_decode_workspace_bytes(int B, int Hq, int DL, int maxp);
cudaError_t launch_latent_append(const LatentAppendArgs &a, cudaStream_t s);
cudaError_t launch_latent_absorb(const float *Wup, const float *WK, const float *WV, float *Ak, float *Av, int Hkv,
                                 int D, int DL, cudaStream_t s);
cudaError_t launch_latent_decode(const LatentDecodeArgs &a, void *workspace, cudaStream_t s);

// Chunked prefill over a cache: gather kernel, attention (chunk mode), then
// the cache append of the chunk.  Buffers of the workspace (see dar_abi.cu).
struct ChunkArgs {
    PrefillArgs pf;        // attention arguments (q, out, Uk, Uv, scale, chunk fields)
    AppendArgs app;        // the append of the chunk (k_new, v_new, Dk, Dv, cache)
    const void *win_k, *win_v;  // the cache ring (read by the gather kernel)
    void *kw, *vw, *kdt, *vdt;  // window and tail buffers
    int32_t *pos0;              // [B] lengths before the chunk
};
cudaError_t launch_prefill_chunk(int dd, const ChunkArgs &c, cudaStream_t s);
// Rows per (sequence, KV head) of the chunk's window and tail buffers.
inline int chunk_window_rows(int w, int n) { return (w + n + 126 + 63) / 64 * 64; }
inline int chunk_tail_rows(int n) { return (n + 127 + 63) / 64 * 64; }

// Split-K geometry of the decode kernel (shared by workspace sizing and launch).
struct DecodeGeometry {
    long long sph;  // stages per (sequence, query head) at full capacity
    int GH, HS;     // query heads per group, groups per KV head
};
// The decode stream kernel runs one CTA of kDecodeWarpsPerCta warps per SM, at
// most kMaxDecodeCtas CTAs.  Its stages fall into ranges -- one per warp, then
// up to kDecodePoolChunks pool chunks if kDecodePoolPercent > 0 -- and each
// range owns 2 slots x 2 types x GH records of kRecFloats floats (acc[64], m,
// l, padding to 16 bytes) in the workspace.
constexpr int kDecodeWarpsPerCta = 8;
constexpr int kMaxDecodeCtas = 160;
constexpr int kDecodePoolPercent = 0;  // share of the stages in the claimable pool (0: no pool)
constexpr int kDecodePoolChunks = 2 * kMaxDecodeCtas * kDecodeWarpsPerCta;  // pool chunks at most
// ranges the workspace holds records for: one per warp, plus the pool's chunks when there is a pool
constexpr int kDecodeRecordRanges = kMaxDecodeCtas * kDecodeWarpsPerCta + (kDecodePoolPercent > 0 ? kDecodePoolChunks : 0);
constexpr int kRecFloats = 68;
DecodeGeometry decode_geometry(dar_dtype dt, int Hq, int Hkv, int dd, int w, int maxp);

// 2-D tensor map of a bf16 row-major [rows][cols] array (cols * 2 = 16, 32, 64
// or 128 bytes, swizzled to match) with boxes of [box_rows][cols].
bool make_tma_2d_bf16(CUtensorMap *map, const void *base, unsigned long long rows, int cols, int box_rows);

// Set the message dar_last_error() returns on this thread.
void set_last_error(const char *msg);

// One-time set-up per device: kernel attributes (such as the shared-memory
// opt-in) apply only to the device that is current when they are set, so each
// device runs the set-up once, with itself current.  Thread-safe; a failed
// set-up keeps its error.
constexpr int kMaxDevices = 64;
struct PerDeviceOnce {
    std::once_flag flag[kMaxDevices];
    cudaError_t err[kMaxDevices] = {};
    int value[kMaxDevices] = {};  // whatever the set-up records (e.g. a CTA count)
};

// Runs fn(dev) once for the current device dev; returns its error and stores
// *value = the value fn recorded (fn returns cudaError_t and may write o.value[dev]).
template <typename F>
cudaError_t per_device_once(PerDeviceOnce &o, F &&fn, int *value = nullptr)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess)
        return e;
    if (dev < 0 || dev >= kMaxDevices)
        return cudaErrorInvalidDevice;
    std::call_once(o.flag[dev], [&] { o.err[dev] = fn(dev); });
    if (value)
        *value = o.value[dev];
    return o.err[dev];
}

}  // namespace dar
