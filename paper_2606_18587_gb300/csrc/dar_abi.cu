// dar_abi.cu -- the extern "C" entry points declared in dar.h: argument
// validation (nothing is launched on a bad argument), workspace layout and
// dispatch to the kernels.
#include <math.h>
#include <stdarg.h>
#include <stdio.h>

#include <string>

#include "dar_common.cuh"
#include "dar_launch.h"

namespace {

thread_local std::string g_err;

dar_status fail(dar_status s, const char *fmt, ...)
{
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    g_err = buf;
    return s;
}

dar_status ok()
{
    g_err.clear();
    return DAR_OK;
}

dar_status from_cuda(cudaError_t e, const char *what)
{
    if (e == cudaSuccess)
        return ok();
    return fail(DAR_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
bool dd_supported(int dd) { return dd == 8 || dd == 16 || dd == 32 || dd == 64; }
bool dtype_valid(int dt) { return dt == DAR_F32 || dt == DAR_BF16; }
size_t esize(dar_dtype dt) { return dt == DAR_F32 ? 4 : 2; }
size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

float default_scale(float scale, int d) { return scale > 0.f ? scale : 1.0f / sqrtf((float)d); }
constexpr float kLog2e = 1.4426950408889634f;

// Common shape checks: returns DAR_OK or an error (message set).
dar_status check_dims(int dt, int d, int dd)
{
    if (!dtype_valid(dt))
        return fail(DAR_ERR_INVALID_ARG, "dtype %d is not DAR_F32 or DAR_BF16", dt);
    if (d != dar::kHeadDim)
        return fail(DAR_ERR_UNSUPPORTED, "head dimension d=%d (only d=64 is built)", d);
    if (!dd_supported(dd))
        return fail(DAR_ERR_UNSUPPORTED, "d_down=%d (built: 8, 16, 32, 64)", dd);
    return DAR_OK;
}

dar_status check_cache(const dar_cache *c)
{
    if (!c)
        return fail(DAR_ERR_INVALID_ARG, "cache is NULL");
    dar_status s = check_dims(c->dtype, c->d, c->d_down);
    if (s != DAR_OK)
        return s;
    if (c->B < 0 || c->Hkv < 1 || c->w < 1 || c->max_pages_per_seq < 0 || c->num_pages < 0)
        return fail(DAR_ERR_INVALID_ARG,
                    "cache shape B=%d Hkv=%d w=%d max_pages_per_seq=%d num_pages=%d (need B>=0, "
                    "Hkv>=1, w>=1, page counts >=0)",
                    c->B, c->Hkv, c->w, c->max_pages_per_seq, c->num_pages);
    if (c->B > 4096)
        return fail(DAR_ERR_UNSUPPORTED, "batch %d > 4096", c->B);
    if (c->B == 0)
        return DAR_OK;
    if (!c->win_k || !c->win_v || !c->seq_lens || !c->status)
        return fail(DAR_ERR_INVALID_ARG, "cache ring, seq_lens or status pointer is NULL");
    if (c->max_pages_per_seq > 0 && (!c->block_table || !c->pool_kd || !c->pool_vd))
        return fail(DAR_ERR_INVALID_ARG, "cache block_table or pool pointer is NULL");
    if (c->max_pages_per_seq > 0 && c->num_pages < 1)
        return fail(DAR_ERR_INVALID_ARG, "max_pages_per_seq=%d but num_pages=0", c->max_pages_per_seq);
    if (!aligned16(c->win_k) || !aligned16(c->win_v) || !aligned16(c->pool_kd) ||
        !aligned16(c->pool_vd))
        return fail(DAR_ERR_INVALID_ARG, "cache buffers must be 16-byte aligned");
    if ((double)c->B * c->Hkv * c->w * c->d > 9.0e18 ||
        (double)c->num_pages * c->Hkv * DAR_PAGE_SIZE * c->d_down > 9.0e18)
        return fail(DAR_ERR_INVALID_ARG, "cache too large");
    return DAR_OK;
}

struct DecodeLayout {
    size_t qt, counters, rec, total;
};

// Workspace of dar_attn_decode: the absorbed queries, one counter per
// (sequence, KV head, head slice) group plus the pool's claim counter, and the
// split-K records of every range the stream kernel can run (one per warp,
// then the pool chunks if there is a pool).  Every call rewrites what it reads.
DecodeLayout decode_layout(const dar_cache *c, int Hq, const dar::DecodeGeometry &gm)
{
    DecodeLayout L;
    L.qt = 0;
    L.counters = L.qt + align256((size_t)c->B * Hq * c->d_down * sizeof(float));
    L.rec = L.counters + align256(((size_t)c->B * c->Hkv * gm.HS + 1) * sizeof(int32_t));
    const size_t recs = (size_t)dar::kDecodeRecordRanges * 4 * gm.GH;
    L.total = L.rec + align256(recs * dar::kRecFloats * sizeof(float));
    return L;
}

// Checks the arguments of dar_cache_append and fills *a; *empty = nothing to launch.
dar_status prepare_append(const dar_cache *cache, const void *k_new, const void *v_new, int32_t n,
                          const int32_t *n_per_seq, const float *Dk, const float *Dv, dar::AppendArgs *a,
                          bool *empty)
{
    dar_status s = check_cache(cache);
    if (s != DAR_OK)
        return s;
    if (n < 0)
        return fail(DAR_ERR_INVALID_ARG, "n=%d", n);
    *empty = cache->B == 0 || n == 0;
    if (*empty)
        return ok();
    if (!k_new || !v_new || !Dk || !Dv)
        return fail(DAR_ERR_INVALID_ARG, "NULL pointer");
    if (!aligned16(k_new) || !aligned16(v_new) || !aligned16(Dk) || !aligned16(Dv))
        return fail(DAR_ERR_INVALID_ARG, "k_new, v_new, Dk and Dv must be 16-byte aligned");
    a->k_new = k_new;
    a->v_new = v_new;
    a->Dk = Dk;
    a->Dv = Dv;
    a->win_k = cache->win_k;
    a->win_v = cache->win_v;
    a->pool_kd = cache->pool_kd;
    a->pool_vd = cache->pool_vd;
    a->block_table = cache->block_table;
    a->n_per_seq = n_per_seq;
    a->seq_lens = cache->seq_lens;
    a->status = cache->status;
    a->B = cache->B;
    a->Hkv = cache->Hkv;
    a->n = n;
    a->w = cache->w;
    a->maxp = cache->max_pages_per_seq;
    a->num_pages = cache->num_pages;
    return ok();
}

// Checks the arguments of dar_attn_decode and fills *a; *empty = nothing to launch.
dar_status prepare_decode(const dar_cache *cache, int32_t Hq, const void *q, const float *Uk, const float *Uv,
                          float scale, void *out, void *workspace, size_t workspace_bytes, dar::DecodeArgs *a,
                          bool *empty)
{
    dar_status s = check_cache(cache);
    if (s != DAR_OK)
        return s;
    if (Hq < cache->Hkv || Hq % cache->Hkv)
        return fail(DAR_ERR_INVALID_ARG, "Hq=%d is not a multiple of Hkv=%d", Hq, cache->Hkv);
    if (cache->B > DAR_DECODE_MAX_BATCH)
        return fail(DAR_ERR_UNSUPPORTED, "decode batch %d > %d", cache->B, DAR_DECODE_MAX_BATCH);
    *empty = cache->B == 0;
    if (*empty)
        return ok();
    if (!q || !Uk || !Uv || !out || !workspace)
        return fail(DAR_ERR_INVALID_ARG, "NULL pointer");
    if (!aligned16(q) || !aligned16(out) || !aligned16(Uk) || !aligned16(Uv) || !aligned16(workspace))
        return fail(DAR_ERR_INVALID_ARG, "q, out, Uk, Uv and workspace must be 16-byte aligned");
    dar::DecodeGeometry gm = dar::decode_geometry(cache->dtype, Hq, cache->Hkv, cache->d_down,
                                                  cache->w, cache->max_pages_per_seq);
    DecodeLayout L = decode_layout(cache, Hq, gm);
    if ((double)cache->B * Hq * gm.sph >= 2147483647.0)
        return fail(DAR_ERR_UNSUPPORTED, "B * Hq * stages = %.0f exceeds the int32 stage index",
                    (double)cache->B * Hq * gm.sph);
    if (workspace_bytes < L.total)
        return fail(DAR_ERR_CAPACITY, "workspace %zu bytes < %zu needed", workspace_bytes, L.total);
    char *ws = static_cast<char *>(workspace);
    a->q = q;
    a->out = out;
    a->win_k = cache->win_k;
    a->win_v = cache->win_v;
    a->pool_kd = cache->pool_kd;
    a->pool_vd = cache->pool_vd;
    a->block_table = cache->block_table;
    a->seq_lens = cache->seq_lens;
    a->status = cache->status;
    a->Uk = Uk;
    a->Uv = Uv;
    a->rec = reinterpret_cast<float *>(ws + L.rec);
    a->qt = reinterpret_cast<float *>(ws + L.qt);
    a->counters = reinterpret_cast<int32_t *>(ws + L.counters);
    a->B = cache->B;
    a->Hq = Hq;
    a->Hkv = cache->Hkv;
    a->G = Hq / cache->Hkv;
    a->GH = gm.GH;
    a->HS = gm.HS;
    a->w = cache->w;
    a->maxp = cache->max_pages_per_seq;
    a->num_pages = cache->num_pages;
    a->qscale = default_scale(scale, cache->d) * kLog2e;
    a->prep_overlaps_prev = 0;
    return ok();
}

struct ChunkLayout {
    size_t pos0, kw, vw, kdt, vdt, total;
};

// Workspace of dar_prefill_chunk: the lengths before the chunk, the window
// buffers (full-d keys / values the chunk's queries can see as local) and the
// tail buffers (bottleneck keys / values near the window edge).
ChunkLayout chunk_layout(const dar_cache *c, int n)
{
    ChunkLayout L;
    const size_t bg = (size_t)c->B * c->Hkv;
    const size_t win = bg * dar::chunk_window_rows(c->w, n) * c->d * sizeof(uint16_t);
    const size_t tail = bg * dar::chunk_tail_rows(n) * c->d_down * sizeof(uint16_t);
    L.pos0 = 0;
    L.kw = align256((size_t)c->B * sizeof(int32_t));
    L.vw = L.kw + align256(win);
    L.kdt = L.vw + align256(win);
    L.vdt = L.kdt + align256(tail);
    L.total = L.vdt + align256(tail);
    return L;
}

}  // namespace

void dar::set_last_error(const char *msg) { g_err = msg ? msg : ""; }

extern "C" {

const char *dar_last_error(void) { return g_err.c_str(); }

dar_status dar_down_project(dar_dtype dtype, int32_t B, int32_t Hkv, int32_t n, int32_t d,
                            int32_t d_down, const void *x, const float *W, void *out, void *stream)
{
    dar_status s = check_dims(dtype, d, d_down);
    if (s != DAR_OK)
        return s;
    if (B < 0 || Hkv < 1 || n < 0)
        return fail(DAR_ERR_INVALID_ARG, "B=%d Hkv=%d n=%d", B, Hkv, n);
    if (B == 0 || n == 0)
        return ok();
    if (!x || !W || !out)
        return fail(DAR_ERR_INVALID_ARG, "NULL pointer");
    if (!aligned16(x) || !aligned16(out) || !aligned16(W))
        return fail(DAR_ERR_INVALID_ARG, "buffers must be 16-byte aligned");
    if ((long long)B * Hkv > 65535)
        return fail(DAR_ERR_UNSUPPORTED, "B*Hkv=%lld > 65535", (long long)B * Hkv);
    return from_cuda(dar::launch_down_project(dtype, d_down, x, W, out, B, Hkv, n, d_down,
                                              static_cast<cudaStream_t>(stream)),
                     "dar_down_project launch");
}

dar_status dar_cache_append(const dar_cache *cache, const void *k_new, const void *v_new,
                            int32_t n, const int32_t *n_per_seq, const float *Dk,
                            const float *Dv, void *stream)
{
    dar::AppendArgs a;
    bool empty = false;
    dar_status s = prepare_append(cache, k_new, v_new, n, n_per_seq, Dk, Dv, &a, &empty);
    if (s != DAR_OK || empty)
        return s;
    return from_cuda(dar::launch_cache_append(cache->dtype, cache->d_down, a,
                                              static_cast<cudaStream_t>(stream)),
                     "dar_cache_append launch");
}

size_t dar_decode_workspace_bytes(const dar_cache *cache, int32_t Hq)
{
    if (check_cache(cache) != DAR_OK || Hq < cache->Hkv || Hq % cache->Hkv)
        return 0;
    dar::DecodeGeometry gm = dar::decode_geometry(cache->dtype, Hq, cache->Hkv, cache->d_down,
                                                  cache->w, cache->max_pages_per_seq);
    return decode_layout(cache, Hq, gm).total;
}

dar_status dar_attn_decode(const dar_cache *cache, int32_t Hq, const void *q, const float *Uk,
                           const float *Uv, float scale, void *out, void *workspace,
                           size_t workspace_bytes, void *stream)
{
    dar::DecodeArgs a;
    bool empty = false;
    dar_status s = prepare_decode(cache, Hq, q, Uk, Uv, scale, out, workspace, workspace_bytes, &a, &empty);
    if (s != DAR_OK || empty)
        return s;
    a.prep_overlaps_prev = 0;  // the kernel before this call is the caller's: wait for it
    return from_cuda(dar::launch_decode(cache->dtype, cache->d_down, a,
                                        static_cast<cudaStream_t>(stream)),
                     "dar_attn_decode launch");
}

dar_status dar_attn_decode_direct(const dar_cache *cache, int32_t Hq, const void *q, const void *qd,
                                  const float *Wo, float scale, float scale_down, void *out,
                                  void *workspace, size_t workspace_bytes, void *stream)
{
    dar::DecodeArgs a;
    bool empty = false;
    // Wo stands in for Uk in the shared checks; Uk is never read here
    dar_status s = prepare_decode(cache, Hq, q, Wo, Wo, scale, out, workspace, workspace_bytes, &a, &empty);
    if (s != DAR_OK || empty)
        return s;
    if (!qd)
        return fail(DAR_ERR_INVALID_ARG, "NULL pointer");
    if (!aligned16(qd))
        return fail(DAR_ERR_INVALID_ARG, "qd must be 16-byte aligned");
    a.qd = qd;
    a.qd_ratio = default_scale(scale_down, cache->d_down) / default_scale(scale, cache->d);
    a.prep_overlaps_prev = 0;
    return from_cuda(dar::launch_decode(cache->dtype, cache->d_down, a, static_cast<cudaStream_t>(stream)),
                     "dar_attn_decode_direct launch");
}

dar_status dar_decode_step(const dar_cache *cache, const void *k_new, const void *v_new, int32_t n,
                           const int32_t *n_per_seq, const float *Dk, const float *Dv, int32_t Hq,
                           const void *q, const float *Uk, const float *Uv, float scale, void *out,
                           void *workspace, size_t workspace_bytes, void *stream)
{
    // every argument of both operations is checked before anything is launched
    dar::AppendArgs ap;
    dar::DecodeArgs dc;
    bool app_empty = false, dec_empty = false;
    dar_status s = prepare_append(cache, k_new, v_new, n, n_per_seq, Dk, Dv, &ap, &app_empty);
    if (s != DAR_OK)
        return s;
    s = prepare_decode(cache, Hq, q, Uk, Uv, scale, out, workspace, workspace_bytes, &dc, &dec_empty);
    if (s != DAR_OK)
        return s;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (!app_empty) {
        s = from_cuda(dar::launch_cache_append(cache->dtype, cache->d_down, ap, st), "dar_decode_step append launch");
        if (s != DAR_OK)
            return s;
    }
    if (dec_empty)
        return ok();
    // the kernel just before the decode is the append above, which writes
    // neither q nor Uk: the decode's query-side set-up may overlap it
    dc.prep_overlaps_prev = app_empty ? 0 : 1;
    return from_cuda(dar::launch_decode(cache->dtype, cache->d_down, dc, st), "dar_decode_step decode launch");
}

size_t dar_prefill_chunk_workspace_bytes(const dar_cache *cache, int32_t n)
{
    if (check_cache(cache) != DAR_OK || n < 0)
        return 0;
    return chunk_layout(cache, n).total;
}

dar_status dar_prefill_chunk(const dar_cache *cache, int32_t Hq, int32_t n, const void *q,
                             const void *k_new, const void *v_new, const float *Dk, const float *Uk,
                             const float *Dv, const float *Uv, float scale, void *out, void *workspace,
                             size_t workspace_bytes, void *stream)
{
    dar::AppendArgs ap;
    bool empty = false;
    dar_status s = prepare_append(cache, k_new, v_new, n, nullptr, Dk, Dv, &ap, &empty);
    if (s != DAR_OK)
        return s;
    if (cache->dtype != DAR_BF16 || cache->d_down < 16)
        return fail(DAR_ERR_UNSUPPORTED, "dar_prefill_chunk: bf16 caches with d_down in {16, 32, 64}");
    if (Hq < cache->Hkv || Hq % cache->Hkv)
        return fail(DAR_ERR_INVALID_ARG, "Hq=%d is not a multiple of Hkv=%d", Hq, cache->Hkv);
    if (empty)
        return ok();
    if (!q || !Uk || !Uv || !out || !workspace)
        return fail(DAR_ERR_INVALID_ARG, "NULL pointer");
    if (!aligned16(q) || !aligned16(out) || !aligned16(Uk) || !aligned16(Uv) || !aligned16(workspace))
        return fail(DAR_ERR_INVALID_ARG, "q, out, Uk, Uv and workspace must be 16-byte aligned");
    if ((long long)cache->B * Hq > 65535 || (long long)cache->B * cache->Hkv > 65535)
        return fail(DAR_ERR_UNSUPPORTED, "B*Hq=%lld > 65535", (long long)cache->B * Hq);
    if ((double)cache->B * Hq * n >= 2147483647.0 ||
        (double)cache->B * cache->Hkv * dar::chunk_window_rows(cache->w, n) >= 2147483647.0 ||
        (double)cache->num_pages * cache->Hkv * DAR_PAGE_SIZE >= 2147483647.0)
        return fail(DAR_ERR_UNSUPPORTED, "dar_prefill_chunk: row indices beyond int32");
    const ChunkLayout L = chunk_layout(cache, n);
    if (workspace_bytes < L.total)
        return fail(DAR_ERR_CAPACITY, "workspace %zu bytes < %zu needed", workspace_bytes, L.total);
    char *ws = static_cast<char *>(workspace);
    dar::ChunkArgs c;
    c.app = ap;
    c.win_k = cache->win_k;
    c.win_v = cache->win_v;
    c.pos0 = reinterpret_cast<int32_t *>(ws + L.pos0);
    c.kw = ws + L.kw;
    c.vw = ws + L.vw;
    c.kdt = ws + L.kdt;
    c.vdt = ws + L.vdt;
    dar::PrefillArgs &a = c.pf;
    a.q = q;
    a.k = a.v = a.kd = a.vd = nullptr;
    a.Uk = Uk;
    a.Uv = Uv;
    a.out = out;
    a.status = cache->status;
    a.B = cache->B;
    a.Hq = Hq;
    a.Hkv = cache->Hkv;
    a.N = 0;
    a.w = cache->w;
    a.dd = cache->d_down;
    a.kd_stride = a.vd_stride = cache->d_down;
    a.qscale = default_scale(scale, cache->d) * kLog2e;
    a.pos0 = c.pos0;
    a.block_table = cache->block_table;
    a.pool_kd = cache->pool_kd;
    a.pool_vd = cache->pool_vd;
    a.n = n;
    a.NW = dar::chunk_window_rows(cache->w, n);
    a.NT = dar::chunk_tail_rows(n);
    a.maxp = cache->max_pages_per_seq;
    a.num_pages = cache->num_pages;
    return from_cuda(dar::launch_prefill_chunk(cache->d_down, c, static_cast<cudaStream_t>(stream)),
                     "dar_prefill_chunk launch");
}

size_t dar_prefill_workspace_bytes(dar_dtype dtype, int32_t B, int32_t Hkv, int32_t N,
                                   int32_t d_down)
{
    if (!dtype_valid(dtype) || B < 0 || Hkv < 0 || N < 0 || d_down < 1)
        return 0;
    const size_t rows = (size_t)B * Hkv * N;
    return align256(rows * dar::prefill_kd_stride(dtype, d_down) * esize(dtype)) +
           align256(rows * dar::prefill_vd_stride(dtype, d_down) * esize(dtype));
}

}  // extern "C"

namespace {

// dar_attn_prefill (qd == NULL: q~ = q Uk^T) and dar_attn_prefill_direct
// (qd given, Uk unused, global scores at scale_down).
dar_status prefill_common(dar_dtype dtype, int32_t B, int32_t Hq, int32_t Hkv, int32_t N, int32_t d,
                          int32_t d_down, int32_t w, const void *q, const void *qd, const void *k,
                          const void *v, const float *Dk, const float *Uk, const float *Dv, const float *Uv,
                          float scale, float scale_down, void *out, void *workspace, size_t workspace_bytes,
                          int32_t *status, void *stream)
{
    dar_status s = check_dims(dtype, d, d_down);
    if (s != DAR_OK)
        return s;
    if (B < 0 || Hkv < 1 || Hq < Hkv || Hq % Hkv || N < 0 || w < 0)
        return fail(DAR_ERR_INVALID_ARG, "B=%d Hq=%d Hkv=%d N=%d w=%d", B, Hq, Hkv, N, w);
    if (B == 0 || N == 0)
        return ok();
    if ((long long)B * Hq > 65535 || (long long)B * Hkv > 65535)
        return fail(DAR_ERR_UNSUPPORTED, "B*Hq=%lld > 65535", (long long)B * Hq);
    if (!Uk)
        Uk = Uv;  // the direct variant has no Uk; never read then
    if (!q || !k || !v || !Dk || !Uk || !Dv || !Uv || !out || !workspace)
        return fail(DAR_ERR_INVALID_ARG, "NULL pointer");
    if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(out) ||
        !aligned16(workspace) || !aligned16(Dk) || !aligned16(Dv) || !aligned16(Uk) ||
        !aligned16(Uv) || (qd && !aligned16(qd)))
        return fail(DAR_ERR_INVALID_ARG, "buffers must be 16-byte aligned");
    const size_t need = dar_prefill_workspace_bytes(dtype, B, Hkv, N, d_down);
    if (workspace_bytes < need)
        return fail(DAR_ERR_CAPACITY, "workspace %zu bytes < %zu needed", workspace_bytes, need);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const int kstride = dar::prefill_kd_stride(dtype, d_down);
    const int vstride = dar::prefill_vd_stride(dtype, d_down);
    char *kd = static_cast<char *>(workspace);
    char *vd = kd + align256((size_t)B * Hkv * N * kstride * esize(dtype));
    cudaError_t e = dar::launch_down_project_kv(dtype, d_down, k, v, Dk, Dv, kd, vd, B, Hkv, N, kstride, vstride,
                                                dar::prefill_vd_ones_col(dtype, d_down), st);
    if (e != cudaSuccess)
        return from_cuda(e, "dar_attn_prefill down-projection launch");
    dar::PrefillArgs a;
    a.q = q;
    a.k = k;
    a.v = v;
    a.kd = kd;
    a.vd = vd;
    a.Uk = Uk;
    a.Uv = Uv;
    a.out = out;
    a.status = status;
    a.B = B;
    a.Hq = Hq;
    a.Hkv = Hkv;
    a.N = N;
    a.w = w;
    a.dd = d_down;
    a.kd_stride = kstride;
    a.vd_stride = vstride;
    a.qscale = default_scale(scale, d) * kLog2e;
    a.qd = qd;
    a.qd_ratio = qd ? default_scale(scale_down, d_down) / default_scale(scale, d) : 1.f;
    if (dtype == DAR_BF16)
        return from_cuda(dar::launch_prefill_tc(d_down, a, st), "dar_attn_prefill (tcgen05) launch");
    return from_cuda(dar::launch_prefill_simt(dtype, d_down, a, st), "dar_attn_prefill launch");
}

}  // namespace

extern "C" {

dar_status dar_attn_prefill(dar_dtype dtype, int32_t B, int32_t Hq, int32_t Hkv, int32_t N,
                            int32_t d, int32_t d_down, int32_t w, const void *q, const void *k,
                            const void *v, const float *Dk, const float *Uk, const float *Dv,
                            const float *Uv, float scale, void *out, void *workspace,
                            size_t workspace_bytes, int32_t *status, void *stream)
{
    if (!Uk && B > 0 && N > 0)
        return fail(DAR_ERR_INVALID_ARG, "NULL pointer");
    return prefill_common(dtype, B, Hq, Hkv, N, d, d_down, w, q, nullptr, k, v, Dk, Uk, Dv, Uv, scale, 0.f, out,
                          workspace, workspace_bytes, status, stream);
}

}  // extern "C"

namespace {

dar_status check_latent(const dar_latent_cache *c)
{
    if (!c)
        return fail(DAR_ERR_INVALID_ARG, "cache is NULL");
    if (c->d != dar::kHeadDim)
        return fail(DAR_ERR_UNSUPPORTED, "head dimension d=%d (only d=64 is built)", c->d);
    if (c->d_lat != 64 && c->d_lat != 128 && c->d_lat != 192 && c->d_lat != 256)
        return fail(DAR_ERR_UNSUPPORTED, "d_lat=%d (built: 64, 128, 192, 256)", c->d_lat);
    if (c->B < 0 || c->Hkv < 1 || c->w < 1 || c->D < 1 || c->max_pages_per_seq < 1 || c->num_pages < 1)
        return fail(DAR_ERR_INVALID_ARG, "latent cache shape B=%d Hkv=%d w=%d D=%d max_pages_per_seq=%d "
                    "num_pages=%d", c->B, c->Hkv, c->w, c->D, c->max_pages_per_seq, c->num_pages);
    if (c->D > 8192)
        return fail(DAR_ERR_UNSUPPORTED, "hidden width D=%d > 8192", c->D);
    if (c->B > 65535)
        return fail(DAR_ERR_UNSUPPORTED, "batch %d > 65535", c->B);
    if (c->B == 0)
        return DAR_OK;
    if (!c->win_k || !c->win_v || !c->pool_c || !c->block_table || !c->seq_lens || !c->status)
        return fail(DAR_ERR_INVALID_ARG, "latent cache pointer is NULL");
    if (!aligned16(c->win_k) || !aligned16(c->win_v) || !aligned16(c->pool_c))
        return fail(DAR_ERR_INVALID_ARG, "latent cache buffers must be 16-byte aligned");
    if ((double)c->num_pages * DAR_PAGE_SIZE >= 2147483647.0 || (double)c->max_pages_per_seq * 64 >= 2147483647.0)
        return fail(DAR_ERR_UNSUPPORTED, "latent pool rows beyond int32");
    return DAR_OK;
}

}  // namespace

extern "C" {

dar_status dar_latent_append(const dar_latent_cache *cache, const void *h_new, const void *k_new,
                             const void *v_new, int32_t n, const int32_t *n_per_seq,
                             const float *W_down, void *stream)
{
    dar_status s = check_latent(cache);
    if (s != DAR_OK)
        return s;
    if (n < 0)
        return fail(DAR_ERR_INVALID_ARG, "n=%d", n);
    if (cache->B == 0 || n == 0)
        return ok();
    if (!h_new || !k_new || !v_new || !W_down)
        return fail(DAR_ERR_INVALID_ARG, "NULL pointer");
    if (!aligned16(h_new) || !aligned16(k_new) || !aligned16(v_new) || !aligned16(W_down))
        return fail(DAR_ERR_INVALID_ARG, "h_new, k_new, v_new and W_down must be 16-byte aligned");
    dar::LatentAppendArgs a;
    a.h = h_new;
    a.k_new = k_new;
    a.v_new = v_new;
    a.Wdown = W_down;
    a.win_k = cache->win_k;
    a.win_v = cache->win_v;
    a.pool_c = cache->pool_c;
    a.block_table = cache->block_table;
    a.n_per_seq = n_per_seq;
    a.seq_lens = cache->seq_lens;
    a.status = cache->status;
    a.B = cache->B;
    a.Hkv = cache->Hkv;
    a.n = n;
    a.D = cache->D;
    a.DL = cache->d_lat;
    a.w = cache->w;
    a.maxp = cache->max_pages_per_seq;
    a.num_pages = cache->num_pages;
    return from_cuda(dar::launch_latent_append(a, static_cast<cudaStream_t>(stream)), "dar_latent_append launch");
}

dar_status dar_latent_absorb(int32_t Hkv, int32_t D, int32_t d, int32_t d_lat, const float *W_up,
                             const float *W_K, const float *W_V, float *A_K, float *A_V, void *stream)
{
    if (d != dar::kHeadDim)
        return fail(DAR_ERR_UNSUPPORTED, "head dimension d=%d (only d=64 is built)", d);
    if (Hkv < 1 || D < 1 || d_lat < 1 || Hkv > 65535 || d_lat > 65535)
        return fail(DAR_ERR_INVALID_ARG, "Hkv=%d D=%d d_lat=%d", Hkv, D, d_lat);
    if (!W_up || !W_K || !W_V || !A_K || !A_V)
        return fail(DAR_ERR_INVALID_ARG, "NULL pointer");
    return from_cuda(dar::launch_latent_absorb(W_up, W_K, W_V, A_K, A_V, Hkv, D, d_lat,
                                               static_cast<cudaStream_t>(stream)),
                     "dar_latent_absorb launch");
}

size_t dar_latent_decode_workspace_bytes(const dar_latent_cache *cache, int32_t Hq)
{
    if (check_latent(cache) != DAR_OK || Hq < cache->Hkv || Hq % cache->Hkv || Hq > 32)
        return 0;
    return dar::latent_decode_workspace_bytes(cache->B, Hq, cache->d_lat, cache->max_pages_per_seq);
}

dar_status dar_latent_decode(const dar_latent_cache *cache, int32_t Hq, const void *q, const float *A_K,
                             const float *A_V, float scale, void *out, void *workspace,
                             size_t workspace_bytes, void *stream)
{
    dar_status s = check_latent(cache);
    if (s != DAR_OK)
        return s;
    if (Hq < cache->Hkv || Hq % cache->Hkv)
        return fail(DAR_ERR_INVALID_ARG, "Hq=%d is not a multiple of Hkv=%d", Hq, cache->Hkv);
    if (Hq > 32)
        return fail(DAR_ERR_UNSUPPORTED, "Hq=%d > 32", Hq);
    if (cache->B > DAR_DECODE_MAX_BATCH)
        return fail(DAR_ERR_UNSUPPORTED, "latent decode batch %d > %d", cache->B, DAR_DECODE_MAX_BATCH);
    if (cache->B == 0)
        return ok();
    if (!q || !A_K || !A_V || !out || !workspace)
        return fail(DAR_ERR_INVALID_ARG, "NULL pointer");
    if (!aligned16(q) || !aligned16(out) || !aligned16(A_K) || !aligned16(A_V) || !aligned16(workspace))
        return fail(DAR_ERR_INVALID_ARG, "q, out, A_K, A_V and workspace must be 16-byte aligned");
    const size_t need = dar::latent_decode_workspace_bytes(cache->B, Hq, cache->d_lat, cache->max_pages_per_seq);
    if (workspace_bytes < need)
        return fail(DAR_ERR_CAPACITY, "workspace %zu bytes < %zu needed", workspace_bytes, need);
    dar::LatentDecodeArgs a;
    a.q = q;
    a.out = out;
    a.win_k = cache->win_k;
    a.win_v = cache->win_v;
    a.pool_c = cache->pool_c;
    a.block_table = cache->block_table;
    a.seq_lens = cache->seq_lens;
    a.status = cache->status;
    a.Ak = A_K;
    a.Av = A_V;
    a.B = cache->B;
    a.Hq = Hq;
    a.Hkv = cache->Hkv;
    a.DL = cache->d_lat;
    a.w = cache->w;
    a.maxp = cache->max_pages_per_seq;
    a.num_pages = cache->num_pages;
    a.scale = default_scale(scale, cache->d);
    return from_cuda(dar::launch_latent_decode(a, workspace, static_cast<cudaStream_t>(stream)),
                     "dar_latent_decode launch");
}

size_t dar_attn_backward_workspace_bytes(dar_dtype dtype, int32_t B, int32_t Hq, int32_t Hkv, int32_t N,
                                         int32_t d_down)
{
    if (!dtype_valid(dtype) || B < 0 || Hkv < 1 || Hq < Hkv || Hq % Hkv || N < 0 || !dd_supported(d_down))
        return 0;
    return dar::backward_workspace_bytes(dtype, B, Hq, Hkv, N, d_down);
}

dar_status dar_attn_backward(dar_dtype dtype, int32_t B, int32_t Hq, int32_t Hkv, int32_t N, int32_t d,
                             int32_t d_down, int32_t w, const void *q, const void *k, const void *v,
                             const float *Dk, const float *Uk, const float *Dv, const float *Uv,
                             const void *out, const void *dout, float scale, void *dq, void *dk, void *dv,
                             float *dDk, float *dUk, float *dDv, float *dUv, void *workspace,
                             size_t workspace_bytes, void *stream)
{
    dar_status s = check_dims(dtype, d, d_down);
    if (s != DAR_OK)
        return s;
    if (B < 0 || Hkv < 1 || Hq < Hkv || Hq % Hkv || N < 0 || w < 0)
        return fail(DAR_ERR_INVALID_ARG, "B=%d Hq=%d Hkv=%d N=%d w=%d", B, Hq, Hkv, N, w);
    if ((long long)B * Hq > 65535 || (long long)B * Hkv > 65535)
        return fail(DAR_ERR_UNSUPPORTED, "B*Hq=%lld > 65535", (long long)B * Hq);
    const void *ptrs[] = {q, k, v, Dk, Uk, Dv, Uv, out, dout, dq, dk, dv, dDk, dUk, dDv, dUv, workspace};
    for (const void *p : ptrs)
        if (!p)
            return fail(DAR_ERR_INVALID_ARG, "NULL pointer");
    for (const void *p : ptrs)
        if (!aligned16(p))
            return fail(DAR_ERR_INVALID_ARG, "buffers must be 16-byte aligned");
    const size_t need = dar::backward_workspace_bytes(dtype, B, Hq, Hkv, N, d_down);
    if (workspace_bytes < need)
        return fail(DAR_ERR_CAPACITY, "workspace %zu bytes < %zu needed", workspace_bytes, need);
    dar::BackwardArgs a;
    a.q = q;
    a.k = k;
    a.v = v;
    a.out = out;
    a.dout = dout;
    a.Dk = Dk;
    a.Uk = Uk;
    a.Dv = Dv;
    a.Uv = Uv;
    a.dq = dq;
    a.dk = dk;
    a.dv = dv;
    a.dDk = dDk;
    a.dUk = dUk;
    a.dDv = dDv;
    a.dUv = dUv;
    a.B = B;
    a.Hq = Hq;
    a.Hkv = Hkv;
    a.N = N;
    a.w = w;
    a.dd = d_down;
    a.scale = default_scale(scale, d);
    return from_cuda(dar::launch_backward(dtype, a, workspace, static_cast<cudaStream_t>(stream)),
                     "dar_attn_backward launch");
}

dar_status dar_attn_prefill_direct(dar_dtype dtype, int32_t B, int32_t Hq, int32_t Hkv, int32_t N,
                                   int32_t d, int32_t d_down, int32_t w, const void *q, const void *qd,
                                   const void *k, const void *v, const float *Dk, const float *Dv,
                                   const float *Wo, float scale, float scale_down, void *out,
                                   void *workspace, size_t workspace_bytes, int32_t *status,
                                   void *stream)
{
    if (!qd && B > 0 && N > 0)
        return fail(DAR_ERR_INVALID_ARG, "NULL pointer");
    return prefill_common(dtype, B, Hq, Hkv, N, d, d_down, w, q, qd, k, v, Dk, nullptr, Dv, Wo, scale, scale_down,
                          out, workspace, workspace_bytes, status, stream);
}

}  // extern "C"
