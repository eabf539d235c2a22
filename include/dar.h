/*
 * dar.h -- C ABI of the GB300 (sm_103a) kernels for Distance-Adaptive
 * Representation (DAR) attention: causal attention in which the last w tokens
 * (the current one included) keep full head-dimension keys and values and
 * older tokens keep only d_down-dimensional bottleneck vectors that are lifted
 * back to d ("Dual Dimensionality for Local and Global Attention", Sec. 2,
 * Eq. 1-4, and the cache scheme of Sec. 5 "Compute and memory efficiency").
 *
 * Conventions shared by every entry point
 *  - All tensor arguments are DEVICE pointers to caller-allocated, caller-owned,
 *    contiguous row-major memory.  The library allocates nothing, frees nothing
 *    and never synchronises: every call enqueues work on `stream` (a
 *    cudaStream_t passed as void*; NULL = the legacy default stream) and returns.
 *  - Storage type T is fp32 (DAR_F32) or bf16 (DAR_BF16) for queries, keys,
 *    values, outputs and the cached vectors.  The projection matrices are
 *    always fp32.  Arithmetic is fp32 on the device.
 *  - Per KV head g the method uses four matrices (the per-head reading of
 *    Eq. 1-2): Dk, Dv = W_down for keys / values, shape [Hkv][d][d_down], and
 *    Uk, Uv = W_up for keys / values, shape [Hkv][d_down][d].  Passing the
 *    same pointers for K and V gives one shared bottleneck.
 *  - GQA: query head h reads KV head g = h / (Hq / Hkv).
 *  - Supported shapes: d = 64; d_down in {8, 16, 32, 64}; Hq a multiple of Hkv.
 *  - Arguments are checked on the host before any launch; a bad argument
 *    returns an error code and launches nothing.  Conditions only the device
 *    can see (a seq_len or block-table entry out of range) are written to the
 *    caller's status word (first error wins) and the affected work is skipped;
 *    the kernels never trap.  dar_last_error() describes the last non-OK
 *    return on the calling thread.
 *  - Every wait a kernel makes on another part of itself (a copy landing, a
 *    tensor-core result) is bounded: after 2 s without progress the waiting
 *    block writes DAR_ERR_DEVICE to the status word, lets its own copies in
 *    flight land, releases its tensor memory and exits, so the caller finds a
 *    stuck kernel on the host instead of a hung device.
 *  - `scale` <= 0 selects the default 1/sqrt(d) of Eq. 4.
 */
#ifndef DAR_H
#define DAR_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    DAR_OK = 0,
    DAR_ERR_INVALID_ARG = 1, /* null pointer, negative size, inconsistent shape   */
    DAR_ERR_UNSUPPORTED = 2, /* valid but not built (d != 64, d_down not listed)  */
    DAR_ERR_CAPACITY = 3,    /* workspace too small / no page for a token         */
    DAR_ERR_CUDA = 4,        /* the CUDA runtime reported an error at launch      */
    DAR_ERR_DEVICE = 5       /* written to a status word: a kernel gave up on a
                                bounded internal wait (see below) and skipped the
                                rest of its work; the context stays usable        */
} dar_status;

typedef enum { DAR_F32 = 0, DAR_BF16 = 1 } dar_dtype;

/* Tokens per page of the bottleneck pool. */
#define DAR_PAGE_SIZE 64

/* Largest batch dar_attn_decode accepts (its per-sequence tables are built by
 * one thread block of 1024 threads, one thread per sequence). */
#define DAR_DECODE_MAX_BATCH 1024

/*
 * Mixed-dimension KV cache (Sec. 5, "Compute and memory efficiency": tokens
 * beyond the window keep only their d_down vectors, so the cache costs
 * O(T d_down + w d) instead of O(T d)).  Host struct holding device pointers.
 *
 *  win_k, win_v   [B][Hkv][w][d] T.  The token at position p of sequence b
 *                 sits in ring slot p % w while L_b - 1 - p < w.
 *  pool_kd,
 *  pool_vd        [num_pages][Hkv][DAR_PAGE_SIZE][d_down] T.  The bottleneck
 *                 vectors k^D = k Dk, v^D = v Dv (Eq. 1) of a token at position
 *                 p that has left the window live in physical page
 *                 block_table[b][p / 64], row p % 64.
 *  block_table    [B][max_pages_per_seq] int32, caller-assigned; entries that
 *                 are needed must lie in [0, num_pages).
 *  seq_lens       [B] int32: tokens held per sequence.  dar_cache_append adds
 *                 to it; the caller zero-fills it for an empty cache.
 *  status         one int32 the kernels set to a dar_status on a device-side
 *                 error (0 = no error); the caller clears it.
 *
 * Requires w >= 1 (the current token is always local, Eq. 3 with i - j = 0).
 */
typedef struct dar_cache {
    dar_dtype dtype;
    int32_t B, Hkv, d, d_down, w;
    int32_t max_pages_per_seq;
    int32_t num_pages;
    void *win_k, *win_v;
    void *pool_kd, *pool_vd;
    int32_t *block_table;
    int32_t *seq_lens;
    int32_t *status;
} dar_cache;

/*
 * Eq. 1, the bottleneck h^D = h W_down, per KV head:
 *   out[b][g][j][c] = round_T( sum_t x[b][g][j][t] * W[g][t][c] )
 * where the sum is ONE fp32 fused-multiply-add chain over t = 0..d-1 starting
 * from +0.0f and the result is rounded once to T (nearest even).  The same
 * chain is used by dar_cache_append and inside dar_attn_prefill, so a token's
 * cached vector is bit-identical whichever call produced it.
 *   x [B][Hkv][n][d] T, W [Hkv][d][d_down] fp32, out [B][Hkv][n][d_down] T.
 */
dar_status dar_down_project(dar_dtype dtype, int32_t B, int32_t Hkv, int32_t n, int32_t d,
                            int32_t d_down, const void *x, const float *W, void *out,
                            void *stream);

/*
 * Append tokens to every sequence of the cache (inference, Sec. 2.3 and the
 * cache scheme of Sec. 5).  k_new, v_new [B][Hkv][n][d] T; sequence b appends
 * its first n_b tokens, n_b = n_per_seq[b] (a device int32[B] with
 * 0 <= n_b <= n) or n_b = n when n_per_seq is NULL.  They take positions
 * seq_lens[b] .. seq_lens[b]+n_b-1.  Every token that leaves the window (its
 * distance from the new last token reaches w) is down-projected with Dk / Dv
 * exactly as dar_down_project and written to its page; the others go to their
 * ring slot.  seq_lens[b] += n_b.  A needed block-table entry outside
 * [0, num_pages), or a length beyond max_pages_per_seq*64 + w, sets
 * *status = DAR_ERR_CAPACITY (an n_b outside [0, n] sets
 * DAR_ERR_INVALID_ARG) and skips that sequence.
 */
dar_status dar_cache_append(const dar_cache *cache, const void *k_new, const void *v_new,
                            int32_t n, const int32_t *n_per_seq, const float *Dk,
                            const float *Dv, void *stream);

/*
 * Bytes of workspace dar_attn_decode needs for this cache shape and Hq query
 * heads.  The workspace needs no initialisation: every call rewrites what it
 * reads.  Calls that share one workspace must not overlap on the device.
 */
size_t dar_decode_workspace_bytes(const dar_cache *cache, int32_t Hq);

/*
 * One decode step (Eq. 3-4 for the query at position i = L_b - 1 of each
 * sequence, L_b = seq_lens[b]): scores against the ring (full d) and the
 * pages (d_down, with W_up absorbed into the query, q~ = q Uk^T), one softmax
 * over both, values lifted once, o = (sum_local p v + (sum_global p v^D) Uv) / sum p.
 *   q [B][Hq][d] T; Uk, Uv [Hkv][d_down][d] fp32; out [B][Hq][d] T; q, out,
 *   Uk, Uv and the workspace 16-byte aligned.
 * A sequence with L_b == 0 gets a zero output.  Split-K over the sequence:
 * two kernels run in order on `stream` (q~ and zeroed counters; streaming,
 * whose warps merge the partial results of each (sequence, KV head) group);
 * the first starts only after all earlier work on the stream has finished.
 * B <= DAR_DECODE_MAX_BATCH and B * Hq * (stages of a full-capacity sequence)
 * < 2^31, else DAR_ERR_UNSUPPORTED.  A length beyond the cache's capacity
 * or a needed block-table entry outside [0, num_pages) sets
 * *status = DAR_ERR_CAPACITY; out is then undefined for that sequence.
 */
dar_status dar_attn_decode(const dar_cache *cache, int32_t Hq, const void *q, const float *Uk,
                           const float *Uv, float scale, void *out, void *workspace,
                           size_t workspace_bytes, void *stream);

/*
 * One serving step (Sec. 2.3 inference with the cache scheme of Sec. 5):
 * dar_cache_append(cache, k_new, v_new, n, n_per_seq, Dk, Dv) followed by
 * dar_attn_decode(cache, Hq, q, Uk, Uv, scale, out, workspace), with the same
 * arguments, requirements and results as those two calls made in turn.  All
 * arguments of both are checked before anything is launched.  The difference
 * is in the ordering on the device: dar_attn_decode alone starts only after
 * all earlier work on the stream has finished, while here the decode's
 * query-side set-up (q~ = q Uk^T) runs while the append is still working,
 * which is safe because the append writes neither q nor Uk.
 */
dar_status dar_decode_step(const dar_cache *cache, const void *k_new, const void *v_new, int32_t n,
                           const int32_t *n_per_seq, const float *Dk, const float *Dv, int32_t Hq,
                           const void *q, const float *Uk, const float *Uv, float scale, void *out,
                           void *workspace, size_t workspace_bytes, void *stream);

/*
 * dar_attn_decode for callers that cannot allocate device memory (the paper
 * has no counterpart; this is an interface convenience).  Some callers have
 * no device allocator to draw a workspace from (code embedded in a host
 * framework that exposes none), or must not allocate once serving has started.
 * This entry point allocates nothing: its scratch is one file-scope device
 * array of DAR_DECODE_NOALLOC_MAX_BYTES that every GPU which loads the library
 * holds until the process exits.  Arguments and results are those of
 * dar_attn_decode; the caller still provides q and out.
 *  - A cache shape whose dar_decode_workspace_bytes() exceeds the maximum is
 *    rejected with DAR_ERR_CAPACITY and nothing is launched.
 *  - The first call on a device looks up the array's device address (with
 *    that device current); make that first call before any stream capture.
 *  - The array needs no clearing (every call rewrites what it reads).  All
 *    calls share the one array, so calls that overlap on the device (other
 *    streams, other threads) race: serialise them.
 */
#define DAR_DECODE_NOALLOC_MAX_BYTES (8u << 20)
dar_status dar_attn_decode_noalloc(const dar_cache *cache, int32_t Hq, const void *q,
                                   const float *Uk, const float *Uv, float scale, void *out,
                                   void *stream);

/* Bytes of workspace dar_attn_prefill needs (the Eq. 1 vectors of all tokens). */
size_t dar_prefill_workspace_bytes(dar_dtype dtype, int32_t B, int32_t Hkv, int32_t N,
                                   int32_t d_down);

/*
 * Causal forward over positions 0..N-1 with no earlier context (the training
 * forward of Sec. 2.3: every token keeps both representations and each query
 * takes the one Eq. 3 selects).
 *   q [B][Hq][N][d], k, v [B][Hkv][N][d] T; Dk, Dv [Hkv][d][d_down] fp32;
 *   Uk, Uv [Hkv][d_down][d] fp32; out [B][Hq][N][d] T.
 * w >= 0; w = 0 is the paper's uniform reduction (no token is local).
 * The workspace (no initialisation needed) receives k^D, v^D; out must not
 * overlap q, k, v or the workspace.  `status` (a device int32,
 * may be NULL) is set to a dar_status if a kernel gives up on a bounded
 * internal wait; the caller clears it.  bf16 runs on the tcgen05 tensor
 * cores, fp32 on the CUDA cores (fp32 FMA, no TF32).
 */
dar_status dar_attn_prefill(dar_dtype dtype, int32_t B, int32_t Hq, int32_t Hkv, int32_t N,
                            int32_t d, int32_t d_down, int32_t w, const void *q, const void *k,
                            const void *v, const float *Dk, const float *Uk, const float *Dv,
                            const float *Uv, float scale, void *out, void *workspace,
                            size_t workspace_bytes, int32_t *status, void *stream);

/*
 * Diagnostic of the failure path every kernel shares (no counterpart in the
 * paper).  Launches one thread block that allocates tensor memory, starts one
 * bulk copy into shared memory and then waits on a barrier that nothing ever
 * completes, with a limit of limit_us microseconds instead of the usual 2 s.
 * When the limit runs out it does what any kernel of this library does when a
 * wait gives up: writes DAR_ERR_DEVICE to *status (a device int32, first error
 * wins), waits for its own copy to land, releases its tensor memory and exits.
 * The device stays usable.  limit_us must lie in [1, 2000000].
 */
dar_status dar_check_bounded_wait(int32_t *status, uint32_t limit_us, void *stream);

/*
 * Chunked prefill over an existing cache (Sec. 2.3 inference with the cache
 * scheme of Sec. 5: a long prompt enters the cache in chunks).  Every sequence
 * b holds L_b = seq_lens[b] tokens and takes n more: k_new, v_new
 * [B][Hkv][n][d] at positions L_b .. L_b + n - 1, with queries q [B][Hq][n][d].
 * out[b][h][r] (same layout as q) is row L_b + r of the causal forward over
 * the whole sequence (Eq. 3-4: local keys i - j < w at full d, the others
 * through the bottleneck), i.e. what dar_attn_prefill would give for those
 * rows over the concatenated sequence.  The call then appends the chunk
 * exactly as dar_cache_append(cache, k_new, v_new, n, NULL, Dk, Dv) does
 * (the cache bytes equal n one-token appends).
 *   bf16 caches with d_down in {16, 32, 64}; Dk, Dv [Hkv][d][d_down] and
 *   Uk, Uv [Hkv][d_down][d] fp32; all pointers 16-byte aligned; workspace of
 *   dar_prefill_chunk_workspace_bytes(cache, n) bytes (no initialisation).
 * Three kernels run in order on `stream`: a gather of the keys the chunk's
 * queries can see (window rows, and bottleneck rows of the tokens the chunk
 * pushes out of the window), the attention, and the append.  A needed
 * block-table entry outside [0, num_pages) or a length beyond the cache's
 * capacity sets *status = DAR_ERR_CAPACITY.
 */
size_t dar_prefill_chunk_workspace_bytes(const dar_cache *cache, int32_t n);
dar_status dar_prefill_chunk(const dar_cache *cache, int32_t Hq, int32_t n, const void *q,
                             const void *k_new, const void *v_new, const float *Dk, const float *Uk,
                             const float *Dv, const float *Uv, float scale, void *out, void *workspace,
                             size_t workspace_bytes, void *stream);

/*
 * Direct lower-dimensional global attention (Sec. 5, "Direct lower-dimensional
 * global attention": the global path runs entirely in d_down instead of
 * lifting h^D back to d).  Local pairs (i - j < w, Eq. 3) are unchanged:
 * scale * q . k_j with full-d keys and values.  Global pairs score
 * scale_down * q^D . k^D_j, where q^D is a d_down query of the row's own
 * (qd) and k^D = k Dk is the cached bottleneck key (Eq. 1); their values
 * v^D_j = v Dv enter as v^D_j Wo, Wo [Hkv][d_down][d] the global path's
 * output map to d.  One softmax covers both paths (Eq. 4 carried over):
 *   o_i = (sum_local p_j v_j + (sum_global p_j v^D_j) Wo) / sum_j p_j.
 * scale_down <= 0 selects 1/sqrt(d_down).  The global path computes
 * scale * (qd * scale_down / scale) . k^D, so on the bf16 tensor-core paths
 * the rescaled qd is rounded to bf16 once, as q~ is in the standard form.
 */

/* As dar_attn_prefill with the direct global path: qd [B][Hq][N][d_down] T,
 * Wo in place of Uv; no Uk.  Same workspace (dar_prefill_workspace_bytes),
 * status and error behaviour. */
dar_status dar_attn_prefill_direct(dar_dtype dtype, int32_t B, int32_t Hq, int32_t Hkv, int32_t N,
                                   int32_t d, int32_t d_down, int32_t w, const void *q, const void *qd,
                                   const void *k, const void *v, const float *Dk, const float *Dv,
                                   const float *Wo, float scale, float scale_down, void *out,
                                   void *workspace, size_t workspace_bytes, int32_t *status,
                                   void *stream);

/* As dar_attn_decode with the direct global path: qd [B][Hq][d_down] T (16-byte
 * aligned), Wo in place of Uv; no Uk.  Same cache (the pages hold k^D, v^D of
 * Eq. 1, written by dar_cache_append), workspace (dar_decode_workspace_bytes)
 * and error behaviour; both kernels start after all earlier work on the
 * stream has finished. */
dar_status dar_attn_decode_direct(const dar_cache *cache, int32_t Hq, const void *q, const void *qd,
                                  const float *Wo, float scale, float scale_down, void *out,
                                  void *workspace, size_t workspace_bytes, void *stream);

/*
 * Gradients of the causal forward of dar_attn_prefill (training, Sec. 2.3:
 * the standard next-token objective; backpropagation updates W_down and W_up
 * from the positions whose queries reach a token through the global path).
 * Given the forward's inputs, its output `out` and the loss gradient `dout`
 * [B][Hq][N][d] T, writes
 *   dq [B][Hq][N][d], dk, dv [B][Hkv][N][d] (T),
 *   dDk, dDv [Hkv][d][d_down], dUk, dUv [Hkv][d_down][d] (fp32),
 * each overwritten (not accumulated).  The derivative is that of Eq. 1-4 with
 * the stored k^D, v^D's rounding to T not differentiated (the bottleneck
 * projections get the gradient of the unrounded product), and D_i = dout_i .
 * out_i taken from the given forward output.  bf16 storage runs the score,
 * dP and gradient contractions on the tensor cores (bf16 operands, P and dS
 * rounded to bf16, fp32 accumulation; d_down = 8 stays on the CUDA cores);
 * fp32 storage runs fp32 arithmetic on the CUDA cores.  The workspace
 * (dar_attn_backward_workspace_bytes, no initialisation) holds per-row and
 * per-token intermediates; outputs must not overlap inputs.  Deterministic:
 * every sum runs in a fixed order.  Shapes as dar_attn_prefill; B*Hq <= 65535.
 */
size_t dar_attn_backward_workspace_bytes(dar_dtype dtype, int32_t B, int32_t Hq, int32_t Hkv,
                                         int32_t N, int32_t d_down);
dar_status dar_attn_backward(dar_dtype dtype, int32_t B, int32_t Hq, int32_t Hkv, int32_t N, int32_t d,
                             int32_t d_down, int32_t w, const void *q, const void *k, const void *v,
                             const float *Dk, const float *Uk, const float *Dv, const float *Uv,
                             const void *out, const void *dout, float scale, void *dq, void *dk, void *dv,
                             float *dDk, float *dUk, float *dDv, float *dUv, void *workspace,
                             size_t workspace_bytes, void *stream);

/*
 * The latent form (the paper's own Eq. 1-3 on hidden states, with the cache
 * scheme of Sec. 5 "Compute and memory efficiency"): every token keeps ONE
 * bottleneck c_j = h_j W_down (Eq. 1, h_j the layer's hidden state of width D),
 * shared by every head and by keys and values; the last w tokens also keep
 * their full per-KV-head keys and values.  A distant token reaches head g as
 * k'_j = (c_j W_up) W_K^g, v'_j = (c_j W_up) W_V^g (Eq. 2-3); with W_up
 * absorbed (A_K^g = W_up W_K^g, A_V^g = W_up W_V^g) the decode scores
 * q . k'_j = (q A_K^gT) . c_j and lifts the weighted sum of the c_j once with
 * A_V^g.  Cache memory is O(T d_lat + w d) for all heads together.
 * Positions are already encoded (no RoPE in the library).  bf16 only;
 * d = 64; d_lat in {64, 128, 192, 256}; Hq <= 32; D <= 8192.
 *
 *  win_k, win_v  [B][Hkv][w][d] bf16, ring slot p % w (as dar_cache)
 *  pool_c        [num_pages][DAR_PAGE_SIZE][d_lat] bf16: c of the token at
 *                position p in page block_table[b][p / 64], row p % 64 --
 *                for EVERY position (window tokens too), so nothing migrates
 *  block_table   [B][max_pages_per_seq] int32; seq_lens [B]; status as dar_cache.
 * Capacity: max_pages_per_seq * 64 tokens per sequence.
 */
typedef struct dar_latent_cache {
    int32_t B, Hkv, d, D, d_lat, w;
    int32_t max_pages_per_seq;
    int32_t num_pages;
    void *win_k, *win_v;
    void *pool_c;
    int32_t *block_table;
    int32_t *seq_lens;
    int32_t *status;
} dar_latent_cache;

/* Append n tokens per sequence (n_b = n_per_seq[b] when given, a device
 * int32[B] with 0 <= n_b <= n): h_new [B][n][D] bf16 their hidden states,
 * k_new, v_new [B][Hkv][n][d] bf16 their keys and values, W_down [D][d_lat]
 * fp32.  Writes c = round_bf16(fp32 FMA chain over e = 0..D-1 of
 * h[e] W_down[e][c], from +0) into each new token's page row (Eq. 1, the same
 * chain order as dar_down_project), ring rows for the tokens that remain in
 * the window, then seq_lens[b] += n_b.  A length beyond capacity or a needed
 * block-table entry outside [0, num_pages) sets *status = DAR_ERR_CAPACITY. */
dar_status dar_latent_append(const dar_latent_cache *cache, const void *h_new, const void *k_new,
                             const void *v_new, int32_t n, const int32_t *n_per_seq,
                             const float *W_down, void *stream);

/* The absorbed maps of Sec. 5: A_K[g] = W_up W_K[g], A_V[g] = W_up W_V[g]
 * (fp32 FMA chains over D).  W_up [d_lat][D], W_K, W_V [Hkv][D][d] fp32.
 * Written: A_K [Hkv][d][d_lat] (stored transposed: element (c, t) of
 * W_up W_K[g] at A_K[g][t][c]) and A_V [Hkv][d_lat][d], both fp32. */
dar_status dar_latent_absorb(int32_t Hkv, int32_t D, int32_t d, int32_t d_lat, const float *W_up,
                             const float *W_K, const float *W_V, float *A_K, float *A_V, void *stream);

/* One decode step of the latent form for the query at position L_b - 1:
 * q [B][Hq][d] bf16, A_K [Hkv][d][d_lat], A_V [Hkv][d_lat][d] fp32 (as
 * dar_latent_absorb writes them),
 * out [B][Hq][d] bf16.  Local keys (the last min(L_b, w) tokens) at full d,
 * distant ones through c, one softmax over both (Eq. 3-4).  Three kernels in
 * order on `stream` (q~ = q A_K^T; split-K over pages of the latent pool and
 * the window; merge and lift).  Workspace of
 * dar_latent_decode_workspace_bytes(cache, Hq) bytes, no initialisation.
 * L_b == 0 gives a zero output.  B <= DAR_DECODE_MAX_BATCH. */
size_t dar_latent_decode_workspace_bytes(const dar_latent_cache *cache, int32_t Hq);
dar_status dar_latent_decode(const dar_latent_cache *cache, int32_t Hq, const void *q, const float *A_K,
                             const float *A_V, float scale, void *out, void *workspace,
                             size_t workspace_bytes, void *stream);

/* Message for the last non-OK return on this thread ("" if none). */
const char *dar_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* DAR_H */
