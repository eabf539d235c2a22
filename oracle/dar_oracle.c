/*
 * dar_oracle.c -- plain, slow CPU oracle for Distance-Adaptive Representation
 * (DAR) attention.  TEST INFRASTRUCTURE ONLY: the tests, the smoke check and
 * the benchmark's CPU-baseline leg call it; the product path never does.
 *
 * It shares no code with the CUDA path.  It follows the method section of
 * "Dual Dimensionality for Local and Global Attention" step by step:
 *
 *   Eq. 1  h^D_j = h_j W_down                (down-projection, per KV head here)
 *   Eq. 2  h'_j  = h^D_j W_up                (lift back to d, done explicitly)
 *   Eq. 3  k_j, v_j = full if i - j < w, lifted otherwise
 *   Eq. 4  o_i = softmax(q_i K_i^T / sqrt(d_k)) V_i   (one softmax over all j <= i)
 *
 * Readings of the paper that this file encodes:
 *   - the projections act per KV head on that head's key/value vectors
 *     (W_down = Dk or Dv, W_up = Uk or Uv), with separate matrices for K and V;
 *   - the query/key inputs are already position-encoded (no RoPE here);
 *   - "local" means i - j < w, so the window holds the current token and the
 *     w - 1 before it; w = 0 makes every token, the current one included,
 *     global (the paper's uniform-reduction baseline, Table 3 row w = 0);
 *   - the down-projected vectors are stored in the storage type T: each output
 *     element is an fp32 fused-multiply-add chain over t = 0..d-1 starting
 *     from +0.0f, rounded once to T with round-to-nearest-even;
 *   - everything after the down-projection is evaluated in fp64;
 *   - GQA: query head h reads KV head g = h / (Hq / Hkv).
 *
 * Parity pins for every function here live in tests/test_oracle_pins.py.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

enum { ORC_F32 = 0, ORC_BF16 = 1 };

/* ---- storage-type helpers ------------------------------------------------ */

static float bf16_bits_to_f32(uint16_t h)
{
    uint32_t u = (uint32_t)h << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return f;
}

/* fp32 -> bf16 bits, round to nearest, ties to even.  NaN stays NaN. */
static uint16_t f32_to_bf16_bits(float f)
{
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    if ((u & 0x7f800000u) == 0x7f800000u && (u & 0x007fffffu) != 0u)
        return (uint16_t)((u >> 16) | 0x0040u);
    uint32_t keep_lsb = (u >> 16) & 1u;
    u += 0x7fffu + keep_lsb;
    return (uint16_t)(u >> 16);
}

static float load_as_f32(const void *p, int dtype, size_t idx)
{
    if (dtype == ORC_F32)
        return ((const float *)p)[idx];
    return bf16_bits_to_f32(((const uint16_t *)p)[idx]);
}

static void store_from_f32(void *p, int dtype, size_t idx, float v)
{
    if (dtype == ORC_F32)
        ((float *)p)[idx] = v;
    else
        ((uint16_t *)p)[idx] = f32_to_bf16_bits(v);
}

/* ---- Eq. 1: down-projection ---------------------------------------------
 * x   [B][Hkv][n][d]   storage type
 * Dw  [Hkv][d][dd]     fp32   (W_down of each KV head)
 * out [B][Hkv][n][dd]  storage type
 * out[b][g][j][c] = round_T( fmaf-chain_{t=0..d-1} x[b][g][j][t] * Dw[g][t][c] )
 */
void dar_oracle_down_project(int dtype, int B, int Hkv, int n, int d, int dd,
                             const void *x, const float *Dw, void *out)
{
    for (int b = 0; b < B; ++b)
        for (int g = 0; g < Hkv; ++g)
            for (int j = 0; j < n; ++j) {
                size_t row = (((size_t)b * Hkv + g) * n + j);
                for (int c = 0; c < dd; ++c) {
                    float acc = 0.0f;
                    for (int t = 0; t < d; ++t) {
                        float xv = load_as_f32(x, dtype, row * d + t);
                        float wv = Dw[((size_t)g * d + t) * dd + c];
                        acc = fmaf(xv, wv, acc);
                    }
                    store_from_f32(out, dtype, row * dd + c, acc);
                }
            }
}

/* Round an fp32 array to bf16 bits (RNE); used by tests to build inputs. */
void dar_oracle_f32_to_bf16(const float *in, uint16_t *out, size_t n)
{
    for (size_t i = 0; i < n; ++i)
        out[i] = f32_to_bf16_bits(in[i]);
}

/* ---- Eq. 2-4: attention over the two representations --------------------- */

typedef struct {
    int dtype, B, Hq, Hkv, N, d, dd, w;
    const void *q;   /* [nrows][d]      storage type, one per row    */
    const void *k;   /* [B][Hkv][N][d]  storage type                  */
    const void *v;   /* [B][Hkv][N][d]  storage type                  */
    const void *kd;  /* [B][Hkv][N][dd] storage type (Eq. 1 output)   */
    const void *vd;  /* [B][Hkv][N][dd] storage type                  */
    const float *Uk; /* [Hkv][dd][d] fp32  (W_up for keys)            */
    const float *Uv; /* [Hkv][dd][d] fp32  (W_up for values)          */
    double scale;    /* 1/sqrt(d_k)                                   */
    long nrows;
    const int *row_b, *row_h, *row_i; /* query rows to evaluate       */
    double *out;     /* [nrows][d]                                    */
    int nthreads;
    int tid;
} attn_job;

/* One (b, g) unit: lift every needed token (Eq. 2), then evaluate each
 * requested query row of this unit with Eq. 3 selection and Eq. 4. */
static void attn_unit(const attn_job *J, int b, int g)
{
    const int d = J->d, dd = J->dd, N = J->N, G = J->Hq / J->Hkv;
    int jmax = -1;
    for (long r = 0; r < J->nrows; ++r)
        if (J->row_b[r] == b && J->row_h[r] / G == g && J->row_i[r] > jmax)
            jmax = J->row_i[r];
    if (jmax < 0)
        return;
    const int n = jmax + 1;

    double *Kfull = malloc(sizeof(double) * (size_t)n * d);
    double *Vfull = malloc(sizeof(double) * (size_t)n * d);
    double *Klift = malloc(sizeof(double) * (size_t)n * d);
    double *Vlift = malloc(sizeof(double) * (size_t)n * d);
    double *s = malloc(sizeof(double) * (size_t)n);
    const size_t base = ((size_t)b * J->Hkv + g) * N;

    for (int j = 0; j < n; ++j) {
        for (int t = 0; t < d; ++t) {
            Kfull[(size_t)j * d + t] = load_as_f32(J->k, J->dtype, (base + j) * d + t);
            Vfull[(size_t)j * d + t] = load_as_f32(J->v, J->dtype, (base + j) * d + t);
        }
        /* Eq. 2: h'_j = h^D_j W_up, explicitly, in fp64. */
        for (int t = 0; t < d; ++t) {
            double ka = 0.0, va = 0.0;
            for (int c = 0; c < dd; ++c) {
                double kdc = load_as_f32(J->kd, J->dtype, (base + j) * dd + c);
                double vdc = load_as_f32(J->vd, J->dtype, (base + j) * dd + c);
                ka += kdc * (double)J->Uk[((size_t)g * dd + c) * d + t];
                va += vdc * (double)J->Uv[((size_t)g * dd + c) * d + t];
            }
            Klift[(size_t)j * d + t] = ka;
            Vlift[(size_t)j * d + t] = va;
        }
    }

    for (long r = 0; r < J->nrows; ++r) {
        if (J->row_b[r] != b || J->row_h[r] / G != g)
            continue;
        const int i = J->row_i[r];
        const size_t qrow = (size_t)r * d;
        double *o = J->out + (size_t)r * d;

        /* Eq. 3 + Eq. 4: scores over j = 0..i, with the key chosen by distance. */
        double smax = -INFINITY;
        for (int j = 0; j <= i; ++j) {
            const double *key = (i - j < J->w) ? &Kfull[(size_t)j * d] : &Klift[(size_t)j * d];
            double dot = 0.0;
            for (int t = 0; t < d; ++t)
                dot += (double)load_as_f32(J->q, J->dtype, qrow + t) * key[t];
            s[j] = J->scale * dot;
            if (s[j] > smax)
                smax = s[j];
        }
        double denom = 0.0;
        for (int j = 0; j <= i; ++j)
            denom += exp(s[j] - smax);
        for (int t = 0; t < d; ++t)
            o[t] = 0.0;
        for (int j = 0; j <= i; ++j) {
            const double p = exp(s[j] - smax) / denom;
            const double *val = (i - j < J->w) ? &Vfull[(size_t)j * d] : &Vlift[(size_t)j * d];
            for (int t = 0; t < d; ++t)
                o[t] += p * val[t];
        }
    }
    free(Kfull);
    free(Vfull);
    free(Klift);
    free(Vlift);
    free(s);
}

static void *attn_worker(void *arg)
{
    const attn_job *J = (const attn_job *)arg;
    const int units = J->B * J->Hkv;
    for (int u = J->tid; u < units; u += J->nthreads)
        attn_unit(J, u / J->Hkv, u % J->Hkv);
    return NULL;
}

/*
 * Evaluate the DAR attention output for an explicit list of query rows.
 * Row r is the query vector q[r] of head row_h[r] of sequence row_b[r] at
 * position row_i[r]; it attends to positions 0..row_i[r] of that sequence.  Prefill asks for
 * every (b, h, i); a decode step asks for i = L_b - 1.  Returns 0, or -1 on a
 * bad argument.  Threads run over (b, g) units.
 */
int dar_oracle_attention(int dtype, int B, int Hq, int Hkv, int N, int d, int dd, int w,
                         const void *q, const void *k, const void *v,
                         const void *kd, const void *vd,
                         const float *Uk, const float *Uv, double scale,
                         long nrows, const int *row_b, const int *row_h, const int *row_i,
                         double *out, int nthreads)
{
    if (B < 1 || Hkv < 1 || Hq < Hkv || Hq % Hkv || N < 1 || d < 1 || dd < 1 || w < 0 ||
        nrows < 0 || (dtype != ORC_F32 && dtype != ORC_BF16))
        return -1;
    for (long r = 0; r < nrows; ++r)
        if (row_b[r] < 0 || row_b[r] >= B || row_h[r] < 0 || row_h[r] >= Hq ||
            row_i[r] < 0 || row_i[r] >= N)
            return -1;
    if (nthreads < 1)
        nthreads = 1;
    attn_job *jobs = malloc(sizeof(attn_job) * (size_t)nthreads);
    pthread_t *th = malloc(sizeof(pthread_t) * (size_t)nthreads);
    for (int t = 0; t < nthreads; ++t) {
        attn_job J = {dtype, B, Hq, Hkv, N, d, dd, w, q, k, v, kd, vd, Uk, Uv, scale,
                      nrows, row_b, row_h, row_i, out, nthreads, t};
        jobs[t] = J;
    }
    for (int t = 1; t < nthreads; ++t)
        pthread_create(&th[t], NULL, attn_worker, &jobs[t]);
    attn_worker(&jobs[0]);
    for (int t = 1; t < nthreads; ++t)
        pthread_join(th[t], NULL);
    free(jobs);
    free(th);
    return 0;
}

/* ---- Sec. 5, "Direct lower-dimensional global attention" ------------------
 * The global path runs in d_down: a query q^D_i of its own (d_down), scored
 * against the d_down keys k^D_j of the distant tokens with scale_down
 * (1/sqrt(d_down) by default), and the weighted d_down values mapped to d by
 * an output map Wo (d_down x d, per KV head).  The local path is unchanged
 * (Eq. 3 selection, scale 1/sqrt(d)), and one softmax covers both paths
 * (Eq. 4 carried over).  Per token the mapped value v^D_j Wo is formed
 * explicitly, in fp64, before the weighted sum. */

typedef struct {
    attn_job base;      /* k, v, kd, vd, q (local query), rows, out, threads */
    const void *qd;     /* [nrows][dd] storage type: the d_down query of each row */
    const float *Wo;    /* [Hkv][dd][d] fp32 */
    double scale_down;
} attn_direct_job;

static void attn_unit_direct(const attn_direct_job *D, int b, int g)
{
    const attn_job *J = &D->base;
    const int d = J->d, dd = J->dd, N = J->N, G = J->Hq / J->Hkv;
    int jmax = -1;
    for (long r = 0; r < J->nrows; ++r)
        if (J->row_b[r] == b && J->row_h[r] / G == g && J->row_i[r] > jmax)
            jmax = J->row_i[r];
    if (jmax < 0)
        return;
    const int n = jmax + 1;

    double *Kfull = malloc(sizeof(double) * (size_t)n * d);
    double *Vfull = malloc(sizeof(double) * (size_t)n * d);
    double *Kdown = malloc(sizeof(double) * (size_t)n * dd);
    double *Vmap = malloc(sizeof(double) * (size_t)n * d);
    double *s = malloc(sizeof(double) * (size_t)n);
    const size_t base = ((size_t)b * J->Hkv + g) * N;

    for (int j = 0; j < n; ++j) {
        for (int t = 0; t < d; ++t) {
            Kfull[(size_t)j * d + t] = load_as_f32(J->k, J->dtype, (base + j) * d + t);
            Vfull[(size_t)j * d + t] = load_as_f32(J->v, J->dtype, (base + j) * d + t);
        }
        for (int c = 0; c < dd; ++c)
            Kdown[(size_t)j * dd + c] = load_as_f32(J->kd, J->dtype, (base + j) * dd + c);
        for (int t = 0; t < d; ++t) {
            double va = 0.0;
            for (int c = 0; c < dd; ++c)
                va += (double)load_as_f32(J->vd, J->dtype, (base + j) * dd + c) *
                      (double)D->Wo[((size_t)g * dd + c) * d + t];
            Vmap[(size_t)j * d + t] = va;
        }
    }

    for (long r = 0; r < J->nrows; ++r) {
        if (J->row_b[r] != b || J->row_h[r] / G != g)
            continue;
        const int i = J->row_i[r];
        double *o = J->out + (size_t)r * d;
        double smax = -INFINITY;
        for (int j = 0; j <= i; ++j) {
            double dot = 0.0;
            if (i - j < J->w) {
                for (int t = 0; t < d; ++t)
                    dot += (double)load_as_f32(J->q, J->dtype, (size_t)r * d + t) * Kfull[(size_t)j * d + t];
                s[j] = J->scale * dot;
            } else {
                for (int c = 0; c < dd; ++c)
                    dot += (double)load_as_f32(D->qd, J->dtype, (size_t)r * dd + c) * Kdown[(size_t)j * dd + c];
                s[j] = D->scale_down * dot;
            }
            if (s[j] > smax)
                smax = s[j];
        }
        double denom = 0.0;
        for (int j = 0; j <= i; ++j)
            denom += exp(s[j] - smax);
        for (int t = 0; t < d; ++t)
            o[t] = 0.0;
        for (int j = 0; j <= i; ++j) {
            const double p = exp(s[j] - smax) / denom;
            const double *val = (i - j < J->w) ? &Vfull[(size_t)j * d] : &Vmap[(size_t)j * d];
            for (int t = 0; t < d; ++t)
                o[t] += p * val[t];
        }
    }
    free(Kfull);
    free(Vfull);
    free(Kdown);
    free(Vmap);
    free(s);
}

static void *attn_direct_worker(void *arg)
{
    const attn_direct_job *D = (const attn_direct_job *)arg;
    const int units = D->base.B * D->base.Hkv;
    for (int u = D->base.tid; u < units; u += D->base.nthreads)
        attn_unit_direct(D, u / D->base.Hkv, u % D->base.Hkv);
    return NULL;
}

/* As dar_oracle_attention, with the global path of Sec. 5's direct variant:
 * qd [nrows][dd] the d_down query of each row, Wo [Hkv][dd][d] the output map
 * of the global path, scale_down the global scores' scale. */
int dar_oracle_attention_direct(int dtype, int B, int Hq, int Hkv, int N, int d, int dd, int w,
                                const void *q, const void *qd, const void *k, const void *v,
                                const void *kd, const void *vd, const float *Wo, double scale,
                                double scale_down, long nrows, const int *row_b, const int *row_h,
                                const int *row_i, double *out, int nthreads)
{
    if (B < 1 || Hkv < 1 || Hq < Hkv || Hq % Hkv || N < 1 || d < 1 || dd < 1 || w < 0 ||
        nrows < 0 || (dtype != ORC_F32 && dtype != ORC_BF16))
        return -1;
    for (long r = 0; r < nrows; ++r)
        if (row_b[r] < 0 || row_b[r] >= B || row_h[r] < 0 || row_h[r] >= Hq ||
            row_i[r] < 0 || row_i[r] >= N)
            return -1;
    if (nthreads < 1)
        nthreads = 1;
    attn_direct_job *jobs = malloc(sizeof(attn_direct_job) * (size_t)nthreads);
    pthread_t *th = malloc(sizeof(pthread_t) * (size_t)nthreads);
    for (int t = 0; t < nthreads; ++t) {
        attn_job J = {dtype, B, Hq, Hkv, N, d, dd, w, q, k, v, kd, vd, NULL, NULL, scale,
                      nrows, row_b, row_h, row_i, out, nthreads, t};
        jobs[t].base = J;
        jobs[t].qd = qd;
        jobs[t].Wo = Wo;
        jobs[t].scale_down = scale_down;
    }
    for (int t = 1; t < nthreads; ++t)
        pthread_create(&th[t], NULL, attn_direct_worker, &jobs[t]);
    attn_direct_worker(&jobs[0]);
    for (int t = 1; t < nthreads; ++t)
        pthread_join(th[t], NULL);
    free(jobs);
    free(th);
    return 0;
}
