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

/* ---- Sec. 2.3, training: gradients of the DAR attention forward -----------
 * The loss is any scalar whose gradient with respect to the outputs o_i is
 * dO_i (given).  Backpropagation runs through the forward's steps in reverse,
 * each written out as its plain derivative, in fp64:
 *
 *   Eq. 4   o_i = sum_j p_ij val_j,  p_i = softmax_j(s_ij),  s_ij = scale q_i . key_j
 *           dP_ij = dO_i . val_j;  dS_ij = p_ij (dP_ij - sum_l p_il dP_il)
 *           dq_i = scale sum_j dS_ij key_j;  dkey_j += scale dS_ij q_i;  dval_j += p_ij dO_i
 *   Eq. 3   key_j / val_j is the full k_j / v_j (i - j < w) or the lifted k'_j / v'_j,
 *           so each (i, j) pair sends its gradient to exactly one of the two
 *   Eq. 2   k'_j = k^D_j Uk:  dk^D_j = dk'_j Uk^T,  dUk += (k^D_j)^T dk'_j   (same for v, Uv)
 *   Eq. 1   k^D_j = k_j Dk:   dk_j += dk^D_j Dk^T,  dDk += k_j^T dk^D_j      (same for v, Dv)
 *
 * The forward stores k^D rounded to the storage type; its derivative is taken
 * as that of the unrounded product (the rounding is not differentiated), so the
 * bottleneck projections receive the gradient of every position that reaches
 * a token through the global path, as Sec. 2.3 describes.  GQA: the gradients
 * of a KV head sum over the query heads that read it. */

typedef struct {
    int dtype, B, Hq, Hkv, N, d, dd, w;
    const void *q, *k, *v, *dout;             /* storage type */
    const float *Dk, *Uk, *Dv, *Uv;           /* fp32 */
    double scale;
    double *dq, *dk, *dv;                     /* [B][Hq|Hkv][N][d] */
    double *wpart;                            /* [B][Hkv][4][d * dd]: dDk, dUk, dDv, dUv of one unit */
    int nthreads, tid;
} bwd_job;

static void bwd_unit(const bwd_job *J, int b, int g)
{
    const int d = J->d, dd = J->dd, N = J->N, G = J->Hq / J->Hkv, w = J->w;
    const size_t base = ((size_t)b * J->Hkv + g) * N;
    const float *Dk = J->Dk + (size_t)g * d * dd, *Dv = J->Dv + (size_t)g * d * dd;
    const float *Uk = J->Uk + (size_t)g * dd * d, *Uv = J->Uv + (size_t)g * dd * d;
    double *K = malloc(sizeof(double) * (size_t)N * d), *V = malloc(sizeof(double) * (size_t)N * d);
    double *KD = malloc(sizeof(double) * (size_t)N * dd), *VD = malloc(sizeof(double) * (size_t)N * dd);
    double *Kl = malloc(sizeof(double) * (size_t)N * d), *Vl = malloc(sizeof(double) * (size_t)N * d);
    double *dKl = calloc((size_t)N * d, sizeof(double)), *dVl = calloc((size_t)N * d, sizeof(double));
    double *p = malloc(sizeof(double) * (size_t)N), *dp = malloc(sizeof(double) * (size_t)N);
    double *Q = malloc(sizeof(double) * (size_t)d), *dO = malloc(sizeof(double) * (size_t)d);
    double *dk = J->dk + base * d, *dv = J->dv + base * d;
    double *wp = J->wpart + ((size_t)b * J->Hkv + g) * 4 * (size_t)d * dd;
    double *dDk = wp, *dUk = wp + (size_t)d * dd, *dDv = wp + 2 * (size_t)d * dd, *dUv = wp + 3 * (size_t)d * dd;

    /* forward quantities: Eq. 1 (stored, rounded to T) and Eq. 2 (explicit lift) */
    for (int j = 0; j < N; ++j) {
        for (int t = 0; t < d; ++t) {
            K[(size_t)j * d + t] = load_as_f32(J->k, J->dtype, (base + j) * d + t);
            V[(size_t)j * d + t] = load_as_f32(J->v, J->dtype, (base + j) * d + t);
        }
        for (int c = 0; c < dd; ++c) {
            float ka = 0.0f, va = 0.0f;
            for (int t = 0; t < d; ++t) {
                ka = fmaf(load_as_f32(J->k, J->dtype, (base + j) * d + t), Dk[(size_t)t * dd + c], ka);
                va = fmaf(load_as_f32(J->v, J->dtype, (base + j) * d + t), Dv[(size_t)t * dd + c], va);
            }
            /* stored in the storage type, as the forward reads them */
            KD[(size_t)j * dd + c] = J->dtype == ORC_BF16 ? bf16_bits_to_f32(f32_to_bf16_bits(ka)) : ka;
            VD[(size_t)j * dd + c] = J->dtype == ORC_BF16 ? bf16_bits_to_f32(f32_to_bf16_bits(va)) : va;
        }
        for (int t = 0; t < d; ++t) {
            double ka = 0.0, va = 0.0;
            for (int c = 0; c < dd; ++c) {
                ka += KD[(size_t)j * dd + c] * (double)Uk[(size_t)c * d + t];
                va += VD[(size_t)j * dd + c] * (double)Uv[(size_t)c * d + t];
            }
            Kl[(size_t)j * d + t] = ka;
            Vl[(size_t)j * d + t] = va;
        }
    }
    memset(dk, 0, sizeof(double) * (size_t)N * d);
    memset(dv, 0, sizeof(double) * (size_t)N * d);

    /* Eq. 4 and Eq. 3 backwards, one query row at a time */
    for (int hh = 0; hh < G; ++hh) {
        const int h = g * G + hh;
        const size_t qbase = ((size_t)b * J->Hq + h) * N;
        for (int i = 0; i < N; ++i) {
            for (int t = 0; t < d; ++t) {
                Q[t] = load_as_f32(J->q, J->dtype, (qbase + i) * d + t);
                dO[t] = load_as_f32(J->dout, J->dtype, (qbase + i) * d + t);
            }
            double smax = -INFINITY;
            for (int j = 0; j <= i; ++j) {
                const double *key = (i - j < w) ? &K[(size_t)j * d] : &Kl[(size_t)j * d];
                double dot = 0.0;
                for (int t = 0; t < d; ++t)
                    dot += Q[t] * key[t];
                p[j] = J->scale * dot;
                if (p[j] > smax)
                    smax = p[j];
            }
            double denom = 0.0;
            for (int j = 0; j <= i; ++j) {
                p[j] = exp(p[j] - smax);
                denom += p[j];
            }
            double Di = 0.0;  /* sum_l p_il dP_il */
            for (int j = 0; j <= i; ++j) {
                p[j] /= denom;
                const double *val = (i - j < w) ? &V[(size_t)j * d] : &Vl[(size_t)j * d];
                double dot = 0.0;
                for (int t = 0; t < d; ++t)
                    dot += dO[t] * val[t];
                dp[j] = dot;
                Di += p[j] * dot;
            }
            double *dqi = J->dq + (qbase + i) * d;
            for (int t = 0; t < d; ++t)
                dqi[t] = 0.0;
            for (int j = 0; j <= i; ++j) {
                const int loc = i - j < w;
                const double ds = p[j] * (dp[j] - Di);
                const double *key = loc ? &K[(size_t)j * d] : &Kl[(size_t)j * d];
                double *dkey = loc ? &dk[(size_t)j * d] : &dKl[(size_t)j * d];
                double *dval = loc ? &dv[(size_t)j * d] : &dVl[(size_t)j * d];
                for (int t = 0; t < d; ++t) {
                    dqi[t] += J->scale * ds * key[t];
                    dkey[t] += J->scale * ds * Q[t];
                    dval[t] += p[j] * dO[t];
                }
            }
        }
    }

    /* Eq. 2 and Eq. 1 backwards, per token */
    memset(wp, 0, sizeof(double) * 4 * (size_t)d * dd);
    double *dkd = malloc(sizeof(double) * (size_t)dd), *dvd = malloc(sizeof(double) * (size_t)dd);
    for (int j = 0; j < N; ++j) {
        for (int c = 0; c < dd; ++c) {
            double a = 0.0, e = 0.0;
            for (int t = 0; t < d; ++t) {
                a += dKl[(size_t)j * d + t] * (double)Uk[(size_t)c * d + t];
                e += dVl[(size_t)j * d + t] * (double)Uv[(size_t)c * d + t];
                dUk[(size_t)c * d + t] += KD[(size_t)j * dd + c] * dKl[(size_t)j * d + t];
                dUv[(size_t)c * d + t] += VD[(size_t)j * dd + c] * dVl[(size_t)j * d + t];
            }
            dkd[c] = a;
            dvd[c] = e;
        }
        for (int t = 0; t < d; ++t)
            for (int c = 0; c < dd; ++c) {
                dk[(size_t)j * d + t] += dkd[c] * (double)Dk[(size_t)t * dd + c];
                dv[(size_t)j * d + t] += dvd[c] * (double)Dv[(size_t)t * dd + c];
                dDk[(size_t)t * dd + c] += K[(size_t)j * d + t] * dkd[c];
                dDv[(size_t)t * dd + c] += V[(size_t)j * d + t] * dvd[c];
            }
    }
    free(dkd);
    free(dvd);
    free(K);
    free(V);
    free(KD);
    free(VD);
    free(Kl);
    free(Vl);
    free(dKl);
    free(dVl);
    free(p);
    free(dp);
    free(Q);
    free(dO);
}

static void *bwd_worker(void *arg)
{
    const bwd_job *J = (const bwd_job *)arg;
    const int units = J->B * J->Hkv;
    for (int u = J->tid; u < units; u += J->nthreads)
        bwd_unit(J, u / J->Hkv, u % J->Hkv);
    return NULL;
}

/*
 * Gradients of the causal forward over positions 0..N-1 (the training forward
 * of Sec. 2.3) for the output gradient dout [B][Hq][N][d] (storage type):
 *   dq [B][Hq][N][d], dk, dv [B][Hkv][N][d], and per KV head
 *   dDk, dDv [Hkv][d][dd], dUk, dUv [Hkv][dd][d], all fp64.
 * Inputs as dar_oracle_attention with Dk, Dv (Eq. 1) in place of kd, vd.
 * Returns 0, or -1 on a bad argument.  Threads run over (b, g) units; the
 * projection gradients are summed over units in a fixed order.
 */
int dar_oracle_backward(int dtype, int B, int Hq, int Hkv, int N, int d, int dd, int w,
                        const void *q, const void *k, const void *v, const float *Dk,
                        const float *Uk, const float *Dv, const float *Uv, const void *dout,
                        double scale, double *dq, double *dk, double *dv, double *dDk,
                        double *dUk, double *dDv, double *dUv, int nthreads)
{
    if (B < 1 || Hkv < 1 || Hq < Hkv || Hq % Hkv || N < 1 || d < 1 || dd < 1 || w < 0 ||
        (dtype != ORC_F32 && dtype != ORC_BF16))
        return -1;
    if (nthreads < 1)
        nthreads = 1;
    const size_t wd = (size_t)d * dd;
    double *wpart = malloc(sizeof(double) * (size_t)B * Hkv * 4 * wd);
    bwd_job *jobs = malloc(sizeof(bwd_job) * (size_t)nthreads);
    pthread_t *th = malloc(sizeof(pthread_t) * (size_t)nthreads);
    for (int t = 0; t < nthreads; ++t) {
        bwd_job J = {dtype, B, Hq, Hkv, N, d, dd, w, q, k, v, dout, Dk, Uk, Dv, Uv, scale,
                     dq, dk, dv, wpart, nthreads, t};
        jobs[t] = J;
    }
    for (int t = 1; t < nthreads; ++t)
        pthread_create(&th[t], NULL, bwd_worker, &jobs[t]);
    bwd_worker(&jobs[0]);
    for (int t = 1; t < nthreads; ++t)
        pthread_join(th[t], NULL);
    for (int g = 0; g < Hkv; ++g)
        for (size_t e = 0; e < wd; ++e) {
            double s0 = 0.0, s1 = 0.0, s2 = 0.0, s3 = 0.0;
            for (int b = 0; b < B; ++b) {
                const double *wp = wpart + ((size_t)b * Hkv + g) * 4 * wd;
                s0 += wp[e];
                s1 += wp[wd + e];
                s2 += wp[2 * wd + e];
                s3 += wp[3 * wd + e];
            }
            dDk[g * wd + e] = s0;
            dUk[g * wd + e] = s1;
            dDv[g * wd + e] = s2;
            dUv[g * wd + e] = s3;
        }
    free(wpart);
    free(jobs);
    free(th);
    return 0;
}

/* ---- Sec. 2 in its latent form, with the cache scheme of Sec. 5 -----------
 * The paper's own form of Eq. 1-3 on hidden states (model width D), with one
 * bottleneck per token shared by every head and by keys and values:
 *   Eq. 1  c_j  = h_j W_down                  (d_lat; given here as stored, c)
 *   Eq. 2  h'_j = c_j W_up                    (back to D, explicitly, fp64)
 *   Eq. 3  k_j = h_j W_K^g,  v_j = h_j W_V^g  inside the window (given: k, v)
 *          k_j = h'_j W_K^g, v_j = h'_j W_V^g beyond it (computed here, fp64)
 *   Eq. 4  one softmax over all j <= i.
 * Positions are already encoded (no RoPE), as in the per-head form.
 *   q    [nrows][d] T        the query of each row
 *   k, v [B][Hkv][N][d] T    full keys / values of every token
 *   c    [B][N][dl] T        the stored bottleneck of every token
 *   Wup  [dl][D] fp32;  WK, WV [Hkv][D][d] fp32 */
typedef struct {
    int dtype, B, Hq, Hkv, N, d, D, dl, w;
    const void *q, *k, *v, *c;
    const float *Wup, *WK, *WV;
    double scale;
    long nrows;
    const int *row_b, *row_h, *row_i;
    double *out;
    int nthreads, tid;
} latent_job;

static void latent_unit(const latent_job *J, int b, int g)
{
    const int d = J->d, D = J->D, dl = J->dl, N = J->N, G = J->Hq / J->Hkv;
    int jmax = -1;
    for (long r = 0; r < J->nrows; ++r)
        if (J->row_b[r] == b && J->row_h[r] / G == g && J->row_i[r] > jmax)
            jmax = J->row_i[r];
    if (jmax < 0)
        return;
    const int n = jmax + 1;
    const size_t base = ((size_t)b * J->Hkv + g) * N;
    double *Kf = malloc(sizeof(double) * (size_t)n * d), *Vf = malloc(sizeof(double) * (size_t)n * d);
    double *Kl = malloc(sizeof(double) * (size_t)n * d), *Vl = malloc(sizeof(double) * (size_t)n * d);
    double *hl = malloc(sizeof(double) * (size_t)D), *s = malloc(sizeof(double) * (size_t)n);
    for (int j = 0; j < n; ++j) {
        for (int t = 0; t < d; ++t) {
            Kf[(size_t)j * d + t] = load_as_f32(J->k, J->dtype, (base + j) * d + t);
            Vf[(size_t)j * d + t] = load_as_f32(J->v, J->dtype, (base + j) * d + t);
        }
        /* Eq. 2: h'_j = c_j W_up */
        for (int e = 0; e < D; ++e) {
            double acc = 0.0;
            for (int a = 0; a < dl; ++a)
                acc += (double)load_as_f32(J->c, J->dtype, ((size_t)b * N + j) * dl + a) *
                       (double)J->Wup[(size_t)a * D + e];
            hl[e] = acc;
        }
        /* Eq. 3, distant branch: k'_j = h'_j W_K^g, v'_j = h'_j W_V^g */
        for (int t = 0; t < d; ++t) {
            double ka = 0.0, va = 0.0;
            for (int e = 0; e < D; ++e) {
                ka += hl[e] * (double)J->WK[((size_t)g * D + e) * d + t];
                va += hl[e] * (double)J->WV[((size_t)g * D + e) * d + t];
            }
            Kl[(size_t)j * d + t] = ka;
            Vl[(size_t)j * d + t] = va;
        }
    }
    for (long r = 0; r < J->nrows; ++r) {
        if (J->row_b[r] != b || J->row_h[r] / G != g)
            continue;
        const int i = J->row_i[r];
        double *o = J->out + (size_t)r * d;
        double smax = -INFINITY;
        for (int j = 0; j <= i; ++j) {
            const double *key = (i - j < J->w) ? &Kf[(size_t)j * d] : &Kl[(size_t)j * d];
            double dot = 0.0;
            for (int t = 0; t < d; ++t)
                dot += (double)load_as_f32(J->q, J->dtype, (size_t)r * d + t) * key[t];
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
            const double *val = (i - j < J->w) ? &Vf[(size_t)j * d] : &Vl[(size_t)j * d];
            for (int t = 0; t < d; ++t)
                o[t] += p * val[t];
        }
    }
    free(Kf);
    free(Vf);
    free(Kl);
    free(Vl);
    free(hl);
    free(s);
}

static void *latent_worker(void *arg)
{
    const latent_job *J = (const latent_job *)arg;
    const int units = J->B * J->Hkv;
    for (int u = J->tid; u < units; u += J->nthreads)
        latent_unit(J, u / J->Hkv, u % J->Hkv);
    return NULL;
}

/* Rows of the latent form (the row list as in dar_oracle_attention). */
int dar_oracle_attention_latent(int dtype, int B, int Hq, int Hkv, int N, int d, int D, int dl, int w,
                                const void *q, const void *k, const void *v, const void *c,
                                const float *Wup, const float *WK, const float *WV, double scale,
                                long nrows, const int *row_b, const int *row_h, const int *row_i,
                                double *out, int nthreads)
{
    if (B < 1 || Hkv < 1 || Hq < Hkv || Hq % Hkv || N < 1 || d < 1 || D < 1 || dl < 1 || w < 0 ||
        nrows < 0 || (dtype != ORC_F32 && dtype != ORC_BF16))
        return -1;
    for (long r = 0; r < nrows; ++r)
        if (row_b[r] < 0 || row_b[r] >= B || row_h[r] < 0 || row_h[r] >= Hq ||
            row_i[r] < 0 || row_i[r] >= N)
            return -1;
    if (nthreads < 1)
        nthreads = 1;
    latent_job *jobs = malloc(sizeof(latent_job) * (size_t)nthreads);
    pthread_t *th = malloc(sizeof(pthread_t) * (size_t)nthreads);
    for (int t = 0; t < nthreads; ++t) {
        latent_job J = {dtype, B, Hq, Hkv, N, d, D, dl, w, q, k, v, c, Wup, WK, WV, scale,
                        nrows, row_b, row_h, row_i, out, nthreads, t};
        jobs[t] = J;
    }
    for (int t = 1; t < nthreads; ++t)
        pthread_create(&th[t], NULL, latent_worker, &jobs[t]);
    latent_worker(&jobs[0]);
    for (int t = 1; t < nthreads; ++t)
        pthread_join(th[t], NULL);
    free(jobs);
    free(th);
    return 0;
}
