/*
 * inputs_gen.c -- seeded synthetic input generator (no arithmetic of the
 * attention method).  Counter-based: element i of stream (seed, stream, sub)
 * is splitmix64(key + (i + 1) * 0x9E3779B97F4A7C15) with key derived from the
 * three ids by splitmix64's finaliser (Steele, Lea & Flood, OOPSLA 2014).  The
 * top 53 bits give a double in [0, 1); normals use Box--Muller over
 * consecutive pairs: element 2k = r cos(2 pi u2), element 2k+1 = r sin(2 pi u2)
 * with r = sqrt(-2 log(1 - u1)), (u1, u2) = (U(2k), U(2k+1)).
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

static uint64_t mix64(uint64_t z)
{
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

uint64_t dargen_key(uint64_t seed, uint64_t stream, uint64_t sub)
{
    uint64_t k = mix64(seed);
    k = mix64(k ^ stream);
    return mix64(k ^ sub);
}

static double unit(uint64_t key, uint64_t i)
{
    uint64_t z = mix64(key + (i + 1) * 0x9E3779B97F4A7C15ull);
    return (double)(z >> 11) * (1.0 / 9007199254740992.0);
}

static uint16_t f32_to_bf16_bits(float f)
{
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    u += 0x7fffu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

typedef struct {
    uint64_t key;
    size_t lo, hi;
    double std;
    int kind; /* 0 float32, 1 bf16 bits, 2 float64, 3 uniform float64 */
    void *out;
} gen_job;

static void *gen_run(void *arg)
{
    const gen_job *J = (const gen_job *)arg;
    for (size_t i = J->lo; i < J->hi; ++i) {
        double x;
        if (J->kind == 3) {
            x = unit(J->key, i);
        } else {
            size_t k = i >> 1;
            double u1 = unit(J->key, 2 * k), u2 = unit(J->key, 2 * k + 1);
            double r = sqrt(-2.0 * log1p(-u1));
            double t = 6.283185307179586 * u2;
            x = ((i & 1) ? r * sin(t) : r * cos(t)) * J->std;
        }
        if (J->kind == 0)
            ((float *)J->out)[i - J->lo] = (float)x;
        else if (J->kind == 1)
            ((uint16_t *)J->out)[i - J->lo] = f32_to_bf16_bits((float)x);
        else
            ((double *)J->out)[i - J->lo] = x;
    }
    return NULL;
}

/* Fill out[0..n) with elements offset..offset+n of the stream. */
void dargen_fill(uint64_t seed, uint64_t stream, uint64_t sub, uint64_t offset, size_t n,
                 double std, int kind, void *out, int nthreads)
{
    if (nthreads < 1)
        nthreads = 1;
    if ((size_t)nthreads > n / 65536 + 1)
        nthreads = (int)(n / 65536 + 1);
    size_t esz = kind == 0 ? 4 : kind == 1 ? 2 : 8;
    gen_job *jobs = malloc(sizeof(gen_job) * (size_t)nthreads);
    pthread_t *th = malloc(sizeof(pthread_t) * (size_t)nthreads);
    uint64_t key = dargen_key(seed, stream, sub);
    for (int t = 0; t < nthreads; ++t) {
        size_t lo = n * (size_t)t / (size_t)nthreads, hi = n * (size_t)(t + 1) / (size_t)nthreads;
        gen_job J = {key, offset + lo, offset + hi, std, kind, (char *)out + lo * esz};
        jobs[t] = J;
    }
    for (int t = 1; t < nthreads; ++t)
        pthread_create(&th[t], NULL, gen_run, &jobs[t]);
    gen_run(&jobs[0]);
    for (int t = 1; t < nthreads; ++t)
        pthread_join(th[t], NULL);
    free(jobs);
    free(th);
}
