/*
 * Oracle-side fast regeneration of synthetic weights, with the oracle's own
 * per-output-row INT8 quantizer. Test infrastructure only: nothing in the
 * product links this file.
 *
 * Generator: counter-based SplitMix64 (Steele, Lea, Flood, OOPSLA 2014) with an
 * Irwin-Hall sum of twelve 16-bit lanes, as specified in synth/gen.py.
 *
 * Quantizer (the paper's "symmetric INT8 weights", Table 1, read per output
 * channel with FP32 scales): for a dense row w, a = max|w|, s = fl32(a / 127),
 * q = clamp(rint(fl32(w / s)), -127, 127); a zero row has s = 0 and q = 0.
 * The groupwise variant (Table 1: group size 128, BF16 scales) applies the same
 * rule to each run of `group` consecutive columns with the scale rounded to
 * BF16 (nearest, ties to even on the FP32 bit pattern) before it divides.
 *
 * Build: gcc -O2 -ffp-contract=off -fno-fast-math -fPIC -shared -pthread.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define OG_GOLDEN 0x9E3779B97F4A7C15ULL

static uint64_t og_mix(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

static uint64_t og_fold(uint64_t z) { return og_mix(z + OG_GOLDEN); }

uint64_t og_stream_key(uint64_t seed, uint64_t tensor, uint64_t layer, uint64_t sub) {
    uint64_t k = og_fold(seed);
    k = og_fold(k ^ tensor);
    k = og_fold(k ^ layer);
    k = og_fold(k ^ sub);
    return k;
}

static float og_normal_at(uint64_t key, uint64_t i) {
    int64_t s = 0;
    for (int k = 0; k < 3; ++k) {
        uint64_t d = og_mix(key + (3 * i + (uint64_t)k + 1) * OG_GOLDEN);
        s += (int64_t)(d & 0xFFFF) + (int64_t)((d >> 16) & 0xFFFF) + (int64_t)((d >> 32) & 0xFFFF) +
             (int64_t)(d >> 48);
    }
    return (float)(s - 393210) * (1.0f / 65536.0f);
}

/* out[i] = fl32(normal(key, start + i) * sigma) for i < count. */
void og_normal(uint64_t key, uint64_t start, int64_t count, float sigma, float* out) {
    for (int64_t i = 0; i < count; ++i) {
        float z = og_normal_at(key, start + (uint64_t)i);
        out[i] = z * sigma;
    }
}

/* Quantize one dense FP32 row of n values. */
void og_quant_row(const float* w, int64_t n, int8_t* q, float* s_out) {
    float a = 0.0f;
    for (int64_t j = 0; j < n; ++j) {
        float v = fabsf(w[j]);
        if (v > a) a = v;
    }
    if (a == 0.0f) {
        *s_out = 0.0f;
        memset(q, 0, (size_t)n);
        return;
    }
    float s = a / 127.0f;
    *s_out = s;
    for (int64_t j = 0; j < n; ++j) {
        float r = rintf(w[j] / s);
        if (r > 127.0f) r = 127.0f;
        if (r < -127.0f) r = -127.0f;
        q[j] = (int8_t)r;
    }
}

/* FP32 -> nearest BF16 value (ties to even), as FP32; finite inputs. */
static float og_bf16(float x) {
    uint32_t u;
    memcpy(&u, &x, 4);
    u = (uint32_t)(((uint64_t)u + 0x7FFFu + ((u >> 16) & 1u)) >> 16) << 16;
    float r;
    memcpy(&r, &u, 4);
    return r;
}

/* Quantize one dense FP32 row of n values in groups of `group` columns (n a multiple of
 * group): q [n], s_out [n / group] (BF16 values held in FP32). */
void og_quant_row_grouped(const float* w, int64_t n, int64_t group, int8_t* q, float* s_out) {
    for (int64_t g0 = 0, gi = 0; g0 < n; g0 += group, ++gi) {
        float a = 0.0f;
        for (int64_t j = g0; j < g0 + group; ++j) {
            float v = fabsf(w[j]);
            if (v > a) a = v;
        }
        float sc = og_bf16(a / 127.0f);
        s_out[gi] = sc;
        if (sc == 0.0f) {
            memset(q + g0, 0, (size_t)group);
            continue;
        }
        for (int64_t j = g0; j < g0 + group; ++j) {
            float r = rintf(w[j] / sc);
            if (r > 127.0f) r = 127.0f;
            if (r < -127.0f) r = -127.0f;
            q[j] = (int8_t)r;
        }
    }
}

typedef struct {
    uint64_t key;
    int64_t abs0; /* absolute index of local row 0 */
    int64_t row0, row1, cols;
    int64_t group; /* 0: one scale per row; else columns per scale group */
    float sigma;
    int8_t* q;
    float* s;
} og_job;

static void* og_worker(void* p) {
    og_job* j = (og_job*)p;
    float* buf = (float*)malloc(sizeof(float) * (size_t)j->cols);
    if (!buf) return (void*)1;
    for (int64_t r = j->row0; r < j->row1; ++r) {
        og_normal(j->key, (uint64_t)(j->abs0 + r) * (uint64_t)j->cols, j->cols, j->sigma, buf);
        if (j->group)
            og_quant_row_grouped(buf, j->cols, j->group, j->q + r * j->cols, j->s + r * (j->cols / j->group));
        else
            og_quant_row(buf, j->cols, j->q + r * j->cols, j->s + r);
    }
    free(buf);
    return 0;
}

static int og_run(uint64_t key, int64_t row0, int64_t nrows, int64_t cols, int64_t group, float sigma, int8_t* q,
                  float* s, int nthreads);

/* Regenerate rows [row0, row0+nrows) of a [rows, cols] N(0, sigma) matrix and quantize
 * each row; q is [nrows, cols], s is [nrows]. Returns 0 on success. */
int og_weight_int8(uint64_t key, int64_t row0, int64_t nrows, int64_t cols, float sigma, int8_t* q,
                   float* s, int nthreads) {
    return og_run(key, row0, nrows, cols, 0, sigma, q, s, nthreads);
}

/* As og_weight_int8 with groupwise scales: s is [nrows, cols / group]. Returns 3 when cols
 * is not a positive multiple of group. */
int og_weight_int8_grouped(uint64_t key, int64_t row0, int64_t nrows, int64_t cols, int64_t group, float sigma,
                           int8_t* q, float* s, int nthreads) {
    if (group < 1 || cols % group) return 3;
    return og_run(key, row0, nrows, cols, group, sigma, q, s, nthreads);
}

static int og_run(uint64_t key, int64_t row0, int64_t nrows, int64_t cols, int64_t group, float sigma, int8_t* q,
                  float* s, int nthreads) {
    if (nthreads < 1) nthreads = 1;
    if (nthreads > 256) nthreads = 256;
    if (nthreads > nrows) nthreads = (int)(nrows > 0 ? nrows : 1);
    pthread_t th[256];
    og_job jobs[256];
    int64_t per = (nrows + nthreads - 1) / nthreads;
    int started = 0, rc = 0;
    for (int t = 0; t < nthreads; ++t) {
        int64_t a = (int64_t)t * per, b = a + per;
        if (b > nrows) b = nrows;
        if (a >= b) break;
        jobs[t].key = key;
        jobs[t].abs0 = row0;
        jobs[t].row0 = a;
        jobs[t].row1 = b;
        jobs[t].cols = cols;
        jobs[t].group = group;
        jobs[t].sigma = sigma;
        jobs[t].q = q;
        jobs[t].s = s;
        if (pthread_create(&th[t], 0, og_worker, &jobs[t]) != 0) {
            rc = 2;
            break;
        }
        ++started;
    }
    for (int t = 0; t < started; ++t) {
        void* ret = 0;
        pthread_join(th[t], &ret);
        if (ret) rc = 1;
    }
    return rc;
}
