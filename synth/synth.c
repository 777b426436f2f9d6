/*
 * Seeded synthetic inputs for the shard-decode workloads.
 *
 * This module produces the INPUTS that both the CUDA library and the CPU
 * oracle consume: Gaussian weights quantised to the packed uint4 format the
 * shard boundary accepts, fp16 KV-cache prefills, fp16 hidden states, token
 * ids, accept patterns and permutations.  It contains none of the shard
 * forward's arithmetic (no GEMV, norm, RoPE, attention or activation); the
 * quantiser here is the offline weight-compression step that happens before
 * a shard is created (the paper's export pipeline, Section 3.2, Step 4).
 *
 * Random numbers come from Philox4x32-10, the counter-based generator of
 * Salmon, Moraes, Dror and Shaw, "Parallel random numbers: as easy as
 * 1, 2, 3" (SC'11), written here from its published definition: a 4x32-bit
 * counter and a 2x32-bit key pass through ten rounds of two 32x32->64
 * multiplies, with the key bumped by the Weyl constants between rounds.
 * Normals use the Box-Muller transform on pairs of 32-bit uniforms.
 *
 * Every stream is addressed by (seed, stream, tag, element index), so any
 * slice of any tensor can be produced independently and in parallel; results
 * do not depend on the thread count.
 *
 * Build: gcc -O2 -fPIC -shared -pthread -ffp-contract=off synth.c -lm
 * (contraction is disabled so x86-64 and aarch64 hosts produce the same bits).
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* ------------------------------------------------------------------------- */
/* Philox4x32-10                                                             */
/* ------------------------------------------------------------------------- */

#define PHILOX_M0 0xD2511F53u
#define PHILOX_M1 0xCD9E8D57u
#define PHILOX_W0 0x9E3779B9u
#define PHILOX_W1 0xBB67AE85u

static void philox_round(uint32_t c[4], const uint32_t k[2]) {
    uint64_t p0 = (uint64_t)PHILOX_M0 * (uint64_t)c[0];
    uint64_t p1 = (uint64_t)PHILOX_M1 * (uint64_t)c[2];
    uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
    uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
    uint32_t n0 = hi1 ^ c[1] ^ k[0];
    uint32_t n1 = lo1;
    uint32_t n2 = hi0 ^ c[3] ^ k[1];
    uint32_t n3 = lo0;
    c[0] = n0; c[1] = n1; c[2] = n2; c[3] = n3;
}

static void philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]) {
    uint32_t c[4] = {ctr[0], ctr[1], ctr[2], ctr[3]};
    uint32_t k[2] = {key[0], key[1]};
    for (int r = 0; r < 10; ++r) {
        philox_round(c, k);
        if (r < 9) { k[0] += PHILOX_W0; k[1] += PHILOX_W1; }
    }
    memcpy(out, c, sizeof(c));
}

/* Exported for known-answer tests. */
void synth_philox4x32_10(const uint32_t* ctr, const uint32_t* key, uint32_t* out) {
    philox4x32_10(ctr, key, out);
}

/* Block b of stream (seed, stream, tag): counter = (b_lo, b_hi, stream, tag),
 * key = (seed_lo, seed_hi). */
static void stream_block(uint64_t seed, uint32_t stream, uint32_t tag, uint64_t b, uint32_t out[4]) {
    uint32_t ctr[4] = {(uint32_t)b, (uint32_t)(b >> 32), stream, tag};
    uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
    philox4x32_10(ctr, key, out);
}

/* ------------------------------------------------------------------------- */
/* fp16 (IEEE binary16) encoding, round to nearest even                      */
/* ------------------------------------------------------------------------- */

static uint16_t f64_to_f16_bits(double x) {
    uint16_t sign = signbit(x) ? 0x8000 : 0;
    double a = fabs(x);
    if (isnan(x)) return (uint16_t)(sign | 0x7E00);
    if (a >= 65520.0) return (uint16_t)(sign | 0x7C00); /* rounds to infinity */
    if (a == 0.0) return sign;
    int e2;
    frexp(a, &e2);           /* a = m * 2^e2, m in [0.5, 1) */
    int e = e2 - 1;          /* a in [2^e, 2^(e+1)) */
    int qexp = (e < -14) ? -24 : e - 10; /* quantum exponent */
    double n = nearbyint(ldexp(a, -qexp)); /* exact scaling, RNE rounding */
    double v = ldexp(n, qexp);
    if (v < ldexp(1.0, -14)) {
        return (uint16_t)(sign | (uint16_t)n); /* subnormal (or rounded up to 2^-14 handled below) */
    }
    frexp(v, &e2);
    e = e2 - 1;
    uint32_t mant = (uint32_t)(ldexp(v, -e) * 1024.0 - 1024.0);
    return (uint16_t)(sign | (uint16_t)((e + 15) << 10) | (uint16_t)mant);
}

static double f16_bits_to_f64(uint16_t h) {
    int sign = (h >> 15) & 1;
    int ex = (h >> 10) & 0x1F;
    int man = h & 0x3FF;
    double v;
    if (ex == 0) v = ldexp((double)man, -24);
    else if (ex == 31) v = man ? NAN : INFINITY;
    else v = ldexp((double)(man + 1024), ex - 25);
    return sign ? -v : v;
}

uint16_t synth_f64_to_f16(double x) { return f64_to_f16_bits(x); }
double synth_f16_to_f64(uint16_t h) { return f16_bits_to_f64(h); }

/* ------------------------------------------------------------------------- */
/* Normals                                                                   */
/* ------------------------------------------------------------------------- */

static const double TWO_PI = 6.283185307179586476925286766559;

/* Four standard normals from one Philox block (two Box-Muller pairs). */
static void block_normals(uint64_t seed, uint32_t stream, uint32_t tag, uint64_t b, double z[4]) {
    uint32_t u[4];
    stream_block(seed, stream, tag, b, u);
    for (int p = 0; p < 2; ++p) {
        double u1 = ((double)u[2 * p] + 1.0) * (1.0 / 4294967296.0); /* (0, 1] */
        double u2 = (double)u[2 * p + 1] * (1.0 / 4294967296.0);     /* [0, 1) */
        double r = sqrt(-2.0 * log(u1));
        double t = TWO_PI * u2;
        z[2 * p] = r * cos(t);
        z[2 * p + 1] = r * sin(t);
    }
}

/* Standard normals for element indices [i0, i1) of a stream, into out[0..). */
static void normals_range(uint64_t seed, uint32_t stream, uint32_t tag, int64_t i0, int64_t i1, double* out) {
    int64_t i = i0;
    while (i < i1) {
        uint64_t b = (uint64_t)i >> 2;
        double z[4];
        block_normals(seed, stream, tag, b, z);
        for (int lane = (int)(i & 3); lane < 4 && i < i1; ++lane, ++i) out[i - i0] = z[lane];
    }
}

/* ------------------------------------------------------------------------- */
/* Thread pool helper                                                        */
/* ------------------------------------------------------------------------- */

typedef void (*range_fn)(void* ctx, int64_t lo, int64_t hi);
typedef struct { range_fn fn; void* ctx; int64_t lo, hi; } range_job;

static void* range_thread(void* p) {
    range_job* j = (range_job*)p;
    if (j->lo < j->hi) j->fn(j->ctx, j->lo, j->hi);
    return NULL;
}

static void parallel_for(int64_t n, int threads, range_fn fn, void* ctx) {
    if (threads < 1) threads = 1;
    if (threads > 256) threads = 256;
    if ((int64_t)threads > n) threads = (int)(n > 0 ? n : 1);
    if (threads == 1) { fn(ctx, 0, n); return; }
    pthread_t tid[256];
    range_job jobs[256];
    int started[256];
    for (int t = 0; t < threads; ++t) {
        jobs[t].fn = fn; jobs[t].ctx = ctx;
        jobs[t].lo = n * t / threads; jobs[t].hi = n * (t + 1) / threads;
        started[t] = pthread_create(&tid[t], NULL, range_thread, &jobs[t]) == 0;
        if (!started[t]) range_thread(&jobs[t]);
    }
    for (int t = 0; t < threads; ++t) if (started[t]) pthread_join(tid[t], NULL);
}

/* ------------------------------------------------------------------------- */
/* Exported generators                                                       */
/* ------------------------------------------------------------------------- */

typedef struct {
    uint64_t seed; uint32_t stream, tag; double sigma, mean;
    float* f32; uint16_t* f16; double* f64;
} normal_ctx;

static void normal_chunk(void* p, int64_t lo, int64_t hi) {
    normal_ctx* c = (normal_ctx*)p;
    enum { CH = 4096 };
    double buf[CH];
    for (int64_t a = lo; a < hi; a += CH) {
        int64_t b = a + CH < hi ? a + CH : hi;
        normals_range(c->seed, c->stream, c->tag, a, b, buf);
        for (int64_t i = a; i < b; ++i) {
            double v = c->mean + c->sigma * buf[i - a];
            if (c->f32) c->f32[i] = (float)v;
            if (c->f16) c->f16[i] = f64_to_f16_bits(v);
            if (c->f64) c->f64[i] = v;
        }
    }
}

/* N(mean, sigma^2) samples, rounded to fp32. */
void synth_normal_f32(float* out, int64_t n, double mean, double sigma, uint64_t seed,
                      uint32_t stream, uint32_t tag, int threads) {
    normal_ctx c = {seed, stream, tag, sigma, mean, out, NULL, NULL};
    parallel_for(n, threads, normal_chunk, &c);
}

/* N(mean, sigma^2) samples, rounded to fp16 (bits). */
void synth_normal_f16(uint16_t* out, int64_t n, double mean, double sigma, uint64_t seed,
                      uint32_t stream, uint32_t tag, int threads) {
    normal_ctx c = {seed, stream, tag, sigma, mean, NULL, out, NULL};
    parallel_for(n, threads, normal_chunk, &c);
}

/* N(mean, sigma^2) samples in fp64. */
void synth_normal_f64(double* out, int64_t n, double mean, double sigma, uint64_t seed,
                      uint32_t stream, uint32_t tag, int threads) {
    normal_ctx c = {seed, stream, tag, sigma, mean, NULL, NULL, out};
    parallel_for(n, threads, normal_chunk, &c);
}

/* Uniform doubles in [0, 1): 53 bits from two 32-bit words; two per block. */
void synth_uniform_f64(double* out, int64_t n, uint64_t seed, uint32_t stream, uint32_t tag) {
    for (int64_t i = 0; i < n; ++i) {
        uint32_t u[4];
        stream_block(seed, stream, tag, (uint64_t)i >> 1, u);
        int p = (int)(i & 1);
        uint64_t hi = u[2 * p] >> 5, lo = u[2 * p + 1] >> 6; /* 27 + 26 bits */
        out[i] = ((double)hi * 67108864.0 + (double)lo) * (1.0 / 9007199254740992.0);
    }
}

/* Uniform integers in [lo, hi] (inclusive), by rejection on 32-bit words so
 * that every value is exactly equally likely.  Word w of the stream is used
 * for attempt w; element i consumes attempts in order from its own
 * sub-stream (tag, i) so elements are independent of each other. */
void synth_uniform_int(int32_t* out, int64_t n, int32_t lo, int32_t hi, uint64_t seed,
                       uint32_t stream, uint32_t tag) {
    uint64_t range = (uint64_t)((int64_t)hi - (int64_t)lo) + 1u;
    uint64_t limit = (4294967296ull / range) * range; /* accept words < limit */
    for (int64_t i = 0; i < n; ++i) {
        uint64_t attempt = 0;
        for (;;) {
            uint32_t u[4];
            /* sub-stream: counter high word carries the element index */
            uint32_t ctr[4] = {(uint32_t)attempt, (uint32_t)i, stream, tag ^ (uint32_t)((uint64_t)i >> 32)};
            uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
            philox4x32_10(ctr, key, u);
            int found = 0;
            for (int w = 0; w < 4; ++w) {
                if ((uint64_t)u[w] < limit) { out[i] = (int32_t)((int64_t)lo + (int64_t)((uint64_t)u[w] % range)); found = 1; break; }
            }
            if (found) break;
            ++attempt;
        }
    }
}

/* ------------------------------------------------------------------------- */
/* Asymmetric uint4 group quantisation and packing                           */
/* ------------------------------------------------------------------------- */
/*
 * Per row and per group of `group` consecutive input columns (the last group
 * of a row may be shorter when cols % group != 0; its range comes from its
 * own elements only):
 *   s   = (max - min) / 15, rounded to fp16 -> s16 (s16 := 1 if it is 0)
 *   z   = clamp(rint(-min / s16), 0, 15)
 *   q_i = clamp(rint(w_i / s16) + z, 0, 15)
 * rint is round-half-to-even.  Packed format (the shard boundary's):
 *   codes  uint8 [rows][ceil(cols/2)], low nibble = even column
 *   scales fp16  [rows][G], G = ceil(cols/group)
 *   zeros  uint8 [rows][ceil(G/2)], low nibble = even group
 */

static void quantize_row(const float* w, int cols, int group, uint8_t* codes, uint16_t* scales, uint8_t* zeros) {
    int G = (cols + group - 1) / group;
    memset(codes, 0, (size_t)(cols + 1) / 2);
    memset(zeros, 0, (size_t)(G + 1) / 2);
    for (int gi = 0; gi < G; ++gi) {
        int c0 = gi * group, c1 = c0 + group < cols ? c0 + group : cols;
        double mn = w[c0], mx = w[c0];
        for (int c = c0 + 1; c < c1; ++c) { if (w[c] < mn) mn = w[c]; if (w[c] > mx) mx = w[c]; }
        uint16_t s16 = f64_to_f16_bits((mx - mn) / 15.0);
        double sd = f16_bits_to_f64(s16);
        if (sd == 0.0) { s16 = 0x3C00; sd = 1.0; }
        double zd = nearbyint(-mn / sd);
        int z = zd < 0 ? 0 : (zd > 15 ? 15 : (int)zd);
        scales[gi] = s16;
        zeros[gi >> 1] |= (uint8_t)(z << (4 * (gi & 1)));
        for (int c = c0; c < c1; ++c) {
            double qd = nearbyint((double)w[c] / sd) + z;
            int q = qd < 0 ? 0 : (qd > 15 ? 15 : (int)qd);
            codes[c >> 1] |= (uint8_t)(q << (4 * (c & 1)));
        }
    }
}

/* Quantise a given fp32 matrix [rows][cols]. */
void synth_quantize(const float* w, int rows, int cols, int group, uint8_t* codes, uint16_t* scales, uint8_t* zeros) {
    int G = (cols + group - 1) / group;
    for (int r = 0; r < rows; ++r)
        quantize_row(w + (size_t)r * cols, cols, group, codes + (size_t)r * ((cols + 1) / 2),
                     scales + (size_t)r * G, zeros + (size_t)r * ((G + 1) / 2));
}

typedef struct {
    int cols, group; double sigma; uint64_t seed; uint32_t stream, tag;
    uint8_t* codes; uint16_t* scales; uint8_t* zeros;
} qmat_ctx;

static void qmat_chunk(void* p, int64_t lo, int64_t hi) {
    qmat_ctx* c = (qmat_ctx*)p;
    int G = (c->cols + c->group - 1) / c->group;
    double* buf = (double*)malloc(sizeof(double) * (size_t)c->cols);
    float* row = (float*)malloc(sizeof(float) * (size_t)c->cols);
    for (int64_t r = lo; r < hi; ++r) {
        normals_range(c->seed, c->stream, c->tag, r * c->cols, (r + 1) * c->cols, buf);
        for (int i = 0; i < c->cols; ++i) row[i] = (float)(c->sigma * buf[i]);
        quantize_row(row, c->cols, c->group, c->codes + (size_t)r * ((c->cols + 1) / 2),
                     c->scales + (size_t)r * G, c->zeros + (size_t)r * ((G + 1) / 2));
    }
    free(buf);
    free(row);
}

/* Weights N(0, sigma^2) in fp32 for a [rows][cols] matrix (element (r, c) is
 * stream element r*cols + c), quantised and packed as above. */
void synth_quant_matrix(uint8_t* codes, uint16_t* scales, uint8_t* zeros, int rows, int cols, int group,
                        double sigma, uint64_t seed, uint32_t stream, uint32_t tag, int threads) {
    qmat_ctx c = {cols, group, sigma, seed, stream, tag, codes, scales, zeros};
    parallel_for(rows, threads, qmat_chunk, &c);
}
