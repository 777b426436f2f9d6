/*
 * ORACLE -- test infrastructure, not part of the product.
 *
 * A plain, slow, fp64 CPU implementation of the decode-step forward of one
 * pipeline shard (a contiguous range of Llama-style layers) over a stateful
 * KV cache, written from the paper's description.  Only the tests, the
 * package's smoke check and the benchmark's CPU-baseline leg may load it.  It
 * shares no code with the CUDA library.
 *
 * What it computes (paper sections in brackets):
 *  - Stateful KV cache [Section 3.4]: each request row keeps, per layer, the
 *    K and V of every cached token; a decode step appends the new tokens' K/V
 *    after the existing entries and attends over the cache.
 *  - beam_idx Gather [Section 4]: before the step, row b of the cache becomes
 *    a copy of row beam_idx[b] (Gather(ReadValue, beam_idx, axis 0)), then the
 *    new K/V are appended to it.  Here the copy is literal and physical.
 *  - Mask-based rewind [Section 5.2]: attention_mask[b][j] = 0 removes cache
 *    entry j of row b from attention on this forward; rejected entries stay
 *    in the cache and new entries append at the next index; RoPE uses the
 *    caller's position_ids (logical positions), not the cache index.
 *  - Physical trim [Section 5.1]: or_trim deletes entries and shifts the
 *    rest down, the operation the mask replaces.
 *  - Packed step [Section 8.6]: or_step_packed runs S query rows over one
 *    cache row with a mask row per query, so slots (regions of the row, an
 *    optional shared prefix) are isolated and same-slot rows form causal
 *    chunks -- continuous batching expressed by the mask layout alone.
 *  - INT4 weights [Section 3.2, Step 4]: W[o][i] = (q - z) * s with uint4
 *    codes q, uint4 zero point z and fp16 scale s per (row, group of inputs).
 *  - Layer math (Llama, Section 3.2 Step 2's attention with precomputed
 *    rotary tables): RMSNorm, q/k/v projections, rotate-half RoPE at
 *    theta^(-2i/d) frequencies, grouped-query softmax attention with scale
 *    1/sqrt(d), output projection + residual, RMSNorm, SwiGLU MLP + residual.
 *  - The final stage's LM head with top-1 compression [Section 6.7]: final
 *    RMSNorm, the INT4 lm_head projection to vocabulary logits, and only the
 *    greedy token (argmax) with its softmax probability leave the stage.
 *
 * Precision: everything is fp64.  With round_points = 1 the result is
 * rounded to fp16 (round to nearest even) at the points where the W4A16 path
 * stores 16-bit data: the activation operand of every projection (normed x,
 * attention output, SwiGLU output), the appended K (after RoPE) and V, and
 * the step's hidden output.  With round_points = 0 only the output is
 * rounded (the K/V cache keeps fp64 values).
 *
 * Softmax skips masked entries entirely (no -inf term), so a masked cache
 * and a physically trimmed one produce identical bits.
 *
 * Build: gcc -O2 -fPIC -shared -fopenmp -ffp-contract=off oracle.c -lm
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

enum { OR_OK = 0, OR_EINVAL = -1, OR_ECAP = -2, OR_ENOMEM = -3 };
enum { MAT_Q = 0, MAT_K, MAT_V, MAT_O, MAT_GATE, MAT_UP, MAT_DOWN, N_MAT };

typedef struct {
    int32_t n_layers, hidden, n_heads, n_kv_heads, head_dim, ffn, group, vocab;
    double rms_eps, rope_theta;
} or_config;

typedef struct {
    const uint8_t* codes;   /* [rows][ceil(cols/2)], low nibble = even column */
    const uint16_t* scales; /* fp16 bits [rows][G] */
    const uint8_t* zeros;   /* [rows][ceil(G/2)], low nibble = even group */
} or_matrix;

typedef struct {
    or_matrix w[N_MAT];
    const uint16_t* attn_norm; /* fp16 bits [H] */
    const uint16_t* ffn_norm;  /* fp16 bits [H] */
} or_layer;

typedef struct {
    or_config cfg;
    or_layer* layers;
    const uint16_t* embedding; /* fp16 bits [V][H] or NULL */
} or_shard;

typedef struct {
    int n_rows, capacity, n_layers, kv_width; /* kv_width = Hkv * d */
    int* len;                                 /* [n_rows] */
    double* k;                                /* [n_rows][n_layers][capacity][kv_width] */
    double* v;
} or_state;

/* ------------------------------------------------------------------------- */
/* fp16 rounding (IEEE binary16, round to nearest even)                      */
/* ------------------------------------------------------------------------- */

double or_f16_to_f64(uint16_t h) {
    int neg = h >> 15, e = (h >> 10) & 31, m = h & 1023;
    double v;
    if (e == 0) v = ldexp((double)m, -24);                 /* subnormal: m * 2^-24 */
    else if (e == 31) v = m ? NAN : INFINITY;
    else v = ldexp(1.0 + m / 1024.0, e - 15);
    return neg ? -v : v;
}

uint16_t or_f64_to_f16(double x) {
    uint16_t sign = signbit(x) ? 0x8000 : 0;
    if (isnan(x)) return sign | 0x7E00;
    double a = fabs(x);
    /* Largest finite fp16 is 65504 = (2 - 2^-10) * 2^15; values from 65520
       (half an ulp above) upward round to infinity. */
    if (a >= 65520.0) return sign | 0x7C00;
    /* Spacing of representable values around a: 2^(e-10) in the normal range
       [2^e, 2^(e+1)), e >= -14; 2^-24 below 2^-14. */
    int e = (a >= ldexp(1.0, -14)) ? ilogb(a) : -14;
    double ulp = ldexp(1.0, e - 10);
    double n = nearbyint(a / ulp);       /* a / ulp is exact; ties to even */
    double r = n * ulp;
    if (r == 0.0) return sign;
    if (r < ldexp(1.0, -14)) return sign | (uint16_t)(r / ldexp(1.0, -24));
    int er = ilogb(r);
    uint16_t frac = (uint16_t)((r / ldexp(1.0, er) - 1.0) * 1024.0);
    return sign | (uint16_t)((er + 15) << 10) | frac;
}

double or_round_f16(double x) { return or_f16_to_f64(or_f64_to_f16(x)); }

/* ------------------------------------------------------------------------- */
/* Threads                                                                   */
/* ------------------------------------------------------------------------- */

static int g_threads = 1;

void or_set_threads(int n) {
    g_threads = n < 1 ? 1 : n;
#ifdef _OPENMP
    omp_set_num_threads(g_threads);
#endif
}

int or_get_threads(void) { return g_threads; }

/* ------------------------------------------------------------------------- */
/* INT4 dequantisation and projection                                        */
/* ------------------------------------------------------------------------- */

/* W[o][i] = (q[o][i] - z[o][i / g]) * s[o][i / g] */
static double dequant(const or_matrix* m, int cols, int group, int o, int i) {
    int G = (cols + group - 1) / group;
    int gi = i / group;
    int q = (m->codes[(size_t)o * ((cols + 1) / 2) + i / 2] >> (4 * (i & 1))) & 15;
    int z = (m->zeros[(size_t)o * ((G + 1) / 2) + gi / 2] >> (4 * (gi & 1))) & 15;
    double s = or_f16_to_f64(m->scales[(size_t)o * G + gi]);
    return (double)(q - z) * s;
}

/* Dense fp64 copy of the dequantised matrix [rows][cols]. */
void or_dequant(const or_matrix* m, int rows, int cols, int group, double* out) {
    for (int o = 0; o < rows; ++o)
        for (int i = 0; i < cols; ++i) out[(size_t)o * cols + i] = dequant(m, cols, group, o, i);
}

/* y[t][o] = sum_i W[o][i] * x[t][i], for t < M tokens; each dot product is
   summed sequentially in i.  Rows run in parallel (results do not depend on
   the thread count). */
void or_gemv(const or_matrix* m, int rows, int cols, int group, const double* x, int M, double* y) {
    #pragma omp parallel num_threads(g_threads)
    {
        double* acc = (double*)malloc(sizeof(double) * (size_t)M);
        #pragma omp for schedule(static)
        for (int o = 0; o < rows; ++o) {
            for (int t = 0; t < M; ++t) acc[t] = 0.0;
            for (int i = 0; i < cols; ++i) {
                double w = dequant(m, cols, group, o, i);
                for (int t = 0; t < M; ++t) acc[t] += w * x[(size_t)t * cols + i];
            }
            for (int t = 0; t < M; ++t) y[(size_t)t * rows + o] = acc[t];
        }
        free(acc);
    }
}

/* ------------------------------------------------------------------------- */
/* Elementwise pieces                                                        */
/* ------------------------------------------------------------------------- */

/* out = x / sqrt(mean(x^2) + eps) * w */
void or_rmsnorm(const double* x, int n, const uint16_t* w, double eps, double* out) {
    double ss = 0.0;
    for (int i = 0; i < n; ++i) ss += x[i] * x[i];
    double inv = 1.0 / sqrt(ss / n + eps);
    for (int i = 0; i < n; ++i) out[i] = x[i] * inv * (w ? or_f16_to_f64(w[i]) : 1.0);
}

/* Rotary embedding on one head vector of dimension d at position pos, in
   the rotate-half form: pairs (i, i + d/2) with frequency
   w_i = theta^(-2i/d) are rotated by the angle pos * w_i. */
void or_rope(double* vec, int d, int pos, double theta) {
    int h = d / 2;
    for (int i = 0; i < h; ++i) {
        double freq = pow(theta, -2.0 * i / d);
        double ang = (double)pos * freq;
        double c = cos(ang), s = sin(ang);
        double a = vec[i], b = vec[i + h];
        vec[i] = a * c - b * s;
        vec[i + h] = b * c + a * s;
    }
}

double or_silu(double x) { return x / (1.0 + exp(-x)); }

/* Softmax attention of one query over n cached entries (rows of K and V with
   stride `stride`), visiting only entries with vis[j] != 0:
   out = sum_j p_j v_j,  p_j = exp(s_j - max) / sum exp(...),
   s_j = q . k_j / sqrt(d).  Returns the number of visible entries. */
int or_attend(const double* q, const double* K, const double* V, int n, int stride, int d,
              const uint8_t* vis, double* out) {
    double scale = 1.0 / sqrt((double)d);
    double mx = -INFINITY;
    int cnt = 0;
    for (int j = 0; j < n; ++j) {
        if (!vis[j]) continue;
        double s = 0.0;
        for (int t = 0; t < d; ++t) s += q[t] * K[(size_t)j * stride + t];
        s *= scale;
        if (s > mx) mx = s;
        ++cnt;
    }
    for (int t = 0; t < d; ++t) out[t] = 0.0;
    if (cnt == 0) return 0;
    double den = 0.0;
    for (int j = 0; j < n; ++j) {
        if (!vis[j]) continue;
        double s = 0.0;
        for (int t = 0; t < d; ++t) s += q[t] * K[(size_t)j * stride + t];
        den += exp(s * scale - mx);
    }
    for (int j = 0; j < n; ++j) {
        if (!vis[j]) continue;
        double s = 0.0;
        for (int t = 0; t < d; ++t) s += q[t] * K[(size_t)j * stride + t];
        double p = exp(s * scale - mx) / den;
        for (int t = 0; t < d; ++t) out[t] += p * V[(size_t)j * stride + t];
    }
    return cnt;
}

/* ------------------------------------------------------------------------- */
/* Shard and state                                                           */
/* ------------------------------------------------------------------------- */

or_shard* or_shard_create(const or_config* cfg, const or_layer* layers, const uint16_t* embedding) {
    if (!cfg || !layers || cfg->n_layers < 1 || cfg->head_dim % 2 || cfg->n_heads % cfg->n_kv_heads) return NULL;
    or_shard* s = (or_shard*)calloc(1, sizeof(or_shard));
    if (!s) return NULL;
    s->cfg = *cfg;
    s->layers = (or_layer*)malloc(sizeof(or_layer) * (size_t)cfg->n_layers);
    if (!s->layers) { free(s); return NULL; }
    memcpy(s->layers, layers, sizeof(or_layer) * (size_t)cfg->n_layers);
    s->embedding = embedding;
    return s;
}

void or_shard_destroy(or_shard* s) {
    if (!s) return;
    free(s->layers);
    free(s);
}

or_state* or_state_create(const or_shard* sh, int n_rows, int capacity) {
    if (!sh || n_rows < 1 || capacity < 1) return NULL;
    or_state* st = (or_state*)calloc(1, sizeof(or_state));
    if (!st) return NULL;
    st->n_rows = n_rows;
    st->capacity = capacity;
    st->n_layers = sh->cfg.n_layers;
    st->kv_width = sh->cfg.n_kv_heads * sh->cfg.head_dim;
    size_t n = (size_t)n_rows * st->n_layers * capacity * st->kv_width;
    st->len = (int*)calloc((size_t)n_rows, sizeof(int));
    st->k = (double*)calloc(n, sizeof(double));
    st->v = (double*)calloc(n, sizeof(double));
    if (!st->len || !st->k || !st->v) {
        free(st->len); free(st->k); free(st->v); free(st);
        return NULL;
    }
    return st;
}

void or_state_destroy(or_state* st) {
    if (!st) return;
    free(st->len); free(st->k); free(st->v); free(st);
}

static size_t kv_off(const or_state* st, int row, int layer, int j) {
    return (((size_t)row * st->n_layers + layer) * st->capacity + j) * st->kv_width;
}

int or_state_length(const or_state* st, int row) {
    if (!st || row < 0 || row >= st->n_rows) return OR_EINVAL;
    return st->len[row];
}

/* Replace one layer of one row with fp16 K/V [len][Hkv][d]; the row's length
   becomes len (all layers of a row share one length). */
int or_state_load(or_state* st, int row, int layer, const uint16_t* k, const uint16_t* v, int len) {
    if (!st || row < 0 || row >= st->n_rows || layer < 0 || layer >= st->n_layers || len < 0) return OR_EINVAL;
    if (len > st->capacity) return OR_ECAP;
    for (int j = 0; j < len; ++j)
        for (int t = 0; t < st->kv_width; ++t) {
            st->k[kv_off(st, row, layer, j) + t] = or_f16_to_f64(k[(size_t)j * st->kv_width + t]);
            st->v[kv_off(st, row, layer, j) + t] = or_f16_to_f64(v[(size_t)j * st->kv_width + t]);
        }
    st->len[row] = len;
    return OR_OK;
}

/* Entries [start, start+n) of one row and layer, as fp16 and/or fp64. */
int or_state_read(const or_state* st, int row, int layer, int start, int n, uint16_t* k16, uint16_t* v16,
                  double* k64, double* v64) {
    if (!st || row < 0 || row >= st->n_rows || layer < 0 || layer >= st->n_layers || start < 0 || n < 0 ||
        start + n > st->len[row])
        return OR_EINVAL;
    for (int j = 0; j < n; ++j)
        for (int t = 0; t < st->kv_width; ++t) {
            double kk = st->k[kv_off(st, row, layer, start + j) + t];
            double vv = st->v[kv_off(st, row, layer, start + j) + t];
            size_t o = (size_t)j * st->kv_width + t;
            if (k16) k16[o] = or_f64_to_f16(kk);
            if (v16) v16[o] = or_f64_to_f16(vv);
            if (k64) k64[o] = kk;
            if (v64) v64[o] = vv;
        }
    return OR_OK;
}

/* Physical trim: keep entry j of the row iff keep[j] != 0 (j < len, where
   len must equal the row's length), shifting kept entries down in order. */
int or_trim(or_state* st, int row, const uint8_t* keep, int len) {
    if (!st || row < 0 || row >= st->n_rows || !keep || len != st->len[row]) return OR_EINVAL;
    int w = 0;
    for (int j = 0; j < len; ++j) {
        if (!keep[j]) continue;
        if (w != j)
            for (int l = 0; l < st->n_layers; ++l) {
                memmove(&st->k[kv_off(st, row, l, w)], &st->k[kv_off(st, row, l, j)], sizeof(double) * st->kv_width);
                memmove(&st->v[kv_off(st, row, l, w)], &st->v[kv_off(st, row, l, j)], sizeof(double) * st->kv_width);
            }
        ++w;
    }
    st->len[row] = w;
    return OR_OK;
}

/* ------------------------------------------------------------------------- */
/* One decode step of the shard                                              */
/* ------------------------------------------------------------------------- */
/*
 * Tokens: M = sum_b n_new[b]; tokens of request b are consecutive, request 0
 * first.  Token t is the i-th new token of its request b.
 * Inputs: hidden_in fp16 [M][H] (or token_ids [M] with the shard's
 * embedding), position_ids [M], attention_mask uint8 [B][mask_stride],
 * beam_idx [B] or NULL (identity).
 * With P_b the length of row b after the beam gather, token i of request b
 * is stored at cache index P_b + i and attends to cache indices j <= P_b + i
 * of row b with attention_mask[b][j] = 1.
 * Output: fp16 [M][H] (round_points or not) and, if out64 is given, the
 * un-rounded fp64 residual stream.
 */
static int step_core(const or_shard* sh, or_state* st, const uint16_t* hidden_in, const int32_t* token_ids,
                     const int32_t* n_new, int B, const int32_t* position_ids, const uint8_t* mask, int mask_stride,
                     const int32_t* beam_idx, int round_points, uint16_t* out16, double* out64, int packed) {
    if (!sh || !st || !n_new || !position_ids || !mask || B < 1 || B > st->n_rows) return OR_EINVAL;
    const or_config* c = &sh->cfg;
    const int H = c->hidden, Hq = c->n_heads, Hkv = c->n_kv_heads, d = c->head_dim, F = c->ffn;
    const int grp = Hq / Hkv, dq = Hq * d, dkv = Hkv * d;
    if ((hidden_in == NULL) == (token_ids == NULL)) return OR_EINVAL;
    if (token_ids && (!sh->embedding || c->vocab < 1)) return OR_EINVAL;

    int M = 0;
    for (int b = 0; b < B; ++b) {
        if (n_new[b] < 1) return OR_EINVAL;
        M += n_new[b];
    }
    int* req = (int*)malloc(sizeof(int) * (size_t)M);
    int* idx = (int*)malloc(sizeof(int) * (size_t)M);
    for (int b = 0, t = 0; b < B; ++b)
        for (int i = 0; i < n_new[b]; ++i, ++t) { req[t] = b; idx[t] = i; }

    /* beam_idx gather: row b <- copy of row beam_idx[b] (all layers, length). */
    if (beam_idx) {
        for (int b = 0; b < B; ++b)
            if (beam_idx[b] < 0 || beam_idx[b] >= B) { free(req); free(idx); return OR_EINVAL; }
        size_t row_elems = (size_t)st->n_layers * st->capacity * st->kv_width;
        double* tk = (double*)malloc(sizeof(double) * row_elems * B);
        double* tv = (double*)malloc(sizeof(double) * row_elems * B);
        int* tl = (int*)malloc(sizeof(int) * B);
        if (!tk || !tv || !tl) { free(tk); free(tv); free(tl); free(req); free(idx); return OR_ENOMEM; }
        for (int b = 0; b < B; ++b) {
            memcpy(tk + row_elems * b, st->k + row_elems * beam_idx[b], sizeof(double) * row_elems);
            memcpy(tv + row_elems * b, st->v + row_elems * beam_idx[b], sizeof(double) * row_elems);
            tl[b] = st->len[beam_idx[b]];
        }
        memcpy(st->k, tk, sizeof(double) * row_elems * B);
        memcpy(st->v, tv, sizeof(double) * row_elems * B);
        memcpy(st->len, tl, sizeof(int) * B);
        free(tk); free(tv); free(tl);
    }

    /* Validate capacity and the mask on the new entries (packed: the mask
       has one row per token, and each token must open its own entry). */
    for (int b = 0; b < B; ++b) {
        int P = st->len[b];
        if (P + n_new[b] > st->capacity) { free(req); free(idx); return OR_ECAP; }
        if (P + n_new[b] > mask_stride) { free(req); free(idx); return OR_EINVAL; }
        for (int i = 0; i < n_new[b]; ++i) {
            const size_t r = packed ? (size_t)i : (size_t)b;
            if (!mask[r * mask_stride + P + i]) { free(req); free(idx); return OR_EINVAL; }
        }
    }

    double* x = (double*)malloc(sizeof(double) * (size_t)M * H);      /* residual stream */
    double* xn = (double*)malloc(sizeof(double) * (size_t)M * H);     /* normed activations */
    double* q = (double*)malloc(sizeof(double) * (size_t)M * dq);
    double* kk = (double*)malloc(sizeof(double) * (size_t)M * dkv);
    double* vv = (double*)malloc(sizeof(double) * (size_t)M * dkv);
    double* att = (double*)malloc(sizeof(double) * (size_t)M * dq);
    double* y = (double*)malloc(sizeof(double) * (size_t)M * (H > F ? H : F));
    double* g = (double*)malloc(sizeof(double) * (size_t)M * F);
    double* u = (double*)malloc(sizeof(double) * (size_t)M * F);
    int maxlen = 0;
    for (int b = 0; b < B; ++b) if (st->len[b] + n_new[b] > maxlen) maxlen = st->len[b] + n_new[b];
    uint8_t* vis = (uint8_t*)malloc((size_t)maxlen + 1);
    int* P0 = (int*)malloc(sizeof(int) * B);
    for (int b = 0; b < B; ++b) P0[b] = st->len[b];

    for (int t = 0; t < M; ++t)
        for (int i = 0; i < H; ++i)
            x[(size_t)t * H + i] = token_ids ? or_f16_to_f64(sh->embedding[(size_t)token_ids[t] * H + i])
                                             : or_f16_to_f64(hidden_in[(size_t)t * H + i]);

#define R1(v) (round_points ? or_round_f16(v) : (v))
    for (int l = 0; l < c->n_layers; ++l) {
        const or_layer* ly = &sh->layers[l];
        /* attention block */
        for (int t = 0; t < M; ++t) {
            or_rmsnorm(x + (size_t)t * H, H, ly->attn_norm, c->rms_eps, xn + (size_t)t * H);
            for (int i = 0; i < H; ++i) xn[(size_t)t * H + i] = R1(xn[(size_t)t * H + i]);
        }
        or_gemv(&ly->w[MAT_Q], dq, H, c->group, xn, M, q);
        or_gemv(&ly->w[MAT_K], dkv, H, c->group, xn, M, kk);
        or_gemv(&ly->w[MAT_V], dkv, H, c->group, xn, M, vv);
        for (int t = 0; t < M; ++t) {
            for (int h = 0; h < Hq; ++h) or_rope(q + (size_t)t * dq + h * d, d, position_ids[t], c->rope_theta);
            for (int h = 0; h < Hkv; ++h) or_rope(kk + (size_t)t * dkv + h * d, d, position_ids[t], c->rope_theta);
            /* append at cache index P_b + i */
            size_t o = kv_off(st, req[t], l, P0[req[t]] + idx[t]);
            for (int e = 0; e < dkv; ++e) {
                st->k[o + e] = R1(kk[(size_t)t * dkv + e]);
                st->v[o + e] = R1(vv[(size_t)t * dkv + e]);
            }
        }
        for (int t = 0; t < M; ++t) {
            /* per request: entries j <= P_b + i with mask[b][j] = 1;
               packed: every entry of the row (old and new) with mask[t][j] = 1 */
            int b = req[t], last = packed ? P0[b] + n_new[b] - 1 : P0[b] + idx[t];
            for (int j = 0; j <= last; ++j)
                vis[j] = mask[(size_t)(packed ? t : b) * mask_stride + j] ? 1 : 0;
            for (int h = 0; h < Hq; ++h) {
                int hk = h / grp;
                const double* K = st->k + kv_off(st, b, l, 0) + hk * d;
                const double* V = st->v + kv_off(st, b, l, 0) + hk * d;
                or_attend(q + (size_t)t * dq + h * d, K, V, last + 1, dkv, d, vis, att + (size_t)t * dq + h * d);
            }
            for (int e = 0; e < dq; ++e) att[(size_t)t * dq + e] = R1(att[(size_t)t * dq + e]);
        }
        or_gemv(&ly->w[MAT_O], H, dq, c->group, att, M, y);
        for (size_t e = 0; e < (size_t)M * H; ++e) x[e] += y[e];
        /* MLP block */
        for (int t = 0; t < M; ++t) {
            or_rmsnorm(x + (size_t)t * H, H, ly->ffn_norm, c->rms_eps, xn + (size_t)t * H);
            for (int i = 0; i < H; ++i) xn[(size_t)t * H + i] = R1(xn[(size_t)t * H + i]);
        }
        or_gemv(&ly->w[MAT_GATE], F, H, c->group, xn, M, g);
        or_gemv(&ly->w[MAT_UP], F, H, c->group, xn, M, u);
        for (size_t e = 0; e < (size_t)M * F; ++e) g[e] = R1(or_silu(g[e]) * u[e]);
        or_gemv(&ly->w[MAT_DOWN], H, F, c->group, g, M, y);
        for (size_t e = 0; e < (size_t)M * H; ++e) x[e] += y[e];
    }
#undef R1
    for (int b = 0; b < B; ++b) st->len[b] = P0[b] + n_new[b];
    for (size_t e = 0; e < (size_t)M * H; ++e) {
        if (out16) out16[e] = or_f64_to_f16(x[e]);
        if (out64) out64[e] = x[e];
    }
    free(x); free(xn); free(q); free(kk); free(vv); free(att); free(y); free(g); free(u);
    free(vis); free(P0); free(req); free(idx);
    return OR_OK;
}

int or_step(const or_shard* sh, or_state* st, const uint16_t* hidden_in, const int32_t* token_ids,
            const int32_t* n_new, int B, const int32_t* position_ids, const uint8_t* mask, int mask_stride,
            const int32_t* beam_idx, int round_points, uint16_t* out16, double* out64) {
    return step_core(sh, st, hidden_in, token_ids, n_new, B, position_ids, mask, mask_stride, beam_idx, round_points,
                     out16, out64, 0);
}

/*
 * Packed step (Section 8.6, continuous batching through the mask layout):
 * S query rows share ONE cache row (row 0 of the state), whose entries the
 * host has partitioned into regions -- an optional shared prefix, then one
 * region per slot.  The S new entries are appended after the existing ones,
 * token t at index P + t, and token t attends to exactly the entries j < P + S
 * with mask2d[t][j] != 0 (mask2d [S][mask_stride]): its own slot's region,
 * the shared prefix, and the new entries of its own slot at or before it, so
 * that several rows of one slot form a causal chunk and rows of different
 * slots are isolated.  Every token must open its own new entry (an idle row
 * opens only that one; a fully masked row would have no softmax).  RoPE uses
 * position_ids, each slot's absolute positions.  Otherwise the layer math is
 * that of or_step.
 */
int or_step_packed(const or_shard* sh, or_state* st, const uint16_t* hidden_in, const int32_t* token_ids, int S,
                   const int32_t* position_ids, const uint8_t* mask2d, int mask_stride, int round_points,
                   uint16_t* out16, double* out64) {
    if (S < 1) return OR_EINVAL;
    const int32_t n_new[1] = {S};
    return step_core(sh, st, hidden_in, token_ids, n_new, 1, position_ids, mask2d, mask_stride, NULL, round_points,
                     out16, out64, 1);
}

/* Test head for greedy-token checks (not part of the shard): logits of the
   tied embedding after an un-weighted RMSNorm,
   logits[t][v] = sum_i E[v][i] * rmsnorm(h[t])[i]. */
void or_logits(const double* h, int M, int H, const uint16_t* E, int V, double eps, double* logits) {
    double* hn = (double*)malloc(sizeof(double) * (size_t)H);
    for (int t = 0; t < M; ++t) {
        or_rmsnorm(h + (size_t)t * H, H, NULL, eps, hn);
        #pragma omp parallel for schedule(static) num_threads(g_threads)
        for (int v = 0; v < V; ++v) {
            double acc = 0.0;
            for (int i = 0; i < H; ++i) acc += or_f16_to_f64(E[(size_t)v * H + i]) * hn[i];
            logits[(size_t)t * V + v] = acc;
        }
    }
    free(hn);
}

/* ------------------------------------------------------------------------- */
/* LM head of a final stage with the top-1 epilogue [Section 6.7]            */
/* ------------------------------------------------------------------------- */

/* For each fp16 hidden row h[t] (t < M):
     x          = rmsnorm(h[t]) * w_norm, rounded to fp16 when round_points
                  (the projection's 16-bit activation operand),
     logits[v]  = sum_i W[v][i] * x[i]   (W the INT4 lm_head, [V][H]),
     token[t]   = the v with the largest logit (the lowest such v on ties),
     p_max[t]   = its softmax probability, 1 / sum_v exp(logits[v] - max),
     margin[t]  = max minus the second largest logit (0 on a tie; for V = 1,
                  +inf).
   Only (token, p_max) are what the final stage sends back in the paper's
   top-1 compression; margin is for tolerance gating in tests.  logits_out
   (nullable) receives [M][V]. */
void or_head_top1(const uint16_t* h16, int M, int H, const uint16_t* w_norm, double eps, const or_matrix* W, int V,
                  int group, int round_points, int32_t* token, double* p_max, double* margin, double* logits_out) {
    double* hx = (double*)malloc(sizeof(double) * (size_t)H);
    double* x = (double*)malloc(sizeof(double) * (size_t)M * H);
    double* lg = (double*)malloc(sizeof(double) * (size_t)M * V);
    for (int t = 0; t < M; ++t) {
        for (int i = 0; i < H; ++i) hx[i] = or_f16_to_f64(h16[(size_t)t * H + i]);
        or_rmsnorm(hx, H, w_norm, eps, x + (size_t)t * H);
        if (round_points)
            for (int i = 0; i < H; ++i) x[(size_t)t * H + i] = or_round_f16(x[(size_t)t * H + i]);
    }
    or_gemv(W, V, H, group, x, M, lg);
    for (int t = 0; t < M; ++t) {
        const double* l = lg + (size_t)t * V;
        int best = 0;
        for (int v = 1; v < V; ++v)
            if (l[v] > l[best]) best = v;
        double second = -INFINITY;
        for (int v = 0; v < V; ++v)
            if (v != best && l[v] > second) second = l[v];
        double den = 0.0;
        for (int v = 0; v < V; ++v) den += exp(l[v] - l[best]);
        token[t] = best;
        p_max[t] = 1.0 / den;
        margin[t] = l[best] - second;
    }
    if (logits_out) memcpy(logits_out, lg, sizeof(double) * (size_t)M * V);
    free(hx);
    free(x);
    free(lg);
}
