/*
 * CPU oracle for one tensor-parallel shard of a Llama-style decoder layer.
 *
 * TEST INFRASTRUCTURE.  Only the tests, the smoke check and the benchmark's CPU-baseline leg
 * load this library.  It shares no code, header, table or constant with the GPU library.
 *
 * Plain loops in fp64.  OpenMP splits only loops whose iterations are independent (output rows
 * of a matrix-vector product, attention heads); every sum is a sequential accumulation in index
 * order.  Citations are to the Voltron paper (arXiv 2607.07046):
 *   - Section 2.1, "LLM Architecture": stacked decoders; attention heads computed independently
 *     with scaled dot-product of Q, K, V; output linear O; FFN projecting up, applying a
 *     nonlinearity and projecting back; GQA shares K/V projections across query-head groups.
 *   - Section 2.1, "LLM Inference": prefill processes the prompt tokens and stores their K and V
 *     in the KV cache; each decode iteration attends to the cache and appends its own K and V.
 *   - Section 3.2.1, tensor parallelism: the main device broadcasts the layer input, each device
 *     computes its shard, and the results are aggregated on the main device.
 * The Llama-specific forms (RMSNorm, rotate-half RoPE, SwiGLU, no biases) follow the workload
 * definitions of the target models; the paper names the models but not these formulas.
 */
#include "oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

#ifdef _OPENMP
#include <omp.h>
#endif

/* ---------------------------------------------------------------- binary16 ---------------- */

/* binary16: 1 sign bit, 5 exponent bits (bias 15), 10 fraction bits.
 * exponent 0 -> subnormal  (-1)^s * f * 2^-24
 * exponent 31 -> inf / nan
 * otherwise   -> (-1)^s * (1024 + f) * 2^(e - 25)                                           */
double or_f16_to_f64(uint16_t h) {
    const int s = h >> 15, e = (h >> 10) & 31, f = h & 1023;
    double mag;
    if (e == 0)
        mag = ldexp((double)f, -24);
    else if (e == 31)
        mag = f ? NAN : INFINITY;
    else
        mag = ldexp((double)(f + 1024), e - 25);
    return s ? -mag : mag;
}

/* Round-to-nearest-even encoding.  rint() rounds to even in the default rounding mode, and the
 * scalings by powers of two are exact, so there is a single rounding. */
uint16_t or_f64_to_f16(double x) {
    if (isnan(x)) return 0x7e00;
    const uint16_t sign = signbit(x) ? 0x8000 : 0;
    const double a = fabs(x);
    if (a >= 65520.0) return sign | 0x7c00;            /* halfway above 65504 rounds to inf */
    if (a < 0x1p-14) {                                  /* subnormal range, quantum 2^-24 */
        const double q = rint(a * 0x1p24);              /* q == 1024 is the smallest normal */
        return sign | (uint16_t)q;
    }
    int k;
    frexp(a, &k);                                       /* a = m 2^k, m in [0.5, 1) */
    int E = k - 1;                                      /* a in [2^E, 2^(E+1)) */
    double q = rint(ldexp(a, 10 - E));                  /* 11-bit significand in [1024, 2048] */
    if (q == 2048.0) {
        q = 1024.0;
        E += 1;
    }
    if (E + 15 >= 31) return sign | 0x7c00;
    return sign | (uint16_t)(((E + 15) << 10) | ((int)q - 1024));
}

/* Decoding table, filled from or_f16_to_f64 when the library is loaded. */
static double g_half[65536];

__attribute__((constructor)) static void or_fill_table(void) {
    for (int i = 0; i < 65536; ++i) g_half[i] = or_f16_to_f64((uint16_t)i);
}

#define HALF(b) (g_half[(b)])

int32_t or_num_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

void or_set_threads(int32_t n) {
#ifdef _OPENMP
    if (n > 0) omp_set_num_threads(n);
#else
    (void)n;
#endif
}

/* ---------------------------------------------------------------- building blocks --------- */

void or_rmsnorm(const double* x, const uint16_t* gain, int32_t n, double eps, double* y) {
    double ss = 0.0;
    for (int32_t i = 0; i < n; ++i) ss += x[i] * x[i];
    const double r = 1.0 / sqrt(ss / (double)n + eps);
    for (int32_t i = 0; i < n; ++i) y[i] = x[i] * r * HALF(gain[i]);
}

void or_rope(double* v, int32_t dh, int64_t pos, double theta) {
    const int32_t half = dh / 2;
    for (int32_t i = 0; i < half; ++i) {
        const double freq = pow(theta, -2.0 * (double)i / (double)dh);
        const double ang = (double)pos * freq;
        const double c = cos(ang), s = sin(ang);
        const double x0 = v[i], x1 = v[i + half];
        v[i] = x0 * c - x1 * s;
        v[i + half] = x0 * s + x1 * c;
    }
}

double or_silu(double z) { return z / (1.0 + exp(-z)); }

void or_attend(const double* q, const uint16_t* k, const uint16_t* v, int64_t n_pos, int32_t dh,
               double* w, double* o) {
    double* s = (double*)malloc(sizeof(double) * (size_t)(n_pos > 0 ? n_pos : 1));
    const double scale = 1.0 / sqrt((double)dh);
    double m = -INFINITY;
    for (int64_t t = 0; t < n_pos; ++t) {
        double acc = 0.0;
        for (int32_t c = 0; c < dh; ++c) acc += q[c] * HALF(k[t * dh + c]);
        s[t] = acc * scale;
        if (s[t] > m) m = s[t];
    }
    double z = 0.0;
    for (int64_t t = 0; t < n_pos; ++t) {
        s[t] = exp(s[t] - m);
        z += s[t];
    }
    for (int32_t c = 0; c < dh; ++c) o[c] = 0.0;
    for (int64_t t = 0; t < n_pos; ++t) {
        const double wt = s[t] / z;
        if (w) w[t] = wt;
        for (int32_t c = 0; c < dh; ++c) o[c] += wt * HALF(v[t * dh + c]);
    }
    free(s);
}

/* y[r] = sum_k W[r * ld + k] * x[k] for r in [0, nrows), k in [0, n). */
static void matvec(const uint16_t* W, int64_t ld, int64_t nrows, const double* x, int64_t n,
                   double* y) {
#pragma omp parallel for schedule(static)
    for (int64_t r = 0; r < nrows; ++r) {
        const uint16_t* row = W + r * ld;
        double acc = 0.0;
        for (int64_t k = 0; k < n; ++k) acc += HALF(row[k]) * x[k];
        y[r] = acc;
    }
}

static void load_row(const uint16_t* src, int32_t n, double* dst) {
    for (int32_t i = 0; i < n; ++i) dst[i] = HALF(src[i]);
}

static int shapes_ok(const or_shapes* s) {
    return s && s->d_model > 0 && s->n_heads > 0 && s->n_kv_heads > 0 && s->d_head > 0 &&
           (s->d_head % 2) == 0 && s->d_ffn >= 0 && (s->n_heads % s->n_kv_heads) == 0;
}

/* ---------------------------------------------------------------- attention block --------- */

int32_t or_kv_append(const or_shapes* s, const or_layer* w, int32_t kvh0, int32_t kvh1,
                     const uint16_t* x, int32_t rows, int64_t pos0, uint16_t* kcache,
                     uint16_t* vcache, int64_t cap) {
    if (!shapes_ok(s) || !w || kvh0 < 0 || kvh1 < kvh0 || kvh1 > s->n_kv_heads || rows < 0 ||
        pos0 < 0 || pos0 + rows > cap)
        return OR_ERR_ARG;
    const int32_t D = s->d_model, dh = s->d_head, nk = kvh1 - kvh0;
    double* xin = (double*)malloc(sizeof(double) * D);
    double* xh = (double*)malloc(sizeof(double) * D);
    double* kk = (double*)malloc(sizeof(double) * (size_t)(nk * dh + 1));
    double* vv = (double*)malloc(sizeof(double) * (size_t)(nk * dh + 1));
    for (int32_t i = 0; i < rows; ++i) {
        const int64_t p = pos0 + i;
        load_row(x + (int64_t)i * D, D, xin);
        or_rmsnorm(xin, w->attn_norm, D, s->rms_eps, xh);
        matvec(w->wk + (int64_t)kvh0 * dh * D, D, (int64_t)nk * dh, xh, D, kk);
        matvec(w->wv + (int64_t)kvh0 * dh * D, D, (int64_t)nk * dh, xh, D, vv);
        for (int32_t j = 0; j < nk; ++j) {
            or_rope(kk + (int64_t)j * dh, dh, p, s->rope_theta);
            uint16_t* kd = kcache + ((int64_t)(kvh0 + j) * cap + p) * dh;
            uint16_t* vd = vcache + ((int64_t)(kvh0 + j) * cap + p) * dh;
            for (int32_t c = 0; c < dh; ++c) {
                kd[c] = or_f64_to_f16(kk[(int64_t)j * dh + c]);
                vd[c] = or_f64_to_f16(vv[(int64_t)j * dh + c]);
            }
        }
    }
    free(xin);
    free(xh);
    free(kk);
    free(vv);
    return OR_OK;
}

int32_t or_attn_partial(const or_shapes* s, const or_layer* w, int32_t h0, int32_t h1,
                        const uint16_t* x, int32_t rows, const int64_t* pos,
                        const uint16_t* kcache, const uint16_t* vcache, int64_t cap,
                        double* partial) {
    return or_attn_partial_window(s, w, h0, h1, x, rows, pos, kcache, vcache, cap, 0, partial);
}

/* Sliding-window attention (Voltron Section 2.1 names it among the attention variants of the
 * evaluated models): row i attends to cache positions [max(0, pos - window + 1), pos]; window <= 0
 * means every position 0..pos. */
int32_t or_attn_partial_window(const or_shapes* s, const or_layer* w, int32_t h0, int32_t h1,
                               const uint16_t* x, int32_t rows, const int64_t* pos,
                               const uint16_t* kcache, const uint16_t* vcache, int64_t cap,
                               int64_t window, double* partial) {
    if (!shapes_ok(s) || !w || h0 < 0 || h1 < h0 || h1 > s->n_heads || rows < 0) return OR_ERR_ARG;
    for (int32_t i = 0; i < rows; ++i)
        if (pos[i] < 0 || pos[i] >= cap) return OR_ERR_ARG;
    const int32_t D = s->d_model, dh = s->d_head, H = s->n_heads, nh = h1 - h0;
    const int32_t group = s->n_heads / s->n_kv_heads;
    double* xin = (double*)malloc(sizeof(double) * D);
    double* xh = (double*)malloc(sizeof(double) * D);
    double* q = (double*)malloc(sizeof(double) * (size_t)(nh * dh + 1));
    double* o = (double*)malloc(sizeof(double) * (size_t)(nh * dh + 1));
    for (int32_t i = 0; i < rows; ++i) {
        double* out = partial + (int64_t)i * D;
        if (nh == 0) {
            for (int32_t d = 0; d < D; ++d) out[d] = 0.0;
            continue;
        }
        load_row(x + (int64_t)i * D, D, xin);
        or_rmsnorm(xin, w->attn_norm, D, s->rms_eps, xh);
        matvec(w->wq + (int64_t)h0 * dh * D, D, (int64_t)nh * dh, xh, D, q);
        for (int32_t h = 0; h < nh; ++h) or_rope(q + (int64_t)h * dh, dh, pos[i], s->rope_theta);
        const int64_t first = window > 0 && pos[i] + 1 > window ? pos[i] + 1 - window : 0;
#pragma omp parallel for schedule(static)
        for (int32_t h = 0; h < nh; ++h) {
            const int32_t j = (h0 + h) / group;
            or_attend(q + (int64_t)h * dh, kcache + ((int64_t)j * cap + first) * dh,
                      vcache + ((int64_t)j * cap + first) * dh, pos[i] + 1 - first, dh, NULL,
                      o + (int64_t)h * dh);
        }
        /* partial[d] = sum over the range's columns of Wo[d][h0*dh + k] * o[k] */
        matvec(w->wo + (int64_t)h0 * dh, (int64_t)H * dh, D, o, (int64_t)nh * dh, out);
    }
    free(xin);
    free(xh);
    free(q);
    free(o);
    return OR_OK;
}

/* ---------------------------------------------------------------- FFN block --------------- */

int32_t or_ffn_partial(const or_shapes* s, const or_layer* w, int32_t c0, int32_t c1,
                       const uint16_t* h, int32_t rows, double* partial) {
    if (!shapes_ok(s) || !w || c0 < 0 || c1 < c0 || c1 > s->d_ffn || rows < 0) return OR_ERR_ARG;
    const int32_t D = s->d_model, F = s->d_ffn, nc = c1 - c0;
    double* hin = (double*)malloc(sizeof(double) * D);
    double* hh = (double*)malloc(sizeof(double) * D);
    double* g = (double*)malloc(sizeof(double) * (size_t)(nc + 1));
    double* u = (double*)malloc(sizeof(double) * (size_t)(nc + 1));
    for (int32_t i = 0; i < rows; ++i) {
        double* out = partial + (int64_t)i * D;
        if (nc == 0) {
            for (int32_t d = 0; d < D; ++d) out[d] = 0.0;
            continue;
        }
        load_row(h + (int64_t)i * D, D, hin);
        or_rmsnorm(hin, w->ffn_norm, D, s->rms_eps, hh);
        matvec(w->w_gate + (int64_t)c0 * D, D, nc, hh, D, g);
        matvec(w->w_up + (int64_t)c0 * D, D, nc, hh, D, u);
        for (int32_t j = 0; j < nc; ++j) g[j] = or_silu(g[j]) * u[j];
        matvec(w->w_down + c0, F, D, g, nc, out);
    }
    free(hin);
    free(hh);
    free(g);
    free(u);
    return OR_OK;
}

/* ---------------------------------------------------------------- aggregation ------------- */

void or_combine(const double* const* partials, int32_t n, int64_t count, const uint16_t* residual,
                uint16_t* out) {
#pragma omp parallel for schedule(static)
    for (int64_t e = 0; e < count; ++e) {
        double acc = residual ? HALF(residual[e]) : 0.0;
        for (int32_t sidx = 0; sidx < n; ++sidx) acc += partials[sidx][e];
        out[e] = or_f64_to_f16(acc);
    }
}

/* ---------------------------------------------------------------- block quantization ------ */
/* Mixed-precision weight shards (Voltron Section 3.2.2, precision heterogeneity; Section 4.2.2;
 * Section 5.1 adopts k-quant formats without defining them).  Reading: each row of a weight
 * matrix is cut into blocks of `block` consecutive weights along the input dimension; a block
 * keeps one binary16 scale d = binary16(amax / qmax), amax the largest |w| of the block, qmax 127
 * (8 bits) or 7 (4 bits), and one signed code per weight, q = round-half-even(w / d) clamped to
 * [-qmax, qmax] (q = 0 when d = 0).  The decision is taken in binary32 arithmetic (the division
 * amax / qmax and w / d), the precision the library's quantizer uses, so both give the same codes.
 * The dequantized weight is q * d. */

int32_t or_quantize_rows(const uint16_t* w, int64_t rows, int64_t k, int32_t bits, int32_t block, int8_t* q,
                         uint16_t* scales) {
    if (!w || !q || !scales || rows < 0 || k < 0 || block < 1 || (bits != 8 && bits != 4)) return OR_ERR_ARG;
    const int32_t qmax = bits == 8 ? 127 : 7;
    const int64_t nb = (k + block - 1) / block;
#pragma omp parallel for schedule(static)
    for (int64_t r = 0; r < rows; ++r) {
        for (int64_t b = 0; b < nb; ++b) {
            const int64_t e0 = b * block, e1 = e0 + block < k ? e0 + block : k;
            float amax = 0.0f;
            for (int64_t e = e0; e < e1; ++e) {
                const float v = fabsf((float)or_f16_to_f64(w[r * k + e]));
                if (v > amax) amax = v;
            }
            const float t = amax / (float)qmax;            /* binary32 division */
            const uint16_t d16 = or_f64_to_f16((double)t);  /* exact widening, then round to binary16 */
            const float d = (float)or_f16_to_f64(d16);
            scales[r * nb + b] = d16;
            for (int64_t e = e0; e < e1; ++e) {
                int32_t c = 0;
                if (d != 0.0f) {
                    const float x = (float)or_f16_to_f64(w[r * k + e]) / d;  /* binary32 division */
                    const float rx = nearbyintf(x);                          /* ties to even */
                    c = rx > (float)qmax ? qmax : (rx < (float)-qmax ? -qmax : (int32_t)rx);
                }
                q[r * k + e] = (int8_t)c;
            }
        }
    }
    return OR_OK;
}

/* y[r] = sum_e (q[r][e] * d[r][e / block]) * x[e] in binary64, e in index order. */
void or_gemv_blockq(const int8_t* q, const uint16_t* scales, int64_t rows, int64_t k, int32_t block,
                    const double* x, double* y) {
    const int64_t nb = (k + block - 1) / block;
#pragma omp parallel for schedule(static)
    for (int64_t r = 0; r < rows; ++r) {
        double acc = 0.0;
        for (int64_t e = 0; e < k; ++e) acc += (double)q[r * k + e] * or_f16_to_f64(scales[r * nb + e / block]) * x[e];
        y[r] = acc;
    }
}

/* ---------------------------------------------------------------- quantized shards -------- */
/* The layer steps of the attention and FFN blocks with every projection by a dequantized,
 * block-quantized matrix (or_gemv_blockq); everything else is as in the binary16 functions above. */

static int qmat_ok(const or_qmat* m, int64_t rows, int64_t k) {
    return m && m->q && m->scales && m->block >= 1 && m->rows == rows && m->k == k;
}

int32_t or_kv_append_q(const or_shapes* s, const uint16_t* attn_norm, const or_qmat* wk, const or_qmat* wv,
                       int32_t kvh0, int32_t kvh1, const uint16_t* x, int32_t rows, int64_t pos0, uint16_t* kcache,
                       uint16_t* vcache, int64_t cap) {
    if (!shapes_ok(s) || !attn_norm || kvh0 < 0 || kvh1 < kvh0 || kvh1 > s->n_kv_heads || rows < 0 || pos0 < 0 ||
        pos0 + rows > cap)
        return OR_ERR_ARG;
    const int32_t D = s->d_model, dh = s->d_head, nk = kvh1 - kvh0;
    if (!qmat_ok(wk, (int64_t)nk * dh, D) || !qmat_ok(wv, (int64_t)nk * dh, D)) return OR_ERR_ARG;
    double* xin = (double*)malloc(sizeof(double) * D);
    double* xh = (double*)malloc(sizeof(double) * D);
    double* kk = (double*)malloc(sizeof(double) * (size_t)(nk * dh + 1));
    double* vv = (double*)malloc(sizeof(double) * (size_t)(nk * dh + 1));
    for (int32_t i = 0; i < rows; ++i) {
        const int64_t p = pos0 + i;
        load_row(x + (int64_t)i * D, D, xin);
        or_rmsnorm(xin, attn_norm, D, s->rms_eps, xh);
        or_gemv_blockq(wk->q, wk->scales, wk->rows, wk->k, wk->block, xh, kk);
        or_gemv_blockq(wv->q, wv->scales, wv->rows, wv->k, wv->block, xh, vv);
        for (int32_t j = 0; j < nk; ++j) {
            or_rope(kk + (int64_t)j * dh, dh, p, s->rope_theta);
            uint16_t* kd = kcache + ((int64_t)(kvh0 + j) * cap + p) * dh;
            uint16_t* vd = vcache + ((int64_t)(kvh0 + j) * cap + p) * dh;
            for (int32_t c = 0; c < dh; ++c) {
                kd[c] = or_f64_to_f16(kk[(int64_t)j * dh + c]);
                vd[c] = or_f64_to_f16(vv[(int64_t)j * dh + c]);
            }
        }
    }
    free(xin);
    free(xh);
    free(kk);
    free(vv);
    return OR_OK;
}

int32_t or_attn_partial_q(const or_shapes* s, const uint16_t* attn_norm, const or_qmat* wq, const or_qmat* wo,
                          int32_t h0, int32_t h1, const uint16_t* x, int32_t rows, const int64_t* pos,
                          const uint16_t* kcache, const uint16_t* vcache, int64_t cap, int64_t window,
                          double* partial) {
    if (!shapes_ok(s) || !attn_norm || h0 < 0 || h1 < h0 || h1 > s->n_heads || rows < 0) return OR_ERR_ARG;
    const int32_t D = s->d_model, dh = s->d_head, nh = h1 - h0;
    const int32_t group = s->n_heads / s->n_kv_heads;
    if (nh > 0 && (!qmat_ok(wq, (int64_t)nh * dh, D) || !qmat_ok(wo, D, (int64_t)nh * dh))) return OR_ERR_ARG;
    for (int32_t i = 0; i < rows; ++i)
        if (pos[i] < 0 || pos[i] >= cap) return OR_ERR_ARG;
    double* xin = (double*)malloc(sizeof(double) * D);
    double* xh = (double*)malloc(sizeof(double) * D);
    double* q = (double*)malloc(sizeof(double) * (size_t)(nh * dh + 1));
    double* o = (double*)malloc(sizeof(double) * (size_t)(nh * dh + 1));
    for (int32_t i = 0; i < rows; ++i) {
        double* out = partial + (int64_t)i * D;
        if (nh == 0) {
            for (int32_t d = 0; d < D; ++d) out[d] = 0.0;
            continue;
        }
        load_row(x + (int64_t)i * D, D, xin);
        or_rmsnorm(xin, attn_norm, D, s->rms_eps, xh);
        or_gemv_blockq(wq->q, wq->scales, wq->rows, wq->k, wq->block, xh, q);
        for (int32_t h = 0; h < nh; ++h) or_rope(q + (int64_t)h * dh, dh, pos[i], s->rope_theta);
        const int64_t first = window > 0 && pos[i] + 1 > window ? pos[i] + 1 - window : 0;
#pragma omp parallel for schedule(static)
        for (int32_t h = 0; h < nh; ++h) {
            const int32_t j = (h0 + h) / group;
            or_attend(q + (int64_t)h * dh, kcache + ((int64_t)j * cap + first) * dh,
                      vcache + ((int64_t)j * cap + first) * dh, pos[i] + 1 - first, dh, NULL, o + (int64_t)h * dh);
        }
        or_gemv_blockq(wo->q, wo->scales, wo->rows, wo->k, wo->block, o, out);
    }
    free(xin);
    free(xh);
    free(q);
    free(o);
    return OR_OK;
}

int32_t or_ffn_partial_q(const or_shapes* s, const uint16_t* ffn_norm, const or_qmat* wg, const or_qmat* wu,
                         const or_qmat* wd, int32_t nc, const uint16_t* h, int32_t rows, double* partial) {
    if (!shapes_ok(s) || !ffn_norm || nc < 0 || rows < 0) return OR_ERR_ARG;
    const int32_t D = s->d_model;
    if (nc > 0 && (!qmat_ok(wg, nc, D) || !qmat_ok(wu, nc, D) || !qmat_ok(wd, D, nc))) return OR_ERR_ARG;
    double* hin = (double*)malloc(sizeof(double) * D);
    double* hh = (double*)malloc(sizeof(double) * D);
    double* g = (double*)malloc(sizeof(double) * (size_t)(nc + 1));
    double* u = (double*)malloc(sizeof(double) * (size_t)(nc + 1));
    for (int32_t i = 0; i < rows; ++i) {
        double* out = partial + (int64_t)i * D;
        if (nc == 0) {
            for (int32_t d = 0; d < D; ++d) out[d] = 0.0;
            continue;
        }
        load_row(h + (int64_t)i * D, D, hin);
        or_rmsnorm(hin, ffn_norm, D, s->rms_eps, hh);
        or_gemv_blockq(wg->q, wg->scales, wg->rows, wg->k, wg->block, hh, g);
        or_gemv_blockq(wu->q, wu->scales, wu->rows, wu->k, wu->block, hh, u);
        for (int32_t j = 0; j < nc; ++j) g[j] = or_silu(g[j]) * u[j];
        or_gemv_blockq(wd->q, wd->scales, wd->rows, wd->k, wd->block, g, out);
    }
    free(hin);
    free(hh);
    free(g);
    free(u);
    return OR_OK;
}

/* ---------------------------------------------------------------- quantized partials ------ */
/* Communication scaling (Voltron Section 4.3.2): activations sent between devices are lowered to
 * INT8 or INT4.  Under tensor parallelism those are the shard partials sent to the main device.
 * Reading: the same block format as the weights (blocks of `block` values, fp16 scale
 * d = fp16(amax / qmax), codes round-half-even(x / d) clamped to [-qmax, qmax], binary32
 * decisions), applied to the binary32 partial as it leaves the device; the main device adds the
 * dequantized partials to the residual. */

int32_t or_quantize_vec(const float* x, int64_t n, int32_t bits, int32_t block, int8_t* q, uint16_t* scales) {
    if (!x || !q || !scales || n < 0 || block < 1 || (bits != 8 && bits != 4)) return OR_ERR_ARG;
    const int32_t qmax = bits == 8 ? 127 : 7;
    const int64_t nb = (n + block - 1) / block;
    for (int64_t b = 0; b < nb; ++b) {
        const int64_t e0 = b * block, e1 = e0 + block < n ? e0 + block : n;
        float amax = 0.0f;
        for (int64_t e = e0; e < e1; ++e)
            if (fabsf(x[e]) > amax) amax = fabsf(x[e]);
        const uint16_t d16 = or_f64_to_f16((double)(amax / (float)qmax));
        const float d = (float)or_f16_to_f64(d16);
        scales[b] = d16;
        for (int64_t e = e0; e < e1; ++e) {
            int32_t c = 0;
            if (d != 0.0f) {
                const float rx = nearbyintf(x[e] / d);
                c = rx > (float)qmax ? qmax : (rx < (float)-qmax ? -qmax : (int32_t)rx);
            }
            q[e] = (int8_t)c;
        }
    }
    return OR_OK;
}

/* out = binary16(residual + sum_s q_s * d_s) elementwise, shards in order s = 0..n-1, binary64
 * sums; q[s] / scales[s] as written by or_quantize_vec for `count` values. */
void or_combine_q(const int8_t* const* q, const uint16_t* const* scales, int32_t n, int64_t count, int32_t block,
                  const uint16_t* residual, uint16_t* out) {
#pragma omp parallel for schedule(static)
    for (int64_t e = 0; e < count; ++e) {
        double acc = residual ? HALF(residual[e]) : 0.0;
        for (int32_t s = 0; s < n; ++s) acc += (double)q[s][e] * or_f16_to_f64(scales[s][e / block]);
        out[e] = or_f64_to_f16(acc);
    }
}
