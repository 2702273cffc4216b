/*
 * CPU oracle for one tensor-parallel shard of a Llama-style decoder layer.
 *
 * TEST INFRASTRUCTURE.  Only the tests, the smoke check and the benchmark's CPU-baseline leg
 * load this library; the GPU library never links or calls it, and the two share no code.
 *
 * What it computes (Voltron, Section 2.1 "LLM Architecture" and "LLM Inference";
 * Section 3.2.1 on tensor parallelism): a decoder layer is an attention block (ATTN) followed by a
 * feed-forward block (FFN).  Under tensor parallelism every device receives the same input,
 * computes its shard (a subset of attention heads, or a subset of FFN intermediate columns) and
 * the shard results are summed on the main device.  The oracle evaluates the plain definition of
 * each block restricted to a head range or a column range, so the full layer is the range that
 * covers every head / column.
 *
 * Arithmetic: fp64 throughout.  fp16 appears only where the data contract fixes it: weights and
 * activations arrive as IEEE binary16 bit patterns, the KV cache stores binary16, and the
 * combined hidden state is rounded to binary16.
 */
#ifndef VT_ORACLE_H
#define VT_ORACLE_H

#include <stdint.h>

typedef struct {
    int32_t d_model;    /* D  */
    int32_t n_heads;    /* H  (query heads) */
    int32_t n_kv_heads; /* Hk (key/value heads; H must be a multiple) */
    int32_t d_head;     /* dh (even) */
    int32_t d_ffn;      /* F  */
    double rms_eps;
    double rope_theta;
} or_shapes;

/* One layer's weights as binary16 bit patterns, nn.Linear layout [out][in], row-major. */
typedef struct {
    const uint16_t* attn_norm; /* [D]        */
    const uint16_t* wq;        /* [H*dh, D]  */
    const uint16_t* wk;        /* [Hk*dh, D] */
    const uint16_t* wv;        /* [Hk*dh, D] */
    const uint16_t* wo;        /* [D, H*dh]  */
    const uint16_t* ffn_norm;  /* [D]        */
    const uint16_t* w_gate;    /* [F, D]     */
    const uint16_t* w_up;      /* [F, D]     */
    const uint16_t* w_down;    /* [D, F]     */
} or_layer;

/* Status codes of the block functions. */
#define OR_OK 0
#define OR_ERR_ARG 1

int32_t or_num_threads(void);
void or_set_threads(int32_t n);

/* IEEE 754-2008 binary16 <-> binary64. Decoding is exact; encoding rounds to nearest even. */
double or_f16_to_f64(uint16_t h);
uint16_t or_f64_to_f16(double x);

/* y = x * g / sqrt(mean(x^2) + eps) over n elements (RMSNorm, Llama form). */
void or_rmsnorm(const double* x, const uint16_t* gain, int32_t n, double eps, double* y);

/* Rotary position embedding of one head vector at position pos, rotate-half pairing:
 * (v_i, v_{i+dh/2}) is turned by the angle pos * theta^(-2i/dh), i < dh/2. */
void or_rope(double* v, int32_t dh, int64_t pos, double theta);

/* silu(z) = z / (1 + exp(-z)). */
double or_silu(double z);

/* One head of scaled dot-product attention over n_pos cached binary16 keys/values (position-major,
 * dh elements per position): w = softmax(q.K^T / sqrt(dh)), o = w.V.  w may be NULL. */
void or_attend(const double* q, const uint16_t* k, const uint16_t* v, int64_t n_pos, int32_t dh,
               double* w, double* o);

/* Key/value projection of `rows` input rows (binary16 [rows, D]) for KV heads [kvh0, kvh1):
 * RMSNorm, k = Wk x^, v = Wv x^, RoPE on k at position pos0 + row, binary16 store into the
 * full-layer caches kcache/vcache [Hk, cap, dh]. */
int32_t or_kv_append(const or_shapes* s, const or_layer* w, int32_t kvh0, int32_t kvh1,
                     const uint16_t* x, int32_t rows, int64_t pos0, uint16_t* kcache,
                     uint16_t* vcache, int64_t cap);

/* Attention-block partial output of query heads [h0, h1) for `rows` rows (binary16 [rows, D]):
 * RMSNorm, q = Wq x^, RoPE at pos[row], causal attention over cache positions 0..pos[row]
 * (KV head of query head h is h / (H/Hk)), then partial = Wo[:, h0*dh : h1*dh] . o.
 * partial is fp64 [rows, D] and excludes the residual. */
int32_t or_attn_partial(const or_shapes* s, const or_layer* w, int32_t h0, int32_t h1,
                        const uint16_t* x, int32_t rows, const int64_t* pos,
                        const uint16_t* kcache, const uint16_t* vcache, int64_t cap,
                        double* partial);

/* The same with a sliding window: row i attends to positions [max(0, pos[i] - window + 1), pos[i]]
 * (window <= 0: all of 0..pos[i]). */
int32_t or_attn_partial_window(const or_shapes* s, const or_layer* w, int32_t h0, int32_t h1,
                               const uint16_t* x, int32_t rows, const int64_t* pos,
                               const uint16_t* kcache, const uint16_t* vcache, int64_t cap,
                               int64_t window, double* partial);

/* FFN-block partial output of intermediate columns [c0, c1) for `rows` rows of h (binary16):
 * RMSNorm, a_j = silu(Wg[j] h^) * (Wu[j] h^), partial = Wd[:, c0:c1] . a (fp64 [rows, D]). */
int32_t or_ffn_partial(const or_shapes* s, const or_layer* w, int32_t c0, int32_t c1,
                       const uint16_t* h, int32_t rows, double* partial);

/* out = binary16(residual + sum_s partials[s]) elementwise, shards summed in order s = 0..n-1.
 * residual may be NULL (treated as zero). */
void or_combine(const double* const* partials, int32_t n, int64_t count, const uint16_t* residual,
                uint16_t* out);

/* Block quantization of binary16 weight rows [rows, k] (Section 3.2.2 / 4.2.2 precision
 * heterogeneity; format reading in oracle.c): codes q [rows, k] (one int8 per weight, in
 * [-127, 127] for bits = 8, [-7, 7] for bits = 4) and binary16 scales [rows, ceil(k / block)]. */
int32_t or_quantize_rows(const uint16_t* w, int64_t rows, int64_t k, int32_t bits, int32_t block, int8_t* q,
                         uint16_t* scales);
/* y = dequantized W . x in binary64 (rows of q, scales as above). */
void or_gemv_blockq(const int8_t* q, const uint16_t* scales, int64_t rows, int64_t k, int32_t block,
                    const double* x, double* y);

/* A block-quantized weight matrix [rows][k] (codes q, one int8 per weight, and binary16 scales
 * [rows][ceil(k / block)], as or_quantize_rows writes them); its dequantized weight is q * d. */
typedef struct {
    const int8_t* q;
    const uint16_t* scales;
    int64_t rows, k;
    int32_t block;
} or_qmat;

/* The attention and FFN blocks of a shard whose projections are block-quantized (mixed-precision
 * shards, Section 3.2.2 / 4.2.2): the same steps as or_kv_append, or_attn_partial_window and
 * or_ffn_partial, every projection by the dequantized matrix.
 *   or_kv_append_q:    wk, wv: rows of KV heads [kvh0, kvh1) of Wk / Wv, [nk*dh][D].
 *   or_attn_partial_q: wq: rows of query heads [h0, h1) of Wq, [nh*dh][D]; wo: columns
 *                      [h0*dh, h1*dh) of Wo, [D][nh*dh]; window as or_attn_partial_window.
 *   or_ffn_partial_q:  wg, wu: rows [c0, c1) of W_gate / W_up, [nc][D]; wd: columns [c0, c1) of
 *                      W_down, [D][nc]. */
int32_t or_kv_append_q(const or_shapes* s, const uint16_t* attn_norm, const or_qmat* wk, const or_qmat* wv,
                       int32_t kvh0, int32_t kvh1, const uint16_t* x, int32_t rows, int64_t pos0, uint16_t* kcache,
                       uint16_t* vcache, int64_t cap);
int32_t or_attn_partial_q(const or_shapes* s, const uint16_t* attn_norm, const or_qmat* wq, const or_qmat* wo,
                          int32_t h0, int32_t h1, const uint16_t* x, int32_t rows, const int64_t* pos,
                          const uint16_t* kcache, const uint16_t* vcache, int64_t cap, int64_t window,
                          double* partial);
int32_t or_ffn_partial_q(const or_shapes* s, const uint16_t* ffn_norm, const or_qmat* wg, const or_qmat* wu,
                         const or_qmat* wd, int32_t nc, const uint16_t* h, int32_t rows, double* partial);

/* Quantized shard partials (Section 4.3.2, communication scaling; reading in oracle.c):
 * codes q [n] and binary16 scales [ceil(n / block)] of a binary32 vector, and the combine of
 * n quantized partials with a binary16 residual (NULL: zero) into binary16 out [count]. */
int32_t or_quantize_vec(const float* x, int64_t n, int32_t bits, int32_t block, int8_t* q, uint16_t* scales);
void or_combine_q(const int8_t* const* q, const uint16_t* const* scales, int32_t n, int64_t count, int32_t block,
                  const uint16_t* residual, uint16_t* out);

#endif
