// Internal declarations shared by the library's translation units (host bookkeeping and kernel
// launchers).  Not part of the C ABI.
#pragma once

#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <string>
#include <vector>

#include "../../include/voltron.h"

namespace vt {

// ------------------------------------------------------------------ decode GEMV geometry
constexpr int kGemvWarps = 8;
constexpr int kGemvThreads = kGemvWarps * 32;
constexpr int kGemvMaxSlabRows = 128;  // rows per CTA (slot array bound)
constexpr int kGemvMaxK = 16384;       // longest row: 8 warps x 32 lanes x 8 chunks x 8 halves


// ------------------------------------------------------------------ decode attention geometry
constexpr int kAttnWarps = 8;
constexpr int kAttnThreads = (kAttnWarps + 1) * 32;  // + one producer warp
// cached positions per pipeline stage: K and V of a stage are two bulk copies of 64 rows; a
// bulk copy carries a fixed engine cost, so copies of 16 KB or more are needed to stream at full
// rate (8 KB copies reach about half of it).
constexpr int kAttnTilePos = 64;
constexpr int kAttnMaxStages = 3;                    // tiles of K and V in flight per CTA
constexpr int kAttnMaxCluster = 16;                  // CTAs per KV head (thread-block cluster)
constexpr int kAttnMaxGroup = 8;  // query heads per KV head supported by the decode kernel

enum GemvEpilogue : int {
    kEpiPlain = 0,   // out[r] = y[r] (fp32)
    kEpiQkvRope = 1, // rows in RoPE-pair order: rotate q/k, append k/v to the cache
    kEpiSwiglu = 2,  // rows (gate, up) interleaved: u[j] = silu(gate) * up
};

struct GemvArgs {
    const __half* w;     // [rows][row_stride]
    int64_t row_stride;  // elements, multiple of 8
    int rows;
    int k;               // used columns (<= row_stride); columns beyond k are never multiplied
    // input: either RMSNorm(x) with gain, or an fp32 vector
    const __half* x;     // fp16 [k] (norm prologue) or nullptr
    const __half* gain;  // fp16 [k]
    float eps;
    const float* vin;    // fp32 [k] when x == nullptr
    // epilogue
    float* out;          // plain: [rows]; swiglu: [rows/2]; qkv: q [h_s*dh]
    // qkv epilogue
    __half* kcache;      // [hk_s][cap][dh]
    __half* vcache;
    int cap;
    const int32_t* len;  // device length of this layer (position of the new token)
    const float2* rope;  // [max_seq][dh/2] (cos, sin)
    int dh;
    int hq;              // query heads of the shard
    int hk;              // KV heads of the shard
    uint32_t* status;
    // 1: the input vector was written at least two launches earlier, so the kernel may read it
    // before griddepcontrol.wait and stream its whole slab while the previous kernel runs.  Such
    // a kernel releases its dependents at once: they may only read, before their own wait, data
    // that was complete when this kernel started (weights, earlier tokens' KV entries, lengths).
    int indep;
};

struct AttnDecodeArgs {
    const float* q;        // [h_s][dh] rotated queries
    const __half* kcache;  // [hk_s][cap][dh]
    const __half* vcache;
    const int32_t* len;
    int cap;
    int hk;                // KV heads of the shard
    int group;             // query heads per KV head
    int dh;
    int stages;            // K/V tiles in flight per CTA (attn_stages)
    float scale_log2;      // log2(e) / sqrt(dh)
    int window;            // > 0: attend to the last `window` positions only (sliding window)
    float* out;            // [h_s][dh] attention output of the shard's query heads
    uint32_t* status;
};

struct CombineArgs {
    float* parts[VT_MAX_DEVICES];  // shard s: one partial of `count` floats (nullptr: none)
    int n;
    int64_t count;
    const __half* residual;  // nullable
    __half* out;
    int clear;               // 1: zero every partial after reading it (consume and clear)
};

constexpr int kFfnMaxCols = 64;  // intermediate columns per CTA of the fused FFN kernel

struct FfnDecodeArgs {
    const __half* x;     // [d] block input (h)
    const __half* gain;  // [d]
    float eps;
    const __half* wgu;   // [2 cols][d] gate/up rows interleaved
    const __half* wdt;   // [cols][d] transposed down slice
    int d, cols;
    float* out;          // [d] shard partial; the kernel adds into it (must start at zero)
    int indep;           // as GemvArgs::indep
};

// ------------------------------------------------------------------ launchers (stream-ordered)
extern bool g_use_pdl;  // programmatic dependent launch between the library's kernels
extern int g_grid_mult; // CTAs per SM of the streaming kernels
extern int g_num_sms;

cudaError_t launch_gemv(int epi, const GemvArgs& a, cudaStream_t st);
int gemv_grid(int rows, int unit);
int gemv_cpl(int k);
cudaError_t launch_attn_decode(const AttnDecodeArgs& a, cudaStream_t st);
size_t attn_decode_smem_bytes(int dh, int group, int stages);
int attn_cluster_size(int hk);
int attn_stages(int cap, int csize);
cudaError_t launch_combine(const CombineArgs& a, cudaStream_t st);
int ffn_grid(int cols);
cudaError_t launch_ffn_decode(const FfnDecodeArgs& a, int grid, cudaStream_t st);
cudaError_t launch_transpose_f16(const __half* src, int64_t src_ld, int rows, int cols, __half* dst,
                                 int64_t dst_ld, cudaStream_t st);
cudaError_t launch_fill_zero_f32(float* p, int64_t n, cudaStream_t st);
cudaError_t launch_kv_advance(int32_t* len, int first, int count, int delta, int cap, uint32_t* status,
                              cudaStream_t st);
cudaError_t launch_rope_table(float2* tab, int max_seq, int dh, double theta, cudaStream_t st);
cudaError_t launch_embed(const __half* table, const int32_t* ids, int n, int d, int vocab,
                         __half* out, uint32_t* status, cudaStream_t st);
cudaError_t launch_gather_rows(const __half* const* src_rows, __half* dst, int n_rows,
                               int64_t row_len, int64_t dst_stride, cudaStream_t st);

// One-time per-process setup of kernel attributes (dynamic shared-memory limits).
cudaError_t init_decode_kernels();
cudaError_t init_prefill_kernels();
cudaError_t init_quant_kernels();

// ------------------------------------------------------------------ prefill path (prefill.cu)
struct PrefillAttnArgs {
    // shard geometry
    int n;                  // rows (tokens) of this call
    int d;                  // d_model
    int dh, hq, hk;         // head dim, query heads and KV heads of the shard
    float eps;
    float scale_log2;       // log2(e) / sqrt(dh)
    const __half* x;        // [n][d] layer input
    const __half* gain;     // [d]
    const __half* wqkv;     // [(hq + 2 hk) * dh][d], RoPE-pair row order
    const __half* wo;       // [d][hq * dh]
    __half* kcache;         // [hk][cap][dh]
    __half* vcache;
    int cap;
    const int32_t* len;     // device length: rows sit at positions len + row_offset + i
    int row_offset;         // rows already processed by earlier chunks of the same call
    int window;             // > 0: row at position p attends to [p - window + 1, p] only
    const float2* rope;     // [max_seq][dh/2]
    // scratch
    __half* xhat;           // [n][2d]: fp16 RMSNorm(x) * gain, then the fp16 rounding of its remainder
    int xhat_ready;         // 1: xhat already holds RMSNorm(x) with this gain (skip the norm)
    __half* q;              // [n][hq][dh]
    __half* attn;           // [n][hq * dh]
    float* out;             // [n][d] partial
    uint32_t* status;
};
struct PrefillFfnArgs {
    int n, d, c;            // rows, d_model, shard columns
    float eps;
    const __half* x;        // [n][d]
    const __half* gain;
    const __half* wgu;      // [2c][d], gate/up rows interleaved
    // Down projection, read in place from the model's Wd [d][F]: wd points at column c0 - ushift
    // (rounded down to a multiple of 8 so the operand starts on a 16-byte boundary), row stride
    // wd_ld = F.  U carries the same shift: column ushift + j of U is shard column j, columns
    // [0, ushift) are zero, so the extra Wd columns contribute nothing.
    const __half* wd;
    int64_t wd_ld;
    int ushift;
    int ldu;                // row stride of u (>= ushift + c, multiple of 8)
    __half* xhat;           // [n][d]
    int xhat_ready;         // as PrefillAttnArgs::xhat_ready
    __half* u;              // [n][ldu]
    float* out;             // [n][d]
    uint32_t* status;
};
vt_status prefill_attn_shard(const PrefillAttnArgs& a, cudaStream_t st, std::string* err);
// the shards of one block at once (all with the same rows and normalised input): one launch per
// GEMM of the block for every shard
vt_status prefill_attn_group(const PrefillAttnArgs* a, int n, cudaStream_t st, std::string* err);
vt_status prefill_ffn_group(const PrefillFfnArgs* a, int n, cudaStream_t st, std::string* err);
// rows x d: out = fp16(residual + sum of partials); with gain, also xhat = RMSNorm(out) * gain.
// split != 0: xhat rows are 2d long, the fp16 value then the fp16 rounding of the remainder.
cudaError_t launch_combine_norm(const CombineArgs& a, int rows, int d, const __half* gain, float eps, __half* xhat,
                                int split, cudaStream_t st);
cudaError_t launch_rmsnorm_rows(const __half* x, const __half* gain, float eps, int rows, int d, __half* y,
                                int split, cudaStream_t st);

// ------------------------------------------------------------------ block-quantized shard weights (quant.cu)
// A matrix [rows][k] stored as codes of 8 or 4 bits with one fp16 scale per block of kQBlock
// weights along k (the dequantized weight is q * d).  Device layout (written by k_quantize_rows):
//   codes: row r at codes + r * row_bytes, row_bytes = nb * 32 (8-bit) or nb * 16 (4-bit),
//          nb = ceil(k / 32); biased codes u = q + 128 (8-bit, one byte each) or u = q + 8 (4-bit:
//          each 32-bit word holds 8 codes, byte i = code i in its low nibble and code i + 4 in its
//          high nibble); positions k .. nb * 32 - 1 hold the code of 0;
//   scales: [rows][nb] fp16.
constexpr int kQBlock = 32;

struct QMatDev {
    uint8_t* codes = nullptr;
    __half* scales = nullptr;
    int rows = 0, k = 0, nb = 0, bits = 16;
    int64_t row_bytes = 0;
};
// Quantizes device fp16 rows (row r at w + r * ld, m.k values) into m's codes and scales, in the
// layout above, with the decisions of vt_quantize_rows (bit-identical codes and scales).
cudaError_t launch_quantize_rows(const __half* w, int64_t ld, const QMatDev& m, cudaStream_t st);

// Host side: bytes of the codes and of the scales of a [rows][k] matrix at `bits`.
size_t qmat_code_bytes(int64_t rows, int64_t k, int bits);
size_t qmat_scale_bytes(int64_t rows, int64_t k);
// The inverse of the packing for the codes: canonical int8 codes [rows][k].
void unpack_qcodes(const uint8_t* codes, int64_t rows, int64_t k, int bits, int8_t* q);
// Host quantizer shared with vt_quantize_rows: codes q [rows][k] (int8) and fp16 scales [rows][nb].
void quantize_rows_host(const __half* w, int64_t rows, int64_t k, int bits, int block, int8_t* q, __half* scales);

struct QGemvArgs {
    QMatDev w;
    // input: RMSNorm(x) * gain (x fp16 [k]) when x is set, else the fp32 vector vin [k]
    const __half* x;
    const __half* gain;
    float eps;
    const float* vin;
    // epilogues as GemvArgs: plain out[rows]; SwiGLU out[rows / 2]; QKV: q to out, K / V appended
    float* out;
    __half* kcache;
    __half* vcache;
    int cap;
    const int32_t* len;
    const float2* rope;
    int dh, hq, hk;
    uint32_t* status;
};
cudaError_t launch_gemv_q(int epi, const QGemvArgs& a, cudaStream_t st);

// Quantized shard partials (communication scaling): x [n] fp32 -> codes (int8 per value at 8
// bits, two 4-bit values per byte) + fp16 scales [ceil(n / 32)]; clear != 0 zeroes x after reading.
cudaError_t launch_quantize_vec(float* x, int64_t n, int bits, uint8_t* codes, __half* scales, int clear,
                                cudaStream_t st);
struct CombineQArgs {
    int bits[VT_MAX_DEVICES];            // per shard: 16 (fp32 partial) or 8 / 4 (codes + scales)
    float* fparts[VT_MAX_DEVICES];       // bits 16
    const uint8_t* codes[VT_MAX_DEVICES];
    const __half* scales[VT_MAX_DEVICES];
    int n;
    int clear;                           // zero the fp32 partials after reading them
    int64_t count;
    const __half* residual;              // nullable
    __half* out;
};
cudaError_t launch_combine_q(const CombineQArgs& a, cudaStream_t st);

// ------------------------------------------------------------------ static-scratch decode attention
// (static_scratch.cu) split-K decode attention whose scratch is one file-scope __device__ array.
constexpr size_t kStaticScratchBytes = (size_t)1 << 20;  // 1 MiB
constexpr int kStaticSplits = 16;                        // position slices per KV head
constexpr int kStaticMaxKvHeads = 64;                    // arrival counters
constexpr int kStaticMaxDevices = 64;                    // cached symbol addresses

struct StaticAttnLayout {  // byte offsets of the regions in the array
    size_t counters, q, attn, part_ml, part_o, bytes;
};
StaticAttnLayout static_attn_layout(int hq, int hk, int dh);
cudaError_t static_scratch_base(void** out);

struct StaticAttnArgs {
    const float* q;        // [hq][dh] rotated queries
    const __half* kcache;  // [hk][cap][dh]
    const __half* vcache;
    const int32_t* len;
    int cap, hk, group, dh;
    float scale_log2;
    int window;            // > 0: sliding window over the last `window` positions
    float* part_ml;        // [hk][kStaticSplits][group][2] (max, sum) of each slice
    float* part_o;         // [hk][kStaticSplits][group][dh] weighted V of each slice
    uint32_t* counters;    // [hk] slices finished; zero between calls
    float* out;            // [hq][dh]
};
cudaError_t launch_attn_decode_static(const StaticAttnArgs& a, cudaStream_t st);
vt_status prefill_ffn_shard(const PrefillFfnArgs& a, cudaStream_t st, std::string* err);


// ------------------------------------------------------------------ persistent decode token (token.cu)
// One cooperative launch computes a whole decode token through every layer of a partition.
constexpr int kTokWarps = 8;                         // consumer warps
constexpr int kTokConsumers = kTokWarps * 32;
// + one warpgroup holding the producer warp (the other three warps leave at once): a whole
// warpgroup, so that it can hand registers to the consumers with setmaxnreg
constexpr int kTokThreads = kTokConsumers + 128;
constexpr int kTokLaunchRegs = 168;                // per thread at launch: 65536 / 384, rounded down to 8
constexpr int kTokProducerRegs = 56, kTokConsumerRegs = 224;
static_assert(128 * kTokProducerRegs + kTokConsumers * kTokConsumerRegs <= kTokThreads * kTokLaunchRegs,
              "the register split must fit in the registers the block is launched with");
constexpr int kTokStageBytes = 32768;                // one stage of the copy ring
constexpr int kTokMinStages = 3, kTokMaxStages = 8;
constexpr int kTokMaxSeg = 2;                        // KV heads a CTA's attention slice touches
constexpr int kTokMaxGroup = 4;                      // query heads per KV head
constexpr int kTokMaxD = 6144;
constexpr int kTokMaxLayers = 256;
constexpr int kTokMaxGrid = 1024;
// words of TokArgs::sync (zero at creation; zeroed again by a status clear)
constexpr int kTokSyncEpoch = 0;                            // barriers completed by earlier launches
constexpr int kTokSyncAbort = 2;                            // nonzero: the token gave up on a wait
constexpr int kTokSyncTestSkip = 4;  // test hook: c + 1 makes CTA c skip its arrival at the launch's first grid barrier
constexpr int kTokSyncTestSpin = 5;  // test hook: nonzero replaces the polls after which a grid-barrier wait gives up
constexpr int kTokSyncFlags = 64;                           // [grid] epoch of each CTA's last arrival
constexpr int kTokSyncWords = kTokSyncFlags + kTokMaxGrid;

struct TokShardPtrs {  // one (layer, device) shard; null weights for an empty block
    const __half* wqkv;  // [(hq + 2 hk) dh][D], RoPE-pair row order
    const __half* wo;    // [D][hq dh]
    const __half* wgu;   // [2c][D], gate/up rows interleaved
    const __half* wdt;   // [c][D]
    __half* kc;          // [hk][cap][dh]
    __half* vc;
};
struct TokLayerPtrs {
    const __half* attn_norm;  // [D]
    const __half* ffn_norm;   // [D]
    int window;               // > 0: sliding attention window of the layer
};

struct TokArgs {
    int n_layers, n_dev, d, dh, group, cap, n_kv, stages, uni_floats, slot_floats, ffn_gcol;
    int hq[VT_MAX_DEVICES], hk[VT_MAX_DEVICES], h0[VT_MAX_DEVICES], kv0[VT_MAX_DEVICES],
        cols[VT_MAX_DEVICES];
    float eps, scale_log2;
    const TokShardPtrs* shard;  // [n_layers][n_dev]
    const TokLayerPtrs* layer;  // [n_layers]
    int32_t* len;               // [n_layers] device KV lengths (advanced by the kernel)
    const float2* rope;         // [max_seq][dh/2]
    const __half* x_in;         // [D]
    __half* x_out;              // [D]
    float* q_all;               // [H][dh] rotated queries of the token
    float* attn_part;           // [n_dev][D]
    float* ffn_part;            // [n_dev][D] (zeroed inside the kernel before use)
    float* states;              // [grid][kTokMaxSeg][group][dh + 2] attention slice states
    float* attn_out;            // [H][dh] merged attention output of the token
    uint32_t* sync;             // kTokSync* words: barrier epoch, abort word, per-CTA arrival flags
    uint32_t* status;
};
// Geometry of the tensor-core GEMV over one 32 KB stage of rows of length K (token_kernel.cuh).
struct MmaGeom {
    int R;    // rows per stage
    int NP;   // row pairs per stage
    int WP;   // warps per row pair (each takes 8 segments of K / WP)
    int L;    // segment length
    int spr;  // partial sums per row (8 WP)
};

__host__ __device__ inline MmaGeom mma_geom(int K) {
    MmaGeom g;
    int r = kTokStageBytes / (2 * K);
    g.R = r < 1 ? 1 : (r > 64 ? 64 : r);
    g.NP = (g.R + 1) / 2;
    g.WP = g.NP >= 5 ? 1 : (g.NP >= 3 ? 2 : (g.NP == 2 ? 4 : 8));
    g.L = K / (8 * g.WP);
    g.spr = 8 * g.WP;
    return g;
}
// The tensor-core path needs whole 16-element steps in every segment.
__host__ __device__ inline bool mma_ok(int K) {
    const MmaGeom g = mma_geom(K);
    return K % (8 * g.WP) == 0 && g.L >= 16 && g.L % 16 == 0;
}

struct TokPlan {  // host-side launch geometry
    int grid = 0, stages = 0, uni_floats = 0, slot_floats = 0, variant = 0, ffn_gcol = 0;
    size_t smem = 0;
};
// One compiled variant of the kernel: tensor-core steps per row segment (STEPS), fp32 chunks per
// thread of a D-vector (MC), head dim, query heads per KV head, and whether the O rows may use the
// shared-memory or CUDA-core paths (shards whose rows do not match STEPS).
struct TokVariant {
    int steps, mc, dh, group;
    bool osmem;
    cudaError_t (*init)(int optin, size_t* dyn_max);
    cudaError_t (*occupancy)(int* per_sm, size_t smem);
    cudaError_t (*launch)(const TokArgs& a, const cudaLaunchConfig_t& cfg);
};
int token_variants_workloads(const TokVariant** out);  // token_v1.cu
int token_variants_small(const TokVariant** out);      // token_v2.cu
// Fills `plan` and returns true when the fused kernel supports the partition's shapes.
bool token_plan(const TokArgs& a, int max_hq, TokPlan* plan, std::string* why);
cudaError_t launch_decode_token(const TokArgs& a, const TokPlan& plan, cudaStream_t st);
size_t token_state_floats(int grid, int group, int dh);
cudaError_t init_token_kernels();

}  // namespace vt
