// C ABI of the library: validation, object lifetime, the shard-sliced weight layout, the KV-cache
// geometry, and the orchestration of the decode and prefill kernels for one shard or the whole
// stack.  Host code only; kernels live in decode.cu and prefill.cu.
//
// The operation follows Voltron (arXiv 2607.07046) Section 3.2.1: tensor parallelism splits each
// layer into shards (attention heads for ATTN, intermediate columns for FFN), every device
// computes its shard from the same broadcast input, and the shard results are aggregated on the
// main device.  Section 4.2.1 allows uneven shares.  Section 4.3.1 ("Pruning") motivates one
// allocation per shard, so one shard's weights can be dropped without touching the others.
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <algorithm>
#include <cmath>
#include <limits>
#include <mutex>
#include <string>
#include <vector>

#include "internal.h"

using namespace vt;

// ================================================================== errors

namespace {

thread_local std::string t_err;

vt_status fail(vt_status st, const char* fmt, ...) {
    char buf[1024];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    t_err = buf;
    return st;
}

vt_status ok() {
    t_err.clear();
    return VT_OK;
}

#define VT_CUDA(expr)                                                                        \
    do {                                                                                     \
        cudaError_t e_ = (expr);                                                             \
        if (e_ != cudaSuccess)                                                               \
            return fail(VT_ERR_CUDA, "%s failed: %s (%s:%d)", #expr, cudaGetErrorString(e_), \
                        __FILE__, __LINE__);                                                 \
    } while (0)

#define VT_TRY(expr)                     \
    do {                                 \
        vt_status s_ = (expr);           \
        if (s_ != VT_OK) return s_;      \
    } while (0)

inline size_t align256(size_t b) { return (b + 255) & ~(size_t)255; }
inline bool aligned16(const void* p) { return ((uintptr_t)p & 15) == 0; }
// True while `st` is being captured into a CUDA graph: calls then record device work only and
// leave the host-side mirror of the KV lengths alone (replays advance the device lengths).
inline bool capturing(cudaStream_t st) {
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(st, &cs) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return cs == cudaStreamCaptureStatusActive;
}
inline int round_up8(int k) { return (k + 7) & ~7; }

// ------------------------------------------------------------------ allocator
struct Allocator {
    vt_allocator a{};
    bool custom = false;
    void* get(size_t bytes) {
        if (bytes == 0) bytes = 256;
        if (custom) return a.alloc(bytes, a.ctx);
        void* p = nullptr;
        if (cudaMalloc(&p, bytes) != cudaSuccess) {
            cudaGetLastError();
            return nullptr;
        }
        return p;
    }
    void put(void* p) {
        if (!p) return;
        if (custom)
            a.free(p, a.ctx);
        else
            cudaFree(p);
    }
};

std::once_flag g_init_once;
cudaError_t g_init_err = cudaSuccess;

cudaError_t init_library() {
    std::call_once(g_init_once, [] {
        const char* e = getenv("VT_NO_PDL");
        g_use_pdl = !(e && e[0] && e[0] != '0');
        const char* gm = getenv("VT_GRID_MULT");
        if (gm && gm[0] >= '1' && gm[0] <= '4') g_grid_mult = gm[0] - '0';
        int dev = 0;
        g_init_err = cudaGetDevice(&dev);
        if (g_init_err != cudaSuccess) return;
        g_init_err = cudaDeviceGetAttribute(&g_num_sms, cudaDevAttrMultiProcessorCount, dev);
        if (g_init_err != cudaSuccess) return;
        g_init_err = init_decode_kernels();
        if (g_init_err != cudaSuccess) return;
        g_init_err = init_prefill_kernels();
        if (g_init_err != cudaSuccess) return;
        g_init_err = init_token_kernels();
        if (g_init_err != cudaSuccess) return;
        g_init_err = init_quant_kernels();
    });
    return g_init_err;
}

}  // namespace

// ================================================================== objects

struct LayerPtrs {
    __half *attn_norm = nullptr, *wq = nullptr, *wk = nullptr, *wv = nullptr, *wo = nullptr,
           *ffn_norm = nullptr, *w_gate = nullptr, *w_up = nullptr, *w_down = nullptr;
};

struct vt_model {
    vt_shapes s{};
    Allocator alloc;
    std::vector<void*> layer_base;
    std::vector<LayerPtrs> layer;
    std::vector<char> loaded;
    __half* embed = nullptr;
    bool embed_loaded = false;
    float2* rope = nullptr;
    uint32_t* status = nullptr;  // device status word of the embedding gather
    std::vector<int32_t> window;  // per layer: sliding attention window (0: all cached positions)
    int n_partitions = 0;         // live partitions (windows are fixed while any exists)
};

struct AttnShard {
    void* base = nullptr;
    __half* norm = nullptr;
    __half* wqkv = nullptr;  // [(hq + 2 hk) dh][D] (fp16 shards)
    __half* wo = nullptr;    // [D][hq dh]          (fp16 shards)
    int h0 = 0, h1 = 0, kv0 = 0, kv1 = 0;
    int bits = 16;           // 16: fp16 weights; 8 / 4: block-quantized (qkv, o)
    QMatDev qkv, o;          // quantized shards: QKV rows [(hq + 2 hk) dh][D] in the same row order, O [D][hq dh]
};

struct FfnShard {
    void* base = nullptr;
    __half* norm = nullptr;
    __half* wgu = nullptr;  // [2c][D], gate/up rows interleaved (fp16 shards)
    __half* wdt = nullptr;  // [c][D], row j = column c0 + j of Wd (fp16 shards)
    int c0 = 0, c1 = 0;
    int bits = 16;          // 16: fp16 weights; 8 / 4: block-quantized (gu, down)
    QMatDev gu, down;       // quantized shards: gate/up rows [2c][D] interleaved, down columns [D][c]
};

struct DecodeScratch {  // per device of the partition
    float* q = nullptr;     // [hq][dh] rotated queries of the token
    float* attn = nullptr;  // [hq][dh] attention output (input of the O projection)
    float* u = nullptr;     // [c] SwiGLU activations (quantized FFN shards)
    int ffn_grid = 0;       // CTAs of the fused FFN kernel
};

constexpr int kPrefillChunk = 1024;  // rows per prefill pass (longer prompts run in chunks)

struct vt_partition {
    vt_model* m = nullptr;
    int n_dev = 0;
    std::vector<vt_range> heads, cols;
    std::vector<AttnShard> attn;  // [layer * n_dev + dev]
    std::vector<FfnShard> ffn;
    std::vector<DecodeScratch> dec;
    std::vector<void*> owned;  // every allocation besides the shard bases
    bool counted = false;      // counted in the model's n_partitions
    mutable int n_kv = 0;      // live KV caches of the partition (precisions are fixed while any exists)
    std::vector<int> comm_bits;   // per device: precision of its partials on the way to the combine (16: fp32)
    uint8_t* pcodes = nullptr;    // [n_dev][D] quantized partials of the whole-token path
    __half* pscales = nullptr;    // [n_dev][ceil(D / 32)]
    uint32_t* status = nullptr;
    // whole-stack buffers
    float* dpart = nullptr;     // [n_dev][D] decode partials (kept zero between blocks)
    float* partials = nullptr;  // [n_dev][kPrefillChunk][D]
    __half* hbuf = nullptr;     // [kPrefillChunk][D]
    __half* xbuf = nullptr;     // [kPrefillChunk][D]
    // prefill scratch
    __half* p_xhat = nullptr;   // [kPrefillChunk][2 D]: ATTN input as fp16 hi / lo halves (FFN: [.][D])
    __half* p_q = nullptr;      // [n_dev] slots of [kPrefillChunk][max_hq][dh], q_slot halves apart
    __half* p_attn = nullptr;   // [n_dev] slots of [kPrefillChunk][max_hq dh]
    __half* p_u = nullptr;      // [n_dev] slots of [kPrefillChunk][max_ld], u_slot halves apart
    int max_hq = 0, max_ld = 0;
    size_t q_slot = 0, u_slot = 0;
    // persistent decode-token kernel: shapes and scratch (the KV object adds its tables)
    bool tok_planned = false;  // the kernel has a plan (and scratch) for the partition's shapes
    bool tok_ok = false;       // ... and every shard is fp16 (quantized shards run per-shard kernels)
    std::string tok_why;
    TokPlan tok_plan;
    TokArgs tok_base{};

    const AttnShard& a(int l, int d) const { return attn[(size_t)l * n_dev + d]; }
    const FfnShard& f(int l, int d) const { return ffn[(size_t)l * n_dev + d]; }
};

struct vt_kv {
    const vt_partition* p = nullptr;
    int cap = 0;
    std::vector<void*> buf;  // [layer * n_dev + dev]: K then V, each [hk][cap][dh]
    int32_t* len = nullptr;  // device [n_layers]
    std::vector<int32_t> h_len;
    uint32_t* status = nullptr;
    void* tok_tab = nullptr;  // device [n_layers][n_dev] TokShardPtrs, then [n_layers] TokLayerPtrs
    Allocator* alloc() const { return &p->m->alloc; }
    __half* k(int l, int d) const { return static_cast<__half*>(buf[(size_t)l * p->n_dev + d]); }
    __half* v(int l, int d) const {
        const AttnShard& s = p->a(l, d);
        return k(l, d) + (size_t)(s.kv1 - s.kv0) * cap * p->m->s.d_head;
    }
};

// ================================================================== validation

extern "C" const char* vt_last_error(void) { return t_err.c_str(); }
extern "C" const char* vt_version(void) { return "0.1.0"; }

extern "C" vt_status vt_shapes_validate(const vt_shapes* s) {
    if (!s) return fail(VT_ERR_INVALID_ARG, "shapes is NULL");
    if (s->n_layers < 1) return fail(VT_ERR_SHAPE, "n_layers must be >= 1");
    if (s->d_model < 64 || s->d_model % 64 != 0 || s->d_model > 16384)
        return fail(VT_ERR_SHAPE, "d_model must be a multiple of 64 in [64, 16384]");
    if (s->n_heads < 1 || s->n_kv_heads < 1 || s->n_heads % s->n_kv_heads != 0)
        return fail(VT_ERR_SHAPE, "n_heads must be a positive multiple of n_kv_heads");
    {
        const int g = s->n_heads / s->n_kv_heads;
        if (g != 1 && g != 2 && g != 4 && g != 8)
            return fail(VT_ERR_SHAPE, "query heads per KV head must be 1, 2, 4 or 8 (got %d)", g);
    }
    if (s->d_head != 64 && s->d_head != 128) return fail(VT_ERR_SHAPE, "d_head must be 64 or 128");
    if ((int64_t)s->n_heads * s->d_head > 16384)
        return fail(VT_ERR_SHAPE, "n_heads * d_head must be <= 16384");
    if (s->d_ffn < 1 || s->d_ffn > kGemvMaxK)
        return fail(VT_ERR_SHAPE, "d_ffn must be in [1, %d]", kGemvMaxK);
    if (s->vocab < 0) return fail(VT_ERR_SHAPE, "vocab must be >= 0");
    if (s->max_seq < 1 || s->max_seq > (1 << 20))
        return fail(VT_ERR_SHAPE, "max_seq must be in [1, 2^20]");
    if (!(s->rms_eps >= 0.f) || !(s->rope_theta > 0.f))
        return fail(VT_ERR_SHAPE, "rms_eps must be >= 0 and rope_theta > 0");
    return ok();
}

// allow_gaps: heads / columns left uncovered are pruned (Section 4.3.1, shard-wise pruning).
static vt_status check_ranges(const vt_range* r, int n, int total, int align, const char* what, bool allow_gaps = false) {
    int expect = 0;
    for (int d = 0; d < n; ++d) {
        if (r[d].begin < 0 || r[d].end > total || r[d].begin > r[d].end)
            return fail(VT_ERR_PARTITION_RANGE, "%s range %d [%d, %d) is not inside [0, %d)", what, d,
                        r[d].begin, r[d].end, total);
        if (allow_gaps && r[d].begin == r[d].end) continue;  // a pruned device: its position does not matter
        if (r[d].begin < expect)
            return fail(VT_ERR_PARTITION_OVERLAP, "%s range %d starts at %d, before %d", what, d,
                        r[d].begin, expect);
        if (r[d].begin > expect && !allow_gaps)
            return fail(VT_ERR_PARTITION_GAP, "%s range %d starts at %d, leaving [%d, %d) unassigned",
                        what, d, r[d].begin, expect, r[d].begin);
        if (align > 1 && (r[d].begin % align != 0 || r[d].end % align != 0))
            return fail(VT_ERR_PARTITION_GQA,
                        "%s range %d [%d, %d) does not align to KV groups of %d heads", what, d,
                        r[d].begin, r[d].end, align);
        if (r[d].end > r[d].begin || !allow_gaps) expect = r[d].end;  // a pruned layout may place empty ranges anywhere
    }
    if (expect != total && !allow_gaps)
        return fail(VT_ERR_PARTITION_GAP, "%s ranges cover [0, %d) of [0, %d)", what, expect, total);
    return VT_OK;
}

extern "C" vt_status vt_partition_validate(const vt_shapes* s, int32_t n, const vt_range* heads,
                                           const vt_range* cols) {
    VT_TRY(vt_shapes_validate(s));
    if (n < 1 || n > VT_MAX_DEVICES)
        return fail(VT_ERR_INVALID_ARG, "n_devices must be in [1, %d]", VT_MAX_DEVICES);
    if (!heads || !cols) return fail(VT_ERR_INVALID_ARG, "range arrays must not be NULL");
    VT_TRY(check_ranges(heads, n, s->n_heads, s->n_heads / s->n_kv_heads, "head"));
    VT_TRY(check_ranges(cols, n, s->d_ffn, 1, "ffn column"));
    return ok();
}

extern "C" vt_status vt_partition_validate_layers(const vt_shapes* s, int32_t n, const vt_range* heads,
                                                  const vt_range* cols, uint32_t flags) {
    VT_TRY(vt_shapes_validate(s));
    if (n < 1 || n > VT_MAX_DEVICES)
        return fail(VT_ERR_INVALID_ARG, "n_devices must be in [1, %d]", VT_MAX_DEVICES);
    if (!heads || !cols) return fail(VT_ERR_INVALID_ARG, "range arrays must not be NULL");
    if (flags & ~VT_PARTITION_PRUNE) return fail(VT_ERR_INVALID_ARG, "unknown partition flags 0x%x", flags);
    const bool gaps = (flags & VT_PARTITION_PRUNE) != 0;
    for (int l = 0; l < s->n_layers; ++l) {
        char what[64];
        snprintf(what, sizeof what, "layer %d head", l);
        VT_TRY(check_ranges(heads + (size_t)l * n, n, s->n_heads, s->n_heads / s->n_kv_heads, what, gaps));
        snprintf(what, sizeof what, "layer %d ffn column", l);
        VT_TRY(check_ranges(cols + (size_t)l * n, n, s->d_ffn, 1, what, gaps));
    }
    return ok();
}

// ================================================================== planning

namespace {

// A block cut into equal units (Voltron Section 4.2.1 assigns TP shards greedily by device
// performance): KV groups for ATTN, `col_unit` FFN columns for FFN.
struct BlockUnits {
    int units, per_unit, total;  // units; heads or columns per unit; heads or columns of the block
    double mem;                  // fp16 bytes a unit occupies (weights, and the K / V cache at max_seq)
    double wbytes;               // weight bytes of a unit
    int kv_heads;                // KV heads of a unit (ATTN: 1)
};

BlockUnits block_units(const vt_shapes& s, vt_block block, int col_unit) {
    const double D = s.d_model, dh = s.d_head;
    const int g = s.n_heads / s.n_kv_heads;
    BlockUnits b{};
    if (block == VT_BLOCK_ATTN) {
        b.units = s.n_kv_heads;
        b.per_unit = g;
        b.total = s.n_heads;
        b.wbytes = 2.0 * ((g + 2) * dh * D + D * g * dh);  // QKV rows and O columns
        b.mem = b.wbytes + 2.0 * 2.0 * s.max_seq * dh;     // + its K and V cache
        b.kv_heads = 1;
    } else {
        b.units = (s.d_ffn + col_unit - 1) / col_unit;
        b.per_unit = col_unit;
        b.total = s.d_ffn;
        b.wbytes = 2.0 * 3.0 * D * col_unit;  // gate, up and down columns
        b.mem = b.wbytes;
        b.kv_heads = 0;
    }
    return b;
}

// Units one at a time to the device that finishes soonest with one more (unit time t[d]; ties:
// the lower index), among those whose remaining memory still holds one more.  False if a unit fits
// nowhere.  For equal units on devices of different speeds this minimises the largest time.
bool greedy_shares(int units, double unit_mem, int n, const double* t, const double* mem_left, int* cnt) {
    for (int d = 0; d < n; ++d) cnt[d] = 0;
    for (int u = 0; u < units; ++u) {
        int best = -1;
        double best_t = 0.0;
        for (int d = 0; d < n; ++d) {
            if (mem_left && (cnt[d] + 1) * unit_mem > mem_left[d]) continue;
            const double tt = (cnt[d] + 1) * t[d];
            if (best < 0 || tt < best_t) {
                best = d;
                best_t = tt;
            }
        }
        if (best < 0) return false;
        ++cnt[best];
    }
    return true;
}

void shares_to_ranges(int n, const int* cnt, int per_unit, int total, vt_range* r) {
    int at = 0;
    for (int d = 0; d < n; ++d) {
        const int e = std::min(total, at + cnt[d] * per_unit);
        r[d].begin = at;
        r[d].end = e;
        at = e;
    }
}

vt_status check_rates(int n, const double* rate, const double* mem) {
    for (int d = 0; d < n; ++d) {
        if (!(rate[d] > 0.0) || !std::isfinite(rate[d]))
            return fail(VT_ERR_INVALID_ARG, "rate[%d] must be finite and positive", d);
        if (mem && !(mem[d] >= 0.0)) return fail(VT_ERR_INVALID_ARG, "mem_bytes[%d] must be >= 0", d);
    }
    return VT_OK;
}

}  // namespace

// Heterogeneity-aware TP shares of one block (Voltron Section 4.2.1).
extern "C" vt_status vt_plan_tp_shares(const vt_shapes* s, vt_block block, int32_t n, const double* rate,
                                       const double* mem, int32_t col_unit, vt_range* ranges,
                                       double* makespan) {
    if (!s || !rate || !ranges) return fail(VT_ERR_INVALID_ARG, "shapes, rate and ranges must not be NULL");
    VT_TRY(vt_shapes_validate(s));
    if (n < 1 || n > VT_MAX_DEVICES) return fail(VT_ERR_INVALID_ARG, "n_devices must be in [1, %d]", VT_MAX_DEVICES);
    if (block != VT_BLOCK_ATTN && block != VT_BLOCK_FFN) return fail(VT_ERR_INVALID_ARG, "unknown block %d", (int)block);
    VT_TRY(check_rates(n, rate, mem));
    if (block == VT_BLOCK_FFN && col_unit < 1) return fail(VT_ERR_INVALID_ARG, "col_unit must be >= 1");
    const BlockUnits b = block_units(*s, block, block == VT_BLOCK_FFN ? col_unit : 1);
    double t[VT_MAX_DEVICES];
    for (int d = 0; d < n; ++d) t[d] = b.mem / rate[d];
    int cnt[VT_MAX_DEVICES];
    if (!greedy_shares(b.units, b.mem, n, t, mem, cnt))
        return fail(VT_ERR_PLAN_MEMORY, "the block's %d units do not fit the memory budgets", b.units);
    shares_to_ranges(n, cnt, b.per_unit, b.total, ranges);
    double worst = 0.0;
    for (int d = 0; d < n; ++d) worst = std::max(worst, cnt[d] * t[d]);
    if (makespan) *makespan = worst;
    return ok();
}

// Layer-wise hybrid parallelism plan (Voltron Section 4.2.1, with the communication pattern of
// MP and TP in Section 3.2.1).
extern "C" vt_status vt_plan_layers(const vt_shapes* s, int32_t n, const double* rate, const double* frate,
                                    const double* mem, double link_bps, double link_lat, int32_t tokens,
                                    int32_t kv_len, vt_block_plan* plans, double* total_s) {
    if (!s || !rate || !plans) return fail(VT_ERR_INVALID_ARG, "shapes, rate and plans must not be NULL");
    VT_TRY(vt_shapes_validate(s));
    if (n < 1 || n > VT_MAX_DEVICES) return fail(VT_ERR_INVALID_ARG, "n_devices must be in [1, %d]", VT_MAX_DEVICES);
    VT_TRY(check_rates(n, rate, mem));
    if (frate)
        for (int d = 0; d < n; ++d)
            if (!(frate[d] > 0.0) || !std::isfinite(frate[d]))
                return fail(VT_ERR_INVALID_ARG, "flop_rate[%d] must be finite and positive", d);
    if (!(link_bps > 0.0) || !std::isfinite(link_bps) || !(link_lat >= 0.0) || !std::isfinite(link_lat))
        return fail(VT_ERR_INVALID_ARG, "the link needs a finite positive rate and a finite latency >= 0");
    if (tokens < 1 || kv_len < 0 || (int64_t)kv_len + tokens > s->max_seq)
        return fail(VT_ERR_INVALID_ARG, "tokens %d at kv_len %d do not fit max_seq %d", tokens, kv_len, s->max_seq);
    const double D = s->d_model, dh = s->d_head, T = tokens, Lkv = kv_len;
    const double act = T * D * 2.0, part = T * D * 4.0;  // fp16 activations, fp32 partials
    auto xfer = [&](double bytes) { return link_lat + bytes / link_bps; };
    std::vector<double> left(n, 0.0);
    for (int d = 0; d < n; ++d) left[d] = mem ? mem[d] : std::numeric_limits<double>::infinity();
    // devices by rate, fastest first (ties: lower index): the order MP tries them in
    std::vector<int> by_rate(n);
    for (int d = 0; d < n; ++d) by_rate[d] = d;
    std::stable_sort(by_rate.begin(), by_rate.end(), [&](int a, int b) { return rate[a] > rate[b]; });
    int holder = 0;
    double total = 0.0;
    for (int bi = 0; bi < 2 * s->n_layers; ++bi) {
        const vt_block blk = (bi & 1) ? VT_BLOCK_FFN : VT_BLOCK_ATTN;
        const BlockUnits b = block_units(*s, blk, 1);
        // per unit: bytes streamed (weights, K / V rows read at kv_len and written for the new rows)
        // and flops over all tokens (2 per weight per token; ATTN also 4 dh per query head and
        // visible position: scores and weighted values)
        double ubytes = b.wbytes, uflops = T * b.wbytes;  // 2 flops per fp16 weight (2 bytes) per token
        if (blk == VT_BLOCK_ATTN) {
            const double g = s->n_heads / s->n_kv_heads;
            ubytes += 2.0 * 2.0 * dh * (Lkv + T);
            uflops += g * 4.0 * dh * (T * Lkv + T * (T + 1) / 2.0);
        }
        double ut[VT_MAX_DEVICES];
        for (int d = 0; d < n; ++d) ut[d] = std::max(ubytes / rate[d], frate ? uflops / frate[d] : 0.0);
        // MP: the fastest device whose remaining memory holds the block
        int mp = -1;
        for (int d : by_rate)
            if (b.units * b.mem <= left[d]) {
                mp = d;
                break;
            }
        const double inf = std::numeric_limits<double>::infinity();
        double mp_comp = inf, mp_comm = 0.0;
        if (mp >= 0) {
            mp_comp = b.units * ut[mp];
            mp_comm = mp != holder ? xfer(act) : 0.0;
        }
        // TP: greedy shares on the remaining memory
        int cnt[VT_MAX_DEVICES];
        const bool tp_ok = greedy_shares(b.units, b.mem, n, ut, left.data(), cnt);
        double tp_comp = inf, tp_comm = 0.0;
        if (tp_ok) {
            tp_comp = 0.0;
            int others = 0;
            for (int d = 0; d < n; ++d) {
                tp_comp = std::max(tp_comp, cnt[d] * ut[d]);
                if (cnt[d] > 0 && d != holder) ++others;
            }
            if (others > 0) tp_comm = xfer(act) + others * xfer(part);
        }
        if (mp < 0 && !tp_ok)
            return fail(VT_ERR_PLAN_MEMORY, "block %d of layer %d fits under neither MP nor TP", bi & 1, bi / 2);
        vt_block_plan& pl = plans[bi];
        pl = vt_block_plan{};
        if (tp_ok && tp_comp + tp_comm < mp_comp + mp_comm) {
            pl.tp = 1;
            pl.device = holder;
            shares_to_ranges(n, cnt, b.per_unit, b.total, pl.ranges);
            pl.compute_s = tp_comp;
            pl.comm_s = tp_comm;
            for (int d = 0; d < n; ++d) left[d] -= cnt[d] * b.mem;
        } else {
            pl.tp = 0;
            pl.device = mp;
            // the whole block on mp: empty ranges before and after it, in device order
            for (int d = 0; d < n; ++d) pl.ranges[d] = vt_range{d <= mp ? 0 : b.total, d < mp ? 0 : b.total};
            pl.compute_s = mp_comp;
            pl.comm_s = mp_comm;
            left[mp] -= b.units * b.mem;
            holder = mp;
        }
        total += pl.compute_s + pl.comm_s;
    }
    if (total_s) *total_s = total;
    return ok();
}

// Importance-aware mixed precision (Voltron Section 4.2.2): blocks lowered one precision step at a
// time in ascending order of importance, the number of steps found by binary search.
namespace {
// bytes of a rows x k weight matrix at `bits` (16: fp16; 8 / 4: codes + one fp16 scale per block of 32)
double matrix_bytes(double rows, double k, int bits) {
    if (bits == 16) return rows * k * 2.0;
    return rows * std::ceil(k / 32.0) * (32.0 * bits / 8.0 + 2.0);
}
struct PrecisionModel {
    const vt_shapes* s;
    int n, nb;
    const vt_block_plan* plans;
    const double *rate, *mem;
    double kv_len;
    std::vector<int> order;  // blocks by ascending importance (ties: lower index)
    // per device: memory and streamed bytes of block b at `bits`
    void block_cost(int b, int d, int bits, double* mem_b, double* stream_b) const {
        const vt_range r = plans[b].ranges[d];
        const double cnt = r.end - r.begin, D = s->d_model, dh = s->d_head;
        if (cnt <= 0) {
            *mem_b = *stream_b = 0.0;
            return;
        }
        if ((b & 1) == 0) {  // ATTN: cnt query heads, cnt / g KV heads
            const double hk = cnt / (s->n_heads / s->n_kv_heads);
            const double w = matrix_bytes((cnt + 2.0 * hk) * dh, D, bits) + matrix_bytes(D, cnt * dh, bits);
            *mem_b = w + 2.0 * 2.0 * hk * s->max_seq * dh;
            *stream_b = w + 2.0 * 2.0 * hk * dh * (kv_len + 1.0);
        } else {  // FFN: cnt columns
            const double w = matrix_bytes(2.0 * cnt, D, bits) + matrix_bytes(D, cnt, bits);
            *mem_b = *stream_b = w;
        }
    }
    // bits of every block after k steps
    void bits_at(int k, int32_t* bits) const {
        for (int b = 0; b < nb; ++b) bits[b] = 16;
        for (int i = 0; i < nb; ++i) {
            if (i < k) bits[order[i]] = 8;
            if (i < k - nb) bits[order[i]] = 4;
        }
    }
    // memory fits every device; total time
    void eval(const int32_t* bits, bool* mem_ok, double* time_s) const {
        std::vector<double> used(n, 0.0);
        double t = 0.0;
        for (int b = 0; b < nb; ++b) {
            double slow = 0.0;
            for (int d = 0; d < n; ++d) {
                double mb, sb;
                block_cost(b, d, bits[b], &mb, &sb);
                used[d] += mb;
                if (sb > 0.0) slow = std::max(slow, sb / rate[d]);
            }
            t += slow + plans[b].comm_s;
        }
        *mem_ok = true;
        if (mem)
            for (int d = 0; d < n; ++d) *mem_ok = *mem_ok && used[d] <= mem[d];
        *time_s = t;
    }
};
}  // namespace

extern "C" vt_status vt_plan_precision(const vt_shapes* s, int32_t n, const vt_block_plan* plans,
                                       const double* importance, const double* rate, const double* mem, double qos_s,
                                       int32_t kv_len, int32_t* bits, int32_t* steps, double* total_s) {
    if (!s || !plans || !importance || !rate || !bits)
        return fail(VT_ERR_INVALID_ARG, "shapes, plans, importance, rate and bits must not be NULL");
    VT_TRY(vt_shapes_validate(s));
    if (n < 1 || n > VT_MAX_DEVICES) return fail(VT_ERR_INVALID_ARG, "n_devices must be in [1, %d]", VT_MAX_DEVICES);
    VT_TRY(check_rates(n, rate, mem));
    if (std::isnan(qos_s)) return fail(VT_ERR_INVALID_ARG, "qos_s is NaN");
    if (kv_len < 0 || kv_len >= s->max_seq) return fail(VT_ERR_INVALID_ARG, "kv_len %d outside [0, max_seq)", kv_len);
    const int nb = 2 * s->n_layers;
    const int g = s->n_heads / s->n_kv_heads;
    for (int b = 0; b < nb; ++b) {
        if (!std::isfinite(importance[b])) return fail(VT_ERR_INVALID_ARG, "importance[%d] is not finite", b);
        const int total = (b & 1) ? s->d_ffn : s->n_heads;
        for (int d = 0; d < n; ++d) {
            const vt_range r = plans[b].ranges[d];
            if (r.begin < 0 || r.end < r.begin || r.end > total)
                return fail(VT_ERR_PARTITION_RANGE, "block %d device %d: range [%d, %d)", b, d, r.begin, r.end);
            if ((b & 1) == 0 && ((r.end - r.begin) % g) != 0)
                return fail(VT_ERR_PARTITION_GQA, "block %d device %d: %d heads are not whole KV groups", b, d,
                            r.end - r.begin);
        }
        if (!(plans[b].comm_s >= 0.0) || !std::isfinite(plans[b].comm_s))
            return fail(VT_ERR_INVALID_ARG, "block %d: comm_s must be finite and >= 0", b);
    }
    PrecisionModel pm{s, n, nb, plans, rate, mem, (double)kv_len, {}};
    pm.order.resize(nb);
    for (int b = 0; b < nb; ++b) pm.order[b] = b;
    std::stable_sort(pm.order.begin(), pm.order.end(), [&](int a, int b) { return importance[a] < importance[b]; });
    const bool timed = qos_s > 0.0 && std::isfinite(qos_s);
    std::vector<int32_t> cand(nb);
    auto feasible = [&](int k, bool* mem_ok, double* t) {
        pm.bits_at(k, cand.data());
        pm.eval(cand.data(), mem_ok, t);
        return *mem_ok && (!timed || *t <= qos_s);
    };
    // memory and time do not grow with k: the smallest feasible k by bisection over [0, 2 nb]
    bool mem_ok;
    double t;
    int lo = 0, hi = 2 * nb;
    if (!feasible(hi, &mem_ok, &t)) {
        pm.bits_at(hi, bits);
        if (steps) *steps = hi;
        if (total_s) *total_s = t;
        if (!mem_ok) return fail(VT_ERR_PLAN_MEMORY, "the memory budgets are missed even with every block at INT4");
        return fail(VT_ERR_PLAN_QOS, "%.6g s with every block at INT4 misses qos_s %.6g s", t, qos_s);
    }
    while (lo < hi) {
        const int mid = lo + (hi - lo) / 2;
        if (feasible(mid, &mem_ok, &t)) hi = mid;
        else lo = mid + 1;
    }
    feasible(lo, &mem_ok, &t);
    pm.bits_at(lo, bits);
    if (steps) *steps = lo;
    if (total_s) *total_s = t;
    return ok();
}

// ================================================================== quantization (host)

// Block quantization of fp16 weight rows (Voltron Sections 3.2.2 / 4.2.2): fp16 scale per block,
// int8 code per weight, every decision in fp32.
extern "C" vt_status vt_quantize_rows(const void* w, int64_t rows, int64_t k, int32_t bits, int32_t block, int8_t* q,
                                      void* scales) {
    if (!w || !q || !scales) return fail(VT_ERR_INVALID_ARG, "w, q and scales must not be NULL");
    if (rows < 0 || k < 0 || block < 1 || (bits != 8 && bits != 4))
        return fail(VT_ERR_INVALID_ARG, "rows %lld, k %lld, block %d, bits %d", (long long)rows, (long long)k, block, bits);
    quantize_rows_host(static_cast<const __half*>(w), rows, k, bits, block, q, static_cast<__half*>(scales));
    return ok();
}

// ================================================================== model

// With `clear`, also re-arms the decode-token kernel's grid barrier and abort word: a token that
// gave up on a wait leaves them in an unknown state (the call that read the flags synchronised the
// device, so no kernel is using them).
static vt_status read_status(uint32_t* dev, uint32_t* flags, int32_t clear, uint32_t* tok_sync) {
    if (!flags) return fail(VT_ERR_INVALID_ARG, "flags is NULL");
    VT_CUDA(cudaDeviceSynchronize());
    VT_CUDA(cudaMemcpy(flags, dev, 4, cudaMemcpyDeviceToHost));
    if (clear) {
        VT_CUDA(cudaMemset(dev, 0, 4));
        if (tok_sync) VT_CUDA(cudaMemset(tok_sync, 0, (size_t)kTokSyncWords * sizeof(uint32_t)));
    }
    return ok();
}


static vt_status upload(void* dst, const void* src, size_t bytes, cudaStream_t st) {
    if (!src) return fail(VT_ERR_INVALID_ARG, "a weight pointer is NULL");
    VT_CUDA(cudaMemcpyAsync(dst, src, bytes, cudaMemcpyHostToDevice, st));
    return VT_OK;
}

extern "C" vt_status vt_model_load_layer(vt_model* m, int32_t l, const vt_layer_weights* w,
                                         vt_stream stream) {
    if (!m || !w) return fail(VT_ERR_INVALID_ARG, "model and weights must not be NULL");
    if (l < 0 || l >= m->s.n_layers) return fail(VT_ERR_INVALID_ARG, "layer %d out of range", l);
    cudaStream_t st = (cudaStream_t)stream;
    const vt_shapes& s = m->s;
    const size_t D = s.d_model, Q = (size_t)s.n_heads * s.d_head, KV = (size_t)s.n_kv_heads * s.d_head,
                 F = s.d_ffn;
    LayerPtrs& L = m->layer[l];
    VT_TRY(upload(L.attn_norm, w->attn_norm, D * 2, st));
    VT_TRY(upload(L.wq, w->wq, Q * D * 2, st));
    VT_TRY(upload(L.wk, w->wk, KV * D * 2, st));
    VT_TRY(upload(L.wv, w->wv, KV * D * 2, st));
    VT_TRY(upload(L.wo, w->wo, D * Q * 2, st));
    VT_TRY(upload(L.ffn_norm, w->ffn_norm, D * 2, st));
    VT_TRY(upload(L.w_gate, w->w_gate, F * D * 2, st));
    VT_TRY(upload(L.w_up, w->w_up, F * D * 2, st));
    VT_TRY(upload(L.w_down, w->w_down, D * F * 2, st));
    VT_CUDA(cudaStreamSynchronize(st));
    m->loaded[l] = 1;
    return ok();
}

extern "C" vt_status vt_model_load_embedding(vt_model* m, const void* embed, vt_stream stream) {
    if (!m || !embed) return fail(VT_ERR_INVALID_ARG, "model and embed must not be NULL");
    if (!m->embed) return fail(VT_ERR_STATE, "the model has no embedding table (vocab == 0)");
    cudaStream_t st = (cudaStream_t)stream;
    VT_TRY(upload(m->embed, embed, (size_t)m->s.vocab * m->s.d_model * 2, st));
    VT_CUDA(cudaStreamSynchronize(st));
    m->embed_loaded = true;
    return ok();
}

extern "C" void vt_model_destroy(vt_model* m) {
    if (!m) return;
    cudaDeviceSynchronize();
    for (void* p : m->layer_base) m->alloc.put(p);
    m->alloc.put(m->embed);
    m->alloc.put(m->rope);
    m->alloc.put(m->status);
    delete m;
}

extern "C" vt_status vt_model_create(const vt_shapes* shapes, const vt_layer_weights* per_layer,
                                     const void* embed, const vt_allocator* allocator,
                                     vt_stream stream, vt_model** out) {
    if (!out) return fail(VT_ERR_INVALID_ARG, "out is NULL");
    *out = nullptr;
    VT_TRY(vt_shapes_validate(shapes));
    if (allocator && (!allocator->alloc || !allocator->free))
        return fail(VT_ERR_INVALID_ARG, "allocator callbacks must not be NULL");
    VT_CUDA(init_library());
    cudaStream_t st = (cudaStream_t)stream;
    vt_model* m = new vt_model();
    m->s = *shapes;
    if (allocator) {
        m->alloc.a = *allocator;
        m->alloc.custom = true;
    }
    const vt_shapes& s = m->s;
    const size_t D = s.d_model, Q = (size_t)s.n_heads * s.d_head, KV = (size_t)s.n_kv_heads * s.d_head,
                 F = s.d_ffn;
    const size_t sizes[9] = {D * 2, Q * D * 2, KV * D * 2, KV * D * 2, D * Q * 2,
                             D * 2, F * D * 2, F * D * 2, D * F * 2};
    size_t total = 0;
    for (size_t b : sizes) total += align256(b);
    m->layer.resize(s.n_layers);
    m->loaded.assign(s.n_layers, 0);
    m->window.assign(s.n_layers, 0);
    for (int l = 0; l < s.n_layers; ++l) {
        uint8_t* base = static_cast<uint8_t*>(m->alloc.get(total));
        if (!base) {
            vt_model_destroy(m);
            return fail(VT_ERR_ALLOC, "allocating %zu bytes for layer %d failed", total, l);
        }
        m->layer_base.push_back(base);
        __half** slots[9] = {&m->layer[l].attn_norm, &m->layer[l].wq, &m->layer[l].wk,
                             &m->layer[l].wv, &m->layer[l].wo, &m->layer[l].ffn_norm,
                             &m->layer[l].w_gate, &m->layer[l].w_up, &m->layer[l].w_down};
        size_t off = 0;
        for (int t = 0; t < 9; ++t) {
            *slots[t] = reinterpret_cast<__half*>(base + off);
            off += align256(sizes[t]);
        }
    }
    if (s.vocab > 0) {
        m->embed = static_cast<__half*>(m->alloc.get((size_t)s.vocab * D * 2));
        if (!m->embed) {
            vt_model_destroy(m);
            return fail(VT_ERR_ALLOC, "allocating the embedding table failed");
        }
    }
    m->status = static_cast<uint32_t*>(m->alloc.get(256));
    if (!m->status) {
        vt_model_destroy(m);
        return fail(VT_ERR_ALLOC, "allocating the model status word failed");
    }
    if (cudaMemsetAsync(m->status, 0, 256, st) != cudaSuccess) {
        vt_model_destroy(m);
        return fail(VT_ERR_CUDA, "clearing the model status word failed");
    }
    const size_t rope_bytes = (size_t)s.max_seq * (s.d_head / 2) * sizeof(float2);
    m->rope = static_cast<float2*>(m->alloc.get(rope_bytes));
    if (!m->rope) {
        vt_model_destroy(m);
        return fail(VT_ERR_ALLOC, "allocating the RoPE table failed");
    }
    cudaError_t e = launch_rope_table(m->rope, s.max_seq, s.d_head, (double)s.rope_theta, st);
    if (e != cudaSuccess) {
        vt_model_destroy(m);
        return fail(VT_ERR_CUDA, "RoPE table launch failed: %s", cudaGetErrorString(e));
    }
    if (per_layer) {
        for (int l = 0; l < s.n_layers; ++l) {
            vt_status r = vt_model_load_layer(m, l, &per_layer[l], stream);
            if (r != VT_OK) {
                std::string keep = t_err;
                vt_model_destroy(m);
                t_err = keep;
                return r;
            }
        }
    }
    if (embed && m->embed) {
        vt_status r = vt_model_load_embedding(m, embed, stream);
        if (r != VT_OK) {
            std::string keep = t_err;
            vt_model_destroy(m);
            t_err = keep;
            return r;
        }
    }
    e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) {
        vt_model_destroy(m);
        return fail(VT_ERR_CUDA, "model setup failed: %s", cudaGetErrorString(e));
    }
    *out = m;
    return ok();
}

extern "C" vt_status vt_model_shapes(const vt_model* m, vt_shapes* out) {
    if (!m || !out) return fail(VT_ERR_INVALID_ARG, "NULL argument");
    *out = m->s;
    return ok();
}

extern "C" vt_status vt_model_set_window(vt_model* m, int32_t layer, int32_t window) {
    if (!m) return fail(VT_ERR_INVALID_ARG, "model is NULL");
    if (layer < -1 || layer >= m->s.n_layers) return fail(VT_ERR_INVALID_ARG, "layer %d out of range", layer);
    if (window < 0) return fail(VT_ERR_INVALID_ARG, "window %d is negative", window);
    if (m->n_partitions > 0)
        return fail(VT_ERR_STATE, "attention windows are fixed while a partition of the model exists");
    for (int l = layer < 0 ? 0 : layer; l < (layer < 0 ? m->s.n_layers : layer + 1); ++l) m->window[l] = window;
    return ok();
}

extern "C" vt_status vt_model_window(const vt_model* m, int32_t layer, int32_t* window) {
    if (!m || !window) return fail(VT_ERR_INVALID_ARG, "NULL argument");
    if (layer < 0 || layer >= m->s.n_layers) return fail(VT_ERR_INVALID_ARG, "layer %d out of range", layer);
    *window = m->window[layer];
    return ok();
}

extern "C" vt_status vt_model_status(vt_model* m, uint32_t* flags, int32_t clear) {
    if (!m) return fail(VT_ERR_INVALID_ARG, "model is NULL");
    return read_status(m->status, flags, clear, nullptr);
}

extern "C" vt_status vt_embed(const vt_model* m, const int32_t* ids, int32_t n, void* out,
                              vt_stream stream) {
    if (!m || (!ids && n > 0) || (!out && n > 0) || n < 0)
        return fail(VT_ERR_INVALID_ARG, "bad vt_embed arguments");
    if (!m->embed || !m->embed_loaded) return fail(VT_ERR_STATE, "no embedding table loaded");
    if (n > 0 && !aligned16(out)) return fail(VT_ERR_INVALID_ARG, "out must be 16-byte aligned");
    VT_CUDA(launch_embed(m->embed, ids, n, m->s.d_model, m->s.vocab, static_cast<__half*>(out), m->status,
                         (cudaStream_t)stream));
    return ok();
}

// ================================================================== partition

extern "C" void vt_partition_destroy(vt_partition* p) {
    if (!p) return;
    cudaDeviceSynchronize();
    Allocator& A = p->m->alloc;
    for (auto& s : p->attn) A.put(s.base);
    for (auto& s : p->ffn) A.put(s.base);
    for (void* q : p->owned) A.put(q);
    if (p->counted) --p->m->n_partitions;
    delete p;
}

namespace {

struct Bump {  // carves one allocation into 256-byte aligned pieces
    uint8_t* base;
    size_t off = 0;
    template <typename T>
    T* take(size_t count) {
        T* r = reinterpret_cast<T*>(base + off);
        off += align256(count * sizeof(T));
        return r;
    }
};

vt_status owned_alloc(vt_partition* p, size_t bytes, void** out) {
    void* q = p->m->alloc.get(bytes);
    if (!q) return fail(VT_ERR_ALLOC, "allocating %zu bytes failed", bytes);
    p->owned.push_back(q);
    *out = q;
    return VT_OK;
}

}  // namespace

// Bytes of the row-pointer table the gather kernel reads while a shard is sliced.
static size_t gather_table_bytes(const vt_shapes& s) {
    const size_t rows = std::max((size_t)(s.n_heads + 2 * s.n_kv_heads) * s.d_head, (size_t)2 * s.d_ffn);
    return rows * sizeof(void*);
}

// The fp16 ATTN shard (l, d) sliced from the model's canonical weights into its own allocation:
// gain, QKV rows (query heads, then K heads, then V heads; each head's rows in RoPE-pair order),
// O columns.  rows_dev: a device table of gather_table_bytes (reused; the stream is synchronized).
static vt_status slice_attn_fp16(vt_partition* p, int l, int d, const __half** rows_dev, cudaStream_t st) {
    const vt_shapes& s = p->m->s;
    const LayerPtrs& L = p->m->layer[l];
    const int D = s.d_model, dh = s.d_head, H = s.n_heads;
    AttnShard& as = p->attn[(size_t)l * p->n_dev + d];
    const int hq = as.h1 - as.h0, hk = as.kv1 - as.kv0;
    const int qkv_rows = (hq + 2 * hk) * dh;
    if (hq == 0) return VT_OK;
    const size_t bytes = align256((size_t)D * 2) + align256((size_t)qkv_rows * D * 2) + align256((size_t)D * hq * dh * 2);
    as.base = p->m->alloc.get(bytes);
    if (!as.base) return fail(VT_ERR_ALLOC, "shard allocation failed");
    Bump b{static_cast<uint8_t*>(as.base)};
    as.norm = b.take<__half>(D);
    as.wqkv = b.take<__half>((size_t)qkv_rows * D);
    as.wo = b.take<__half>((size_t)D * hq * dh);
    as.bits = 16;
    VT_CUDA(cudaMemcpyAsync(as.norm, L.attn_norm, (size_t)D * 2, cudaMemcpyDeviceToDevice, st));
    std::vector<const __half*> rows_host;
    for (int blk = 0; blk < hq + 2 * hk; ++blk) {
        const __half* src;
        int head;
        if (blk < hq) {
            src = L.wq;
            head = as.h0 + blk;
        } else if (blk < hq + hk) {
            src = L.wk;
            head = as.kv0 + blk - hq;
        } else {
            src = L.wv;
            head = as.kv0 + blk - hq - hk;
        }
        for (int i = 0; i < dh / 2; ++i) {
            rows_host.push_back(src + ((size_t)head * dh + i) * D);
            rows_host.push_back(src + ((size_t)head * dh + i + dh / 2) * D);
        }
    }
    VT_CUDA(cudaMemcpyAsync(rows_dev, rows_host.data(), rows_host.size() * sizeof(void*), cudaMemcpyHostToDevice, st));
    VT_CUDA(launch_gather_rows(rows_dev, as.wqkv, (int)rows_host.size(), D, D, st));
    VT_CUDA(cudaStreamSynchronize(st));  // rows_host / rows_dev are reused
    VT_CUDA(cudaMemcpy2DAsync(as.wo, (size_t)hq * dh * 2, L.wo + (size_t)as.h0 * dh, (size_t)H * dh * 2,
                              (size_t)hq * dh * 2, D, cudaMemcpyDeviceToDevice, st));
    return VT_OK;
}

// The fp16 FFN shard (l, d): gain, gate/up rows interleaved, the transposed down columns.
static vt_status slice_ffn_fp16(vt_partition* p, int l, int d, const __half** rows_dev, cudaStream_t st) {
    const vt_shapes& s = p->m->s;
    const LayerPtrs& L = p->m->layer[l];
    const int D = s.d_model, F = s.d_ffn;
    FfnShard& fs = p->ffn[(size_t)l * p->n_dev + d];
    const int c = fs.c1 - fs.c0;
    if (c == 0) return VT_OK;
    const size_t bytes = align256((size_t)D * 2) + align256((size_t)2 * c * D * 2) + align256((size_t)c * D * 2);
    fs.base = p->m->alloc.get(bytes);
    if (!fs.base) return fail(VT_ERR_ALLOC, "shard allocation failed");
    Bump b{static_cast<uint8_t*>(fs.base)};
    fs.norm = b.take<__half>(D);
    fs.wgu = b.take<__half>((size_t)2 * c * D);
    fs.wdt = b.take<__half>((size_t)c * D);
    fs.bits = 16;
    VT_CUDA(cudaMemcpyAsync(fs.norm, L.ffn_norm, (size_t)D * 2, cudaMemcpyDeviceToDevice, st));
    std::vector<const __half*> rows_host;
    for (int j = 0; j < c; ++j) {
        rows_host.push_back(L.w_gate + (size_t)(fs.c0 + j) * D);
        rows_host.push_back(L.w_up + (size_t)(fs.c0 + j) * D);
    }
    VT_CUDA(cudaMemcpyAsync(rows_dev, rows_host.data(), rows_host.size() * sizeof(void*), cudaMemcpyHostToDevice, st));
    VT_CUDA(launch_gather_rows(rows_dev, fs.wgu, (int)rows_host.size(), D, D, st));
    VT_CUDA(cudaStreamSynchronize(st));
    VT_CUDA(launch_transpose_f16(L.w_down + fs.c0, F, D, c, fs.wdt, D, st));
    return VT_OK;
}

// heads / cols: [n_layers][n] ranges (per-layer partition table).
static vt_status partition_create(vt_model* m, int32_t n, const vt_range* heads, const vt_range* cols, uint32_t flags,
                                  vt_stream stream, vt_partition** out) {
    if (!out || !m) return fail(VT_ERR_INVALID_ARG, "NULL argument");
    *out = nullptr;
    VT_TRY(vt_partition_validate_layers(&m->s, n, heads, cols, flags));
    for (int l = 0; l < m->s.n_layers; ++l)
        if (!m->loaded[l]) return fail(VT_ERR_STATE, "layer %d weights were never loaded", l);
    cudaStream_t st = (cudaStream_t)stream;
    const vt_shapes& s = m->s;
    const int D = s.d_model, dh = s.d_head, H = s.n_heads, F = s.d_ffn;
    const int g = s.n_heads / s.n_kv_heads;
    vt_partition* p = new vt_partition();
    p->m = m;
    p->n_dev = n;
    p->counted = true;
    ++m->n_partitions;
    p->heads.assign(heads, heads + (size_t)m->s.n_layers * n);
    p->cols.assign(cols, cols + (size_t)m->s.n_layers * n);
    p->attn.resize((size_t)s.n_layers * n);
    p->ffn.resize((size_t)s.n_layers * n);
    Allocator& A = m->alloc;

    auto bail = [&](vt_status r) {
        std::string keep = t_err;
        vt_partition_destroy(p);
        t_err = keep;
        return r;
    };

    // host staging of row-pointer tables for the gather kernel (per layer)
    const __half** rows_dev = static_cast<const __half**>(A.get(gather_table_bytes(s)));
    if (!rows_dev) return bail(fail(VT_ERR_ALLOC, "allocating the gather table failed"));
    vt_status r = VT_OK;
    for (int l = 0; l < s.n_layers && r == VT_OK; ++l)
        for (int d = 0; d < n && r == VT_OK; ++d) {
            AttnShard& as = p->attn[(size_t)l * n + d];
            as.h0 = heads[(size_t)l * n + d].begin;
            as.h1 = heads[(size_t)l * n + d].end;
            as.kv0 = as.h0 / g;
            as.kv1 = as.h1 / g;
            FfnShard& fs = p->ffn[(size_t)l * n + d];
            fs.c0 = cols[(size_t)l * n + d].begin;
            fs.c1 = cols[(size_t)l * n + d].end;
            if ((r = slice_attn_fp16(p, l, d, rows_dev, st)) == VT_OK) r = slice_ffn_fp16(p, l, d, rows_dev, st);
        }
    A.put(rows_dev);
    if (r != VT_OK) return bail(r);

    // ------------------------------------------------------------------ decode scratch
    p->dec.resize(n);
    for (int d = 0; d < n; ++d) {
        // sized for this device's largest shard over the layers
        int hq = 0, c = 0;
        for (int l = 0; l < s.n_layers; ++l) {
            hq = std::max(hq, p->a(l, d).h1 - p->a(l, d).h0);
            c = std::max(c, p->f(l, d).c1 - p->f(l, d).c0);
            p->max_ld = std::max(p->max_ld, round_up8(p->f(l, d).c1 - p->f(l, d).c0 + p->f(l, d).c0 % 8));
        }
        const int hk = hq / g;
        DecodeScratch& ds = p->dec[d];
        ds.ffn_grid = ffn_grid(c);
        const size_t bytes = align256((size_t)std::max(hq, 1) * dh * 4) * 2 + align256((size_t)std::max(c, 1) * 4);
        void* q;
        if ((r = owned_alloc(p, bytes, &q)) != VT_OK) return bail(r);
        Bump b{static_cast<uint8_t*>(q)};
        ds.q = b.take<float>((size_t)std::max(hq, 1) * dh);
        ds.attn = b.take<float>((size_t)std::max(hq, 1) * dh);
        ds.u = b.take<float>((size_t)std::max(c, 1));
        VT_CUDA(cudaMemsetAsync(q, 0, bytes, st));
        p->max_hq = std::max(p->max_hq, hq);
        (void)hk;
    }
    // ------------------------------------------------------------------ stack + prefill scratch
    {
        const size_t R = kPrefillChunk;
        // q, attention output and u: one slot per shard, so the shards of a block run together
        p->q_slot = align256(R * std::max(p->max_hq, 1) * dh * 2) / 2;
        p->u_slot = align256(R * std::max(p->max_ld, 8) * 2) / 2;
        const size_t bytes = align256(4) + align256((size_t)n * D * 4) + align256((size_t)n * R * D * 4) + 2 * align256(R * D * 2) +
                             align256(R * 2 * D * 2) + 2 * (size_t)n * p->q_slot * 2 + (size_t)n * p->u_slot * 2;
        void* q;
        if ((r = owned_alloc(p, bytes, &q)) != VT_OK) return bail(r);
        Bump b{static_cast<uint8_t*>(q)};
        p->status = b.take<uint32_t>(1);
        p->dpart = b.take<float>((size_t)n * D);
        p->partials = b.take<float>((size_t)n * R * D);
        p->hbuf = b.take<__half>(R * D);
        p->xbuf = b.take<__half>(R * D);
        p->p_xhat = b.take<__half>(R * 2 * D);
        p->p_q = b.take<__half>((size_t)n * p->q_slot);
        p->p_attn = b.take<__half>((size_t)n * p->q_slot);
        p->p_u = b.take<__half>((size_t)n * p->u_slot);
        VT_CUDA(cudaMemsetAsync(q, 0, bytes, st));
    }
    // ------------------------------------------------------------------ quantized partials (communication scaling)
    {
        p->comm_bits.assign(n, 16);
        const size_t nbq = (size_t)(D + kQBlock - 1) / kQBlock;
        void* q;
        if ((r = owned_alloc(p, align256((size_t)n * D) + align256((size_t)n * nbq * 2), &q)) != VT_OK) return bail(r);
        Bump b{static_cast<uint8_t*>(q)};
        p->pcodes = b.take<uint8_t>((size_t)n * D);
        p->pscales = b.take<__half>((size_t)n * nbq);
    }
    // ------------------------------------------------------------------ decode-token kernel
    {
        TokArgs& t = p->tok_base;
        t = TokArgs{};
        t.n_layers = s.n_layers;
        t.n_dev = n;
        t.d = D;
        t.dh = dh;
        t.group = g;
        t.n_kv = s.n_kv_heads;
        t.eps = s.rms_eps;
        t.scale_log2 = (float)(1.4426950408889634 / sqrt((double)dh));
        t.rope = m->rope;
        for (int d = 0; d < n; ++d) {
            t.hq[d] = heads[d].end - heads[d].begin;
            t.hk[d] = t.hq[d] / g;
            t.h0[d] = heads[d].begin;
            t.kv0[d] = heads[d].begin / g;
            t.cols[d] = cols[d].end - cols[d].begin;
        }
        // the fused kernel takes one partition for every layer, covering every head and column
        bool uniform = (flags & VT_PARTITION_PRUNE) == 0;
        for (int l = 1; l < s.n_layers && uniform; ++l)
            for (int d = 0; d < n; ++d)
                uniform &= heads[(size_t)l * n + d].begin == heads[d].begin && heads[(size_t)l * n + d].end == heads[d].end &&
                           cols[(size_t)l * n + d].begin == cols[d].begin && cols[(size_t)l * n + d].end == cols[d].end;
        if (uniform) {
            p->tok_ok = p->tok_planned = token_plan(t, p->max_hq, &p->tok_plan, &p->tok_why);
        } else {
            p->tok_ok = p->tok_planned = false;
            p->tok_why = (flags & VT_PARTITION_PRUNE) ? "a pruned partition runs on the per-shard kernels"
                                                      : "a per-layer partition runs on the per-shard kernels";
        }
        if (p->tok_ok) {
            const size_t bytes = 2 * align256((size_t)H * dh * 4) + 2 * align256((size_t)n * D * 4) +
                                 align256(token_state_floats(p->tok_plan.grid, g, dh) * 4) +
                                 align256((size_t)kTokSyncWords * 4);
            void* q;
            if ((r = owned_alloc(p, bytes, &q)) != VT_OK) return bail(r);
            Bump b{static_cast<uint8_t*>(q)};
            t.q_all = b.take<float>((size_t)H * dh);
            t.attn_part = b.take<float>((size_t)n * D);
            t.ffn_part = b.take<float>((size_t)n * D);
            t.states = b.take<float>(token_state_floats(p->tok_plan.grid, g, dh));
            t.attn_out = b.take<float>((size_t)H * dh);
            t.sync = b.take<uint32_t>(kTokSyncWords);
            VT_CUDA(cudaMemsetAsync(q, 0, bytes, st));
        }
    }
    VT_CUDA(cudaStreamSynchronize(st));
    *out = p;
    return ok();
}

extern "C" vt_status vt_partition_create(vt_model* m, int32_t n, const vt_range* heads, const vt_range* cols,
                                         vt_stream stream, vt_partition** out) {
    if (!out || !m) return fail(VT_ERR_INVALID_ARG, "NULL argument");
    *out = nullptr;
    VT_TRY(vt_partition_validate(&m->s, n, heads, cols));
    std::vector<vt_range> hl((size_t)m->s.n_layers * n), cl((size_t)m->s.n_layers * n);
    for (int l = 0; l < m->s.n_layers; ++l)
        for (int d = 0; d < n; ++d) {
            hl[(size_t)l * n + d] = heads[d];
            cl[(size_t)l * n + d] = cols[d];
        }
    return partition_create(m, n, hl.data(), cl.data(), 0, stream, out);
}

extern "C" vt_status vt_partition_create_layers(vt_model* m, int32_t n, const vt_range* heads, const vt_range* cols,
                                                uint32_t flags, vt_stream stream, vt_partition** out) {
    return partition_create(m, n, heads, cols, flags, stream, out);
}

extern "C" int32_t vt_partition_devices(const vt_partition* p) { return p ? p->n_dev : 0; }

extern "C" vt_status vt_partition_status(vt_partition* p, uint32_t* flags, int32_t clear) {
    if (!p) return fail(VT_ERR_INVALID_ARG, "partition is NULL");
    return read_status(p->status, flags, clear, p->tok_base.sync);
}

static vt_status check_shard(const vt_partition* p, vt_shard sh) {
    if (!p) return fail(VT_ERR_INVALID_ARG, "partition is NULL");
    if (sh.layer < 0 || sh.layer >= p->m->s.n_layers || sh.device < 0 || sh.device >= p->n_dev ||
        (sh.block != VT_BLOCK_ATTN && sh.block != VT_BLOCK_FFN))
        return fail(VT_ERR_INVALID_ARG, "shard (layer %d, device %d, block %d) out of range",
                    sh.layer, sh.device, sh.block);
    return VT_OK;
}

extern "C" vt_status vt_shard_weight_layout(const vt_partition* p, vt_shard sh, int32_t which,
                                            int64_t* rows, int64_t* stride) {
    VT_TRY(check_shard(p, sh));
    if (!rows || !stride) return fail(VT_ERR_INVALID_ARG, "NULL output");
    const vt_shapes& s = p->m->s;
    const AttnShard& a = p->a(sh.layer, sh.device);
    const FfnShard& f = p->f(sh.layer, sh.device);
    const int hq = a.h1 - a.h0, hk = a.kv1 - a.kv0, c = f.c1 - f.c0;
    if (((which == 1 || which == 2) && a.bits != 16) || ((which == 4 || which == 5) && f.bits != 16))
        return fail(VT_ERR_STATE, "tensor %d of the shard is block-quantized: read it with vt_shard_qweights_read", which);
    switch (which) {
        case 0: *rows = hq > 0; *stride = s.d_model; break;
        case 1: *rows = (int64_t)(hq + 2 * hk) * s.d_head; *stride = s.d_model; break;
        case 2: *rows = hq > 0 ? s.d_model : 0; *stride = (int64_t)hq * s.d_head; break;
        case 3: *rows = c > 0; *stride = s.d_model; break;
        case 4: *rows = 2 * (int64_t)c; *stride = s.d_model; break;
        case 5: *rows = c; *stride = s.d_model; break;
        default: return fail(VT_ERR_INVALID_ARG, "unknown tensor %d", which);
    }
    return ok();
}

extern "C" vt_status vt_shard_weights_read(const vt_partition* p, vt_shard sh, int32_t which,
                                           void* dst, size_t bytes, size_t* size_out) {
    int64_t rows = 0, stride = 0;
    VT_TRY(vt_shard_weight_layout(p, sh, which, &rows, &stride));
    const AttnShard& a = p->a(sh.layer, sh.device);
    const FfnShard& f = p->f(sh.layer, sh.device);
    const __half* src = nullptr;
    switch (which) {
        case 0: src = a.norm; break;
        case 1: src = a.wqkv; break;
        case 2: src = a.wo; break;
        case 3: src = f.norm; break;
        case 4: src = f.wgu; break;
        default: src = f.wdt; break;
    }
    const size_t size = (size_t)rows * stride * 2;
    if (size_out) *size_out = size;
    const size_t nb = std::min(bytes, size);
    if (nb > 0) {
        if (!dst) return fail(VT_ERR_INVALID_ARG, "dst is NULL");
        VT_CUDA(cudaDeviceSynchronize());
        VT_CUDA(cudaMemcpy(dst, src, nb, cudaMemcpyDeviceToHost));
    }
    return ok();
}

// ------------------------------------------------------------------ shard precision

// Quantized matrix storage for `rows` x `k` at `bits` carved from a Bump.
static QMatDev take_qmat(Bump& b, int rows, int k, int bits) {
    QMatDev m;
    m.rows = rows;
    m.k = k;
    m.nb = (k + kQBlock - 1) / kQBlock;
    m.bits = bits;
    m.row_bytes = (int64_t)m.nb * (bits == 8 ? 32 : 16);
    m.codes = b.take<uint8_t>(qmat_code_bytes(rows, k, bits));
    m.scales = b.take<__half>((size_t)rows * m.nb);
    return m;
}

static size_t qmat_bytes(int rows, int k, int bits) {
    return align256(qmat_code_bytes(rows, k, bits)) + align256(qmat_scale_bytes(rows, k));
}

static void update_token_kernel(vt_partition* p) {
    bool quantized = false, comm = false;
    for (const AttnShard& a : p->attn) quantized |= a.bits != 16;
    for (const FfnShard& f : p->ffn) quantized |= f.bits != 16;
    for (int b : p->comm_bits) comm |= b != 16;
    p->tok_ok = p->tok_planned && !quantized && !comm;
    if (p->tok_planned && quantized) p->tok_why = "a shard is block-quantized: the token runs on the per-shard kernels";
    else if (p->tok_planned && comm) p->tok_why = "partials are quantized for transmission: the token runs on the per-shard kernels";
}

extern "C" vt_status vt_partition_set_precision(vt_partition* p, vt_shard sh, int32_t bits, vt_stream stream) {
    VT_TRY(check_shard(p, sh));
    if (bits != 16 && bits != 8 && bits != 4) return fail(VT_ERR_INVALID_ARG, "bits %d must be 16, 8 or 4", bits);
    if (p->n_kv > 0) return fail(VT_ERR_STATE, "shard precisions are fixed while a KV cache of the partition exists");
    cudaStream_t st = (cudaStream_t)stream;
    const vt_shapes& s = p->m->s;
    const int D = s.d_model, dh = s.d_head, l = sh.layer, d = sh.device;
    Allocator& A = p->m->alloc;
    const __half** rows_dev = nullptr;
    auto table = [&]() -> const __half** {
        if (!rows_dev) rows_dev = static_cast<const __half**>(A.get(gather_table_bytes(s)));
        return rows_dev;
    };
    vt_status r = VT_OK;
    if (sh.block == VT_BLOCK_ATTN) {
        AttnShard& a = p->attn[(size_t)l * p->n_dev + d];
        const int hq = a.h1 - a.h0, hk = a.kv1 - a.kv0, K = hq * dh, rows = (hq + 2 * hk) * dh;
        if (hq == 0 || bits == a.bits) {
            // an empty shard stores nothing and stays fp16
        } else {
            if (a.bits != 16) {  // back to the fp16 slices first
                VT_CUDA(cudaStreamSynchronize(st));
                A.put(a.base);
                a.base = nullptr;
                if (!table()) return fail(VT_ERR_ALLOC, "allocating the gather table failed");
                r = slice_attn_fp16(p, l, d, rows_dev, st);
            }
            if (r == VT_OK && bits != 16) {
                void* nb = A.get(align256((size_t)D * 2) + qmat_bytes(rows, D, bits) + qmat_bytes(D, K, bits));
                if (!nb) {
                    r = fail(VT_ERR_ALLOC, "allocating the quantized shard failed");
                } else {
                    Bump b{static_cast<uint8_t*>(nb)};
                    __half* norm = b.take<__half>(D);
                    const QMatDev qkv = take_qmat(b, rows, D, bits), o = take_qmat(b, D, K, bits);
                    cudaError_t e = cudaMemcpyAsync(norm, a.norm, (size_t)D * 2, cudaMemcpyDeviceToDevice, st);
                    if (e == cudaSuccess) e = launch_quantize_rows(a.wqkv, D, qkv, st);
                    if (e == cudaSuccess) e = launch_quantize_rows(a.wo, K, o, st);
                    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
                    if (e != cudaSuccess) {
                        A.put(nb);
                        r = fail(VT_ERR_CUDA, "quantizing the shard failed: %s", cudaGetErrorString(e));
                    } else {
                        A.put(a.base);
                        a.base = nb;
                        a.norm = norm;
                        a.wqkv = a.wo = nullptr;
                        a.qkv = qkv;
                        a.o = o;
                        a.bits = bits;
                    }
                }
            }
        }
    } else {
        FfnShard& f = p->ffn[(size_t)l * p->n_dev + d];
        const int c = f.c1 - f.c0;
        if (c == 0 || bits == f.bits) {
            // an empty shard stores nothing and stays fp16
        } else {
            if (f.bits != 16) {
                VT_CUDA(cudaStreamSynchronize(st));
                A.put(f.base);
                f.base = nullptr;
                if (!table()) return fail(VT_ERR_ALLOC, "allocating the gather table failed");
                r = slice_ffn_fp16(p, l, d, rows_dev, st);
            }
            if (r == VT_OK && bits != 16) {
                void* nb = A.get(align256((size_t)D * 2) + qmat_bytes(2 * c, D, bits) + qmat_bytes(D, c, bits));
                if (!nb) {
                    r = fail(VT_ERR_ALLOC, "allocating the quantized shard failed");
                } else {
                    Bump b{static_cast<uint8_t*>(nb)};
                    __half* norm = b.take<__half>(D);
                    const QMatDev gu = take_qmat(b, 2 * c, D, bits), dn = take_qmat(b, D, c, bits);
                    cudaError_t e = cudaMemcpyAsync(norm, f.norm, (size_t)D * 2, cudaMemcpyDeviceToDevice, st);
                    if (e == cudaSuccess) e = launch_quantize_rows(f.wgu, D, gu, st);
                    // the down projection is quantized along the shard's columns: rows of Wd[:, c0:c1]
                    if (e == cudaSuccess) e = launch_quantize_rows(p->m->layer[l].w_down + f.c0, s.d_ffn, dn, st);
                    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
                    if (e != cudaSuccess) {
                        A.put(nb);
                        r = fail(VT_ERR_CUDA, "quantizing the shard failed: %s", cudaGetErrorString(e));
                    } else {
                        A.put(f.base);
                        f.base = nb;
                        f.norm = norm;
                        f.wgu = f.wdt = nullptr;
                        f.gu = gu;
                        f.down = dn;
                        f.bits = bits;
                    }
                }
            }
        }
    }
    if (rows_dev) A.put(rows_dev);
    update_token_kernel(p);
    if (r != VT_OK) return r;
    return ok();
}

extern "C" int32_t vt_shard_precision(const vt_partition* p, vt_shard sh) {
    if (check_shard(p, sh) != VT_OK) return 0;
    return sh.block == VT_BLOCK_ATTN ? p->a(sh.layer, sh.device).bits : p->f(sh.layer, sh.device).bits;
}

extern "C" vt_status vt_shard_qweights_read(const vt_partition* p, vt_shard sh, int32_t which, int8_t* codes,
                                            void* scales) {
    VT_TRY(check_shard(p, sh));
    const bool attn = which == 1 || which == 2, ffn = which == 4 || which == 5;
    if (!attn && !ffn) return fail(VT_ERR_INVALID_ARG, "tensor %d has no quantized form", which);
    if ((attn && sh.block != VT_BLOCK_ATTN) || (ffn && sh.block != VT_BLOCK_FFN))
        return fail(VT_ERR_INVALID_ARG, "tensor %d does not belong to block %d", which, sh.block);
    const QMatDev* m = nullptr;
    if (attn) {
        const AttnShard& a = p->a(sh.layer, sh.device);
        if (a.bits == 16 || a.h1 == a.h0) return fail(VT_ERR_STATE, "the shard is not block-quantized");
        m = which == 1 ? &a.qkv : &a.o;
    } else {
        const FfnShard& f = p->f(sh.layer, sh.device);
        if (f.bits == 16 || f.c1 == f.c0) return fail(VT_ERR_STATE, "the shard is not block-quantized");
        m = which == 4 ? &f.gu : &f.down;
    }
    if (!codes || !scales) return fail(VT_ERR_INVALID_ARG, "codes and scales must not be NULL");
    std::vector<uint8_t> raw(qmat_code_bytes(m->rows, m->k, m->bits));
    VT_CUDA(cudaDeviceSynchronize());
    VT_CUDA(cudaMemcpy(raw.data(), m->codes, raw.size(), cudaMemcpyDeviceToHost));
    VT_CUDA(cudaMemcpy(scales, m->scales, qmat_scale_bytes(m->rows, m->k), cudaMemcpyDeviceToHost));
    unpack_qcodes(raw.data(), m->rows, m->k, m->bits, codes);
    return ok();
}

// ================================================================== KV cache

extern "C" void vt_kv_destroy(vt_kv* kv) {
    if (!kv) return;
    cudaDeviceSynchronize();
    --kv->p->n_kv;
    Allocator* A = kv->alloc();
    for (void* b : kv->buf) A->put(b);
    A->put(kv->len);
    A->put(kv->tok_tab);
    delete kv;
}

extern "C" vt_status vt_kv_create(const vt_partition* p, int32_t cap, vt_stream stream, vt_kv** out) {
    if (!p || !out) return fail(VT_ERR_INVALID_ARG, "NULL argument");
    *out = nullptr;
    const vt_shapes& s = p->m->s;
    if (cap < 1 || cap > s.max_seq)
        return fail(VT_ERR_INVALID_ARG, "capacity %d must be in [1, max_seq = %d]", cap, s.max_seq);
    cudaStream_t st = (cudaStream_t)stream;
    vt_kv* kv = new vt_kv();
    kv->p = p;
    kv->cap = cap;
    ++p->n_kv;
    kv->buf.assign((size_t)s.n_layers * p->n_dev, nullptr);
    Allocator* A = kv->alloc();
    for (int l = 0; l < s.n_layers; ++l)
        for (int d = 0; d < p->n_dev; ++d) {
            const AttnShard& a = p->a(l, d);
            const int hk = a.kv1 - a.kv0;
            if (hk == 0) continue;
            const size_t bytes = (size_t)2 * hk * cap * s.d_head * 2;
            void* b = A->get(bytes);
            if (!b) {
                vt_kv_destroy(kv);
                return fail(VT_ERR_ALLOC, "allocating the KV cache of layer %d device %d failed", l, d);
            }
            kv->buf[(size_t)l * p->n_dev + d] = b;
            cudaError_t e = cudaMemsetAsync(b, 0, bytes, st);
            if (e != cudaSuccess) {
                vt_kv_destroy(kv);
                return fail(VT_ERR_CUDA, "cudaMemsetAsync failed: %s", cudaGetErrorString(e));
            }
        }
    const size_t meta = align256((size_t)s.n_layers * 4) + 256;
    uint8_t* mb = static_cast<uint8_t*>(A->get(meta));
    if (!mb) {
        vt_kv_destroy(kv);
        return fail(VT_ERR_ALLOC, "allocating KV lengths failed");
    }
    kv->len = reinterpret_cast<int32_t*>(mb);
    kv->status = reinterpret_cast<uint32_t*>(mb + align256((size_t)s.n_layers * 4));
    kv->h_len.assign(s.n_layers, 0);
    // pointer tables of the decode-token kernel (host copies live until the synchronise below)
    std::vector<TokShardPtrs> tsh;
    std::vector<TokLayerPtrs> tly;
    if (p->tok_ok) {
        const int L = s.n_layers, n = p->n_dev;
        tsh.resize((size_t)L * n);
        tly.resize(L);
        for (int l = 0; l < L; ++l) {
            tly[l].attn_norm = p->m->layer[l].attn_norm;
            tly[l].ffn_norm = p->m->layer[l].ffn_norm;
            tly[l].window = p->m->window[l];
            for (int d = 0; d < n; ++d) {
                const AttnShard& a = p->a(l, d);
                const FfnShard& f = p->f(l, d);
                TokShardPtrs& t = tsh[(size_t)l * n + d];
                t.wqkv = a.wqkv;
                t.wo = a.wo;
                t.wgu = f.wgu;
                t.wdt = f.wdt;
                t.kc = a.kv1 > a.kv0 ? kv->k(l, d) : nullptr;
                t.vc = a.kv1 > a.kv0 ? kv->v(l, d) : nullptr;
            }
        }
        const size_t tb = align256(tsh.size() * sizeof(TokShardPtrs)) + tly.size() * sizeof(TokLayerPtrs);
        kv->tok_tab = A->get(tb);
        if (!kv->tok_tab) {
            vt_kv_destroy(kv);
            return fail(VT_ERR_ALLOC, "allocating the decode-token tables failed");
        }
        uint8_t* tp = static_cast<uint8_t*>(kv->tok_tab);
        cudaError_t te = cudaMemcpyAsync(tp, tsh.data(), tsh.size() * sizeof(TokShardPtrs), cudaMemcpyHostToDevice, st);
        if (te == cudaSuccess)
            te = cudaMemcpyAsync(tp + align256(tsh.size() * sizeof(TokShardPtrs)), tly.data(),
                                 tly.size() * sizeof(TokLayerPtrs), cudaMemcpyHostToDevice, st);
        if (te != cudaSuccess) {
            vt_kv_destroy(kv);
            return fail(VT_ERR_CUDA, "uploading the decode-token tables failed: %s", cudaGetErrorString(te));
        }
    }
    cudaError_t e = cudaMemsetAsync(mb, 0, meta, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) {
        vt_kv_destroy(kv);
        return fail(VT_ERR_CUDA, "KV setup failed: %s", cudaGetErrorString(e));
    }
    *out = kv;
    return ok();
}

extern "C" int32_t vt_kv_capacity(const vt_kv* kv) { return kv ? kv->cap : 0; }

extern "C" vt_status vt_kv_advance(vt_kv* kv, int32_t layer, int32_t n, vt_stream stream) {
    if (!kv) return fail(VT_ERR_INVALID_ARG, "kv is NULL");
    const int L = kv->p->m->s.n_layers;
    if (layer < -1 || layer >= L) return fail(VT_ERR_INVALID_ARG, "layer %d out of range", layer);
    const int first = layer < 0 ? 0 : layer, count = layer < 0 ? L : 1;
    const bool cap_mode = capturing((cudaStream_t)stream);
    if (!cap_mode)  // while capturing, the device clamps and flags instead (the mirror is stale)
        for (int l = first; l < first + count; ++l)
            if ((int64_t)kv->h_len[l] + n > kv->cap || (int64_t)kv->h_len[l] + n < 0)
                return fail(VT_ERR_KV_CAPACITY, "advancing layer %d from %d by %d leaves [0, %d]", l,
                            kv->h_len[l], n, kv->cap);
    VT_CUDA(launch_kv_advance(kv->len, first, count, n, kv->cap, kv->status, (cudaStream_t)stream));
    if (!cap_mode)
        for (int l = first; l < first + count; ++l) kv->h_len[l] += n;
    return ok();
}

extern "C" vt_status vt_kv_set_length(vt_kv* kv, int32_t layer, int32_t len, vt_stream stream) {
    if (!kv) return fail(VT_ERR_INVALID_ARG, "kv is NULL");
    const int L = kv->p->m->s.n_layers;
    if (layer < -1 || layer >= L) return fail(VT_ERR_INVALID_ARG, "layer %d out of range", layer);
    if (len < 0 || len > kv->cap) return fail(VT_ERR_KV_CAPACITY, "length %d outside [0, %d]", len, kv->cap);
    const int first = layer < 0 ? 0 : layer, count = layer < 0 ? L : 1;
    cudaStream_t st = (cudaStream_t)stream;
    std::vector<int32_t> v(count, len);
    VT_CUDA(cudaMemcpyAsync(kv->len + first, v.data(), count * 4, cudaMemcpyHostToDevice, st));
    VT_CUDA(cudaStreamSynchronize(st));
    for (int l = first; l < first + count; ++l) kv->h_len[l] = len;
    return ok();
}

extern "C" vt_status vt_kv_length(vt_kv* kv, int32_t layer, vt_stream stream, int32_t* out) {
    if (!kv || !out) return fail(VT_ERR_INVALID_ARG, "NULL argument");
    if (layer < 0 || layer >= kv->p->m->s.n_layers)
        return fail(VT_ERR_INVALID_ARG, "layer %d out of range", layer);
    cudaStream_t st = (cudaStream_t)stream;
    VT_CUDA(cudaMemcpyAsync(out, kv->len + layer, 4, cudaMemcpyDeviceToHost, st));
    VT_CUDA(cudaStreamSynchronize(st));
    kv->h_len[layer] = *out;
    return ok();
}

extern "C" vt_status vt_kv_status(vt_kv* kv, uint32_t* flags, int32_t clear) {
    if (!kv) return fail(VT_ERR_INVALID_ARG, "kv is NULL");
    return read_status(kv->status, flags, clear, kv->p->tok_base.sync);
}

static vt_status kv_copy(const vt_kv* kv, int32_t l, int32_t d, int32_t n_pos, void* kh,
                         const void* kh_in, void* vh, const void* vh_in) {
    if (!kv) return fail(VT_ERR_INVALID_ARG, "kv is NULL");
    const vt_partition* p = kv->p;
    if (l < 0 || l >= p->m->s.n_layers || d < 0 || d >= p->n_dev)
        return fail(VT_ERR_INVALID_ARG, "(layer %d, device %d) out of range", l, d);
    if (n_pos < 0 || n_pos > kv->cap) return fail(VT_ERR_KV_CAPACITY, "n_pos %d outside [0, %d]", n_pos, kv->cap);
    const AttnShard& a = p->a(l, d);
    const int hk = a.kv1 - a.kv0, dh = p->m->s.d_head;
    if (hk == 0 || n_pos == 0) return ok();
    VT_CUDA(cudaDeviceSynchronize());
    const size_t row = (size_t)n_pos * dh * 2, pitch = (size_t)kv->cap * dh * 2;
    if (kh_in) {
        VT_CUDA(cudaMemcpy2D(kv->k(l, d), pitch, kh_in, row, row, hk, cudaMemcpyHostToDevice));
        VT_CUDA(cudaMemcpy2D(kv->v(l, d), pitch, vh_in, row, row, hk, cudaMemcpyHostToDevice));
    } else {
        VT_CUDA(cudaMemcpy2D(kh, row, kv->k(l, d), pitch, row, hk, cudaMemcpyDeviceToHost));
        VT_CUDA(cudaMemcpy2D(vh, row, kv->v(l, d), pitch, row, hk, cudaMemcpyDeviceToHost));
    }
    return ok();
}

extern "C" vt_status vt_kv_read(const vt_kv* kv, int32_t l, int32_t d, int32_t n_pos, void* kh,
                                void* vh) {
    if (!kh || !vh) return fail(VT_ERR_INVALID_ARG, "NULL host buffer");
    return kv_copy(kv, l, d, n_pos, kh, nullptr, vh, nullptr);
}

extern "C" vt_status vt_kv_write_raw(vt_kv* kv, int32_t l, int32_t d, int32_t n_pos,
                                     const void* kh, const void* vh) {
    if (!kh || !vh) return fail(VT_ERR_INVALID_ARG, "NULL host buffer");
    return kv_copy(kv, l, d, n_pos, nullptr, kh, nullptr, vh);
}

// ================================================================== shard compute

// QKV projection of ATTN shard (l, d) with RoPE and the K/V append at the layer's length: the
// fp16 GEMV or, for a block-quantized shard, the dequantizing one.  q: [hq][dh] rotated queries.
// indep: the caller guarantees that `x` was written at least two kernel launches before (the
// fp16 GEMV may then read it before griddepcontrol.wait).
static cudaError_t attn_qkv(const vt_partition* p, int l, int d, const __half* x, vt_kv* kv, float* q,
                            cudaStream_t st, int indep) {
    const vt_shapes& s = p->m->s;
    const AttnShard& a = p->a(l, d);
    const int hq = a.h1 - a.h0, hk = a.kv1 - a.kv0, dh = s.d_head, D = s.d_model;
    if (a.bits != 16) {
        QGemvArgs g{};
        g.w = a.qkv;
        g.x = x;
        g.gain = a.norm;
        g.eps = s.rms_eps;
        g.out = q;
        g.kcache = kv->k(l, d);
        g.vcache = kv->v(l, d);
        g.cap = kv->cap;
        g.len = kv->len + l;
        g.rope = p->m->rope;
        g.dh = dh;
        g.hq = hq;
        g.hk = hk;
        g.status = kv->status;
        return launch_gemv_q(kEpiQkvRope, g, st);
    }
    GemvArgs g{};
    g.w = a.wqkv;
    g.row_stride = D;
    g.rows = (hq + 2 * hk) * dh;
    g.k = D;
    g.x = x;
    g.gain = a.norm;
    g.eps = s.rms_eps;
    g.out = q;
    g.kcache = kv->k(l, d);
    g.vcache = kv->v(l, d);
    g.cap = kv->cap;
    g.len = kv->len + l;
    g.rope = p->m->rope;
    g.dh = dh;
    g.hq = hq;
    g.hk = hk;
    g.status = kv->status;
    g.indep = indep;
    return launch_gemv(kEpiQkvRope, g, st);
}

// O projection of ATTN shard (l, d): out [D] = Wo_s . attn (fp32), fp16 or block-quantized.
static cudaError_t attn_o(const vt_partition* p, int l, int d, const float* attn, float* out, uint32_t* status,
                          cudaStream_t st) {
    const vt_shapes& s = p->m->s;
    const AttnShard& a = p->a(l, d);
    const int hq = a.h1 - a.h0, dh = s.d_head, D = s.d_model;
    if (a.bits != 16) {
        QGemvArgs o{};
        o.w = a.o;
        o.vin = attn;
        o.out = out;
        o.status = status;
        return launch_gemv_q(kEpiPlain, o, st);
    }
    GemvArgs o{};
    o.w = a.wo;
    o.row_stride = (int64_t)hq * dh;
    o.rows = D;
    o.k = hq * dh;
    o.vin = attn;
    o.out = out;
    o.status = status;
    return launch_gemv(kEpiPlain, o, st);
}

// indep: the caller guarantees that `x` was written at least two kernel launches before this
// shard's first kernel, so that kernel may read it before griddepcontrol.wait (see k_gemv).
static vt_status decode_attn(const vt_partition* p, int l, int d, const __half* x, vt_kv* kv,
                             float* out, cudaStream_t st, int indep = 0) {
    const vt_shapes& s = p->m->s;
    const AttnShard& a = p->a(l, d);
    const DecodeScratch& ds = p->dec[d];
    const int hq = a.h1 - a.h0, hk = a.kv1 - a.kv0, dh = s.d_head, D = s.d_model;
    if (hq == 0) {
        VT_CUDA(launch_fill_zero_f32(out, D, st));
        return VT_OK;
    }
    VT_CUDA(attn_qkv(p, l, d, x, kv, ds.q, st, indep));

    AttnDecodeArgs t{};
    t.q = ds.q;
    t.kcache = kv->k(l, d);
    t.vcache = kv->v(l, d);
    t.len = kv->len + l;
    t.cap = kv->cap;
    t.hk = hk;
    t.group = s.n_heads / s.n_kv_heads;
    t.dh = dh;
    t.stages = attn_stages(kv->cap, attn_cluster_size(hk));
    t.scale_log2 = (float)(1.4426950408889634 / sqrt((double)dh));
    t.window = p->m->window[l];
    t.out = ds.attn;
    t.status = kv->status;
    VT_CUDA(launch_attn_decode(t, st));
    VT_CUDA(attn_o(p, l, d, ds.attn, out, kv->status, st));
    return VT_OK;
}

// FFN shard decode: the fused column-split kernel adds every CTA's partial into `out`, which
// must hold zeros; `zero_first` clears it in stream order before the kernel runs.
static vt_status decode_ffn(const vt_partition* p, int l, int d, const __half* x, float* out,
                            cudaStream_t st, int indep = 0, bool zero_first = true) {
    const vt_shapes& s = p->m->s;
    const FfnShard& f = p->f(l, d);
    const DecodeScratch& ds = p->dec[d];
    const int c = f.c1 - f.c0, D = s.d_model;
    if (f.bits != 16 && c > 0) {
        // block-quantized shard: gate/up rows with the SwiGLU epilogue, then the down columns (the
        // partial is written, not added)
        QGemvArgs g{};
        g.w = f.gu;
        g.x = x;
        g.gain = f.norm;
        g.eps = s.rms_eps;
        g.out = ds.u;
        g.status = p->status;
        VT_CUDA(launch_gemv_q(kEpiSwiglu, g, st));
        QGemvArgs o{};
        o.w = f.down;
        o.vin = ds.u;
        o.out = out;
        o.status = p->status;
        VT_CUDA(launch_gemv_q(kEpiPlain, o, st));
        return VT_OK;
    }
    if (zero_first) VT_CUDA(launch_fill_zero_f32(out, D, st));
    if (c == 0) return VT_OK;
    FfnDecodeArgs g{};
    g.x = x;
    g.gain = f.norm;
    g.eps = s.rms_eps;
    g.wgu = f.wgu;
    g.wdt = f.wdt;
    g.d = D;
    g.cols = c;
    g.out = out;
    g.indep = indep;
    VT_CUDA(launch_ffn_decode(g, ds.ffn_grid, st));
    return VT_OK;
}

extern "C" vt_status vt_decode_step(const vt_partition* p, vt_shard sh, const void* x, vt_kv* kv,
                                    float* out, vt_stream stream) {
    VT_TRY(check_shard(p, sh));
    if (!x || !out) return fail(VT_ERR_INVALID_ARG, "x and out_partial must not be NULL");
    if (!aligned16(x)) return fail(VT_ERR_INVALID_ARG, "x must be 16-byte aligned");
    cudaStream_t st = (cudaStream_t)stream;
    if (sh.block == VT_BLOCK_ATTN) {
        if (!kv || kv->p != p) return fail(VT_ERR_INVALID_ARG, "an ATTN shard needs this partition's KV cache");
        if (kv->h_len[sh.layer] + 1 > kv->cap)
            return fail(VT_ERR_KV_CAPACITY, "layer %d holds %d of %d positions", sh.layer,
                        kv->h_len[sh.layer], kv->cap);
        VT_TRY(decode_attn(p, sh.layer, sh.device, static_cast<const __half*>(x), kv, out, st));
    } else {
        VT_TRY(decode_ffn(p, sh.layer, sh.device, static_cast<const __half*>(x), out, st));
    }
    return ok();
}

// ATTN shard step with every intermediate in the module's static scratch array: the same QKV and
// O kernels as decode_attn, with the split-K attention kernel of static_scratch.cu between them.
// Touches neither the partition's decode scratch nor any allocator.
extern "C" vt_status vt_decode_step_static(const vt_partition* p, vt_shard sh, const void* x, vt_kv* kv,
                                           float* out, vt_stream stream) {
    VT_TRY(check_shard(p, sh));
    if (sh.block != VT_BLOCK_ATTN)
        return fail(VT_ERR_INVALID_ARG, "vt_decode_step_static runs ATTN shards only (an FFN shard uses no scratch: call vt_decode_step)");
    if (!x || !out) return fail(VT_ERR_INVALID_ARG, "x and out_partial must not be NULL");
    if (!aligned16(x)) return fail(VT_ERR_INVALID_ARG, "x must be 16-byte aligned");
    if (!kv || kv->p != p) return fail(VT_ERR_INVALID_ARG, "an ATTN shard needs this partition's KV cache");
    if (kv->h_len[sh.layer] + 1 > kv->cap)
        return fail(VT_ERR_KV_CAPACITY, "layer %d holds %d of %d positions", sh.layer, kv->h_len[sh.layer], kv->cap);
    const vt_shapes& s = p->m->s;
    const AttnShard& a = p->a(sh.layer, sh.device);
    const int hq = a.h1 - a.h0, hk = a.kv1 - a.kv0, dh = s.d_head, D = s.d_model, l = sh.layer, d = sh.device;
    cudaStream_t st = (cudaStream_t)stream;
    if (hq == 0) {
        VT_CUDA(launch_fill_zero_f32(out, D, st));
        return ok();
    }
    const StaticAttnLayout lay = static_attn_layout(hq, hk, dh);
    if (hk > kStaticMaxKvHeads || lay.bytes > kStaticScratchBytes)
        return fail(VT_ERR_INVALID_ARG,
                    "shard (layer %d, device %d) needs %zu bytes of static scratch for %d query and %d KV "
                    "heads of dim %d; the array holds %zu bytes and %d KV heads",
                    l, d, lay.bytes, hq, hk, dh, kStaticScratchBytes, kStaticMaxKvHeads);
    void* base = nullptr;
    cudaError_t ce = static_scratch_base(&base);
    if (ce != cudaSuccess)
        return fail(VT_ERR_CUDA, "looking up the static scratch address failed: %s", cudaGetErrorString(ce));
    uint8_t* b = static_cast<uint8_t*>(base);
    float* q = reinterpret_cast<float*>(b + lay.q);
    float* attn = reinterpret_cast<float*>(b + lay.attn);

    VT_CUDA(attn_qkv(p, l, d, static_cast<const __half*>(x), kv, q, st, 0));

    StaticAttnArgs t{};
    t.q = q;
    t.kcache = kv->k(l, d);
    t.vcache = kv->v(l, d);
    t.len = kv->len + l;
    t.cap = kv->cap;
    t.hk = hk;
    t.group = s.n_heads / s.n_kv_heads;
    t.dh = dh;
    t.scale_log2 = (float)(1.4426950408889634 / sqrt((double)dh));
    t.window = p->m->window[l];
    t.part_ml = reinterpret_cast<float*>(b + lay.part_ml);
    t.part_o = reinterpret_cast<float*>(b + lay.part_o);
    t.counters = reinterpret_cast<uint32_t*>(b + lay.counters);
    t.out = attn;
    VT_CUDA(launch_attn_decode_static(t, st));

    VT_CUDA(attn_o(p, l, d, attn, out, kv->status, st));
    return ok();
}

extern "C" vt_status vt_combine(const float* const* partials, int32_t n, int32_t rows, int32_t d,
                                const void* residual, void* out, vt_stream stream) {
    if (!partials || !out || n < 1 || n > VT_MAX_DEVICES || rows < 0 || d < 0)
        return fail(VT_ERR_INVALID_ARG, "bad vt_combine arguments");
    CombineArgs c{};
    for (int s = 0; s < n; ++s) {
        if (!partials[s]) return fail(VT_ERR_INVALID_ARG, "partial %d is NULL", s);
        c.parts[s] = const_cast<float*>(partials[s]);
    }
    c.n = n;
    c.count = (int64_t)rows * d;
    c.residual = static_cast<const __half*>(residual);
    c.out = static_cast<__half*>(out);
    VT_CUDA(launch_combine(c, (cudaStream_t)stream));
    return ok();
}

// ------------------------------------------------------------------ prefill

// Arguments of one shard's prefill.  xhat_ready: the partition's xhat scratch already holds
// RMSNorm(x) with this block's gain (the whole-stack path computes it once per block, in the
// combine that produced x).  slot: the shard's q / attention / u scratch slot.
static void attn_args(const vt_partition* p, vt_shard sh, const __half* x, int n, vt_kv* kv, float* out,
                      int row_offset, bool xhat_ready, int slot, PrefillAttnArgs* t) {
    const vt_shapes& s = p->m->s;
    const AttnShard& a = p->a(sh.layer, sh.device);
    *t = PrefillAttnArgs{};
    t->n = n;
    t->d = s.d_model;
    t->dh = s.d_head;
    t->hq = a.h1 - a.h0;
    t->hk = a.kv1 - a.kv0;
    t->eps = s.rms_eps;
    t->scale_log2 = (float)(1.4426950408889634 / sqrt((double)s.d_head));
    t->x = x;
    t->gain = a.norm;
    t->wqkv = a.wqkv;
    t->wo = a.wo;
    t->kcache = kv->k(sh.layer, sh.device);
    t->vcache = kv->v(sh.layer, sh.device);
    t->cap = kv->cap;
    t->len = kv->len + sh.layer;
    t->row_offset = row_offset;
    t->window = p->m->window[sh.layer];
    t->rope = p->m->rope;
    t->xhat = p->p_xhat;
    t->xhat_ready = xhat_ready;
    t->q = p->p_q + (size_t)slot * p->q_slot;
    t->attn = p->p_attn + (size_t)slot * p->q_slot;
    t->out = out;
    t->status = kv->status;
}

static void ffn_args(const vt_partition* p, vt_shard sh, const __half* x, int n, float* out, bool xhat_ready,
                     int slot, PrefillFfnArgs* t) {
    const vt_shapes& s = p->m->s;
    const FfnShard& f = p->f(sh.layer, sh.device);
    *t = PrefillFfnArgs{};
    t->n = n;
    t->d = s.d_model;
    t->c = f.c1 - f.c0;
    t->eps = s.rms_eps;
    t->x = x;
    t->gain = f.norm;
    t->wgu = f.wgu;
    t->ushift = f.c0 % 8;
    t->wd = p->m->layer[sh.layer].w_down + (f.c0 - t->ushift);
    t->wd_ld = s.d_ffn;
    t->ldu = p->max_ld;
    t->xhat = p->p_xhat;
    t->xhat_ready = xhat_ready;
    t->u = p->p_u + (size_t)slot * p->u_slot;
    t->out = out;
    t->status = p->status;
}

static vt_status prefill_shard(const vt_partition* p, vt_shard sh, const __half* x, int n, vt_kv* kv,
                               float* out, int row_offset, cudaStream_t st, bool xhat_ready = false) {
    const vt_shapes& s = p->m->s;
    if ((sh.block == VT_BLOCK_ATTN ? p->a(sh.layer, sh.device).bits : p->f(sh.layer, sh.device).bits) != 16)
        return fail(VT_ERR_STATE, "prefill runs on fp16 shards; shard (layer %d, device %d, block %d) is block-quantized",
                    sh.layer, sh.device, sh.block);
    const int D = s.d_model;
    std::string err;
    if (sh.block == VT_BLOCK_ATTN) {
        const AttnShard& a = p->a(sh.layer, sh.device);
        if (a.h1 == a.h0) {
            VT_CUDA(launch_fill_zero_f32(out, (int64_t)n * D, st));
            return VT_OK;
        }
        PrefillAttnArgs t;
        attn_args(p, sh, x, n, kv, out, row_offset, xhat_ready, 0, &t);
        vt_status r = prefill_attn_shard(t, st, &err);
        if (r != VT_OK) return fail(r, "%s", err.c_str());
    } else {
        const FfnShard& f = p->f(sh.layer, sh.device);
        if (f.c1 == f.c0) {
            VT_CUDA(launch_fill_zero_f32(out, (int64_t)n * D, st));
            return VT_OK;
        }
        if (s.d_ffn % 8 != 0) return fail(VT_ERR_SHAPE, "prefill needs d_ffn to be a multiple of 8");
        PrefillFfnArgs t;
        ffn_args(p, sh, x, n, out, xhat_ready, 0, &t);
        vt_status r = prefill_ffn_shard(t, st, &err);
        if (r != VT_OK) return fail(r, "%s", err.c_str());
    }
    return VT_OK;
}

// Every shard of one block of layer l, on `rows` rows whose normalised input is in p_xhat: the
// shards' GEMMs run as one launch per GEMM of the block (empty shards get a zero partial).
static vt_status prefill_block(const vt_partition* p, int l, vt_block block, const __half* x, int rows, vt_kv* kv,
                               int row_offset, cudaStream_t st) {
    const vt_shapes& s = p->m->s;
    const int D = s.d_model;
    PrefillAttnArgs at[VT_MAX_DEVICES];
    PrefillFfnArgs ft[VT_MAX_DEVICES];
    int n = 0;
    for (int d = 0; d < p->n_dev; ++d) {
        float* out = p->partials + (size_t)d * kPrefillChunk * D;
        const vt_shard sh{l, d, block};
        const bool empty = block == VT_BLOCK_ATTN ? p->a(l, d).h1 == p->a(l, d).h0 : p->f(l, d).c1 == p->f(l, d).c0;
        if (empty) {
            VT_CUDA(launch_fill_zero_f32(out, (int64_t)rows * D, st));
            continue;
        }
        if (block == VT_BLOCK_ATTN) attn_args(p, sh, x, rows, kv, out, row_offset, true, d, &at[n++]);
        else ffn_args(p, sh, x, rows, out, true, d, &ft[n++]);
    }
    if (block == VT_BLOCK_FFN && n > 0 && s.d_ffn % 8 != 0)
        return fail(VT_ERR_SHAPE, "prefill needs d_ffn to be a multiple of 8");
    std::string err;
    const vt_status r = block == VT_BLOCK_ATTN ? prefill_attn_group(at, n, st, &err) : prefill_ffn_group(ft, n, st, &err);
    if (r != VT_OK) return fail(r, "%s", err.c_str());
    return VT_OK;
}

extern "C" vt_status vt_prefill(const vt_partition* p, vt_shard sh, const void* x, int32_t n,
                                vt_kv* kv, float* out, vt_stream stream) {
    VT_TRY(check_shard(p, sh));
    if (!x || !out || n < 1) return fail(VT_ERR_INVALID_ARG, "x, out_partial must be set and n >= 1");
    if (!aligned16(x) || !aligned16(out)) return fail(VT_ERR_INVALID_ARG, "x and out_partial must be 16-byte aligned");
    if (n > p->m->s.max_seq) return fail(VT_ERR_INVALID_ARG, "n %d exceeds max_seq", n);
    cudaStream_t st = (cudaStream_t)stream;
    if (sh.block == VT_BLOCK_ATTN) {
        if (!kv || kv->p != p) return fail(VT_ERR_INVALID_ARG, "an ATTN shard needs this partition's KV cache");
        if ((int64_t)kv->h_len[sh.layer] + n > kv->cap)
            return fail(VT_ERR_KV_CAPACITY, "layer %d holds %d of %d positions; %d more do not fit",
                        sh.layer, kv->h_len[sh.layer], kv->cap, n);
    }
    const int D = p->m->s.d_model;
    for (int r0 = 0; r0 < n; r0 += kPrefillChunk) {
        const int rows = std::min(kPrefillChunk, n - r0);
        VT_TRY(prefill_shard(p, sh, static_cast<const __half*>(x) + (size_t)r0 * D, rows, kv,
                             out + (size_t)r0 * D, r0, st));
    }
    return ok();
}

// ------------------------------------------------------------------ whole stack

static vt_status check_token_args(const vt_partition* p, vt_kv* kv, const void* x_in, const void* x_out) {
    if (!p || !kv || kv->p != p || !x_in || !x_out)
        return fail(VT_ERR_INVALID_ARG, "bad vt_decode_token arguments");
    if (!aligned16(x_in)) return fail(VT_ERR_INVALID_ARG, "x_in must be 16-byte aligned");
    const vt_shapes& s = p->m->s;
    for (int l = 0; l < s.n_layers; ++l)
        if (kv->h_len[l] + 1 > kv->cap)
            return fail(VT_ERR_KV_CAPACITY, "layer %d holds %d of %d positions", l, kv->h_len[l], kv->cap);
    return VT_OK;
}

extern "C" int32_t vt_decode_token_fused_available(const vt_partition* p, const char** why) {
    if (why) *why = p ? (p->tok_ok ? "" : p->tok_why.c_str()) : "partition is NULL";
    return p && p->tok_ok ? 1 : 0;
}

extern "C" vt_status vt_token_partials_read(const vt_partition* p, int32_t block, float* host_dst) {
    if (!p || !host_dst || (block != VT_BLOCK_ATTN && block != VT_BLOCK_FFN))
        return fail(VT_ERR_INVALID_ARG, "bad vt_token_partials_read arguments");
    if (!p->tok_ok) return fail(VT_ERR_STATE, "the partition has no fused decode-token kernel: %s", p->tok_why.c_str());
    const float* src = block == VT_BLOCK_ATTN ? p->tok_base.attn_part : p->tok_base.ffn_part;
    VT_CUDA(cudaDeviceSynchronize());
    VT_CUDA(cudaMemcpy(host_dst, src, (size_t)p->n_dev * p->m->s.d_model * 4, cudaMemcpyDeviceToHost));
    return ok();
}

extern "C" vt_status vt_token_test_barrier(vt_partition* p, int32_t cta, uint32_t spin_polls, vt_stream stream) {
    if (!p || cta < -1) return fail(VT_ERR_INVALID_ARG, "bad vt_token_test_barrier arguments");
    if (!p->tok_ok) return fail(VT_ERR_STATE, "the partition has no fused decode-token kernel: %s", p->tok_why.c_str());
    if (cta >= p->tok_plan.grid) return fail(VT_ERR_INVALID_ARG, "cta %d is outside the grid of %d", cta, p->tok_plan.grid);
    // two consecutive words of the sync area: the skipping CTA + 1, then the poll limit
    const uint32_t words[2] = {(uint32_t)(cta + 1), spin_polls};
    static_assert(kTokSyncTestSpin == kTokSyncTestSkip + 1, "test words are adjacent");
    VT_CUDA(cudaMemcpyAsync(p->tok_base.sync + kTokSyncTestSkip, words, sizeof(words), cudaMemcpyHostToDevice,
                            (cudaStream_t)stream));
    VT_CUDA(cudaStreamSynchronize((cudaStream_t)stream));
    return ok();
}

extern "C" vt_status vt_decode_token(const vt_partition* p, vt_kv* kv, const void* x_in, void* x_out,
                                     vt_stream stream) {
    VT_TRY(check_token_args(p, kv, x_in, x_out));
    if (!p->tok_ok || !kv->tok_tab || !aligned16(x_out)) return vt_decode_token_sharded(p, kv, x_in, x_out, stream);
    const vt_shapes& s = p->m->s;
    TokArgs t = p->tok_base;
    t.cap = kv->cap;
    t.shard = static_cast<const TokShardPtrs*>(kv->tok_tab);
    t.layer = reinterpret_cast<const TokLayerPtrs*>(static_cast<const uint8_t*>(kv->tok_tab) +
                                                    align256((size_t)s.n_layers * p->n_dev * sizeof(TokShardPtrs)));
    t.len = kv->len;
    t.x_in = static_cast<const __half*>(x_in);
    t.x_out = static_cast<__half*>(x_out);
    t.status = kv->status;
    VT_CUDA(launch_decode_token(t, p->tok_plan, (cudaStream_t)stream));
    if (!capturing((cudaStream_t)stream))
        for (int l = 0; l < s.n_layers; ++l) kv->h_len[l] += 1;
    return ok();
}

// The combine of one block of the whole-token path: the plain fp32 combine, or, when some
// device's partials travel quantized (communication scaling), each such partial quantized as it
// leaves its shard and the combine of the dequantized values (both clear the fp32 partials).
static vt_status combine_block(const vt_partition* p, int l, vt_block block, const CombineArgs& c, cudaStream_t st) {
    bool any = false;
    for (int b : p->comm_bits) any |= b != 16;
    if (!any) {
        VT_CUDA(launch_combine(c, st));
        return VT_OK;
    }
    const int D = p->m->s.d_model, nbq = (D + kQBlock - 1) / kQBlock;
    CombineQArgs q{};
    q.n = p->n_dev;
    q.clear = 1;
    q.count = D;
    q.residual = c.residual;
    q.out = c.out;
    for (int d = 0; d < p->n_dev; ++d) {
        const bool empty = block == VT_BLOCK_ATTN ? p->a(l, d).h1 == p->a(l, d).h0 : p->f(l, d).c1 == p->f(l, d).c0;
        q.bits[d] = empty ? 16 : p->comm_bits[d];
        q.fparts[d] = c.parts[d];
        q.codes[d] = p->pcodes + (size_t)d * D;
        q.scales[d] = p->pscales + (size_t)d * nbq;
        if (q.bits[d] != 16)
            VT_CUDA(launch_quantize_vec(c.parts[d], D, q.bits[d], p->pcodes + (size_t)d * D, p->pscales + (size_t)d * nbq, 1, st));
    }
    VT_CUDA(launch_combine_q(q, st));
    return VT_OK;
}

extern "C" vt_status vt_partition_set_comm_bits(vt_partition* p, int32_t device, int32_t bits) {
    if (!p) return fail(VT_ERR_INVALID_ARG, "partition is NULL");
    if (device < -1 || device >= p->n_dev) return fail(VT_ERR_INVALID_ARG, "device %d out of range", device);
    if (bits != 16 && bits != 8 && bits != 4) return fail(VT_ERR_INVALID_ARG, "bits %d must be 16, 8 or 4", bits);
    for (int d = 0; d < p->n_dev; ++d)
        if (device < 0 || d == device) p->comm_bits[d] = bits;
    update_token_kernel(p);
    return ok();
}

extern "C" size_t vt_partial_code_bytes(int64_t count, int32_t bits) {
    if (count < 0 || (bits != 8 && bits != 4)) return 0;
    return bits == 8 ? (size_t)count : (size_t)((count + 1) / 2);
}

extern "C" vt_status vt_quantize_partial(const float* partial, int64_t count, int32_t bits, void* codes, void* scales,
                                         vt_stream stream) {
    if (count < 0 || (bits != 8 && bits != 4)) return fail(VT_ERR_INVALID_ARG, "count %lld, bits %d", (long long)count, bits);
    if (count > 0 && (!partial || !codes || !scales)) return fail(VT_ERR_INVALID_ARG, "NULL pointer");
    VT_CUDA(launch_quantize_vec(const_cast<float*>(partial), count, bits, static_cast<uint8_t*>(codes),
                                static_cast<__half*>(scales), 0, (cudaStream_t)stream));
    return ok();
}

extern "C" vt_status vt_combine_q(const void* const* codes, const void* const* scales, int32_t n, int64_t count,
                                  int32_t bits, const void* residual, void* out, vt_stream stream) {
    if (!codes || !scales || !out || n < 1 || n > VT_MAX_DEVICES || count < 0 || (bits != 8 && bits != 4))
        return fail(VT_ERR_INVALID_ARG, "bad vt_combine_q arguments");
    CombineQArgs q{};
    q.n = n;
    q.count = count;
    q.residual = static_cast<const __half*>(residual);
    q.out = static_cast<__half*>(out);
    for (int s = 0; s < n; ++s) {
        if (!codes[s] || !scales[s]) return fail(VT_ERR_INVALID_ARG, "codes or scales of partial %d are NULL", s);
        q.bits[s] = bits;
        q.codes[s] = static_cast<const uint8_t*>(codes[s]);
        q.scales[s] = static_cast<const __half*>(scales[s]);
    }
    VT_CUDA(launch_combine_q(q, (cudaStream_t)stream));
    return ok();
}

extern "C" vt_status vt_decode_token_sharded(const vt_partition* p, vt_kv* kv, const void* x_in, void* x_out,
                                             vt_stream stream) {
    VT_TRY(check_token_args(p, kv, x_in, x_out));
    const vt_shapes& s = p->m->s;
    cudaStream_t st = (cudaStream_t)stream;
    const int D = s.d_model, n = p->n_dev;
    // One fp32 partial buffer per shard serves both blocks: the O projection stores the ATTN
    // partial; the ATTN combine reads and clears it; the FFN kernels add into it; the FFN combine
    // reads and clears it again (buffers start zeroed, so empty shards contribute zeros).
    CombineArgs c{};
    c.n = n;
    c.count = D;
    c.clear = 1;
    for (int d = 0; d < n; ++d) c.parts[d] = p->dpart + (size_t)d * D;
    const __half* cur = static_cast<const __half*>(x_in);
    for (int l = 0; l < s.n_layers; ++l) {
        // After the first launched shard of a block, a shard's input was written by the combine
        // at least two launches earlier, so its first kernel may read it before waiting.
        bool launched = false;
        for (int d = 0; d < n; ++d) {
            const AttnShard& as = p->a(l, d);
            if (as.h1 == as.h0) continue;
            VT_TRY(decode_attn(p, l, d, cur, kv, p->dpart + (size_t)d * D, st, launched));
            launched = true;
        }
        c.residual = cur;
        c.out = p->hbuf;
        VT_TRY(combine_block(p, l, VT_BLOCK_ATTN, c, st));
        launched = false;
        for (int d = 0; d < n; ++d) {
            const FfnShard& fs = p->f(l, d);
            if (fs.c1 == fs.c0) continue;
            VT_TRY(decode_ffn(p, l, d, p->hbuf, p->dpart + (size_t)d * D, st, launched, false));
            launched = true;
        }
        __half* dst = (l == s.n_layers - 1) ? static_cast<__half*>(x_out) : p->xbuf;
        c.residual = p->hbuf;
        c.out = dst;
        VT_TRY(combine_block(p, l, VT_BLOCK_FFN, c, st));
        cur = dst;
    }
    VT_CUDA(launch_kv_advance(kv->len, 0, s.n_layers, 1, kv->cap, kv->status, st));
    if (!capturing(st))
        for (int l = 0; l < s.n_layers; ++l) kv->h_len[l] += 1;
    return ok();
}

extern "C" vt_status vt_prefill_tokens(const vt_partition* p, vt_kv* kv, const void* x_in, int32_t n,
                                       void* x_out, vt_stream stream) {
    if (!p || !kv || kv->p != p || !x_in || !x_out || n < 1)
        return fail(VT_ERR_INVALID_ARG, "bad vt_prefill_tokens arguments");
    if (!aligned16(x_in) || !aligned16(x_out))
        return fail(VT_ERR_INVALID_ARG, "x_in and x_out must be 16-byte aligned");
    const vt_shapes& s = p->m->s;
    for (int l = 0; l < s.n_layers; ++l)
        if ((int64_t)kv->h_len[l] + n > kv->cap)
            return fail(VT_ERR_KV_CAPACITY, "layer %d holds %d of %d positions; %d more do not fit", l,
                        kv->h_len[l], kv->cap, n);
    for (const AttnShard& a : p->attn)
        if (a.bits != 16 && a.h1 > a.h0) return fail(VT_ERR_STATE, "prefill runs on fp16 shards; an ATTN shard is block-quantized");
    for (const FfnShard& f : p->ffn)
        if (f.bits != 16 && f.c1 > f.c0) return fail(VT_ERR_STATE, "prefill runs on fp16 shards; an FFN shard is block-quantized");
    cudaStream_t st = (cudaStream_t)stream;
    const int D = s.d_model, nd = p->n_dev;
    for (int r0 = 0; r0 < n; r0 += kPrefillChunk) {
        const int rows = std::min(kPrefillChunk, n - r0);
        CombineArgs c{};
        c.n = nd;
        c.count = (int64_t)rows * D;
        for (int d = 0; d < nd; ++d) c.parts[d] = p->partials + (size_t)d * kPrefillChunk * D;
        const __half* cur = static_cast<const __half*>(x_in) + (size_t)r0 * D;
        // Every shard of a block normalises the same input with the same gain: the norm runs once
        // per block, fused into the combine that produced the block's input.
        VT_CUDA(launch_rmsnorm_rows(cur, p->m->layer[0].attn_norm, s.rms_eps, rows, D, p->p_xhat, 1, st));
        for (int l = 0; l < s.n_layers; ++l) {
            VT_TRY(prefill_block(p, l, VT_BLOCK_ATTN, cur, rows, kv, r0, st));
            c.residual = cur;
            c.out = p->hbuf;
            VT_CUDA(launch_combine_norm(c, rows, D, p->m->layer[l].ffn_norm, s.rms_eps, p->p_xhat, 0, st));
            VT_TRY(prefill_block(p, l, VT_BLOCK_FFN, p->hbuf, rows, kv, r0, st));
            const bool last = l == s.n_layers - 1;
            __half* dst = last ? static_cast<__half*>(x_out) + (size_t)r0 * D : p->xbuf;
            c.residual = p->hbuf;
            c.out = dst;
            VT_CUDA(launch_combine_norm(c, rows, D, last ? nullptr : p->m->layer[l + 1].attn_norm, s.rms_eps,
                                        p->p_xhat, 1, st));
            cur = dst;
        }
    }
    VT_CUDA(launch_kv_advance(kv->len, 0, s.n_layers, n, kv->cap, kv->status, st));
    if (!capturing(st))
        for (int l = 0; l < s.n_layers; ++l) kv->h_len[l] += n;
    return ok();
}
