/*
 * voltron.h - C ABI of the GB300 (sm_103a) library for the per-device tensor-parallel shard of a
 * Llama-style decoder layer.
 *
 * Source of the operation: Voltron (arXiv 2607.07046), Section 3.2.1: under tensor parallelism a
 * layer is split into shards; the main device broadcasts the layer input, every device computes
 * its shard with that input, and the shard results are aggregated on the main device, once per
 * layer.  Section 2.1 fixes what a layer holds: an attention block (independent heads computing
 * scaled dot-product attention over Q, K, V, then an output linear O; GQA shares K/V heads among
 * groups of query heads) and a feed-forward block (project up, nonlinearity, project back), and
 * the two inference phases: prefill (the prompt in parallel, K/V written to the KV cache) and
 * decode (one token per step, attending to the cache and appending its own K/V).  Section 4.2.1
 * assigns uneven shares to heterogeneous devices, so partitions are arbitrary contiguous ranges.
 *
 * Here every "device" of a partition is a shard executed on the one GPU, one after another; the
 * broadcast is every shard reading the same device buffer, and the aggregation is vt_combine, an
 * on-device sum.
 *
 * Conventions
 *  - Dtypes: weights, activations, hidden states and the KV cache are IEEE binary16 ("fp16",
 *    passed as void*); partial outputs are fp32.  Decode computes in fp32 from fp16 data; prefill
 *    feeds fp16 operands to the tensor cores with fp32 accumulation.
 *  - Layouts: row-major.  Linear weights use the nn.Linear layout [out][in].  A hidden-state batch
 *    is [rows][d_model].
 *  - Ownership: the library copies weights into its own device buffers, allocated through the
 *    caller's vt_allocator (or cudaMalloc when it is NULL) and released by the matching destroy
 *    call.  Every other device pointer is the caller's and must stay valid until the work queued
 *    on the given stream has finished.
 *  - Asynchrony: compute calls only enqueue work on `stream` and return.  Host-detectable errors
 *    (bad arguments, bad shapes or partitions, KV capacity from the host-side length mirror, a
 *    failed launch) return a nonzero vt_status before anything is enqueued, with a message in
 *    vt_last_error().  Nothing aborts or traps.  Problems only a kernel can see (a KV length past
 *    capacity during graph replay, a wait that gave up) set bits in a device status word, read
 *    with vt_kv_status / vt_partition_status.
 *  - Threads: objects are not internally locked; use one object from one host thread at a time.
 *  - Streams and graphs: every compute call except vt_decode_step_static can be captured into a
 *    CUDA graph; positions come from device-resident KV lengths, so a replayed graph appends at
 *    the right place.  (No claim is made for vt_decode_step_static.)  While the stream is being
 *    captured, calls record device work only and leave the host-side mirror of the KV lengths
 *    unchanged; replays advance the device lengths alone, and vt_kv_length refreshes the mirror.
 *    vt_kv_set_length and the synchronous test hooks cannot be captured.
 *  - Citations: each declaration names the section of Voltron that defines its operation; calls
 *    that are library plumbing (object lifetime, status words, test hooks) say so.
 */
#ifndef VOLTRON_H
#define VOLTRON_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#if defined(__GNUC__)
#define VT_API __attribute__((visibility("default")))
#else
#define VT_API
#endif

typedef int32_t vt_status;
#define VT_OK 0
#define VT_ERR_INVALID_ARG 1      /* null pointer, negative size, unknown enum */
#define VT_ERR_SHAPE 2            /* vt_shapes not supported (see vt_shapes_validate) */
#define VT_ERR_PARTITION_OVERLAP 3 /* range d starts before range d-1 ends */
#define VT_ERR_PARTITION_GAP 4    /* range d starts after range d-1 ends, or the union is short */
#define VT_ERR_PARTITION_GQA 5    /* a head range does not start and end on a KV-group boundary */
#define VT_ERR_PARTITION_RANGE 6  /* begin > end, or a bound outside [0, H] / [0, F] */
#define VT_ERR_KV_CAPACITY 7      /* the call would write past the KV-cache capacity */
#define VT_ERR_CUDA 8             /* a CUDA runtime call failed (text in vt_last_error) */
#define VT_ERR_ALLOC 9            /* the allocator returned NULL */
#define VT_ERR_STATE 10           /* object not ready (e.g. a layer's weights never loaded) */
#define VT_ERR_PLAN_MEMORY 11     /* the devices' memory budgets cannot hold the block */
#define VT_ERR_PLAN_QOS 12        /* no precision configuration meets the time budget */

#define VT_MAX_DEVICES 16

/* Bits of the device status word. */
#define VT_DEV_KV_OVERFLOW 1u     /* a kernel saw a KV length at or past capacity and skipped */
#define VT_DEV_WAIT_TIMEOUT 2u    /* a kernel gave up waiting on an asynchronous copy */
#define VT_DEV_BAD_TOKEN 4u       /* the embedding gather saw a token id outside [0, vocab) */

typedef void* vt_stream; /* a cudaStream_t; NULL is the legacy default stream */

typedef struct {
    int32_t n_layers;
    int32_t d_model;    /* D, multiple of 64 */
    int32_t n_heads;    /* H, query heads */
    int32_t n_kv_heads; /* Hk, divides H (H == Hk is MHA) */
    int32_t d_head;     /* dh, 64 or 128 */
    int32_t d_ffn;      /* F, SwiGLU intermediate width */
    int32_t vocab;      /* rows of the embedding table (0: no table) */
    int32_t max_seq;    /* largest position + 1 that any KV cache may hold */
    float rms_eps;      /* RMSNorm epsilon (inside the square root) */
    float rope_theta;   /* RoPE base */
} vt_shapes;

/* Half-open range [begin, end). */
typedef struct {
    int32_t begin, end;
} vt_range;

/* Device-memory allocator.  alloc(bytes, ctx) returns a device pointer aligned to 256 bytes or
 * NULL; free(ptr, ctx) releases it.  Both may be called from the thread that calls the library. */
typedef struct {
    void* (*alloc)(size_t bytes, void* ctx);
    void (*free)(void* ptr, void* ctx);
    void* ctx;
} vt_allocator;

/* One layer's weights, fp16 host pointers, nn.Linear layout.  Read only during the call. */
typedef struct {
    const void* attn_norm; /* [D]        RMSNorm gain of the attention block */
    const void* wq;        /* [H*dh, D]  */
    const void* wk;        /* [Hk*dh, D] */
    const void* wv;        /* [Hk*dh, D] */
    const void* wo;        /* [D, H*dh]  */
    const void* ffn_norm;  /* [D]        RMSNorm gain of the FFN block */
    const void* w_gate;    /* [F, D]     */
    const void* w_up;      /* [F, D]     */
    const void* w_down;    /* [D, F]     */
} vt_layer_weights;

typedef enum { VT_BLOCK_ATTN = 0, VT_BLOCK_FFN = 1 } vt_block;

/* One shard: the `block` of layer `layer` assigned to device `device` of a partition. */
typedef struct {
    int32_t layer;
    int32_t device;
    int32_t block; /* vt_block */
} vt_shard;

typedef struct vt_model vt_model;
typedef struct vt_partition vt_partition;
typedef struct vt_kv vt_kv;

/* Library plumbing (no paper counterpart).  Text of the last error on the calling thread ("" if
 * none).  Valid until the next call. */
VT_API const char* vt_last_error(void);

/* Library plumbing.  Library version, "major.minor.patch". */
VT_API const char* vt_version(void);

/* Host-only checks (no GPU needed).  vt_shapes_validate returns VT_OK or VT_ERR_SHAPE: the
 * decoder-layer shapes of Section 2.1 ("LLM Architecture": attention heads, GQA groups, FFN) that
 * the kernels support.  vt_partition_validate applies the partition rules of vt_partition below
 * (Section 3.2.1 head/column shards, Section 4.2.1 uneven shares). */
VT_API vt_status vt_shapes_validate(const vt_shapes* shapes);
VT_API vt_status vt_partition_validate(const vt_shapes* shapes, int32_t n_devices,
                                const vt_range* head_ranges, const vt_range* ffn_col_ranges);

/* ---------------------------------------------------------------- planning (host only) --------
 * vt_plan_tp_shares: the heterogeneity-aware tensor-parallel split of one block (Voltron Section
 * 4.2.1, layer allocation under TP: shards are assigned greedily to devices by their performance,
 * to balance the execution time across devices and so limit stragglers; within each device's
 * memory budget, Section 4.2.1 and Fig. 5).
 *
 * The block is cut into equal units: for VT_BLOCK_ATTN one KV group (n_heads / n_kv_heads query
 * heads with their KV head); for VT_BLOCK_FFN `col_unit` FFN columns (the last unit is shorter
 * when col_unit does not divide d_ffn; col_unit is ignored for ATTN).  A unit's bytes are its
 * fp16 weights (ATTN: its QKV rows and O columns, plus its K and V cache at max_seq positions;
 * FFN: its gate, up and down columns).  Decode streams every shard byte once per token, so device
 * d takes units_d * unit_bytes / rate[d] seconds (rate: bytes per second, > 0).  Units are given
 * one at a time to the device that would finish its share soonest with one more unit (ties: the
 * lower device index), among the devices whose share still fits in mem_bytes[d] (nullable: no
 * limit); for equal units this minimises the slowest device's time.  The shares are written as
 * contiguous ranges in device order (ranges[n_devices]: query heads for ATTN, columns for FFN;
 * a device may get an empty range), valid for vt_partition_create.  makespan (nullable) receives
 * the slowest device's time in seconds.
 * Errors: VT_ERR_INVALID_ARG (NULL shapes / rate / ranges, n_devices outside [1, VT_MAX_DEVICES],
 * a rate that is not finite and positive, a negative or NaN budget, col_unit < 1 for FFN),
 * VT_ERR_SHAPE (invalid shapes), VT_ERR_PLAN_MEMORY (some unit fits on no device).  Nothing is
 * written on error. */
VT_API vt_status vt_plan_tp_shares(const vt_shapes* shapes, vt_block block, int32_t n_devices,
                                   const double* rate, const double* mem_bytes, int32_t col_unit,
                                   vt_range* ranges, double* makespan);

/* vt_plan_layers: the layer-wise hybrid parallelism plan (Voltron Section 4.2.1): the blocks of
 * the stack (ATTN then FFN of layer 0, then of layer 1, ...) are planned one after another.  For
 * each block both strategies are estimated and the one with the lower time is kept (ties: MP):
 *   MP: the whole block on the device with the highest rate whose remaining memory holds it; if the
 *       activations are on another device they are sent first (one transfer of tokens * D fp16).
 *   TP: shares from vt_plan_tp_shares on the remaining memory; the device holding the input
 *       broadcasts it once (one transfer), the devices with a share compute at the same time, and
 *       every other participant sends its fp32 partial [tokens * D] back to it (one transfer each,
 *       one after another: the devices share one link).  The input holder keeps the activations.
 * A transfer of b bytes takes link_latency_s + b / link_bytes_per_s.  A device's compute time for
 * its part of a block is max(bytes / rate[d], flops / flop_rate[d]) (flop_rate nullable: bytes
 * only), where bytes are its fp16 weights plus, for ATTN, the K / V rows read at kv_len and
 * written for the `tokens` new rows, and flops are 2 per weight per token plus the attention
 * scores and weighted values over kv_len + tokens positions.  Memory (mem_bytes nullable: no
 * limit) holds weights and the K / V cache at max_seq.  The input starts on device 0.
 * plans[2 * n_layers] receives the plan of every block (ATTN of layer l at 2 l, FFN at 2 l + 1);
 * total_s (nullable) the sum of the blocks' compute and transfer times.
 * Errors: as vt_plan_tp_shares, plus VT_ERR_INVALID_ARG for tokens < 1, kv_len < 0 or
 * kv_len + tokens > max_seq, or a link rate that is not finite and positive or a negative latency;
 * VT_ERR_PLAN_MEMORY when a block fits under neither strategy. */
typedef struct {
    int32_t tp;                      /* 0: MP, 1: TP */
    int32_t device;                  /* MP: the device; TP: the input holder, which gathers the partials */
    vt_range ranges[VT_MAX_DEVICES]; /* query heads (ATTN) or FFN columns of each device */
    double compute_s, comm_s;        /* slowest participant's compute; transfers */
} vt_block_plan;
VT_API vt_status vt_plan_layers(const vt_shapes* shapes, int32_t n_devices, const double* rate,
                                const double* flop_rate, const double* mem_bytes, double link_bytes_per_s,
                                double link_latency_s, int32_t tokens, int32_t kv_len, vt_block_plan* plans,
                                double* total_s);

/* vt_plan_precision (host only): importance-aware mixed precision (Voltron Section 4.2.2).  Given
 * the blocks' plan (plans[2 n_layers], e.g. from vt_plan_layers: each device's heads or columns
 * of every block, and the block's transfer time comm_s) and an importance score per block
 * (importance[2 n_layers], ATTN of layer l at 2 l, FFN at 2 l + 1; higher = more important; the
 * scores are the caller's, the paper's come from offline perplexity profiling), blocks are lowered
 * one precision step at a time in ascending order of importance (ties: lower block index).
 * Configuration k (0 <= k <= 4 n_layers) has the min(k, 2 n_layers) least important blocks at
 * INT8 at least and the first k - 2 n_layers of them at INT4; every block of a configuration is
 * at one precision on all its devices.  A device's memory (its shards' weights at their
 * precision: fp16, or codes plus one fp16 scale per 32 weights along the contraction axis, as
 * vt_partition_set_precision stores them, plus the fp16 K / V cache of its KV heads at max_seq)
 * and the stack's time (per block the slowest device's streamed bytes / rate[d]: its weights and,
 * for ATTN, the K / V rows of kv_len + 1 positions; plus the block's comm_s) do not grow with k,
 * so the smallest k that fits every mem_bytes[d] (nullable: no limit) and qos_s (<= 0 or
 * infinite: no limit) is found by binary search over k.
 * bits[2 n_layers] receives 16, 8 or 4 per block; steps (nullable) the chosen k; total_s
 * (nullable) that configuration's time.  The plan's parallelism is kept: re-planning with the new
 * precisions is the caller's choice.
 * Errors: VT_ERR_INVALID_ARG (null pointers, non-finite importance or comm_s, kv_len outside
 * [0, max_seq), bad rates or budgets), VT_ERR_PARTITION_RANGE / VT_ERR_PARTITION_GQA for a plan
 * range outside the block or not in whole KV groups; VT_ERR_PLAN_MEMORY or VT_ERR_PLAN_QOS when
 * even configuration 4 n_layers (every block INT4) misses a budget, with bits, steps and total_s
 * describing that configuration. */
VT_API vt_status vt_plan_precision(const vt_shapes* shapes, int32_t n_devices, const vt_block_plan* plans,
                                   const double* importance, const double* rate, const double* mem_bytes,
                                   double qos_s, int32_t kv_len, int32_t* bits, int32_t* steps, double* total_s);

/* vt_quantize_rows (host only): block quantization of fp16 weight rows for mixed-precision shards
 * (Voltron Section 3.2.2 and Section 4.2.2, precision heterogeneity; Section 5.1 names k-quant
 * formats without defining them).  Each row of w (host fp16 [rows][k], row-major) is cut into
 * blocks of `block` consecutive weights (the last one may be shorter); a block gets the fp16
 * scale d = fp16(amax / qmax) (amax: its largest |w|; qmax: 127 for bits = 8, 7 for bits = 4) and
 * every weight the code q = round-half-even(w / d) clamped to [-qmax, qmax] (0 when d = 0), both
 * divisions in fp32.  Outputs (host, caller-owned): q int8 [rows][k]; scales fp16
 * [rows][ceil(k / block)].  The dequantized weight is q * d.
 * Errors: VT_ERR_INVALID_ARG (NULL pointer, rows or k < 0, block < 1, bits not 8 or 4). */
VT_API vt_status vt_quantize_rows(const void* w, int64_t rows, int64_t k, int32_t bits, int32_t block, int8_t* q,
                                  void* scales);

/* ---------------------------------------------------------------- model ------------------------
 * vt_model_create (Section 2.1, "LLM Architecture": the decoder layers the shards are cut from;
 * the weights are the unpartitioned layer before Section 3.2.1 splits it): allocates device storage for every layer in the canonical (unpartitioned)
 * layout, the RoPE table for positions [0, max_seq) and, if vocab > 0, the embedding table, on
 * the current CUDA device.  per_layer (nullable) holds n_layers host weight sets, copied now;
 * embed (nullable) is the host fp16 table [vocab, D].  Layers not given here are loaded later
 * with vt_model_load_layer.  Synchronizes `stream` before returning (host buffers may be reused).
 */
VT_API vt_status vt_model_create(const vt_shapes* shapes, const vt_layer_weights* per_layer,
                          const void* embed, const vt_allocator* allocator, vt_stream stream,
                          vt_model** out);
/* Library plumbing for vt_model_create: load one layer's weights (copied now, synchronizes the
 * stream), load the embedding table, read the shapes back, free everything. */
VT_API vt_status vt_model_load_layer(vt_model* model, int32_t layer, const vt_layer_weights* weights,
                              vt_stream stream);
VT_API vt_status vt_model_load_embedding(vt_model* model, const void* embed, vt_stream stream);
VT_API vt_status vt_model_shapes(const vt_model* model, vt_shapes* out);
VT_API void vt_model_destroy(vt_model* model);
/* vt_model_set_window (Section 2.1, "LLM Architecture": sliding-window attention is one of the
 * attention variants of the evaluated models; gemma-3 uses a window of 1024 on most layers):
 * layer `layer` (or every layer when -1) attends, for a row at position p, only to positions
 * [max(0, p - window + 1), p] (window = 0, the default: every position 0..p).  Applies to every
 * decode and prefill entry point.  Windows are fixed while a partition of the model exists:
 * set them before vt_partition_create (VT_ERR_STATE otherwise).  VT_ERR_INVALID_ARG for a
 * negative window or a layer out of range.  Host only.
 * vt_model_window reads one layer's window back. */
VT_API vt_status vt_model_set_window(vt_model* model, int32_t layer, int32_t window);
VT_API vt_status vt_model_window(const vt_model* model, int32_t layer, int32_t* window);
/* Library plumbing.  Reads the model's device status word (VT_DEV_BAD_TOKEN from vt_embed),
 * synchronizing the device; clear != 0 resets it. */
VT_API vt_status vt_model_status(vt_model* model, uint32_t* flags, int32_t clear);

/* Embedding gather (Section 2.1, "LLM Architecture": token ids enter the stack as embedding
 * rows): out[i, :] = E[ids[i], :] for i < n, copied bit for bit.  ids: device int32 [n]; out:
 * device fp16 [n, D], 16-byte aligned.  An id outside [0, vocab) gives a zero row and sets
 * VT_DEV_BAD_TOKEN in the model's status word (vt_model_status); the call itself still returns
 * VT_OK, since the ids are only seen on the device.  VT_ERR_STATE without a loaded table. */
VT_API vt_status vt_embed(const vt_model* model, const int32_t* ids, int32_t n, void* out,
                   vt_stream stream);

/* ---------------------------------------------------------------- partition --------------------
 * vt_partition: splits every layer among n_devices shards (Section 3.2.1; uneven shares as in
 * Section 4.2.1).  Device d gets query heads head_ranges[d] of every attention block (and the KV
 * heads of their groups) and FFN intermediate columns ffn_col_ranges[d] of every FFN block.
 * Rules: the ranges of each kind are listed in device order, contiguous, disjoint, and cover
 * [0, H) and [0, F) exactly; empty ranges are allowed (that shard's partial is all zeros); under
 * GQA every head range starts and ends on a multiple of H/Hk.  Violations return
 * VT_ERR_PARTITION_* before any device work.  Each (layer, block, device) shard gets its own
 * allocation holding its weights in the shard-sliced layout, so a shard can be dropped alone.
 * The model must outlive the partition.  Synchronizes `stream`.
 */
VT_API vt_status vt_partition_create(vt_model* model, int32_t n_devices, const vt_range* head_ranges,
                              const vt_range* ffn_col_ranges, vt_stream stream,
                              vt_partition** out);
/* vt_partition_create_layers (Section 4.2.1: the plan is made layer by layer, ATTN and FFN as
 * separate layers, each run by one device (MP) or split among devices (TP); Section 4.3.1: shards
 * are pruned, the same number from every layer, to fit a shrinking memory budget): a partition
 * with its own ranges per layer.  heads, cols: [n_layers][n_devices] ranges (layer-major); each
 * layer follows vt_partition's rules (a block on one device with empty ranges elsewhere is MP).
 * flags VT_PARTITION_PRUNE: a layer's ranges may leave heads / columns uncovered; those are pruned
 * (their terms are omitted from the layer, as a dropped shard's would be) and an empty range may
 * sit anywhere.  Each (layer, block, device) shard gets its own allocation, as in vt_partition.
 * The fused decode kernel takes one partition for every layer: vt_decode_token runs a per-layer or
 * pruned partition on the per-shard kernels.  vt_partition_validate_layers checks the same rules
 * on the host.  Errors: as vt_partition_create; VT_ERR_INVALID_ARG for unknown flags. */
#define VT_PARTITION_PRUNE 1u
VT_API vt_status vt_partition_create_layers(vt_model* model, int32_t n_devices, const vt_range* head_ranges,
                                            const vt_range* ffn_col_ranges, uint32_t flags, vt_stream stream,
                                            vt_partition** out);
VT_API vt_status vt_partition_validate_layers(const vt_shapes* shapes, int32_t n_devices, const vt_range* head_ranges,
                                              const vt_range* ffn_col_ranges, uint32_t flags);
/* Library plumbing: the partition's device count; its device status word (VT_DEV_* bits of
 * kernels that have no KV cache; synchronizes the device; clear != 0 resets it and re-arms the
 * fused decode kernel's grid barrier); destruction (the model must still exist). */
VT_API int32_t vt_partition_devices(const vt_partition* part);
VT_API vt_status vt_partition_status(vt_partition* part, uint32_t* flags, int32_t clear);
VT_API void vt_partition_destroy(vt_partition* part);

/* Test hook (library plumbing; the slicing itself is Section 3.2.1's head/column split): copies
 * one tensor of a shard's sliced weights to host memory.  which: 0 = attention
 * RMSNorm gain, 1 = fused QKV rows, 2 = O columns, 3 = FFN RMSNorm gain, 4 = fused gate/up rows,
 * 5 = down columns.  Copies min(bytes, size) bytes; *size_out (nullable) receives the size.
 * Layouts are documented beside vt_shard_weight_layout.  Synchronous. */
VT_API vt_status vt_shard_weights_read(const vt_partition* part, vt_shard shard, int32_t which,
                                void* host_dst, size_t bytes, size_t* size_out);
/* Geometry of a shard's sliced tensor: rows and row stride (elements) of tensor `which`.
 *  which 1 (QKV): rows = (h_s + 2 hk_s) * dh; head block b (q heads, then k heads, then v heads)
 *    occupies rows [b*dh, (b+1)*dh) and stores, at row b*dh + 2i, the source row of dimension i
 *    and at row b*dh + 2i + 1 the source row of dimension i + dh/2 (RoPE partners adjacent).
 *  which 2 (O): rows = D, stride = h_s*dh: columns [h0*dh, h1*dh) of Wo.
 *  which 4 (gate/up): rows = 2 * c_s: row 2j = gate row c0 + j, row 2j + 1 = up row c0 + j.
 *  which 5 (down, transposed): rows = c_s, stride = D: row j = column c0 + j of Wd.
 *  which 0, 3: one row of D. */
VT_API vt_status vt_shard_weight_layout(const vt_partition* part, vt_shard shard, int32_t which,
                                 int64_t* rows, int64_t* row_stride);

/* vt_partition_set_precision (Section 3.2.2, precision heterogeneity: a device holds its shard at
 * its own precision; Section 4.2.2 allocates the precision per layer; Section 5.1 names k-quant
 * formats without defining them): stores shard `shard` at `bits` = 8 or 4 (block-quantized) or
 * 16 (fp16, sliced again from the model).  Format (the library's reading of k-quant): every weight
 * row is cut into blocks of 32 weights along its input axis; a block keeps the fp16 scale
 * d = fp16(amax / qmax) (qmax 127 or 7) and each weight the code round-half-even(w / d) clamped to
 * [-qmax, qmax], both divisions in fp32 (the codes of vt_quantize_rows, bit for bit).  Quantized
 * tensors: ATTN: the QKV rows (rows along D) and the O columns (rows of Wo_s [D][h_s dh] along the
 * shard's columns); FFN: the gate/up rows (along D) and the down projection as Wd[:, c0:c1]
 * ([D][c] rows along the shard's columns).  Codes are stored packed (one byte per 8-bit code, two
 * 4-bit codes per byte) with the fp16 scales, replacing the shard's fp16 weights (its bytes halve
 * or quarter, plus one scale per 32 weights).  Decode (vt_decode_step, vt_decode_step_static,
 * vt_decode_token_sharded) runs quantized shards with a dequantizing kernel; vt_decode_token then
 * runs the per-shard kernels (vt_decode_token_fused_available says why); prefill needs fp16
 * shards (VT_ERR_STATE).  Precisions are fixed while a KV cache of the partition exists
 * (VT_ERR_STATE): set them before vt_kv_create.  An empty shard stores nothing and stays fp16.
 * Synchronizes `stream`.  Errors: VT_ERR_INVALID_ARG (bad shard or bits), VT_ERR_ALLOC, VT_ERR_CUDA.
 * vt_shard_precision returns a shard's bits (16, 8 or 4; 0 for a bad shard). */
VT_API vt_status vt_partition_set_precision(vt_partition* part, vt_shard shard, int32_t bits, vt_stream stream);
VT_API int32_t vt_shard_precision(const vt_partition* part, vt_shard shard);
/* Test hook (library plumbing): the codes and scales of a block-quantized shard tensor, synchronous.
 * which: 1 = QKV rows [(h_s + 2 hk_s) dh][D] (rows in the order of vt_shard_weight_layout), 2 = O
 * [D][h_s dh], 4 = gate/up rows [2 c][D] (interleaved), 5 = down [D][c] (columns c0 .. c1 - 1 of
 * Wd, not transposed).  codes: host int8 [rows][k]; scales: host fp16 [rows][ceil(k / 32)].
 * VT_ERR_STATE when the tensor is not quantized. */
VT_API vt_status vt_shard_qweights_read(const vt_partition* part, vt_shard shard, int32_t which, int8_t* codes,
                                        void* scales);

/* ---------------------------------------------------------------- KV cache ---------------------
 * vt_kv_create (Section 2.1, "LLM Inference": the KV cache that prefill fills and every decode
 * step appends to; split by KV head among the devices as tensor parallelism splits the heads,
 * Section 3.2.1): per (layer, device) fp16 caches K and V, each [hk_s][capacity][dh] for that
 * device's KV heads (tensor parallelism splits the cache by head), plus one device-resident length
 * per layer (initially 0) and a host mirror of it.  capacity <= max_seq.  Contents start zeroed.
 */
VT_API vt_status vt_kv_create(const vt_partition* part, int32_t capacity, vt_stream stream, vt_kv** out);
/* Library plumbing: destruction and the capacity given at creation. */
VT_API void vt_kv_destroy(vt_kv* kv);
VT_API int32_t vt_kv_capacity(const vt_kv* kv);
/* Cache bookkeeping (Section 2.1: each decode step appends one position, a prefill n).  Adds n
 * to the length of `layer` (or of every layer when layer == -1), on the device (in stream
 * order) and in the host mirror.  Decode and prefill append at the current length without
 * advancing it: advance once per layer after all of that layer's attention shards ran.
 * VT_ERR_KV_CAPACITY when the mirror says a length would leave [0, capacity].  While the stream
 * is being captured the mirror is not consulted: the device clamps a length that would leave
 * [0, capacity] into it and sets VT_DEV_KV_OVERFLOW. */
VT_API vt_status vt_kv_advance(vt_kv* kv, int32_t layer, int32_t n, vt_stream stream);
/* Cache bookkeeping: sets the length of `layer` (or all when -1) to len, device and host
 * mirror; synchronizes the stream (not capturable). */
VT_API vt_status vt_kv_set_length(vt_kv* kv, int32_t layer, int32_t len, vt_stream stream);
/* Cache bookkeeping: reads the device length of `layer` (synchronizes the stream) and refreshes
 * the host mirror. */
VT_API vt_status vt_kv_length(vt_kv* kv, int32_t layer, vt_stream stream, int32_t* len);
/* Library plumbing: reads (and with clear != 0 resets) the device status word of kernels that
 * used this cache. */
VT_API vt_status vt_kv_status(vt_kv* kv, uint32_t* flags, int32_t clear);
/* Test hooks, synchronous: copy positions [0, n_pos) of the (layer, device) cache between device
 * and host.  Host layout [hk_s][n_pos][dh] fp16 for K and for V. */
VT_API vt_status vt_kv_read(const vt_kv* kv, int32_t layer, int32_t device, int32_t n_pos, void* k_host,
                     void* v_host);
VT_API vt_status vt_kv_write_raw(vt_kv* kv, int32_t layer, int32_t device, int32_t n_pos,
                          const void* k_host, const void* v_host);

/* ---------------------------------------------------------------- shard compute ----------------
 * vt_decode_step (Section 2.1, decode phase; Section 3.2.1, one device's shard of a tensor-
 * parallel layer, the ATTN and FFN blocks being separate layers as in Section 4.2.1): one decode
 * token through one shard.
 *   ATTN shard (kv required): x^ = RMSNorm(x); q, k, v of the shard's heads; RoPE on q and k at
 *   position p = current length of the layer; k, v appended at p; attention of each query head
 *   over positions 0..p (split-K flash decoding); out_partial = Wo[:, shard cols] . attn.
 *   FFN shard (kv ignored, may be NULL): x^ = RMSNorm(x); u = silu(Wg x^) * (Wu x^) over the shard's
 *   columns; out_partial = Wd[:, shard cols] . u.
 *   x: device fp16 [D] (the block input, identical for every shard); out_partial: device fp32 [D],
 *   excluding the residual.  Does not advance the KV length.
 */
VT_API vt_status vt_decode_step(const vt_partition* part, vt_shard shard, const void* x, vt_kv* kv,
                         float* out_partial, vt_stream stream);

/* vt_decode_step_static: vt_decode_step for an ATTN shard with no allocation and no allocated
 * scratch.  The paper has no counterpart; it is a library convenience.
 *   Who needs it: callers that cannot allocate device memory when they run decoding.  For
 *   example, a host whose memory plan has given all of HBM to the weights and the KV cache, or
 *   one whose allocator cannot be entered from the thread that drives decoding.  The step keeps
 *   every intermediate in one file-scope __device__ array of 1 MiB (1048576 bytes) that is part
 *   of the library's device image.  It calls no cudaMalloc, cudaFree or other allocating routine.
 *   It does not use the partition's decode scratch.
 *   Computation: as vt_decode_step for the ATTN shard.  Attention runs as split-K over 16 slices
 *   per KV head.  The slices are merged by the last one to finish, so results match
 *   vt_decode_step to rounding, not bit for bit.
 *   Arguments, layouts, ownership: as vt_decode_step.  kv is required.  Does not advance the KV
 *   length.
 *   Limits: the shard needs 256 + 8*h_s*dh + 64*hk_s*G*(dh+2) bytes (each region rounded up to
 *   256 bytes; G = query heads per KV head), at most 1 MiB, and hk_s <= 64.  A larger shard
 *   returns VT_ERR_INVALID_ARG with the byte count in vt_last_error().  An FFN shard returns
 *   VT_ERR_INVALID_ARG (it uses no scratch; call vt_decode_step).
 *   First call on a device: looks up the array's device address with cudaGetSymbolAddress, with
 *   that device current, and keeps it.  Any failure is VT_ERR_CUDA.  Make that first call before
 *   any stream capture on that device begins.  The kept address is the array's for the life of
 *   the device's primary context: do not use the library across a cudaDeviceReset (the module
 *   would load again and the array could move).
 *   Must start at zero: only the 64 per-KV-head arrival counters at the start of the array.  The
 *   module loader zeroes them, and every call leaves them at zero.
 *   Races: the array is shared by every call in the process on that device.  Two calls in flight
 *   at once, on different streams or host threads, corrupt each other.  Order them. */
VT_API vt_status vt_decode_step_static(const vt_partition* part, vt_shard shard, const void* x, vt_kv* kv,
                                float* out_partial, vt_stream stream);

/* vt_prefill (Section 2.1, prefill phase: the prompt in parallel, K/V written to the cache;
 * Section 3.2.1 shard): n prompt rows through one shard (n >= 1).
 *   ATTN shard: rows sit at positions p0..p0+n-1 with p0 = current length of the layer; row i
 *   attends causally to positions 0..p0+i (earlier turns' cache included).  K and V of all rows
 *   are appended.  FFN shard: as decode, row by row.
 *   x: device fp16 [n, D]; out_partial: device fp32 [n, D]; n <= max_seq.  Does not advance.
 */
VT_API vt_status vt_prefill(const vt_partition* part, vt_shard shard, const void* x, int32_t n,
                     vt_kv* kv, float* out_partial, vt_stream stream);

/* vt_combine (Section 3.2.1: the shard results are aggregated on the main device): the sum.
 *   out[e] = fp16(residual[e] + sum_{s=0}^{n-1} partials[s][e]), e < rows*d, summed in fp32 in
 *   the order s = 0..n-1.  partials: host array of n device pointers to fp32 [rows, d];
 *   residual: device fp16 [rows, d] or NULL; out: device fp16 [rows, d] (may alias residual).
 *   1 <= n <= VT_MAX_DEVICES. */
VT_API vt_status vt_combine(const float* const* partials, int32_t n, int32_t rows, int32_t d,
                     const void* residual, void* out, vt_stream stream);

/* ---------------------------------------------------------------- communication scaling -------
 * Section 4.3.2: the activations sent between devices are lowered to INT8 or INT4 when the link
 * is too slow; under tensor parallelism those are the shard partials on their way to the main
 * device.  Format (the library's reading): blocks of 32 values, fp16 scale d = fp16(amax / qmax)
 * (qmax 127 or 7) and codes round-half-even(x / d) clamped to [-qmax, qmax], decisions in fp32;
 * codes stored as one int8 per value (8 bits) or two per byte (4 bits: value 2i in the low nibble,
 * 2i + 1 in the high nibble, each stored as q + 8).
 * vt_partial_code_bytes: bytes of the codes of `count` values (0 for bad arguments).
 * vt_quantize_partial: device fp32 partial [count] -> device codes and fp16 scales
 *   [ceil(count / 32)] (the partial is not modified).
 * vt_combine_q: out[e] = fp16(residual[e] + sum_{s=0}^{n-1} q_s[e] d_s[e / 32]) summed in fp32 in
 *   shard order; codes / scales: host arrays of n device pointers; residual nullable; out may
 *   alias residual.
 * vt_partition_set_comm_bits: device `device` (or every device when -1) sends its partials at
 *   `bits` (16: fp32, the default; 8; 4) in the whole-token path: each such partial is quantized
 *   as its shard finishes and the combine adds the dequantized values.  vt_decode_token then runs
 *   the per-shard kernels.  May change between tokens.
 * Errors: VT_ERR_INVALID_ARG for NULL pointers, bad counts, devices or bits. */
VT_API size_t vt_partial_code_bytes(int64_t count, int32_t bits);
VT_API vt_status vt_quantize_partial(const float* partial, int64_t count, int32_t bits, void* codes, void* scales,
                                     vt_stream stream);
VT_API vt_status vt_combine_q(const void* const* codes, const void* const* scales, int32_t n, int64_t count,
                              int32_t bits, const void* residual, void* out, vt_stream stream);
VT_API vt_status vt_partition_set_comm_bits(vt_partition* part, int32_t device, int32_t bits);

/* ---------------------------------------------------------------- whole stack ------------------
 * vt_decode_token: one decode token through every layer (Voltron Section 2.1, decode phase; the
 *   tensor-parallel layer of Section 3.2.1): for each layer, every ATTN shard (as vt_decode_step)
 *   and the combine with the residual; every FFN shard and the combine; then every layer's KV
 *   length advances by one.
 *   x_in, x_out: device fp16 [D], 16-byte aligned; they may be the same buffer.  Uses buffers
 *   owned by the partition, so one partition runs one vt_decode_token / vt_prefill_tokens at a
 *   time (stream-ordered).
 *   When vt_decode_token_fused_available() says so, the whole token is ONE cooperative kernel
 *   launch (one CTA per SM): each CTA streams its share of every shard's weights and cached K/V
 *   through a shared-memory ring, shards are processed in order within each phase, and the CTAs
 *   meet at four grid barriers per layer.  Results equal the per-shard kernels' within fp32
 *   rounding (the FFN partials are summed by bulk reductions in the L2 in arrival order, so they
 *   repeat only to fp32 rounding).
 *   Every wait in that kernel is bounded: a CTA that gives up sets VT_DEV_WAIT_TIMEOUT in the KV
 *   status word, the token's output is then undefined, and vt_kv_status(..., clear = 1) (or
 *   vt_partition_status) must be called before the next token to re-arm the grid barrier.
 *   Otherwise (unsupported shapes, or x_out not 16-byte aligned) it runs vt_decode_token_sharded.
 *   The launch can be captured in a CUDA graph.
 */
VT_API vt_status vt_decode_token(const vt_partition* part, vt_kv* kv, const void* x_in, void* x_out,
                          vt_stream stream);
/* The same token (Sections 2.1 and 3.2.1, as vt_decode_token) as a sequence of per-shard
 * kernels (3 per ATTN shard, 1 per FFN shard, one combine per block, one length update), linked
 * by programmatic dependent launch: vt_decode_step for every shard, one after another, and
 * vt_combine per block. */
VT_API vt_status vt_decode_token_sharded(const vt_partition* part, vt_kv* kv, const void* x_in,
                                         void* x_out, vt_stream stream);
/* Library plumbing: 1 if vt_decode_token runs as one fused kernel for this partition, else 0; *why (optional)
 * receives the reason when it does not (valid while the partition lives).  Fused needs a
 * device with cooperative launch, d_model a multiple of 8 and at most 6144, d_head 64 or 128,
 * 1, 2 or 4 query heads per KV head, at most as many KV heads as SMs, at most 256 layers, and
 * at most 256 QKV rows per SM. */
VT_API int32_t vt_decode_token_fused_available(const vt_partition* part, const char** why);
/* Test hook (library plumbing): copies the fp32 shard partials [n_devices][D] of the last layer
 * that the fused decode-token kernel computed (block VT_BLOCK_ATTN: the O-projection partials;
 * VT_BLOCK_FFN: the down-projection partials) to host memory, after synchronizing the device.
 * Valid after a vt_decode_token that ran fused; VT_ERR_STATE when the partition has no fused
 * kernel. */
VT_API vt_status vt_token_partials_read(const vt_partition* part, int32_t block, float* host_dst);
/* Test hook (library plumbing) for the bounded waits of the fused decode-token kernel: in the
 * next vt_decode_token launches, CTA `cta` (0 <= cta < grid; -1: none) does not publish its
 * arrival at the launch's first grid barrier, and a grid-barrier wait gives up after
 * `spin_polls` polls (0: the built-in limit, several seconds).  The other CTAs then give up
 * waiting, the kernel returns with VT_DEV_WAIT_TIMEOUT in the KV status word and the token's
 * output and appended K/V undefined (the lengths still advance by one).  vt_kv_status or
 * vt_partition_status with clear = 1 removes both settings and re-arms the barrier.
 * Synchronous.  VT_ERR_STATE when the partition has no fused kernel. */
VT_API vt_status vt_token_test_barrier(vt_partition* part, int32_t cta, uint32_t spin_polls, vt_stream stream);
/* vt_prefill_tokens (Section 2.1, prefill phase, through the tensor-parallel layers of Section
 * 3.2.1): n prompt rows through every layer (same order as vt_decode_token), then every layer's
 * KV length advances by n.  x_in, x_out: device fp16 [n, D], may be the same.  The shards of a
 * block run together: one tensor-core GEMM launch per projection covers every shard (each with
 * its own partial), then the combine adds them in shard order.  Prompts longer than 1024 rows run
 * in chunks of 1024.  Every shard must be fp16: VT_ERR_STATE when one is block-quantized. */
VT_API vt_status vt_prefill_tokens(const vt_partition* part, vt_kv* kv, const void* x_in, int32_t n,
                            void* x_out, vt_stream stream);

#ifdef __cplusplus
}
#endif

#endif /* VOLTRON_H */
