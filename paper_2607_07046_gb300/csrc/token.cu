// Persistent decode-token kernel (sm_103a): one cooperative launch computes one decode token
// through every layer of a tensor-parallel partition.
//
// What it computes is what the per-shard decode kernels compute, in the same order of shards
// (Voltron Section 2.1, decoder layer and decode phase; Section 3.2.1, tensor parallelism): for
// every layer, each ATTN shard's RMSNorm, QKV projection with RoPE and KV append, attention over
// its KV heads and partial O projection; the combine h = x + sum of ATTN partials (fp16); each
// FFN shard's RMSNorm, SwiGLU and partial down projection; the combine x_next = h + sum of FFN
// partials (fp16).
//
// Why one kernel.  A decode token streams every weight once through small, dependent
// matrix-vector products: as separate kernels that is hundreds of launches of 5-20 us, and the
// ramp-up and tail of each leave HBM idle for a large share of the token.  Here every CTA (one
// per SM) streams a fixed slice of every layer's weights, and of the cached K/V rows, through a
// ring of shared-memory stages that a producer warp (the one working warp of a third warpgroup,
// which hands its registers to the consumers) fills with bulk copies.  The copies depend on
// nothing the token computes, so the producer runs ahead of the arithmetic.  Eight consumer warps
// do the arithmetic and meet the other CTAs at four grid barriers per layer (after QKV, after
// attention, after O, after the FFN); while they wait, the ring keeps filling.
//
// Work split: CTA c of G CTAs takes the c-th of G near-equal contiguous ranges of
//   QKV        row pairs of all shards' Wqkv, shard after shard (pair = RoPE rotation pair)
//   attention  (KV head, position) pairs over all KV heads; each CTA stores the online-softmax
//              state (max, sum, weighted V) of each KV head it touched, and every CTA that
//              projects a shard's O rows merges the states of that shard's heads with
//              log-sum-exp weights
//   O          rows of all shards' Wo, shard after shard, into the shard partials
//   FFN        intermediate columns of all shards: gate/up rows, SwiGLU, then the matching rows
//              of the transposed down slice, accumulated per CTA and added into the shard
//              partial with one bulk reduction (so FFN partials repeat only to fp32 rounding)
// The matrix-vector products run on the tensor cores (mma.sync; see the tensor-core GEMV notes
// below); the FFN down projection, a sum of scaled rows, runs on the CUDA cores.
// Every shard's partial depends on that shard's weights only, and the combines add the shards in
// index order.  Each CTA recomputes the combines it needs (the layer input and h) from the
// partials, which live in L2, instead of waiting for one CTA to publish them.
//
// Files: token_kernel.cuh holds the device code, templated on the tensor-core steps per row
// segment, the chunks per thread of a D-vector, the head dim, the query heads per KV head and
// whether the shared-memory O path is compiled in; token_v1.cu and token_v2.cu instantiate the
// variants (each carries a single attention path, which keeps it small in the instruction cache,
// a measured 11% of the token time for the 7B shapes); this file chooses and launches a variant.
//
// Waits.  The grid barrier and every stage wait give up after a bounded number of polls; the CTA
// that gives up sets the token's abort word and VT_DEV_WAIT_TIMEOUT, every other CTA sees the
// abort word at its next wait, and all of them run the rest of the schedule without waiting or
// computing, so the named barriers between consumer warps still line up.  The producer never
// leaves with a copy in flight.
#include <cuda_runtime.h>

#include <algorithm>
#include <string>

#include "internal.h"

namespace vt {

size_t token_state_floats(int grid, int group, int dh) { return (size_t)grid * kTokMaxSeg * group * (dh + 4); }

static size_t token_smem(const TokArgs& a, int stages, int uni_floats, int slot_floats) {
    return 1024 + (size_t)stages * kTokStageBytes + (((size_t)a.d * 2 + 127) & ~(size_t)127) +
           (((size_t)uni_floats * 4 + 127) & ~(size_t)127) + (((size_t)slot_floats * 4 + 127) & ~(size_t)127) +
           128 * 4 + 64 * 4 + (size_t)kTokMaxLayers * 4 + (size_t)2 * stages * 8;
}

static const TokVariant* g_tok_var[16];
static size_t g_tok_dyn_max[16];
static int g_tok_nvar = 0;
static int g_tok_coop = 0;

cudaError_t init_token_kernels() {
    int dev = 0, optin = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&g_tok_coop, cudaDevAttrCooperativeLaunch, dev);
    if (e != cudaSuccess) return e;
    g_tok_nvar = 0;
    for (auto get : {token_variants_workloads, token_variants_small}) {
        const TokVariant* v = nullptr;
        const int n = get(&v);
        for (int i = 0; i < n && g_tok_nvar < 16; ++i) {
            if ((e = v[i].init(optin, &g_tok_dyn_max[g_tok_nvar])) != cudaSuccess) return e;
            g_tok_var[g_tok_nvar++] = &v[i];
        }
    }
    return cudaSuccess;
}

bool token_plan(const TokArgs& a, int max_hq, TokPlan* plan, std::string* why) {
    auto no = [&](const char* w) {
        if (why) *why = w;
        return false;
    };
    if (!g_tok_coop) return no("the device cannot launch cooperative kernels");
    if (a.d % 64 != 0 || a.d > kTokMaxD) return no("d_model must be a multiple of 64 and at most 6144");
    if (a.dh != 64 && a.dh != 128) return no("d_head must be 64 or 128");
    if (a.group != 1 && a.group != 2 && a.group != 4) return no("query heads per KV head must be 1, 2 or 4");
    if (a.n_layers < 1 || a.n_layers > kTokMaxLayers) return no("too many layers");
    if (a.n_dev < 1 || a.n_dev > VT_MAX_DEVICES) return no("bad device count");
    const int grid = g_num_sms;
    if (grid < 1 || grid > kTokMaxGrid || a.n_kv > grid) return no("more KV heads than SMs");
    if (!mma_ok(a.d)) return no("d_model does not split into whole tensor-core steps");
    const MmaGeom gd = mma_geom(a.d);
    const int steps = gd.L / 16, mc = (a.d / 8 + kTokConsumers - 1) / kTokConsumers;
    // O rows whose length does not split into the kernel's steps need a variant with the
    // shared-memory (or CUDA-core) O path
    bool need_osmem = false;
    for (int s = 0; s < a.n_dev; ++s)
        if (a.hq[s] > 0 && !(mma_ok(a.hq[s] * a.dh) && mma_geom(a.hq[s] * a.dh).L == 16 * steps)) need_osmem = true;
    int vi = -1;
    for (int i = 0; i < g_tok_nvar; ++i) {
        const TokVariant& v = *g_tok_var[i];
        if (v.steps != steps || v.mc != mc || v.dh != a.dh || v.group != a.group || (need_osmem && !v.osmem)) continue;
        if (vi < 0 || (g_tok_var[vi]->osmem && !v.osmem)) vi = i;  // prefer the variant without the extra paths
    }
    if (vi < 0) return no("no compiled kernel variant for these shapes");
    // partial-sum slots: QKV rows of a CTA, the gate/up rows of an FFN column group, O rows of a
    // CTA (with the slice table of the KV heads beside them)
    int64_t pairs = 0;
    int max_k = 1;
    for (int s = 0; s < a.n_dev; ++s) {
        pairs += (int64_t)(a.hq[s] + 2 * a.hk[s]) * a.dh / 2;
        if (a.hq[s] > 0) max_k = std::max(max_k, a.hq[s] * a.dh);
    }
    int o_spr = 8;
    for (int s = 0; s < a.n_dev; ++s)
        if (a.hq[s] > 0 && mma_ok(a.hq[s] * a.dh)) o_spr = std::max(o_spr, mma_geom(a.hq[s] * a.dh).spr);
    int64_t n_o = 0;
    for (int s = 0; s < a.n_dev; ++s) n_o += a.hq[s] > 0 ? a.d : 0;
    const int64_t qkv_rows = 2 * ((pairs + grid - 1) / grid), o_rows = (n_o + grid - 1) / grid + 1;
    int64_t ffn_tot = 0;
    for (int s = 0; s < a.n_dev; ++s) ffn_tot += a.cols[s];
    const int gcol = (int)std::min<int64_t>((ffn_tot + grid - 1) / grid + 1, 128);
    int64_t slot = qkv_rows * gd.spr;
    slot = std::max<int64_t>(slot, (int64_t)2 * gcol * gd.spr);
    slot = std::max<int64_t>(slot, o_rows * o_spr);
    // merge scratch: (max, sum) of every slice of every KV head of a shard, then their offsets
    // the second half of the slots holds the slice table of every KV head during the O phase,
    // while the O rows' partial sums use the first half
    const int64_t table = (int64_t)a.n_kv * (grid / std::max(1, a.n_kv) + 3);
    slot = std::max<int64_t>(slot, 2 * std::max<int64_t>(table, o_rows * o_spr));
    slot = std::max<int64_t>(slot, a.d);  // the FFN phase stages a D-vector there for its bulk reduction
    if (slot > 16384) return no("too much per-CTA work for the partial-sum slots");
    const int uni = std::max(max_hq * a.dh, kTokWarps * a.group * (a.dh + 2));
    int stages = kTokMaxStages;
    while (stages >= kTokMinStages && token_smem(a, stages, uni, (int)slot) > g_tok_dyn_max[vi]) --stages;
    if (stages < kTokMinStages) return no("not enough shared memory");
    const size_t smem = token_smem(a, stages, uni, (int)slot);
    int per_sm = 0;
    cudaError_t e = g_tok_var[vi]->occupancy(&per_sm, smem);
    if (e != cudaSuccess || per_sm < 1) {
        cudaGetLastError();
        return no("the kernel does not fit on an SM");
    }
    plan->grid = grid;
    plan->stages = stages;
    plan->uni_floats = uni;
    plan->slot_floats = (int)slot;
    plan->ffn_gcol = gcol;
    plan->variant = vi;
    plan->smem = smem;
    return true;
}

cudaError_t launch_decode_token(const TokArgs& args, const TokPlan& plan, cudaStream_t st) {
    TokArgs a = args;
    a.stages = plan.stages;
    a.uni_floats = plan.uni_floats;
    a.slot_floats = plan.slot_floats;
    a.ffn_gcol = plan.ffn_gcol;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(plan.grid);
    cfg.blockDim = dim3(kTokThreads);
    cfg.dynamicSmemBytes = plan.smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return g_tok_var[plan.variant]->launch(a, cfg);
}

}  // namespace vt
