// Decode attention whose scratch is a fixed array of the module, not an allocation.
//
// The ordinary ATTN decode step keeps its intermediates (rotated queries, attention output) in
// per-device buffers that vt_partition_create allocated, and merges its split-K slices inside a
// thread-block cluster.  This file holds a variant of the attention kernel for callers that must
// not allocate device memory: its intermediates and its split-K partial states all live in one
// file-scope __device__ array, which the CUDA loader places in device memory together with the
// module's code, before any call.
//
// What it computes is the same as k_attn_decode (Voltron Section 2.1, attention of one decode
// token over positions 0..p of the shard's KV heads): each CTA of a (split, KV head) grid scores
// one slice of the cached positions for every query head of the group and keeps the online
// softmax state (max, sum, weighted V) in fp32; it stores that state in the scratch, and the last
// CTA of the head to finish (an arrival counter per head) merges the slices with log-sum-exp
// weights.
//
// Zero at start: only the arrival counters.  A __device__ array is zero when the module is
// loaded, and the merging CTA puts its head's counter back to zero, so every call finds them at
// zero.  The other regions are written before they are read within a call.
// Races: two calls in flight at once (two streams, or two host threads) share the one array and
// corrupt each other's intermediates and counters; calls must be ordered.
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include <mutex>

#include "device.cuh"
#include "internal.h"

namespace vt {

static __device__ __align__(256) uint8_t g_static_scratch[kStaticScratchBytes];

static size_t round256(size_t b) { return (b + 255) & ~(size_t)255; }

StaticAttnLayout static_attn_layout(int hq, int hk, int dh) {
    StaticAttnLayout L{};
    const int group = hk > 0 ? hq / hk : 1;
    L.counters = 0;
    L.q = round256((size_t)kStaticMaxKvHeads * 4);
    L.attn = L.q + round256((size_t)hq * dh * 4);
    L.part_ml = L.attn + round256((size_t)hq * dh * 4);
    L.part_o = L.part_ml + round256((size_t)hk * kStaticSplits * group * 2 * 4);
    L.bytes = L.part_o + round256((size_t)hk * kStaticSplits * group * dh * 4);
    return L;
}

// The device address of the array, looked up once per device (with that device current) and kept.
cudaError_t static_scratch_base(void** out) {
    static std::mutex mu;
    static void* addr[kStaticMaxDevices] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kStaticMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(mu);
    if (!addr[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_static_scratch);
        if (e != cudaSuccess) return e;
        if (!p) return cudaErrorInvalidSymbol;
        addr[dev] = p;
    }
    *out = addr[dev];
    return cudaSuccess;
}

constexpr int kSplitWarps = 4;

// grid (kStaticSplits, hk), kSplitWarps warps.  Warp w of a CTA takes positions t0 + w, t0 + w + 4,
// ... of its slice, one at a time; the warps' states merge in fixed order in shared memory.
template <int DH, int G>
__global__ void __launch_bounds__(kSplitWarps * 32) k_attn_decode_split(const __grid_constant__ StaticAttnArgs a) {
    constexpr int EPL = DH / 32;
    __shared__ float sm_m[kSplitWarps][G], sm_l[kSplitWarps][G];
    __shared__ float sm_o[kSplitWarps][G][DH];
    __shared__ int s_last;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int split = blockIdx.x, nsplit = gridDim.x, j = blockIdx.y;

    // the preceding QKV kernel wrote the queries and appended this token's K and V
    pdl_wait();
    const int len = *a.len;
    const bool ok = len >= 0 && len < a.cap;
    const int n_pos = ok ? len + 1 : min(max(len, 0), a.cap);
    const int t_lo = (a.window > 0 && n_pos > a.window) ? n_pos - a.window : 0;  // sliding window
    const int n_att = n_pos - t_lo;
    const int chunk = (n_att + nsplit - 1) / nsplit;
    const int t0 = t_lo + min(split * chunk, n_att), t1 = min(n_pos, t0 + chunk);
    const __half* kbase = a.kcache + (int64_t)j * a.cap * DH;
    const __half* vbase = a.vcache + (int64_t)j * a.cap * DH;

    float q[G][EPL], m[G], l[G], o[G][EPL];
#pragma unroll
    for (int h = 0; h < G; ++h) {
        m[h] = -INFINITY;
        l[h] = 0.f;
#pragma unroll
        for (int e = 0; e < EPL; ++e) {
            q[h][e] = __ldcg(a.q + (j * G + h) * DH + lane * EPL + e);
            o[h][e] = 0.f;
        }
    }
    // one vector load per lane for its EPL elements of a K row and of a V row (8 or 4 bytes)
    auto load_row = [&](const __half* row, float (&dst)[EPL]) {
        if constexpr (EPL == 4) {
            const uint2 u = __ldcg(reinterpret_cast<const uint2*>(row + lane * 4));
            const float2 f0 = h2_to_f2(u.x), f1 = h2_to_f2(u.y);
            dst[0] = f0.x; dst[1] = f0.y; dst[2] = f1.x; dst[3] = f1.y;
        } else {
            const float2 f0 = h2_to_f2(__ldcg(reinterpret_cast<const unsigned int*>(row + lane * 2)));
            dst[0] = f0.x; dst[1] = f0.y;
        }
    };
    for (int p = t0 + warp; p < t1; p += kSplitWarps) {
        float kv[EPL], vv[EPL];
        load_row(kbase + (int64_t)p * DH, kv);
        load_row(vbase + (int64_t)p * DH, vv);
#pragma unroll
        for (int h = 0; h < G; ++h) {
            float sc = 0.f;
#pragma unroll
            for (int e = 0; e < EPL; ++e) sc = fmaf(q[h][e], kv[e], sc);
            sc = warp_sum(sc) * a.scale_log2;
            const float mn = fmaxf(m[h], sc);
            const float corr = exp2f(m[h] - mn), pw = exp2f(sc - mn);
            l[h] = l[h] * corr + pw;
#pragma unroll
            for (int e = 0; e < EPL; ++e) o[h][e] = fmaf(o[h][e], corr, pw * vv[e]);
            m[h] = mn;
        }
    }
#pragma unroll
    for (int h = 0; h < G; ++h) {
        if (lane == 0) {
            sm_m[warp][h] = m[h];
            sm_l[warp][h] = l[h];
        }
#pragma unroll
        for (int e = 0; e < EPL; ++e) sm_o[warp][h][lane * EPL + e] = o[h][e];
    }
    __syncthreads();

    // this CTA's slice state -> scratch, slot (j, split)
    float* part_m = a.part_ml + ((size_t)j * nsplit + split) * G * 2;
    float* part_o = a.part_o + ((size_t)j * nsplit + split) * G * DH;
    for (int f = tid; f < G * DH; f += kSplitWarps * 32) {
        const int h = f / DH, d = f - h * DH;
        float M = -INFINITY;
        for (int w = 0; w < kSplitWarps; ++w) M = fmaxf(M, sm_m[w][h]);
        float L = 0.f, O = 0.f;
        if (M != -INFINITY)
            for (int w = 0; w < kSplitWarps; ++w) {
                const float s = exp2f(sm_m[w][h] - M);
                L += sm_l[w][h] * s;
                O += sm_o[w][h][d] * s;
            }
        part_o[f] = O;
        if (d == 0) {
            part_m[2 * h] = M;
            part_m[2 * h + 1] = L;
        }
    }
    // publish the state, then count this slice in; the last slice of the head merges
    __threadfence();
    __syncthreads();
    if (tid == 0) s_last = atomicAdd(a.counters + j, 1u) == (unsigned)(nsplit - 1);
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    const float* hm = a.part_ml + (size_t)j * nsplit * G * 2;
    const float* ho = a.part_o + (size_t)j * nsplit * G * DH;
    for (int f = tid; f < G * DH; f += kSplitWarps * 32) {
        const int h = f / DH, d = f - h * DH;
        float M = -INFINITY;
        for (int c = 0; c < nsplit; ++c) M = fmaxf(M, __ldcg(hm + (c * G + h) * 2));
        float L = 0.f, O = 0.f;
        if (M != -INFINITY)
            for (int c = 0; c < nsplit; ++c) {
                const float mc = __ldcg(hm + (c * G + h) * 2);
                const float s = mc == -INFINITY ? 0.f : exp2f(mc - M);
                L += __ldcg(hm + (c * G + h) * 2 + 1) * s;
                O += __ldcg(ho + (size_t)c * G * DH + f) * s;
            }
        a.out[(j * G + h) * DH + d] = L > 0.f ? O / L : 0.f;
    }
    // leave the counter at zero for the next call
    if (tid == 0) atomicExch(a.counters + j, 0u);
}

template <int DH, int G>
static cudaError_t launch_split(const StaticAttnArgs& a, cudaStream_t st) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(kStaticSplits, a.hk);
    cfg.blockDim = dim3(kSplitWarps * 32);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = g_use_pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, k_attn_decode_split<DH, G>, a);
}

template <int DH>
static cudaError_t launch_split_dh(const StaticAttnArgs& a, cudaStream_t st) {
    switch (a.group) {
        case 1: return launch_split<DH, 1>(a, st);
        case 2: return launch_split<DH, 2>(a, st);
        case 4: return launch_split<DH, 4>(a, st);
        case 8: return launch_split<DH, 8>(a, st);
        default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_attn_decode_static(const StaticAttnArgs& a, cudaStream_t st) {
    if (a.hk <= 0) return cudaSuccess;
    if (a.hk > kStaticMaxKvHeads) return cudaErrorInvalidValue;
    if (a.dh == 128) return launch_split_dh<128>(a, st);
    if (a.dh == 64) return launch_split_dh<64>(a, st);
    return cudaErrorInvalidValue;
}

}  // namespace vt
