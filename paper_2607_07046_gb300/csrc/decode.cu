// Decode-path kernels for one tensor-parallel shard (batch 1), sm_103a.
//
// What they compute (Voltron Section 2.1, per shard as in Section 3.2.1):
//   k_gemv        y = W . v for the shard's rows of a linear layer, with
//                   - an RMSNorm prologue (v = x * g / sqrt(mean(x^2) + eps)) for the QKV
//                     projection,
//                   - epilogues: RoPE + KV-cache append (QKV) or a plain fp32 partial (O).
//   k_attn_decode split-K flash decoding: one thread-block cluster per KV head; each CTA scores
//                 one slice of the cached positions for all query heads of the group, keeps
//                 (max, sum, weighted V) in fp32, and the slices are merged with log-sum-exp
//                 weights through distributed shared memory.
//   k_ffn         the whole FFN block of a shard in one launch: RMSNorm, gate/up GEMV with
//                 SwiGLU for a few columns per CTA, then those columns' rows of the transposed
//                 down slice, reduced into the fp32 partial.
//   k_combine     the aggregation on the main device: residual + sum of partials, in shard order,
//                 clearing the partials it consumed.
//
// All of them are HBM-bound (one fp16 weight or cache element read per two flops); the design
// notes are at each kernel.
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include <utility>

#include "device.cuh"
#include "internal.h"

namespace vt {

bool g_use_pdl = true;
int g_grid_mult = 1;
int g_num_sms = 0;

template <typename... KArgs, typename... Args>
static cudaError_t launch_k(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                            cudaStream_t st, Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = g_use_pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...);
}

// ============================================================== GEMV
//
// Geometry.  A CTA of 8 warps owns a contiguous slab of rows (pairs of rows for the paired
// epilogues).  The row length k is cut into 16-byte chunks; each lane owns CPL chunks of a row
// (chunk (slice * CPL + q) * 32 + lane), WPR = ceil(chunks / (32 CPL)) warps cover one row, and
// the 8 warps form RG = 8 / WPR row groups that walk the slab's rows in lockstep.  A lane's input
// values (x^ or v) are therefore fixed for the whole slab and stay in registers.
//
// Pipeline.  Weights move with 16-byte LDG.128 loads straight into registers, two batches of R
// rows (R * CPL chunks per lane) in flight.  Both batches are issued before griddepcontrol.wait:
// they do not depend on the previous kernel, so a kernel streams its first 64 KB per SM while
// the previous kernel finishes.  After a batch is consumed, its R row partials per lane are
// reduced across the warp with a multi-row butterfly (R rows in 9 shuffles for R = 8 rather than
// 5 per row), and each (row, slice) total goes to a shared-memory slot; the epilogue sums the
// WPR slots of a row in slice order, so results are deterministic.

static __host__ __device__ __forceinline__ int round_up8(int k) { return (k + 7) & ~7; }

// Chunks per lane for a row of `k` columns: the choice with the best use of the 8 warps' lanes.
int gemv_cpl(int k) {
    const int nch = round_up8(k) / 8;
    static const int cand[] = {1, 2, 3, 4, 8};
    int best = 8;
    double bs = -1.0;
    for (int c : cand) {
        const int wpr = (nch + 32 * c - 1) / (32 * c);
        if (wpr > kGemvWarps) continue;
        const int rg = kGemvWarps / wpr;
        const double score = (double)(rg * wpr) / kGemvWarps * (double)nch / (double)(wpr * 32 * c);
        if (score > bs + 1e-9) {
            bs = score;
            best = c;
        }
    }
    return best;
}

int gemv_grid(int rows, int unit) {
    const int units = rows / unit;
    if (units <= 0) return 0;
    int g = (g_num_sms > 0 ? g_num_sms : 148) * g_grid_mult;
    const int per = kGemvMaxSlabRows / unit;
    const int need = (units + per - 1) / per;
    if (g < need) g = need;
    if (g > units) g = units;
    return g;
}

template <int EPI, int CPL, int R>
__global__ void __launch_bounds__(kGemvThreads, (CPL <= 4 ? 2 : 1))
    k_gemv(const __grid_constant__ GemvArgs a) {
    constexpr int NB = R * CPL;  // chunks per lane per batch
    __shared__ float slots[kGemvMaxSlabRows * kGemvWarps];
    __shared__ float red[kGemvWarps + 1];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    constexpr int unit = (EPI == kEpiPlain) ? 1 : 2;
    const int units = a.rows / unit;
    const int r0 = (int)(((int64_t)blockIdx.x * units) / gridDim.x) * unit;
    const int r1 = (int)(((int64_t)(blockIdx.x + 1) * units) / gridDim.x) * unit;
    const int nrows = r1 - r0;
    const int nch = round_up8(a.k) >> 3;
    const int wpr = (nch + 32 * CPL - 1) / (32 * CPL);
    const int rg = kGemvWarps / wpr;
    const int slice = warp % wpr, grp = warp / wpr;
    const bool active = grp < rg;
    const int n_my = active ? max(0, (nrows - grp + rg - 1) / rg) : 0;
    const __half* wbase = a.w + (int64_t)(r0 + grp) * a.row_stride;
    const int64_t rstep = (int64_t)rg * a.row_stride;

    auto load = [&](uint4 (&b)[NB], int i0) {
#pragma unroll
        for (int j = 0; j < R; ++j)
#pragma unroll
            for (int q = 0; q < CPL; ++q) {
                const int i = i0 + j, ch = (slice * CPL + q) * 32 + lane;
                b[j * CPL + q] = (i < n_my && ch < nch) ? ldg_stream(wbase + i * rstep + ch * 8)
                                                        : make_uint4(0u, 0u, 0u, 0u);
            }
    };
    uint4 b0[NB], b1[NB];
    load(b0, 0);  // weights are constant: stream them before waiting on the previous kernel
    load(b1, R);
    if (!a.indep) pdl_wait();
    else pdl_launch_dependents();

    // this lane's input values
    float xr[CPL][8];
    if (a.x != nullptr) {
        float ss = 0.f;
        for (int i = tid * 8; i < a.k; i += kGemvThreads * 8) {
            const uint4 u = *reinterpret_cast<const uint4*>(a.x + i);
            const float2 p0 = h2_to_f2(u.x), p1 = h2_to_f2(u.y), p2 = h2_to_f2(u.z), p3 = h2_to_f2(u.w);
            ss += p0.x * p0.x + p0.y * p0.y + p1.x * p1.x + p1.y * p1.y + p2.x * p2.x + p2.y * p2.y +
                  p3.x * p3.x + p3.y * p3.y;
        }
        ss = warp_sum(ss);
        if (lane == 0) red[warp] = ss;
        __syncthreads();
        if (tid == 0) {
            float tot = 0.f;
            for (int w = 0; w < kGemvWarps; ++w) tot += red[w];
            red[kGemvWarps] = 1.0f / sqrtf(tot / (float)a.k + a.eps);
        }
        __syncthreads();
        const float rinv = red[kGemvWarps];
#pragma unroll
        for (int q = 0; q < CPL; ++q) {
            const int ch = (slice * CPL + q) * 32 + lane;
            if (ch < nch) {
                const uint4 u = *reinterpret_cast<const uint4*>(a.x + ch * 8);
                const uint4 g = *reinterpret_cast<const uint4*>(a.gain + ch * 8);
                const uint32_t uu[4] = {u.x, u.y, u.z, u.w}, gg[4] = {g.x, g.y, g.z, g.w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float2 xv = h2_to_f2(uu[e]), gv = h2_to_f2(gg[e]);
                    xr[q][2 * e] = xv.x * rinv * gv.x;
                    xr[q][2 * e + 1] = xv.y * rinv * gv.y;
                }
            } else {
#pragma unroll
                for (int e = 0; e < 8; ++e) xr[q][e] = 0.f;
            }
        }
    } else {
#pragma unroll
        for (int q = 0; q < CPL; ++q) {
            const int ch = (slice * CPL + q) * 32 + lane;
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                const int idx = ch * 8 + e;
                xr[q][e] = (ch < nch && idx < a.k) ? __ldcg(a.vin + idx) : 0.f;
            }
        }
    }
    if (!a.indep) pdl_launch_dependents();

    constexpr int per = 32 / R;
    auto consume = [&](uint4 (&b)[NB], int i0) {
        float v[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) v[j] = 0.f;
#pragma unroll
        for (int j = 0; j < R; ++j) {
            float acc = 0.f;
#pragma unroll
            for (int q = 0; q < CPL; ++q) acc += dot8(b[j * CPL + q], xr[q]);
            v[j] = acc;
        }
        load(b, i0 + 2 * R);
        const float t = multi_row_sum<R>(v, lane);
        const int i = i0 + lane / per;
        if ((lane % per) == 0 && i < n_my) slots[(grp + rg * i) * kGemvWarps + slice] = t;
    };
    for (int i = 0; i < n_my; i += 2 * R) {
        consume(b0, i);
        if (i + R < n_my) consume(b1, i + R);
    }
    if (a.indep) pdl_wait();  // all reads done; publish only after the previous kernel
    __syncthreads();

    // -------------------------------------------------------------- epilogues
    auto row_value = [&](int r) {
        float y = 0.f;
        for (int w = 0; w < wpr; ++w) y += slots[r * kGemvWarps + w];
        return y;
    };
    if constexpr (EPI == kEpiPlain) {
        for (int r = tid; r < nrows; r += kGemvThreads) a.out[r0 + r] = row_value(r);
    } else if constexpr (EPI == kEpiSwiglu) {
        for (int t = tid; t < nrows / 2; t += kGemvThreads) {
            const float g = row_value(2 * t), u = row_value(2 * t + 1);
            a.out[r0 / 2 + t] = silu(g) * u;
        }
    } else {  // kEpiQkvRope
        const int p = *a.len;
        const bool ok = p >= 0 && p < a.cap;
        if (!ok && tid == 0) set_status(a.status, VT_DEV_KV_OVERFLOW);
        const int half = a.dh >> 1;
        for (int t = tid; t < nrows / 2; t += kGemvThreads) {
            const float ye = row_value(2 * t), yo = row_value(2 * t + 1);
            const int gr = r0 + 2 * t;
            const int b = gr / a.dh;
            const int i = (gr - b * a.dh) >> 1;
            if (b < a.hq + a.hk) {
                const float2 cs = ok ? a.rope[(int64_t)p * half + i] : make_float2(1.f, 0.f);
                const float re = ye * cs.x - yo * cs.y;
                const float ro = ye * cs.y + yo * cs.x;
                if (b < a.hq) {
                    a.out[b * a.dh + i] = re;
                    a.out[b * a.dh + i + half] = ro;
                } else if (ok) {
                    __half* kd = a.kcache + ((int64_t)(b - a.hq) * a.cap + p) * a.dh;
                    kd[i] = __float2half_rn(re);
                    kd[i + half] = __float2half_rn(ro);
                }
            } else if (ok) {
                __half* vd = a.vcache + ((int64_t)(b - a.hq - a.hk) * a.cap + p) * a.dh;
                vd[i] = __float2half_rn(ye);
                vd[i + half] = __float2half_rn(yo);
            }
        }
    }
}

// ============================================================== fused FFN shard (decode)
//
// One kernel per FFN shard, column-split: CTA g owns intermediate columns [j0, j1) of the shard.
//   phase A  a_j = silu(Wg[j] . x^) * (Wu[j] . x^)   (gate/up rows 2j, 2j+1; same machinery as
//            k_gemv, RMSNorm prologue, activations kept in shared memory)
//   phase B  p_g = sum_{j in [j0, j1)} a_j * WdT[j, :]  (rows of the transposed down slice)
// so the shard's partial Wd[:, c0:c1] . a is sum_g p_g, which the combine adds in CTA order.
// Nothing in the kernel waits on another CTA.  The WdT rows a CTA will need are prefetched into
// L2 with one bulk prefetch at kernel start, so phase B streams from L2 while phase A streams
// gate/up rows from HBM.
__device__ __forceinline__ void prefetch_l2_bulk(const void* p, uint32_t bytes) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}

int ffn_grid(int cols) {
    if (cols <= 0) return 0;
    int g = (g_num_sms > 0 ? g_num_sms : 148) * g_grid_mult;
    const int need = (cols + kFfnMaxCols - 1) / kFfnMaxCols;
    if (g < need) g = need;
    if (g > cols) g = cols;
    return g;
}

template <int CPL, int R, int MC>
__global__ void __launch_bounds__(kGemvThreads, 2) k_ffn(const __grid_constant__ FfnDecodeArgs a) {
    constexpr int NB = R * CPL;
    __shared__ float slots[2 * kFfnMaxCols * kGemvWarps];
    __shared__ float act[kFfnMaxCols];
    __shared__ float red[kGemvWarps + 1];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int j0 = (int)(((int64_t)blockIdx.x * a.cols) / gridDim.x);
    const int j1 = (int)(((int64_t)(blockIdx.x + 1) * a.cols) / gridDim.x);
    const int ncol = j1 - j0;
    const int nrows = 2 * ncol;
    const int D = a.d;
    if (tid == 0 && ncol > 0)  // phase B rows: contiguous in the transposed slice
        for (int64_t off = 0, tot = (int64_t)ncol * D * 2; off < tot; off += 65536)
            prefetch_l2_bulk(reinterpret_cast<const uint8_t*>(a.wdt + (int64_t)j0 * D) + off,
                             (uint32_t)(tot - off < 65536 ? tot - off : 65536));

    // ---------------------------------------------------------------- phase A: gate/up rows
    const int nch = D >> 3;
    const int wpr = (nch + 32 * CPL - 1) / (32 * CPL);
    const int rg = kGemvWarps / wpr;
    const int slice = warp % wpr, grp = warp / wpr;
    const bool active = grp < rg;
    const int n_my = active ? max(0, (nrows - grp + rg - 1) / rg) : 0;
    const __half* wbase = a.wgu + (int64_t)(2 * j0 + grp) * D;
    const int64_t rstep = (int64_t)rg * D;
    auto load = [&](uint4 (&b)[NB], int i0) {
#pragma unroll
        for (int j = 0; j < R; ++j)
#pragma unroll
            for (int q = 0; q < CPL; ++q) {
                const int i = i0 + j, ch = (slice * CPL + q) * 32 + lane;
                b[j * CPL + q] = (i < n_my && ch < nch) ? ldg_stream(wbase + i * rstep + ch * 8)
                                                        : make_uint4(0u, 0u, 0u, 0u);
            }
    };
    uint4 b0[NB], b1[NB];
    load(b0, 0);
    load(b1, R);
    if (!a.indep) pdl_wait();
    else pdl_launch_dependents();
    float xr[CPL][8];
    {
        float ss = 0.f;
        for (int i = tid * 8; i < D; i += kGemvThreads * 8) {
            const uint4 u = *reinterpret_cast<const uint4*>(a.x + i);
            const float2 p0 = h2_to_f2(u.x), p1 = h2_to_f2(u.y), p2 = h2_to_f2(u.z), p3 = h2_to_f2(u.w);
            ss += p0.x * p0.x + p0.y * p0.y + p1.x * p1.x + p1.y * p1.y + p2.x * p2.x + p2.y * p2.y +
                  p3.x * p3.x + p3.y * p3.y;
        }
        ss = warp_sum(ss);
        if (lane == 0) red[warp] = ss;
        __syncthreads();
        if (tid == 0) {
            float tot = 0.f;
            for (int w = 0; w < kGemvWarps; ++w) tot += red[w];
            red[kGemvWarps] = 1.0f / sqrtf(tot / (float)D + a.eps);
        }
        __syncthreads();
        const float rinv = red[kGemvWarps];
#pragma unroll
        for (int q = 0; q < CPL; ++q) {
            const int ch = (slice * CPL + q) * 32 + lane;
            if (ch < nch) {
                const uint4 u = *reinterpret_cast<const uint4*>(a.x + ch * 8);
                const uint4 g = *reinterpret_cast<const uint4*>(a.gain + ch * 8);
                const uint32_t uu[4] = {u.x, u.y, u.z, u.w}, gg[4] = {g.x, g.y, g.z, g.w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float2 xv = h2_to_f2(uu[e]), gv = h2_to_f2(gg[e]);
                    xr[q][2 * e] = xv.x * rinv * gv.x;
                    xr[q][2 * e + 1] = xv.y * rinv * gv.y;
                }
            } else {
#pragma unroll
                for (int e = 0; e < 8; ++e) xr[q][e] = 0.f;
            }
        }
    }
    if (!a.indep) pdl_launch_dependents();
    constexpr int per = 32 / R;
    auto consume = [&](uint4 (&b)[NB], int i0) {
        float v[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) v[j] = 0.f;
#pragma unroll
        for (int j = 0; j < R; ++j) {
            float acc = 0.f;
#pragma unroll
            for (int q = 0; q < CPL; ++q) acc += dot8(b[j * CPL + q], xr[q]);
            v[j] = acc;
        }
        load(b, i0 + 2 * R);
        const float t = multi_row_sum<R>(v, lane);
        const int i = i0 + lane / per;
        if ((lane % per) == 0 && i < n_my) slots[(grp + rg * i) * kGemvWarps + slice] = t;
    };
    for (int i = 0; i < n_my; i += 2 * R) {
        consume(b0, i);
        if (i + R < n_my) consume(b1, i + R);
    }
    __syncthreads();
    for (int t = tid; t < ncol; t += kGemvThreads) {
        float g = 0.f, u = 0.f;
        for (int w = 0; w < wpr; ++w) {
            g += slots[(2 * t) * kGemvWarps + w];
            u += slots[(2 * t + 1) * kGemvWarps + w];
        }
        act[t] = silu(g) * u;
    }
    __syncthreads();

    // ---------------------------------------------------------------- phase B: WdT rows
    // thread t owns output chunks t + 256 m (8 outputs each); RB columns per batch, 2 in flight
    constexpr int RB = (8 / MC) > 0 ? (8 / MC) : 1;
    const int nchd = D >> 3;
    float acc[MC][8];
#pragma unroll
    for (int m = 0; m < MC; ++m)
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[m][e] = 0.f;
    const __half* wd0 = a.wdt + (int64_t)j0 * D;
    auto loadb = [&](uint4 (&b)[RB * MC], int c0) {
#pragma unroll
        for (int jj = 0; jj < RB; ++jj)
#pragma unroll
            for (int m = 0; m < MC; ++m) {
                const int col = c0 + jj, ch = tid + kGemvThreads * m;
                b[jj * MC + m] = (col < ncol && ch < nchd) ? ldg_stream(wd0 + (int64_t)col * D + ch * 8)
                                                           : make_uint4(0u, 0u, 0u, 0u);
            }
    };
    auto accum = [&](uint4 (&b)[RB * MC], int c0) {
#pragma unroll
        for (int jj = 0; jj < RB; ++jj) {
            const float s = (c0 + jj < ncol) ? act[c0 + jj] : 0.f;
#pragma unroll
            for (int m = 0; m < MC; ++m) {
                const uint4 w = b[jj * MC + m];
                const float2 w0 = h2_to_f2(w.x), w1 = h2_to_f2(w.y), w2 = h2_to_f2(w.z), w3 = h2_to_f2(w.w);
                acc[m][0] = fmaf(w0.x, s, acc[m][0]);
                acc[m][1] = fmaf(w0.y, s, acc[m][1]);
                acc[m][2] = fmaf(w1.x, s, acc[m][2]);
                acc[m][3] = fmaf(w1.y, s, acc[m][3]);
                acc[m][4] = fmaf(w2.x, s, acc[m][4]);
                acc[m][5] = fmaf(w2.y, s, acc[m][5]);
                acc[m][6] = fmaf(w3.x, s, acc[m][6]);
                acc[m][7] = fmaf(w3.y, s, acc[m][7]);
            }
        }
    };
    {
        uint4 c0b[RB * MC], c1b[RB * MC];
        loadb(c0b, 0);
        loadb(c1b, RB);
        for (int c = 0; c < ncol; c += 2 * RB) {
            accum(c0b, c);
            loadb(c0b, c + 2 * RB);
            if (c + RB < ncol) {
                accum(c1b, c + RB);
                loadb(c1b, c + 3 * RB);
            }
        }
    }
    // the CTA's partial goes through shared memory into one bulk add onto the shard partial
    extern __shared__ __align__(16) float pbuf[];  // [d]
#pragma unroll
    for (int m = 0; m < MC; ++m) {
        const int ch = tid + kGemvThreads * m;
        if (ch < nchd) {
            reinterpret_cast<float4*>(pbuf + ch * 8)[0] = make_float4(acc[m][0], acc[m][1], acc[m][2], acc[m][3]);
            reinterpret_cast<float4*>(pbuf + ch * 8)[1] = make_float4(acc[m][4], acc[m][5], acc[m][6], acc[m][7]);
        }
    }
    fence_proxy_async_smem();
    __syncthreads();
    if (a.indep) pdl_wait();
    if (tid == 0 && ncol > 0) bulk_reduce_add_f32(a.out, pbuf, (uint32_t)D * 4);
    __syncthreads();
}

template <int CPL, int R>
static cudaError_t launch_ffn_cpl(const FfnDecodeArgs& a, int grid, cudaStream_t st) {
    const int mc = ((a.d >> 3) + kGemvThreads - 1) / kGemvThreads;
    const dim3 g(grid), b(kGemvThreads);
    const size_t sm = (size_t)a.d * 4;
    if (mc <= 1) return launch_k(k_ffn<CPL, R, 1>, g, b, sm, st, a);
    if (mc <= 2) return launch_k(k_ffn<CPL, R, 2>, g, b, sm, st, a);
    if (mc <= 3) return launch_k(k_ffn<CPL, R, 3>, g, b, sm, st, a);
    if (mc <= 4) return launch_k(k_ffn<CPL, R, 4>, g, b, sm, st, a);
    return launch_k(k_ffn<CPL, R, 8>, g, b, sm, st, a);
}

cudaError_t launch_ffn_decode(const FfnDecodeArgs& a, int grid, cudaStream_t st) {
    if (grid <= 0) return cudaSuccess;
    switch (gemv_cpl(a.d)) {
        case 1: return launch_ffn_cpl<1, 8>(a, grid, st);
        case 2: return launch_ffn_cpl<2, 4>(a, grid, st);
        case 3: return launch_ffn_cpl<3, 2>(a, grid, st);
        case 4: return launch_ffn_cpl<4, 2>(a, grid, st);
        default: return launch_ffn_cpl<8, 1>(a, grid, st);
    }
}

template <int EPI>
static cudaError_t launch_gemv_epi(const GemvArgs& a, int grid, cudaStream_t st) {
    const dim3 g(grid), b(kGemvThreads);
    switch (gemv_cpl(a.k)) {
        case 1: return launch_k(k_gemv<EPI, 1, 8>, g, b, 0, st, a);
        case 2: return launch_k(k_gemv<EPI, 2, 4>, g, b, 0, st, a);
        case 3: return launch_k(k_gemv<EPI, 3, 2>, g, b, 0, st, a);
        case 4: return launch_k(k_gemv<EPI, 4, 2>, g, b, 0, st, a);
        default: return launch_k(k_gemv<EPI, 8, 1>, g, b, 0, st, a);
    }
}

cudaError_t launch_gemv(int epi, const GemvArgs& a, cudaStream_t st) {
    const int unit = epi == kEpiPlain ? 1 : 2;
    const int grid = gemv_grid(a.rows, unit);
    if (grid == 0) return cudaSuccess;
    switch (epi) {
        case kEpiPlain: return launch_gemv_epi<kEpiPlain>(a, grid, st);
        case kEpiQkvRope: return launch_gemv_epi<kEpiQkvRope>(a, grid, st);
        default: return launch_gemv_epi<kEpiSwiglu>(a, grid, st);
    }
}

// ============================================================== split-K flash decoding
//
// One thread-block cluster per KV head of the shard.  CTA r of the cluster scores a contiguous
// slice of the cached positions for every query head of the KV head's group, keeping the
// online-softmax state (running max m in log2 units, sum l of 2^(s - m), weighted sum o of V)
// in fp32.  Slices merge on chip: after a cluster barrier, CTA r combines feature slice r of
// all CTAs' states through distributed shared memory, out = sum_c 2^(m_c - M) o_c /
// sum_c 2^(m_c - M) l_c with M = max_c m_c, and writes it; a second barrier keeps every CTA's
// state alive until all reads finished.  Cached positions other than the token's own are
// streamed into shared memory by one producer thread with bulk copies before
// griddepcontrol.wait (they were written by earlier tokens); the new position is read after it.

// per-warp states + gather buffers of the cluster merge (csize <= kAttnMaxCluster slices of the
// CTA's feature range, plus their max and sum per head)
static __host__ __device__ __forceinline__ size_t attn_state_floats(int dh, int group) {
    const int fpr = (group * dh + 7) / 8;  // features per CTA for the smallest cluster (8)
    return (size_t)2 * kAttnWarps * group + (size_t)kAttnWarps * group * dh +
           (size_t)kAttnMaxCluster * (2 * group + fpr);
}

size_t attn_decode_smem_bytes(int dh, int group, int stages) {
    const size_t tiles = (size_t)stages * kAttnTilePos * dh * 2 * 2;
    const size_t st = attn_state_floats(dh, group) * 4;
    return tiles + ((st + 15) & ~(size_t)15) + (size_t)2 * stages * 8;
}

int g_attn_cluster = 16;  // set at init: 16 when a 16-CTA cluster can be scheduled, else 8

int attn_cluster_size(int hk) {
    (void)hk;
    return g_attn_cluster;
}

int attn_stages(int cap, int csize) {
    const int per = (cap + csize - 1) / csize;
    int t = (per + kAttnTilePos - 1) / kAttnTilePos;
    return t < 2 ? 2 : (t > kAttnMaxStages ? kAttnMaxStages : t);
}

template <int DH, int G>
__global__ void __launch_bounds__(kAttnThreads) k_attn_decode(const __grid_constant__ AttnDecodeArgs a) {
    extern __shared__ __align__(128) uint8_t smem[];
    constexpr int EPL = DH / 32;  // elements per lane
    constexpr int TILE_BYTES = kAttnTilePos * DH * 2;
    const int S = a.stages;
    uint8_t* ring = smem;  // stage s: K tile at s*2*TILE_BYTES, V tile after it
    float* wm = reinterpret_cast<float*>(smem + (size_t)S * 2 * TILE_BYTES);  // [warps][G]
    float* wl = wm + kAttnWarps * G;                                           // [warps][G]
    float* wo = wl + kAttnWarps * G;                                           // [warps][G][DH]
    constexpr int FMAX = (G * DH + 7) / 8;                                     // features per CTA (csize >= 8)
    float* gm = wo + kAttnWarps * G * DH;                                      // [kAttnMaxCluster][G]
    float* gl = gm + kAttnMaxCluster * G;                                      // [kAttnMaxCluster][G]
    float* go = gl + kAttnMaxCluster * G;                                      // [kAttnMaxCluster][FMAX]
    const size_t st_bytes = (attn_state_floats(DH, G) * 4 + 15) & ~(size_t)15;
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + (size_t)S * 2 * TILE_BYTES + st_bytes);
    uint64_t* empty = full + S;
    __shared__ int s_abort;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int rank = (int)cluster_rank(), csize = (int)cluster_size();  // csize is 8 or 16
    const int j = blockIdx.y;
    // The length was written by a kernel that completed before this one started (see device.cuh).
    const int len = *a.len;
    const bool ok = len >= 0 && len < a.cap;
    const int n_pos = ok ? len + 1 : min(max(len, 0), a.cap);
    const int pnew = ok ? len : -1;
    // sliding window: only the last `window` positions (ending at the new token) are attended
    const int t_lo = (a.window > 0 && n_pos > a.window) ? n_pos - a.window : 0;
    const int n_att = n_pos - t_lo;
    const int chunk = (n_att + csize - 1) / csize;
    const int t0 = t_lo + min(rank * chunk, n_att), t1 = min(n_pos, t0 + chunk);
    const int old_end = pnew >= 0 ? min(t1, pnew) : t1;
    const int n_old = max(old_end - t0, 0);
    const int ntiles = (n_old + kAttnTilePos - 1) / kAttnTilePos;
    const __half* kbase = a.kcache + (int64_t)j * a.cap * DH;
    const __half* vbase = a.vcache + (int64_t)j * a.cap * DH;

    if (tid == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], kAttnWarps);
        }
        s_abort = 0;
        fence_mbar_init();
    }
    cluster_arrive_relaxed();  // matched by cluster_wait() before the first remote store
    __syncthreads();

    if (warp == kAttnWarps) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            int issued = 0;
            for (int t = 0; t < ntiles; ++t) {
                const int s = t % S;
                if (t >= S && !mbar_wait(&empty[s], ((t / S) - 1) & 1)) {
                    s_abort = 1;
                    set_status(a.status, VT_DEV_WAIT_TIMEOUT);
                    break;
                }
                if (*(volatile int*)&s_abort) break;
                const int p0 = t0 + t * kAttnTilePos;
                const int np = min(kAttnTilePos, old_end - p0);
                const uint32_t bytes = (uint32_t)np * DH * 2;
                mbar_arrive_expect_tx(&full[s], 2 * bytes);
                uint8_t* dst = ring + s * 2 * TILE_BYTES;
                bulk_g2s(dst, kbase + (int64_t)p0 * DH, bytes, &full[s]);
                bulk_g2s(dst + TILE_BYTES, vbase + (int64_t)p0 * DH, bytes, &full[s]);
                issued = t + 1;
            }
            // never leave with copies in flight: wait for the last fill of every stage
            for (int t = max(0, issued - S); t < issued; ++t)
                if (!mbar_wait(&full[t % S], (t / S) & 1)) set_status(a.status, VT_DEV_WAIT_TIMEOUT);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------ consumers
        constexpr int NC = kAttnWarps * 32;
        pdl_wait();
        // the rotated queries and (in the CTA whose slice holds it) the token appended by the
        // preceding QKV kernel: all loads issued together, through L2
        const bool has_new = warp == 0 && pnew >= t0 && pnew < t1;
        float q[G][EPL], kn[EPL], vn[EPL];
#pragma unroll
        for (int h = 0; h < G; ++h)
#pragma unroll
            for (int e = 0; e < EPL; ++e) q[h][e] = __ldcg(a.q + (j * G + h) * DH + lane * EPL + e);
#pragma unroll
        for (int e = 0; e < EPL; ++e) {
            kn[e] = has_new ? __half2float(__ldcg(kbase + (int64_t)pnew * DH + lane * EPL + e)) : 0.f;
            vn[e] = has_new ? __half2float(__ldcg(vbase + (int64_t)pnew * DH + lane * EPL + e)) : 0.f;
        }
        pdl_launch_dependents();

        float m[G], l[G], o[G][EPL];
#pragma unroll
        for (int h = 0; h < G; ++h) {
            m[h] = -INFINITY;
            l[h] = 0.f;
#pragma unroll
            for (int e = 0; e < EPL; ++e) o[h][e] = 0.f;
        }
        // Online softmax over batches of P = 8 / G positions: the G x P scores of a batch are
        // reduced across the warp together (one multi-row butterfly), so the dependency chain
        // per batch is one reduction and one rescale instead of one per position.
        constexpr int P = 8 / G;
        auto load_lane = [&](const __half* row, float (&dst)[EPL]) {
            if constexpr (EPL == 4) {
                const uint2 u = *reinterpret_cast<const uint2*>(row + lane * 4);
                const float2 f0 = h2_to_f2(u.x), f1 = h2_to_f2(u.y);
                dst[0] = f0.x; dst[1] = f0.y; dst[2] = f1.x; dst[3] = f1.y;
            } else {
                const float2 f0 = h2_to_f2(*reinterpret_cast<const uint32_t*>(row + lane * 2));
                dst[0] = f0.x; dst[1] = f0.y;
            }
        };
        // kp[i] / vp[i]: rows of batch position i (nullptr: padding, score -inf)
        auto update_batch = [&](const __half* const (&kp)[P], const __half* const (&vp)[P]) {
            float kv[P][EPL], vv[P][EPL];
#pragma unroll
            for (int i = 0; i < P; ++i) {
                if (kp[i]) {
                    load_lane(kp[i], kv[i]);
                    load_lane(vp[i], vv[i]);
                } else {
#pragma unroll
                    for (int e = 0; e < EPL; ++e) kv[i][e] = vv[i][e] = 0.f;
                }
            }
            float part[8];
#pragma unroll
            for (int h = 0; h < G; ++h)
#pragma unroll
                for (int i = 0; i < P; ++i) {
                    float sc = 0.f;
#pragma unroll
                    for (int e = 0; e < EPL; ++e) sc = fmaf(q[h][e], kv[i][e], sc);
                    part[h * P + i] = sc;
                }
            const float mine = multi_row_sum<8>(part, lane);  // lane 4r holds row r = h * P + i
            float sc[G][P];
#pragma unroll
            for (int r = 0; r < 8; ++r) sc[r / P][r % P] = __shfl_sync(0xffffffffu, mine, 4 * r) * a.scale_log2;
#pragma unroll
            for (int h = 0; h < G; ++h) {
                float mb = m[h];
#pragma unroll
                for (int i = 0; i < P; ++i)
                    if (kp[i]) mb = fmaxf(mb, sc[h][i]);
                const float corr = exp2f(m[h] - mb);
                float lsum = l[h] * corr;
                float acc[EPL];
#pragma unroll
                for (int e = 0; e < EPL; ++e) acc[e] = o[h][e] * corr;
#pragma unroll
                for (int i = 0; i < P; ++i) {
                    const float pw = kp[i] ? exp2f(sc[h][i] - mb) : 0.f;
                    lsum += pw;
#pragma unroll
                    for (int e = 0; e < EPL; ++e) acc[e] = fmaf(pw, vv[i][e], acc[e]);
                }
                l[h] = lsum;
#pragma unroll
                for (int e = 0; e < EPL; ++e) o[h][e] = acc[e];
                m[h] = mb;
            }
        };
        for (int t = 0; t < ntiles; ++t) {
            const int s = t % S;
            if (!mbar_wait(&full[s], (t / S) & 1)) {
                s_abort = 1;
                set_status(a.status, VT_DEV_WAIT_TIMEOUT);
                break;
            }
            const int np = min(kAttnTilePos, old_end - (t0 + t * kAttnTilePos));
            const __half* kt = reinterpret_cast<const __half*>(ring + s * 2 * TILE_BYTES);
            const __half* vt = reinterpret_cast<const __half*>(ring + s * 2 * TILE_BYTES + TILE_BYTES);
            // warp w takes positions w*P + i + 4*P*k of the tile
            for (int b0 = warp * P; b0 < np; b0 += kAttnWarps * P) {
                const __half* kp[P];
                const __half* vp[P];
#pragma unroll
                for (int i = 0; i < P; ++i) {
                    const int pos = b0 + i;
                    kp[i] = pos < np ? kt + pos * DH : nullptr;
                    vp[i] = pos < np ? vt + pos * DH : nullptr;
                }
                update_batch(kp, vp);
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty[s]);
        }
        if (has_new) {
#pragma unroll
            for (int h = 0; h < G; ++h) {
                float sc = 0.f;
#pragma unroll
                for (int e = 0; e < EPL; ++e) sc = fmaf(q[h][e], kn[e], sc);
                sc = warp_sum(sc) * a.scale_log2;
                const float mn = fmaxf(m[h], sc);
                const float corr = exp2f(m[h] - mn);
                const float pw = exp2f(sc - mn);
                l[h] = l[h] * corr + pw;
#pragma unroll
                for (int e = 0; e < EPL; ++e) o[h][e] = fmaf(o[h][e], corr, pw * vn[e]);
                m[h] = mn;
            }
        }
        // per-warp states, merged in fixed order below
#pragma unroll
        for (int h = 0; h < G; ++h) {
            if (lane == 0) {
                wm[warp * G + h] = m[h];
                wl[warp * G + h] = l[h];
            }
#pragma unroll
            for (int e = 0; e < EPL; ++e) wo[(warp * G + h) * DH + lane * EPL + e] = o[h][e];
        }
        consumer_bar(1, NC);
        // Merge the warps (fixed order) and push the CTA's state to the CTAs that own each
        // feature: feature f of the G x DH output goes to rank f / fpr, slot `rank`; the max and
        // sum of head h go to every rank (thread d < csize of head h sends them to rank d).
        // Remote stores need no reply; the cluster barrier below makes them visible.
        cluster_wait();  // every CTA of the cluster has started
        const bool dead = s_abort != 0;  // an aborted CTA contributes an empty slice
        const int fpr = (G * DH + csize - 1) / csize;
        for (int idx = tid; idx < G * DH; idx += NC) {
            const int h = idx / DH, d = idx - h * DH;
            float M = -INFINITY;
            if (!dead)
                for (int w = 0; w < kAttnWarps; ++w) M = fmaxf(M, wm[w * G + h]);
            float L = 0.f, O = 0.f;
            if (M != -INFINITY) {
                for (int w = 0; w < kAttnWarps; ++w) {
                    const float f = exp2f(wm[w * G + h] - M);
                    L += wl[w * G + h] * f;
                    O += wo[(w * G + h) * DH + d] * f;
                }
            }
            const int owner = idx / fpr;
            dsmem_st(dsmem_addr(&go[rank * FMAX + (idx - owner * fpr)], owner), O);
            if (d < csize) {
                dsmem_st(dsmem_addr(&gm[rank * G + h], d), M);
                dsmem_st(dsmem_addr(&gl[rank * G + h], d), L);
            }
        }
    }
    if (warp == kAttnWarps) cluster_wait();
    cluster_sync();
    // merge: this CTA owns features [f0, f1); every slice c of the cluster pushed its values
    if (warp < kAttnWarps) {
        const int nf = G * DH, fpr = (nf + csize - 1) / csize;
        const int f0 = rank * fpr, f1 = min(nf, f0 + fpr);
        for (int f = f0 + tid; f < f1; f += kAttnWarps * 32) {
            const int h = f / DH, d = f - h * DH;
            float M = -INFINITY;
            for (int c = 0; c < csize; ++c) M = fmaxf(M, gm[c * G + h]);
            float L = 0.f, O = 0.f;
            if (M != -INFINITY) {
                for (int c = 0; c < csize; ++c) {
                    const float mc = gm[c * G + h];
                    const float w = mc == -INFINITY ? 0.f : exp2f(mc - M);
                    L += gl[c * G + h] * w;
                    O += go[c * FMAX + (f - f0)] * w;
                }
            }
            a.out[(j * G + h) * DH + d] = L > 0.f ? O / L : 0.f;
        }
    }
}

template <int DH, int G>
static cudaError_t launch_attn_dhg(const AttnDecodeArgs& a, cudaStream_t st) {
    const int cs = attn_cluster_size(a.hk);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(cs, a.hk);
    cfg.blockDim = dim3(kAttnThreads);
    cfg.dynamicSmemBytes = attn_decode_smem_bytes(DH, G, a.stages);
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = cs;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = g_use_pdl ? 2 : 1;
    return cudaLaunchKernelEx(&cfg, k_attn_decode<DH, G>, a);
}

template <int DH>
static cudaError_t launch_attn_dh(const AttnDecodeArgs& a, cudaStream_t st) {
    switch (a.group) {
        case 1: return launch_attn_dhg<DH, 1>(a, st);
        case 2: return launch_attn_dhg<DH, 2>(a, st);
        case 4: return launch_attn_dhg<DH, 4>(a, st);
        case 8: return launch_attn_dhg<DH, 8>(a, st);
        default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_attn_decode(const AttnDecodeArgs& a, cudaStream_t st) {
    if (a.hk <= 0) return cudaSuccess;
    if (a.dh == 128) return launch_attn_dh<128>(a, st);
    if (a.dh == 64) return launch_attn_dh<64>(a, st);
    return cudaErrorInvalidValue;
}

// ============================================================== small kernels

// out[e] = fp16(residual[e] + sum_s parts[s][e]), shards added in order s = 0..n-1 in fp32.
// With `clear`, every partial element is zeroed right after it is read (the partial buffers are
// then ready for the bulk reductions of the next block).
__global__ void __launch_bounds__(256) k_combine(const __grid_constant__ CombineArgs a) {
    pdl_wait();
    pdl_launch_dependents();
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < a.count; e += stride) {
        float v[VT_MAX_DEVICES];
#pragma unroll
        for (int s = 0; s < VT_MAX_DEVICES; ++s)
            v[s] = (s < a.n && a.parts[s] != nullptr) ? __ldcg(a.parts[s] + e) : 0.f;
        float acc = a.residual ? __half2float(a.residual[e]) : 0.f;
#pragma unroll
        for (int s = 0; s < VT_MAX_DEVICES; ++s)
            if (s < a.n) acc += v[s];
        a.out[e] = __float2half_rn(acc);
        if (a.clear) {
#pragma unroll
            for (int s = 0; s < VT_MAX_DEVICES; ++s)
                if (s < a.n && a.parts[s] != nullptr) a.parts[s][e] = 0.f;
        }
    }
}

cudaError_t launch_combine(const CombineArgs& a, cudaStream_t st) {
    if (a.count <= 0) return cudaSuccess;
    int64_t blocks = (a.count + 255) / 256;
    const int64_t cap = (int64_t)(g_num_sms > 0 ? g_num_sms : 148) * 8;
    if (blocks > cap) blocks = cap;
    return launch_k(k_combine, dim3((unsigned)blocks), dim3(256), 0, st, a);
}

__global__ void k_fill_zero_f32(float* p, int64_t n) {
    pdl_wait();
    pdl_launch_dependents();
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) p[i] = 0.f;
}

cudaError_t launch_fill_zero_f32(float* p, int64_t n, cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    int64_t blocks = (n + 255) / 256;
    if (blocks > 1024) blocks = 1024;
    return launch_k(k_fill_zero_f32, dim3((unsigned)blocks), dim3(256), 0, st, p, n);
}

// len[l] += delta for the layers [first, first + count); a result outside [0, cap] is clamped
// into it and flagged VT_DEV_KV_OVERFLOW (the host checks this before launch, except while a
// stream is being captured, when its length mirror does not follow the device).
__global__ void k_kv_advance(int32_t* len, int first, int count, int delta, int cap, uint32_t* status) {
    pdl_wait();
    pdl_launch_dependents();
    for (int i = threadIdx.x; i < count; i += blockDim.x) {
        const int64_t v = (int64_t)len[first + i] + delta;
        if (v < 0 || v > cap) set_status(status, VT_DEV_KV_OVERFLOW);
        len[first + i] = (int32_t)(v < 0 ? 0 : (v > cap ? cap : v));
    }
}

cudaError_t launch_kv_advance(int32_t* len, int first, int count, int delta, int cap, uint32_t* status,
                              cudaStream_t st) {
    return launch_k(k_kv_advance, dim3(1), dim3(128), 0, st, len, first, count, delta, cap, status);
}

__global__ void k_rope_table(float2* tab, int max_seq, int half, int dh, double theta) {
    pdl_wait();
    pdl_launch_dependents();
    const int64_t n = (int64_t)max_seq * half;
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < n;
         e += (int64_t)gridDim.x * blockDim.x) {
        const int p = (int)(e / half), i = (int)(e - (int64_t)p * half);
        const double freq = pow(theta, -2.0 * (double)i / (double)dh);
        double s, c;
        sincos((double)p * freq, &s, &c);
        tab[e] = make_float2((float)c, (float)s);
    }
}

cudaError_t launch_rope_table(float2* tab, int max_seq, int dh, double theta, cudaStream_t st) {
    const int half = dh / 2;
    const int64_t n = (int64_t)max_seq * half;
    int64_t blocks = (n + 255) / 256;
    if (blocks > 4096) blocks = 4096;
    if (blocks < 1) blocks = 1;
    return launch_k(k_rope_table, dim3((unsigned)blocks), dim3(256), 0, st, tab, max_seq, half,
                    dh, theta);
}

// One CTA per row: 16-byte chunks of the table row (d is a multiple of 8, out 16-byte aligned).
// An id outside [0, vocab) gives a zero row and sets VT_DEV_BAD_TOKEN.
__global__ void k_embed(const __half* table, const int32_t* ids, int n, int d, int vocab, __half* out,
                        uint32_t* status) {
    pdl_wait();
    pdl_launch_dependents();
    const int row = blockIdx.x;
    if (row >= n) return;
    const int id = ids[row];
    const bool ok = id >= 0 && id < vocab;
    if (!ok && threadIdx.x == 0) set_status(status, VT_DEV_BAD_TOKEN);
    const uint4* src = reinterpret_cast<const uint4*>(table + (int64_t)(ok ? id : 0) * d);
    uint4* dst = reinterpret_cast<uint4*>(out + (int64_t)row * d);
    for (int c = threadIdx.x; c < d / 8; c += blockDim.x) dst[c] = ok ? src[c] : make_uint4(0u, 0u, 0u, 0u);
}

cudaError_t launch_embed(const __half* table, const int32_t* ids, int n, int d, int vocab, __half* out,
                         uint32_t* status, cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    if (d % 8 != 0) return cudaErrorInvalidValue;
    return launch_k(k_embed, dim3(n), dim3(256), 0, st, table, ids, n, d, vocab, out, status);
}

// dst[c][r] = src[r][c] for r < rows, c < cols (32 x 32 tiles through shared memory)
__global__ void k_transpose_f16(const __half* src, int64_t src_ld, int rows, int cols, __half* dst,
                                int64_t dst_ld) {
    __shared__ __half tile[32][33];
    pdl_wait();
    pdl_launch_dependents();
    const int r0 = blockIdx.y * 32, c0 = blockIdx.x * 32;
    for (int i = threadIdx.y; i < 32; i += blockDim.y) {
        const int r = r0 + i, c = c0 + threadIdx.x;
        if (r < rows && c < cols) tile[i][threadIdx.x] = src[(int64_t)r * src_ld + c];
    }
    __syncthreads();
    for (int i = threadIdx.y; i < 32; i += blockDim.y) {
        const int c = c0 + i, r = r0 + threadIdx.x;
        if (r < rows && c < cols) dst[(int64_t)c * dst_ld + r] = tile[threadIdx.x][i];
    }
}

cudaError_t launch_transpose_f16(const __half* src, int64_t src_ld, int rows, int cols, __half* dst,
                                 int64_t dst_ld, cudaStream_t st) {
    if (rows <= 0 || cols <= 0) return cudaSuccess;
    const dim3 grid((cols + 31) / 32, (rows + 31) / 32), block(32, 8);
    return launch_k(k_transpose_f16, grid, block, 0, st, src, src_ld, rows, cols, dst, dst_ld);
}

__global__ void k_gather_rows(const __half* const* src_rows, __half* dst, int n_rows,
                              int64_t row_len, int64_t dst_stride) {
    pdl_wait();
    pdl_launch_dependents();
    for (int r = blockIdx.x; r < n_rows; r += gridDim.x) {
        const __half* s = src_rows[r];
        __half* d = dst + (int64_t)r * dst_stride;
        for (int64_t c = threadIdx.x; c < row_len; c += blockDim.x) d[c] = s[c];
    }
}

cudaError_t launch_gather_rows(const __half* const* src_rows, __half* dst, int n_rows,
                               int64_t row_len, int64_t dst_stride, cudaStream_t st) {
    if (n_rows <= 0) return cudaSuccess;
    const int blocks = n_rows < 4096 ? n_rows : 4096;
    return launch_k(k_gather_rows, dim3(blocks), dim3(256), 0, st, src_rows, dst, n_rows, row_len,
                    dst_stride);
}

}  // namespace vt

namespace vt {

// Raises a kernel's dynamic shared-memory limit to `want` bytes, capped by the device's
// per-block opt-in limit minus the kernel's static shared memory.
template <typename K>
static cudaError_t allow_smem(K kern, size_t want, bool max_carveout = false) {
    int dev = 0, optin = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    if (e != cudaSuccess) return e;
    cudaFuncAttributes fa{};
    if ((e = cudaFuncGetAttributes(&fa, kern)) != cudaSuccess) return e;
    const size_t cap = (size_t)optin > fa.sharedSizeBytes ? (size_t)optin - fa.sharedSizeBytes : 0;
    if ((e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)(want < cap ? want : cap))) != cudaSuccess)
        return e;
    // The QKV GEMV and the attention kernel that follows it ask for the largest shared-memory
    // carveout: an SM configured that way while the GEMV runs can already host the attention
    // CTAs (and their prefetch of cached K/V) without draining to change its carveout.
    if (!max_carveout) return cudaSuccess;
    return cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout,
                                (int)cudaSharedmemCarveoutMaxShared);
}

cudaError_t init_decode_kernels() {
    cudaError_t e;
#define VT_GEMV_ATTR(EPI)                                                         \
    if ((e = allow_smem(k_gemv<EPI, 1, 8>, 0)) != cudaSuccess) return e;          \
    if ((e = allow_smem(k_gemv<EPI, 2, 4>, 0)) != cudaSuccess) return e;          \
    if ((e = allow_smem(k_gemv<EPI, 3, 2>, 0)) != cudaSuccess) return e;          \
    if ((e = allow_smem(k_gemv<EPI, 4, 2>, 0)) != cudaSuccess) return e;          \
    if ((e = allow_smem(k_gemv<EPI, 8, 1>, 0)) != cudaSuccess) return e;
    VT_GEMV_ATTR(kEpiPlain) VT_GEMV_ATTR(kEpiSwiglu)
#undef VT_GEMV_ATTR
    if ((e = allow_smem(k_gemv<kEpiQkvRope, 1, 8>, 0, true)) != cudaSuccess) return e;
    if ((e = allow_smem(k_gemv<kEpiQkvRope, 2, 4>, 0, true)) != cudaSuccess) return e;
    if ((e = allow_smem(k_gemv<kEpiQkvRope, 3, 2>, 0, true)) != cudaSuccess) return e;
    if ((e = allow_smem(k_gemv<kEpiQkvRope, 4, 2>, 0, true)) != cudaSuccess) return e;
    if ((e = allow_smem(k_gemv<kEpiQkvRope, 8, 1>, 0, true)) != cudaSuccess) return e;
    if ((e = allow_smem(k_combine, 0)) != cudaSuccess) return e;
    if ((e = allow_smem(k_fill_zero_f32, 0)) != cudaSuccess) return e;
    if ((e = allow_smem(k_kv_advance, 0)) != cudaSuccess) return e;
#define VT_FFN_ATTR(CPL, R)                                                                       \
    if ((e = allow_smem(k_ffn<CPL, R, 1>, 1 * kGemvThreads * 32)) != cudaSuccess) return e;       \
    if ((e = allow_smem(k_ffn<CPL, R, 2>, 2 * kGemvThreads * 32)) != cudaSuccess) return e;       \
    if ((e = allow_smem(k_ffn<CPL, R, 3>, 3 * kGemvThreads * 32)) != cudaSuccess) return e;       \
    if ((e = allow_smem(k_ffn<CPL, R, 4>, 4 * kGemvThreads * 32)) != cudaSuccess) return e;       \
    if ((e = allow_smem(k_ffn<CPL, R, 8>, 8 * kGemvThreads * 32)) != cudaSuccess) return e;
    VT_FFN_ATTR(1, 8) VT_FFN_ATTR(2, 4) VT_FFN_ATTR(3, 2) VT_FFN_ATTR(4, 2) VT_FFN_ATTR(8, 1)
#undef VT_FFN_ATTR
#define VT_ATTN_ATTR(DH, G)                                                                       \
    if ((e = allow_smem(k_attn_decode<DH, G>, attn_decode_smem_bytes(DH, G, kAttnMaxStages), true)) != \
        cudaSuccess)                                                                              \
        return e;                                                                                 \
    if ((e = cudaFuncSetAttribute(k_attn_decode<DH, G>,                                           \
                                  cudaFuncAttributeNonPortableClusterSizeAllowed, 1)) != cudaSuccess) \
        return e;
    VT_ATTN_ATTR(64, 1) VT_ATTN_ATTR(64, 2) VT_ATTN_ATTR(64, 4) VT_ATTN_ATTR(64, 8)
    VT_ATTN_ATTR(128, 1) VT_ATTN_ATTR(128, 2) VT_ATTN_ATTR(128, 4) VT_ATTN_ATTR(128, 8)
#undef VT_ATTN_ATTR
    {
        // 16-CTA clusters need the non-portable size; fall back to 8 when none can be scheduled
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(16, 1);
        cfg.blockDim = dim3(kAttnThreads);
        cfg.dynamicSmemBytes = attn_decode_smem_bytes(128, 8, kAttnMaxStages);
        cudaLaunchAttribute at[1];
        at[0].id = cudaLaunchAttributeClusterDimension;
        at[0].val.clusterDim.x = 16;
        at[0].val.clusterDim.y = 1;
        at[0].val.clusterDim.z = 1;
        cfg.attrs = at;
        cfg.numAttrs = 1;
        int nclusters = 0;
        if (cudaOccupancyMaxActiveClusters(&nclusters, k_attn_decode<128, 8>, &cfg) != cudaSuccess ||
            nclusters < 1) {
            cudaGetLastError();
            g_attn_cluster = 8;
        }
    }
    return cudaSuccess;
}

}  // namespace vt
