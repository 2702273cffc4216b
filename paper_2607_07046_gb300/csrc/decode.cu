// Decode-path kernels for one tensor-parallel shard (batch 1), sm_103a.
//
// What they compute (Voltron Section 2.1, per shard as in Section 3.2.1):
//   k_gemv        y = W . v for the shard's rows of a linear layer, with
//                   - an RMSNorm prologue (v = x * g / sqrt(mean(x^2) + eps)) for the QKV and
//                     gate/up projections,
//                   - epilogues: RoPE + KV-cache append (QKV), SwiGLU (gate/up), or a plain fp32
//                     partial (O and down projections, the shard's contribution to the layer).
//   k_attn_decode split-K flash decoding: each CTA scores one slice of the cached positions of one
//                 KV head for all query heads of its group, keeps (max, sum, weighted V) in fp32,
//                 and the last CTA of the head merges the slices with log-sum-exp weights.
//   k_combine     the aggregation on the main device: residual + sum of partials, in shard order.
//
// The GEMV is HBM-bound (one fp16 weight read per two flops); its design notes are at k_gemv.
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include <utility>

#include "device.cuh"
#include "internal.h"

namespace vt {

bool g_use_pdl = true;
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

__device__ __forceinline__ void consumer_bar(int id, int nthreads) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
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

__device__ __forceinline__ uint4 ldg_stream(const void* p) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

// R row partials per lane -> lane l with l % (32 / R) == 0 returns the warp total of row
// l / (32 / R).  Each level halves the values a lane carries: lanes whose bit `o` is set keep the
// upper half and send the lower half to their partner, and vice versa.
template <int R>
__device__ __forceinline__ float multi_row_sum(float (&v)[8], int lane) {
    if constexpr (R == 8) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const bool hi = lane & 16;
            const float send = hi ? v[i] : v[i + 4];
            v[i] = (hi ? v[i + 4] : v[i]) + __shfl_xor_sync(0xffffffffu, send, 16);
        }
    }
    if constexpr (R >= 4) {
        constexpr int o = R == 8 ? 8 : 16;
#pragma unroll
        for (int i = 0; i < 2; ++i) {
            const bool hi = lane & o;
            const float send = hi ? v[i] : v[i + 2];
            v[i] = (hi ? v[i + 2] : v[i]) + __shfl_xor_sync(0xffffffffu, send, o);
        }
    }
    if constexpr (R >= 2) {
        constexpr int o = R == 8 ? 4 : (R == 4 ? 8 : 16);
        const bool hi = lane & o;
        const float send = hi ? v[0] : v[1];
        v[0] = (hi ? v[1] : v[0]) + __shfl_xor_sync(0xffffffffu, send, o);
    }
    constexpr int first = R == 8 ? 2 : (R == 4 ? 4 : (R == 2 ? 8 : 16));
#pragma unroll
    for (int o = first; o >= 1; o >>= 1) v[0] += __shfl_xor_sync(0xffffffffu, v[0], o);
    return v[0];
}

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
    int g = g_num_sms > 0 ? g_num_sms : 148;
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
    if (a.indep) {  // all reads done; complete only after the previous kernel, then publish
        pdl_wait();
        pdl_launch_dependents();
    }
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

size_t attn_decode_smem_bytes(int dh) {
    return (size_t)kAttnStages * kAttnTilePos * dh * 2 * 2 +           // K and V tiles
           (size_t)kAttnWarps * kAttnMaxGroup * (dh + 2) * 4 +         // per-warp states
           2 * kAttnStages * 8 + 128;
}

template <int DH, int G>
__global__ void __launch_bounds__(kAttnThreads) k_attn_decode(const __grid_constant__ AttnDecodeArgs a) {
    extern __shared__ __align__(128) uint8_t smem[];
    constexpr int EPL = DH / 32;  // elements per lane
    constexpr int TILE_BYTES = kAttnTilePos * DH * 2;
    uint8_t* ring = smem;  // stage s: K tile at s*2*TILE_BYTES, V tile after it
    float* wst = reinterpret_cast<float*>(smem + kAttnStages * 2 * TILE_BYTES);
    float* wm = wst;                                   // [warps][G]
    float* wl = wm + kAttnWarps * kAttnMaxGroup;       // [warps][G]
    float* wo = wl + kAttnWarps * kAttnMaxGroup;       // [warps][G][DH]
    uint64_t* full = reinterpret_cast<uint64_t*>(wo + kAttnWarps * kAttnMaxGroup * DH);
    uint64_t* empty = full + kAttnStages;
    __shared__ int s_abort, s_last;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int j = blockIdx.y, c = blockIdx.x;
    // The length was written by a kernel at least two launches back (see device.cuh).
    const int len = *a.len;
    const bool ok = len >= 0 && len < a.cap;
    const int n_pos = ok ? len + 1 : min(max(len, 0), a.cap);
    const int pnew = ok ? len : -1;
    const int chunk = (n_pos + a.nsplit - 1) / a.nsplit;
    const int t0 = min(c * chunk, n_pos), t1 = min(n_pos, t0 + chunk);
    const int old_end = pnew >= 0 ? min(t1, pnew) : t1;
    const int n_old = max(old_end - t0, 0);
    const int ntiles = (n_old + kAttnTilePos - 1) / kAttnTilePos;
    const __half* kbase = a.kcache + (int64_t)j * a.cap * DH;
    const __half* vbase = a.vcache + (int64_t)j * a.cap * DH;

    if (tid == 0) {
        for (int s = 0; s < kAttnStages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], kAttnWarps);
        }
        s_abort = 0;
        fence_mbar_init();
    }
    __syncthreads();

    if (warp == kAttnWarps) {
        if (lane == 0) {
            int last_issued[kAttnStages];
            for (int s = 0; s < kAttnStages; ++s) last_issued[s] = -1;
            for (int t = 0; t < ntiles; ++t) {
                const int s = t % kAttnStages;
                if (t >= kAttnStages && !mbar_wait(&empty[s], ((t / kAttnStages) - 1) & 1)) {
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
                last_issued[s] = t;
            }
            for (int s = 0; s < kAttnStages; ++s)
                if (last_issued[s] >= 0 && !mbar_wait(&full[s], (last_issued[s] / kAttnStages) & 1))
                    set_status(a.status, VT_DEV_WAIT_TIMEOUT);
        }
        return;
    }

    constexpr int NC = kAttnWarps * 32;
    pdl_wait();
    float q[G][EPL];
#pragma unroll
    for (int h = 0; h < G; ++h)
#pragma unroll
        for (int e = 0; e < EPL; ++e) q[h][e] = a.q[(j * G + h) * DH + lane * EPL + e];
    pdl_launch_dependents();

    float m[G], l[G], o[G][EPL];
#pragma unroll
    for (int h = 0; h < G; ++h) {
        m[h] = -INFINITY;
        l[h] = 0.f;
#pragma unroll
        for (int e = 0; e < EPL; ++e) o[h][e] = 0.f;
    }
    // online softmax update with one cached position (kv, vv: this lane's EPL elements)
    auto update = [&](const float (&kv)[EPL], const float (&vv)[EPL]) {
#pragma unroll
        for (int h = 0; h < G; ++h) {
            float s = 0.f;
#pragma unroll
            for (int e = 0; e < EPL; ++e) s = fmaf(q[h][e], kv[e], s);
            s = warp_sum(s) * a.scale_log2;
            const float mn = fmaxf(m[h], s);
            const float corr = exp2f(m[h] - mn);
            const float p = exp2f(s - mn);
            l[h] = l[h] * corr + p;
#pragma unroll
            for (int e = 0; e < EPL; ++e) o[h][e] = fmaf(o[h][e], corr, p * vv[e]);
            m[h] = mn;
        }
    };
    auto load_lane = [&](const __half* row, float (&dst)[EPL]) {
        if constexpr (EPL == 4) {
            const uint2 u = *reinterpret_cast<const uint2*>(row + lane * 4);
            const float2 t0 = h2_to_f2(u.x), t1 = h2_to_f2(u.y);
            dst[0] = t0.x; dst[1] = t0.y; dst[2] = t1.x; dst[3] = t1.y;
        } else {
            const float2 t0 = h2_to_f2(*reinterpret_cast<const uint32_t*>(row + lane * 2));
            dst[0] = t0.x; dst[1] = t0.y;
        }
    };

    bool aborted = false;
    for (int t = 0; t < ntiles; ++t) {
        const int s = t % kAttnStages;
        if (!mbar_wait(&full[s], (t / kAttnStages) & 1)) {
            s_abort = 1;
            aborted = true;
            set_status(a.status, VT_DEV_WAIT_TIMEOUT);
            break;
        }
        const int np = min(kAttnTilePos, old_end - (t0 + t * kAttnTilePos));
        const __half* kt = reinterpret_cast<const __half*>(ring + s * 2 * TILE_BYTES);
        const __half* vt = reinterpret_cast<const __half*>(ring + s * 2 * TILE_BYTES + TILE_BYTES);
        for (int pl = warp; pl < np; pl += kAttnWarps) {
            float kv[EPL], vv[EPL];
            load_lane(kt + pl * DH, kv);
            load_lane(vt + pl * DH, vv);
            update(kv, vv);
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty[s]);
    }
    // the token appended by the preceding QKV kernel: read through L2 (never cached in L1 here)
    if (!aborted && warp == 0 && pnew >= t0 && pnew < t1) {
        float kv[EPL], vv[EPL];
#pragma unroll
        for (int e = 0; e < EPL; ++e) {
            kv[e] = __half2float(__ldcg(kbase + (int64_t)pnew * DH + lane * EPL + e));
            vv[e] = __half2float(__ldcg(vbase + (int64_t)pnew * DH + lane * EPL + e));
        }
        update(kv, vv);
    }
    // merge the four warps' states (fixed order)
#pragma unroll
    for (int h = 0; h < G; ++h) {
        if (lane == 0) {
            wm[warp * kAttnMaxGroup + h] = m[h];
            wl[warp * kAttnMaxGroup + h] = l[h];
        }
#pragma unroll
        for (int e = 0; e < EPL; ++e) wo[(warp * kAttnMaxGroup + h) * DH + lane * EPL + e] = o[h][e];
    }
    consumer_bar(1, NC);
    // An aborted CTA still writes an empty slice and takes its ticket, so the merge stays in step.
    const bool dead = s_abort != 0;
    for (int idx = tid; idx < G * DH; idx += NC) {
        const int h = idx / DH, d = idx - h * DH;
        float M = -INFINITY;
        if (!dead)
            for (int w = 0; w < kAttnWarps; ++w) M = fmaxf(M, wm[w * kAttnMaxGroup + h]);
        float L = 0.f, O = 0.f;
        if (M != -INFINITY) {
            for (int w = 0; w < kAttnWarps; ++w) {
                const float f = exp2f(wm[w * kAttnMaxGroup + h] - M);
                L += wl[w * kAttnMaxGroup + h] * f;
                O += wo[(w * kAttnMaxGroup + h) * DH + d] * f;
            }
        }
        const int hl = j * G + h;
        a.part_o[((int64_t)hl * a.nsplit + c) * DH + d] = O;
        if (d == 0) {
            a.part_ml[((int64_t)hl * a.nsplit + c) * 2 + 0] = M;
            a.part_ml[((int64_t)hl * a.nsplit + c) * 2 + 1] = L;
        }
    }
    __threadfence();
    consumer_bar(1, NC);
    if (tid == 0) {
        const int old = atomicAdd(&a.tickets[j], 1);
        s_last = (old == a.nsplit - 1);
    }
    consumer_bar(1, NC);
    if (!s_last) return;
    __threadfence();
    // Merge the nsplit slices of the group's heads.  Slice weights exp2(m_c - M) / L are computed
    // once per (head, slice) into shared memory (the tile ring is free by now), then every
    // (head, dim) output is a weighted sum over the slices.
    float* wts = reinterpret_cast<float*>(ring);  // [G][nsplit]
    for (int h = warp; h < G; h += kAttnWarps) {
        const float* ml = a.part_ml + (int64_t)(j * G + h) * a.nsplit * 2;
        float M = -INFINITY;
        for (int cc = lane; cc < a.nsplit; cc += 32) M = fmaxf(M, __ldcg(ml + 2 * cc));
        M = warp_max(M);
        float L = 0.f;
        for (int cc = lane; cc < a.nsplit; cc += 32) {
            const float mc = __ldcg(ml + 2 * cc);
            const float f = mc == -INFINITY ? 0.f : exp2f(mc - M);
            wts[h * a.nsplit + cc] = f;
            L += __ldcg(ml + 2 * cc + 1) * f;
        }
        L = warp_sum(L);
        const float inv = L > 0.f ? 1.0f / L : 0.f;
        __syncwarp();
        for (int cc = lane; cc < a.nsplit; cc += 32) wts[h * a.nsplit + cc] *= inv;
    }
    consumer_bar(1, NC);
    for (int idx = tid; idx < G * DH; idx += NC) {
        const int h = idx / DH, d = idx - h * DH;
        const int hl = j * G + h;
        const float* po = a.part_o + (int64_t)hl * a.nsplit * DH + d;
        const float* w = wts + h * a.nsplit;
        float O0 = 0.f, O1 = 0.f, O2 = 0.f, O3 = 0.f;
        int cc = 0;
        for (; cc + 4 <= a.nsplit; cc += 4) {
            O0 += w[cc] * __ldcg(po + (int64_t)cc * DH);
            O1 += w[cc + 1] * __ldcg(po + (int64_t)(cc + 1) * DH);
            O2 += w[cc + 2] * __ldcg(po + (int64_t)(cc + 2) * DH);
            O3 += w[cc + 3] * __ldcg(po + (int64_t)(cc + 3) * DH);
        }
        for (; cc < a.nsplit; ++cc) O0 += w[cc] * __ldcg(po + (int64_t)cc * DH);
        a.out[hl * DH + d] = (O0 + O1) + (O2 + O3);
    }
    if (tid == 0) a.tickets[j] = 0;
}

template <int DH>
static cudaError_t launch_attn_dh(const AttnDecodeArgs& a, cudaStream_t st) {
    const dim3 grid(a.nsplit, a.hk), block(kAttnThreads);
    const size_t smem = attn_decode_smem_bytes(DH);
    switch (a.group) {
        case 1: return launch_k(k_attn_decode<DH, 1>, grid, block, smem, st, a);
        case 2: return launch_k(k_attn_decode<DH, 2>, grid, block, smem, st, a);
        case 4: return launch_k(k_attn_decode<DH, 4>, grid, block, smem, st, a);
        case 8: return launch_k(k_attn_decode<DH, 8>, grid, block, smem, st, a);
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

__global__ void k_combine(const __grid_constant__ CombineArgs a) {
    pdl_wait();
    pdl_launch_dependents();
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < a.count; e += stride) {
        float acc = a.residual ? __half2float(a.residual[e]) : 0.f;
        for (int s = 0; s < a.n; ++s) acc += a.parts[s][e];
        a.out[e] = __float2half_rn(acc);
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

__global__ void k_kv_advance(int32_t* len, int first, int count, int delta) {
    pdl_wait();
    pdl_launch_dependents();
    for (int i = threadIdx.x; i < count; i += blockDim.x) len[first + i] += delta;
}

cudaError_t launch_kv_advance(int32_t* len, int first, int count, int delta, cudaStream_t st) {
    return launch_k(k_kv_advance, dim3(1), dim3(128), 0, st, len, first, count, delta);
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

__global__ void k_embed(const __half* table, const int32_t* ids, int n, int d, int vocab,
                        __half* out) {
    pdl_wait();
    pdl_launch_dependents();
    const int row = blockIdx.x;
    if (row >= n) return;
    const int id = ids[row];
    const bool ok = id >= 0 && id < vocab;
    for (int c = threadIdx.x; c < d; c += blockDim.x)
        out[(int64_t)row * d + c] = ok ? table[(int64_t)id * d + c] : __float2half(0.f);
}

cudaError_t launch_embed(const __half* table, const int32_t* ids, int n, int d, int vocab,
                         __half* out, cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    return launch_k(k_embed, dim3(n), dim3(256), 0, st, table, ids, n, d, vocab, out);
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
static cudaError_t allow_smem(K kern, size_t want) {
    int dev = 0, optin = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    if (e != cudaSuccess) return e;
    cudaFuncAttributes fa{};
    if ((e = cudaFuncGetAttributes(&fa, kern)) != cudaSuccess) return e;
    const size_t cap = (size_t)optin > fa.sharedSizeBytes ? (size_t)optin - fa.sharedSizeBytes : 0;
    return cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)(want < cap ? want : cap));
}

cudaError_t init_decode_kernels() {
    cudaError_t e;
#define VT_ATTN_ATTR(DH, G) \
    if ((e = allow_smem(k_attn_decode<DH, G>, attn_decode_smem_bytes(DH))) != cudaSuccess) return e;
    VT_ATTN_ATTR(64, 1) VT_ATTN_ATTR(64, 2) VT_ATTN_ATTR(64, 4) VT_ATTN_ATTR(64, 8)
    VT_ATTN_ATTR(128, 1) VT_ATTN_ATTR(128, 2) VT_ATTN_ATTR(128, 4) VT_ATTN_ATTR(128, 8)
#undef VT_ATTN_ATTR
    return cudaSuccess;
}

}  // namespace vt
