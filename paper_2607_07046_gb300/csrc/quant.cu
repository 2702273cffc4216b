// Block-quantized (INT8 / INT4) shard weights for decode: the host quantizer and packer, and the
// dequantizing matrix-vector kernel, sm_103a.
//
// What they compute (Voltron Section 3.2.2, precision heterogeneity: a device may hold its shard
// at a reduced precision; Section 4.2.2 allocates precisions per layer; Section 5.1 names k-quant
// formats without defining them).  Format: each weight row is cut into blocks of 32 consecutive
// weights along the input axis; a block keeps the fp16 scale d = fp16(amax / qmax) (qmax 127 for
// 8 bits, 7 for 4 bits) and every weight the code q = round-half-even(w / d) clamped to
// [-qmax, qmax] (0 when d = 0), both divisions in fp32.  A projection is y = sum_e (q_e d) x_e.
//
// The kernel streams the codes with 16-byte loads and rebuilds each code as an fp32 integer with
// one byte permute (0x4B000000 | u is the float 2^23 + u, u the biased code) and one subtraction,
// then multiplies with the input in fp32 pairs (packed f32x2 arithmetic, two lanes of the FMA
// pipe per instruction).  The bias is removed once per chunk: sum_e u_e x_e - bias * sum_e x_e,
// with the input's chunk sums computed once per CTA.  Decode at batch 1 is bound by HBM, and this
// keeps the CUDA-core work per byte low enough for 8-bit codes (2 instructions per code) and close
// enough for 4-bit codes.
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include <algorithm>
#include <cmath>

#include "device.cuh"
#include "internal.h"

namespace vt {

// ================================================================== host: quantizer and packer

void quantize_rows_host(const __half* w, int64_t rows, int64_t k, int bits, int block, int8_t* q, __half* scales) {
    const int qmax = bits == 8 ? 127 : 7;
    const int64_t nb = (k + block - 1) / block;
    for (int64_t r = 0; r < rows; ++r)
        for (int64_t b = 0; b < nb; ++b) {
            const int64_t e0 = b * block, e1 = std::min(k, e0 + block);
            float amax = 0.0f;
            for (int64_t e = e0; e < e1; ++e) amax = std::max(amax, std::fabs(__half2float(w[r * k + e])));
            const __half d16 = __float2half_rn(amax / (float)qmax);  // fp32 division, one rounding to fp16
            const float d = __half2float(d16);
            scales[r * nb + b] = d16;
            for (int64_t e = e0; e < e1; ++e) {
                int c = 0;
                if (d != 0.0f) {
                    const float x = std::nearbyint(__half2float(w[r * k + e]) / d);  // fp32 division, ties to even
                    c = x > (float)qmax ? qmax : (x < (float)-qmax ? -qmax : (int)x);
                }
                q[r * k + e] = (int8_t)c;
            }
        }
}

static int64_t qmat_nb(int64_t k) { return (k + kQBlock - 1) / kQBlock; }

size_t qmat_code_bytes(int64_t rows, int64_t k, int bits) {
    return (size_t)rows * (size_t)qmat_nb(k) * (bits == 8 ? 32 : 16);
}

size_t qmat_scale_bytes(int64_t rows, int64_t k) { return (size_t)rows * (size_t)qmat_nb(k) * 2; }

void unpack_qcodes(const uint8_t* codes, int64_t rows, int64_t k, int bits, int8_t* q) {
    const int64_t nb = qmat_nb(k);
    const int64_t rb = nb * (bits == 8 ? 32 : 16);
    for (int64_t r = 0; r < rows; ++r) {
        const uint8_t* row = codes + r * rb;
        for (int64_t e = 0; e < k; ++e) {
            int u;
            if (bits == 8) {
                u = row[e] - 128;
            } else {
                const int64_t g = e / 8, i = e % 8;
                const uint8_t byte = row[g * 4 + (i & 3)];
                u = (i < 4 ? (byte & 15) : (byte >> 4)) - 8;
            }
            q[r * k + e] = (int8_t)u;
        }
    }
}

// ================================================================== device: dequantizing GEMV
//
// Geometry.  A warp takes groups of kQRows consecutive rows; the 16-byte chunks of a row (16
// codes at 8 bits, one block of 32 at 4 bits) are spread over the lanes (chunk 32 i + lane), so
// every load instruction of the warp reads 512 contiguous bytes of one row, and the input values
// of a chunk (from shared memory) serve all kQRows rows.  Row partials are reduced across the
// warp with the multi-row butterfly; a CTA owns a contiguous range of row groups.  The next
// step's codes and scales are loaded while the current step computes (two register buffers), and
// the first two steps are issued before griddepcontrol.wait: the weights do not depend on the
// preceding kernel.
constexpr int kQWarps = 8;
constexpr int kQThreads = kQWarps * 32;
constexpr int kQRows = 8;

__device__ __forceinline__ float2 codes_f2(uint32_t u, int b0) {
    // bytes b0, b0 + 1 of u as the floats 2^23 + byte, then minus 2^23: the byte's value, exactly
    const float2 f = make_float2(__int_as_float((int)__byte_perm(u, 0x4B000000u, 0x7540u + (unsigned)b0)),
                                 __int_as_float((int)__byte_perm(u, 0x4B000000u, 0x7541u + (unsigned)b0)));
    return __fadd2_rn(f, make_float2(-8388608.0f, -8388608.0f));
}

// sum over the chunk's codes of (biased code) * x; x: the chunk's input values in shared memory
template <int BITS>
__device__ __forceinline__ float chunk_dot(const uint4& c, const float* x) {
    const uint32_t w[4] = {c.x, c.y, c.z, c.w};
    float2 s0 = make_float2(0.f, 0.f), s1 = make_float2(0.f, 0.f);
    if constexpr (BITS == 8) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float4 xv = *reinterpret_cast<const float4*>(x + 4 * i);
            s0 = __ffma2_rn(codes_f2(w[i], 0), make_float2(xv.x, xv.y), s0);
            s1 = __ffma2_rn(codes_f2(w[i], 2), make_float2(xv.z, xv.w), s1);
        }
    } else {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const uint32_t lo = w[i] & 0x0F0F0F0Fu, hi = (w[i] >> 4) & 0x0F0F0F0Fu;
            const float4 xa = *reinterpret_cast<const float4*>(x + 8 * i);
            const float4 xb = *reinterpret_cast<const float4*>(x + 8 * i + 4);
            s0 = __ffma2_rn(codes_f2(lo, 0), make_float2(xa.x, xa.y), s0);
            s1 = __ffma2_rn(codes_f2(lo, 2), make_float2(xa.z, xa.w), s1);
            s0 = __ffma2_rn(codes_f2(hi, 0), make_float2(xb.x, xb.y), s0);
            s1 = __ffma2_rn(codes_f2(hi, 2), make_float2(xb.z, xb.w), s1);
        }
    }
    return (s0.x + s0.y) + (s1.x + s1.y);
}

template <int EPI, int BITS>
__global__ void __launch_bounds__(kQThreads) k_gemv_q(const __grid_constant__ QGemvArgs a) {
    constexpr int CPC = BITS == 8 ? 16 : 32;  // codes per 16-byte chunk
    constexpr float BIAS = BITS == 8 ? 128.f : 8.f;
    extern __shared__ __align__(16) float qsm[];
    __shared__ float red[kQWarps + 1];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const QMatDev& W = a.w;
    const int kp = W.nb * kQBlock;                 // padded row length of the input
    const int nch = (int)(W.row_bytes >> 4);       // chunks per row
    float* xs = qsm;                               // [kp] input (zero past k)
    float* cs = qsm + kp;                          // [nch] input sum of each chunk
    const int ngroups = (W.rows + kQRows - 1) / kQRows;
    const int g0 = (int)(((int64_t)blockIdx.x * ngroups) / gridDim.x);
    const int g1 = (int)(((int64_t)(blockIdx.x + 1) * ngroups) / gridDim.x);
    const int nbi = (nch + 31) / 32;               // chunk rounds per row
    const int my_groups = g1 - g0 > warp ? (g1 - g0 - warp + kQWarps - 1) / kQWarps : 0;
    const int n_steps = my_groups * nbi;

    auto load = [&](uint4 (&b)[kQRows], __half (&d)[kQRows], int s) {
        const int gi = s / nbi, bi = s - gi * nbi;
        const int row0 = (g0 + warp + kQWarps * gi) * kQRows, ch = bi * 32 + lane;
        const bool on = s < n_steps && ch < nch;
        const int sidx = BITS == 8 ? ch >> 1 : ch;
#pragma unroll
        for (int r = 0; r < kQRows; ++r) {
            const bool ok = on && row0 + r < W.rows;
            b[r] = ok ? ldg_stream(W.codes + (int64_t)(row0 + r) * W.row_bytes + (int64_t)ch * 16) : make_uint4(0u, 0u, 0u, 0u);
            d[r] = ok ? W.scales[(int64_t)(row0 + r) * W.nb + sidx] : __float2half(0.f);
        }
    };
    uint4 b0[kQRows], b1[kQRows];
    __half d0[kQRows], d1[kQRows];
    load(b0, d0, 0);
    load(b1, d1, 1);
    pdl_wait();

    // ---------------------------------------------------------------- input into shared memory
    if (a.x != nullptr) {
        float ss = 0.f;
        for (int i = tid; i < W.k; i += kQThreads) {
            const float v = __half2float(a.x[i]);
            ss = fmaf(v, v, ss);
        }
        ss = warp_sum(ss);
        if (lane == 0) red[warp] = ss;
        __syncthreads();
        if (tid == 0) {
            float tot = 0.f;
            for (int w = 0; w < kQWarps; ++w) tot += red[w];
            red[kQWarps] = 1.0f / sqrtf(tot / (float)W.k + a.eps);
        }
        __syncthreads();
        const float rinv = red[kQWarps];
        for (int i = tid; i < kp; i += kQThreads)
            xs[i] = i < W.k ? __half2float(a.x[i]) * rinv * __half2float(a.gain[i]) : 0.f;
    } else {
        for (int i = tid; i < kp; i += kQThreads) xs[i] = i < W.k ? __ldcg(a.vin + i) : 0.f;
    }
    __syncthreads();
    for (int c = tid; c < nch; c += kQThreads) {
        float t = 0.f;
        for (int e = 0; e < CPC; ++e) t += xs[c * CPC + e];
        cs[c] = t;
    }
    __syncthreads();
    pdl_launch_dependents();

    float acc[kQRows];
    auto consume = [&](const uint4 (&b)[kQRows], const __half (&d)[kQRows], int s) {
        const int gi = s / nbi, bi = s - gi * nbi;
        const int row0 = (g0 + warp + kQWarps * gi) * kQRows, ch = bi * 32 + lane;
        if (bi == 0)
#pragma unroll
            for (int r = 0; r < kQRows; ++r) acc[r] = 0.f;
        if (ch < nch) {
            const float* x = xs + ch * CPC;
            const float bsum = BIAS * cs[ch];
#pragma unroll
            for (int r = 0; r < kQRows; ++r) acc[r] = fmaf(__half2float(d[r]), chunk_dot<BITS>(b[r], x) - bsum, acc[r]);
        }
        if (bi == nbi - 1) {
            float v[8];
#pragma unroll
            for (int r = 0; r < kQRows; ++r) v[r] = acc[r];
            const float t = multi_row_sum<kQRows>(v, lane);  // lane 4 r holds row row0 + r
            const float t_odd = __shfl_down_sync(0xffffffffu, t, 4);  // the next row's total
            const int r = lane >> 2, row = row0 + r;
            if ((lane & 3) == 0 && row < W.rows) {
                if constexpr (EPI == kEpiPlain) {
                    a.out[row] = t;
                } else if ((r & 1) == 0 && row + 1 < W.rows) {
                    if constexpr (EPI == kEpiSwiglu) {
                        a.out[row >> 1] = silu(t) * t_odd;
                    } else {  // kEpiQkvRope: rows (row, row + 1) are the RoPE pair (i, i + dh / 2)
                        const int p = *a.len;
                        const bool ok = p >= 0 && p < a.cap;
                        if (!ok && row == 0) set_status(a.status, VT_DEV_KV_OVERFLOW);
                        const int half = a.dh >> 1;
                        const int blk = row / a.dh, i = (row - blk * a.dh) >> 1;
                        if (blk < a.hq + a.hk) {
                            const float2 cs2 = ok ? a.rope[(int64_t)p * half + i] : make_float2(1.f, 0.f);
                            const float re = t * cs2.x - t_odd * cs2.y;
                            const float ro = t * cs2.y + t_odd * cs2.x;
                            if (blk < a.hq) {
                                a.out[blk * a.dh + i] = re;
                                a.out[blk * a.dh + i + half] = ro;
                            } else if (ok) {
                                __half* kd = a.kcache + ((int64_t)(blk - a.hq) * a.cap + p) * a.dh;
                                kd[i] = __float2half_rn(re);
                                kd[i + half] = __float2half_rn(ro);
                            }
                        } else if (ok) {
                            __half* vd = a.vcache + ((int64_t)(blk - a.hq - a.hk) * a.cap + p) * a.dh;
                            vd[i] = __float2half_rn(t);
                            vd[i + half] = __float2half_rn(t_odd);
                        }
                    }
                }
            }
        }
    };
    for (int s = 0; s < n_steps; s += 2) {
        consume(b0, d0, s);
        load(b0, d0, s + 2);
        if (s + 1 < n_steps) {
            consume(b1, d1, s + 1);
            load(b1, d1, s + 3);
        }
    }
}

// ================================================================== device: quantizer
//
// One thread per block of 32 weights of a row: the fp16 scale and the biased codes of the format
// above, packed into the kernel layout.  Every decision is the host quantizer's: IEEE fp32
// division (amax / qmax and w / d), one rounding of the scale to fp16, round-half-even of w / d,
// so the codes equal those of vt_quantize_rows bit for bit.
template <int BITS>
__global__ void k_quantize_rows(const __half* __restrict__ w, int64_t ld, int rows, int k, int nb,
                                uint8_t* __restrict__ codes, int64_t row_bytes, __half* __restrict__ scales) {
    constexpr int QMAX = BITS == 8 ? 127 : 7, BIAS = BITS == 8 ? 128 : 8;
    const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (t >= (int64_t)rows * nb) return;
    const int r = (int)(t / nb), b = (int)(t - (int64_t)r * nb);
    const __half* src = w + (int64_t)r * ld + (int64_t)b * kQBlock;
    const int n = min(kQBlock, k - b * kQBlock);
    float amax = 0.f;
    for (int e = 0; e < n; ++e) amax = fmaxf(amax, fabsf(__half2float(src[e])));
    const __half d16 = __float2half_rn(amax / (float)QMAX);
    const float d = __half2float(d16);
    scales[(int64_t)r * nb + b] = d16;
    uint32_t u[kQBlock];
#pragma unroll
    for (int e = 0; e < kQBlock; ++e) {
        int c = 0;
        if (e < n && d != 0.f) {
            const float x = rintf(__half2float(src[e]) / d);
            c = x > (float)QMAX ? QMAX : (x < (float)-QMAX ? -QMAX : (int)x);
        }
        u[e] = (uint32_t)(c + BIAS);
    }
    uint8_t* dst = codes + (int64_t)r * row_bytes + (int64_t)b * (BITS == 8 ? 32 : 16);
    if constexpr (BITS == 8) {
        uint32_t wd[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) wd[i] = u[4 * i] | (u[4 * i + 1] << 8) | (u[4 * i + 2] << 16) | (u[4 * i + 3] << 24);
        reinterpret_cast<uint4*>(dst)[0] = make_uint4(wd[0], wd[1], wd[2], wd[3]);
        reinterpret_cast<uint4*>(dst)[1] = make_uint4(wd[4], wd[5], wd[6], wd[7]);
    } else {
        uint32_t wd[4];
#pragma unroll
        for (int g = 0; g < 4; ++g) {
            uint32_t v = 0;
#pragma unroll
            for (int i = 0; i < 4; ++i) v |= ((u[8 * g + i] & 15u) | ((u[8 * g + i + 4] & 15u) << 4)) << (8 * i);
            wd[g] = v;
        }
        *reinterpret_cast<uint4*>(dst) = make_uint4(wd[0], wd[1], wd[2], wd[3]);
    }
}

cudaError_t launch_quantize_rows(const __half* w, int64_t ld, const QMatDev& m, cudaStream_t st) {
    const int64_t n = (int64_t)m.rows * m.nb;
    if (n <= 0) return cudaSuccess;
    const int threads = 128;
    const unsigned blocks = (unsigned)((n + threads - 1) / threads);
    if (m.bits == 8)
        k_quantize_rows<8><<<blocks, threads, 0, st>>>(w, ld, m.rows, m.k, m.nb, m.codes, m.row_bytes, m.scales);
    else if (m.bits == 4)
        k_quantize_rows<4><<<blocks, threads, 0, st>>>(w, ld, m.rows, m.k, m.nb, m.codes, m.row_bytes, m.scales);
    else
        return cudaErrorInvalidValue;
    return cudaGetLastError();
}

template <int EPI>
static cudaError_t launch_q_epi(const QGemvArgs& a, cudaStream_t st) {
    const int ngroups = (a.w.rows + kQRows - 1) / kQRows;
    int grid = (g_num_sms > 0 ? g_num_sms : 148) * 2;
    grid = std::min(grid, std::max(ngroups, 1));
    const size_t smem = ((size_t)a.w.nb * kQBlock + (size_t)(a.w.row_bytes >> 4)) * sizeof(float);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kQThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = g_use_pdl ? 1 : 0;
    if (a.w.bits == 8) return cudaLaunchKernelEx(&cfg, k_gemv_q<EPI, 8>, a);
    if (a.w.bits == 4) return cudaLaunchKernelEx(&cfg, k_gemv_q<EPI, 4>, a);
    return cudaErrorInvalidValue;
}

cudaError_t launch_gemv_q(int epi, const QGemvArgs& a, cudaStream_t st) {
    if (a.w.rows <= 0) return cudaSuccess;
    const size_t smem = ((size_t)a.w.nb * kQBlock + (size_t)(a.w.row_bytes >> 4)) * sizeof(float);
    if (smem > 200 * 1024) return cudaErrorInvalidValue;
    switch (epi) {
        case kEpiPlain: return launch_q_epi<kEpiPlain>(a, st);
        case kEpiSwiglu: return launch_q_epi<kEpiSwiglu>(a, st);
        case kEpiQkvRope: return launch_q_epi<kEpiQkvRope>(a, st);
        default: return cudaErrorInvalidValue;
    }
}

// ================================================================== quantized shard partials
//
// Communication scaling (Voltron Section 4.3.2): the activations sent between devices are lowered
// to 8 or 4 bits.  Under tensor parallelism those are the fp32 shard partials sent to the main
// device.  Format: blocks of 32 values, fp16 scale d = fp16(amax / qmax) and codes
// round-half-even(x / d) clamped to [-qmax, qmax], fp32 decisions (the oracle's vector format);
// stored as one int8 per value (8 bits) or two per byte (4 bits: value 2 i in the low nibble and
// 2 i + 1 in the high nibble, each as q + 8).

// One thread per block of 32 values.  clear: zero the partial after reading it (the partials of the
// whole-token path are accumulated into zeroed buffers).
template <int BITS>
__global__ void k_quantize_vec(float* __restrict__ x, int64_t n, uint8_t* __restrict__ codes, __half* __restrict__ scales,
                               int clear) {
    constexpr int QMAX = BITS == 8 ? 127 : 7;
    pdl_wait();
    const int64_t b = (int64_t)blockIdx.x * blockDim.x + threadIdx.x, nb = (n + kQBlock - 1) / kQBlock;
    if (b < nb) {
        const int64_t e0 = b * kQBlock;
        const int m = (int)(n - e0 < (int64_t)kQBlock ? n - e0 : (int64_t)kQBlock);
        float v[kQBlock];
        float amax = 0.f;
#pragma unroll
        for (int e = 0; e < kQBlock; ++e) {
            v[e] = e < m ? x[e0 + e] : 0.f;
            amax = fmaxf(amax, fabsf(v[e]));
        }
        const __half d16 = __float2half_rn(amax / (float)QMAX);
        const float d = __half2float(d16);
        scales[b] = d16;
        int q[kQBlock];
#pragma unroll
        for (int e = 0; e < kQBlock; ++e) {
            int c = 0;
            if (d != 0.f) {
                const float r = rintf(v[e] / d);
                c = r > (float)QMAX ? QMAX : (r < (float)-QMAX ? -QMAX : (int)r);
            }
            q[e] = c;
        }
        if constexpr (BITS == 8) {
            for (int e = 0; e < m; ++e) codes[e0 + e] = (uint8_t)(int8_t)q[e];
        } else {
            for (int e = 0; e < m; e += 2) {
                const uint32_t lo = (uint32_t)(q[e] + 8), hi = e + 1 < m ? (uint32_t)(q[e + 1] + 8) : 8u;
                codes[(e0 + e) >> 1] = (uint8_t)(lo | (hi << 4));
            }
        }
        if (clear)
            for (int e = 0; e < m; ++e) x[e0 + e] = 0.f;
    }
    pdl_launch_dependents();
}

cudaError_t launch_quantize_vec(float* x, int64_t n, int bits, uint8_t* codes, __half* scales, int clear,
                                cudaStream_t st) {
    const int64_t nb = (n + kQBlock - 1) / kQBlock;
    if (nb <= 0) return cudaSuccess;
    const unsigned grid = (unsigned)((nb + 127) / 128);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(128);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = g_use_pdl ? 1 : 0;
    if (bits == 8) return cudaLaunchKernelEx(&cfg, k_quantize_vec<8>, x, n, codes, scales, clear);
    if (bits == 4) return cudaLaunchKernelEx(&cfg, k_quantize_vec<4>, x, n, codes, scales, clear);
    return cudaErrorInvalidValue;
}

// out[e] = fp16(residual[e] + sum_s p_s[e]) with shards in order, fp32: p_s is the fp32 partial
// (bits 16; zeroed after reading when clear is set) or the dequantized code q_s[e] d_s[e / 32].
__global__ void k_combine_q(const __grid_constant__ CombineQArgs a) {
    pdl_wait();
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < a.count; e += (int64_t)gridDim.x * blockDim.x) {
        float acc = a.residual ? __half2float(a.residual[e]) : 0.f;
        for (int s = 0; s < a.n; ++s) {
            const int bits = a.bits[s];
            if (bits == 16) {
                acc += __ldcg(a.fparts[s] + e);
                if (a.clear) a.fparts[s][e] = 0.f;
                continue;
            }
            int q;
            if (bits == 8) {
                q = (int)(int8_t)a.codes[s][e];
            } else {
                const uint8_t byte = a.codes[s][e >> 1];
                q = (int)((e & 1) ? (byte >> 4) : (byte & 15)) - 8;
            }
            acc = fmaf((float)q, __half2float(a.scales[s][e / kQBlock]), acc);
        }
        a.out[e] = __float2half_rn(acc);
    }
    pdl_launch_dependents();
}

cudaError_t launch_combine_q(const CombineQArgs& a, cudaStream_t st) {
    if (a.count <= 0) return cudaSuccess;
    const int64_t blocks = std::min<int64_t>((a.count + 255) / 256, (int64_t)(g_num_sms > 0 ? g_num_sms : 148) * 8);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)blocks);
    cfg.blockDim = dim3(256);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = g_use_pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, k_combine_q, a);
}

cudaError_t init_quant_kernels() {
    const int lim = 200 * 1024;
    cudaError_t e;
#define VT_Q_ATTR(EPI)                                                                                            \
    if ((e = cudaFuncSetAttribute(k_gemv_q<EPI, 8>, cudaFuncAttributeMaxDynamicSharedMemorySize, lim)) != cudaSuccess) \
        return e;                                                                                                 \
    if ((e = cudaFuncSetAttribute(k_gemv_q<EPI, 4>, cudaFuncAttributeMaxDynamicSharedMemorySize, lim)) != cudaSuccess) \
        return e;
    VT_Q_ATTR(kEpiPlain)
    VT_Q_ATTR(kEpiSwiglu)
    VT_Q_ATTR(kEpiQkvRope)
#undef VT_Q_ATTR
    return cudaSuccess;
}

}  // namespace vt
