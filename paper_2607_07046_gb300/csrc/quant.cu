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
// The kernel keeps the codes as integers and multiplies them on the tensor cores (integer MMA
// against an exact three-digit int8 split of the input), so the work per code is a small fraction
// of an instruction and the GEMV streams at the memory rate (details at the kernel).
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
// Integer tensor-core GEMV.  Decode at batch 1 is bound by HBM only if the work per weight code
// stays far below one instruction; rebuilding codes as floats costs more than that.  So the codes
// stay integers and go to `mma.sync m16n8k32` (u8 codes x s8 input, s32 accumulate), one MMA per
// block of 32 weights of 16 rows:
//   - the input x^ (fp32) of block b is split into three int8 digits at scales s, s / 254 and
//     s / 254^2 (s = max|x^| / 127 over the block), which reproduce it to 2^-24 of the block's
//     largest value; the digits are the MMA's B columns 0, 1, 2, so one MMA gives all three
//     integer dot products of each row with the block;
//   - the code bias leaves in integers: sum (u - bias) q = D - bias * Q, Q = sum q over the block;
//   - a row's block term is s * (D1 - bias Q1) + s / 254 * (D2 - ...) + ..., times the block's
//     fp16 weight scale, accumulated in fp32.
// Within a block the k order is permuted the same way for A and B: lane (g, t) of the MMA loads
// the 8 codes of rows g and g + 8 at positions 8t .. 8t + 7 (one 8-byte load per row at 8 bits;
// one 4-byte word at 4 bits, whose nibbles unpack to the same positions), which become its
// fragment's k = 4t .. 4t + 3 and 16 + 4t .. 16 + 4t + 3; the B fragment of lane (n, t) is loaded
// from the same positions of digit n, stored in the block's natural order.
// Work split: a CTA takes 64 rows (four MMA row tiles) and one part of the blocks, and computes the
// input digits of its part only; warp w takes row tile w % 4 and half w / 4 of the part.  The
// parts of a row tile form a thread-block cluster: after a cluster barrier rank 0 adds the
// parts' row sums in rank order (distributed shared memory) and runs the epilogue, and a second
// cluster barrier keeps the other ranks until it has read them.  No global scratch, no flags.
// The first codes are loaded before griddepcontrol.wait: weights do not depend on the preceding
// kernel.
constexpr int kQWarps = 8;
constexpr int kQThreads = kQWarps * 32;
constexpr int kQRows = 64;  // rows per CTA
constexpr int kQUnroll = 4; // blocks in flight per warp and buffer
constexpr int kQMaxParts = 8;

__device__ __forceinline__ void mma_u8s8(int (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k32.row.col.s32.u8.s8.s32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
        : "+r"(d[0]), "+r"(d[1]), "+r"(d[2]), "+r"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Blocks of part `part` of `parts` over nb blocks.
__device__ __forceinline__ void part_blocks(int nb, int part, int parts, int& b0, int& b1) {
    b0 = (int)(((int64_t)part * nb) / parts);
    b1 = (int)(((int64_t)(part + 1) * nb) / parts);
}
// shared-memory bytes of a CTA whose part has at most `pb` blocks: per block 3 x 32 digits, then
// 16 bytes of scales (s1, s2, s3) and 16 of bias-scaled digit sums
static size_t gemv_q_smem(int pb) { return (size_t)pb * (96 + 16 + 16) + 16; }

template <int EPI, int BITS>
__global__ void __launch_bounds__(kQThreads) k_gemv_q(const __grid_constant__ QGemvArgs a) {
    constexpr int BIAS = BITS == 8 ? 128 : 8;
    extern __shared__ __align__(16) uint8_t qsm[];
    __shared__ float red[kQWarps + 1];
    __shared__ float rsum[kQWarps][16];
    __shared__ float rows_sum[kQRows];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, g = lane >> 2, t = lane & 3;
    const QMatDev& W = a.w;
    const int nb = W.nb;
    const int parts = (int)gridDim.x, part = (int)blockIdx.x;  // cluster (parts, 1, 1): rank = part
    int pb0, pb1;
    part_blocks(nb, part, parts, pb0, pb1);
    const int npb = pb1 - pb0;
    int8_t* xq = reinterpret_cast<int8_t*>(qsm);                           // [npb][3][32]
    float4* xsc = reinterpret_cast<float4*>(qsm + (size_t)npb * 96);       // [npb] (s1, s2, s3, -)
    int4* xsum = reinterpret_cast<int4*>(xsc + npb);                       // [npb] bias * digit sums
    const int tile = warp & 3, half = warp >> 2;
    const int row0 = (int)blockIdx.y * kQRows + tile * 16;
    const int ra = row0 + g, rb = row0 + g + 8;
    const bool oka = ra < W.rows, okb = rb < W.rows;
    // this warp's blocks: half `half` of the part
    const int wb0 = pb0 + (half == 0 ? 0 : npb / 2), wb1 = half == 0 ? pb0 + npb / 2 : pb1;
    const uint8_t* ca = W.codes + (int64_t)(oka ? ra : 0) * W.row_bytes;
    const uint8_t* cb = W.codes + (int64_t)(okb ? rb : 0) * W.row_bytes;
    const __half* sa = W.scales + (int64_t)(oka ? ra : 0) * nb;
    const __half* sb = W.scales + (int64_t)(okb ? rb : 0) * nb;

    // codes of rows g, g + 8 (8 bytes each at 8 bits, a word at 4) and, in lane t = 0, the rows'
    // weight scales, for kQUnroll blocks from block bb
    auto load = [&](uint2 (&va)[kQUnroll], uint2 (&vb)[kQUnroll], __half2 (&dv)[kQUnroll], int bb) {
#pragma unroll
        for (int u = 0; u < kQUnroll; ++u) {
            const int b = bb + u;
            const bool on = b < wb1;
            if constexpr (BITS == 8) {
                va[u] = on && oka ? ldg_stream_u2(ca + (int64_t)b * 32 + 8 * t) : make_uint2(0u, 0u);
                vb[u] = on && okb ? ldg_stream_u2(cb + (int64_t)b * 32 + 8 * t) : make_uint2(0u, 0u);
            } else {
                va[u].x = on && oka ? ldg_stream_u1(ca + (int64_t)b * 16 + 4 * t) : 0u;
                vb[u].x = on && okb ? ldg_stream_u1(cb + (int64_t)b * 16 + 4 * t) : 0u;
                va[u].y = vb[u].y = 0u;
            }
            const __half z = __float2half(0.f);
            dv[u] = __halves2half2(on && oka && t == 0 ? sa[b] : z, on && okb && t == 0 ? sb[b] : z);
        }
    };
    uint2 pa[2][kQUnroll], pb[2][kQUnroll];
    __half2 pd[2][kQUnroll];
    load(pa[0], pb[0], pd[0], wb0);
    load(pa[1], pb[1], pd[1], wb0 + kQUnroll);
    pdl_wait();

    // ---------------------------------------------------------------- input digits of the part
    float rinv = 1.f;
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
            float s = 0.f;
            for (int w = 0; w < kQWarps; ++w) s += red[w];
            red[kQWarps] = 1.0f / sqrtf(s / (float)W.k + a.eps);
        }
        __syncthreads();
        rinv = red[kQWarps];
    }
    for (int j = warp; j < npb; j += kQWarps) {
        const int i = (pb0 + j) * kQBlock + lane;
        float v = 0.f;
        if (i < W.k) v = a.x != nullptr ? __half2float(a.x[i]) * rinv * __half2float(a.gain[i]) : __ldcg(a.vin + i);
        // the block's largest magnitude (non-negative floats order as their bit patterns)
        const float amax = __uint_as_float(__reduce_max_sync(0xffffffffu, __float_as_uint(fabsf(v))));
        const float s1 = amax / 127.0f, s2 = s1 / 254.0f, s3 = s2 / 254.0f;
        const float i1 = amax > 0.f ? 127.0f / amax : 0.f, i2 = i1 * 254.0f, i3 = i2 * 254.0f;
        // three digits: each takes the remainder of the ones before, to within half its step
        const float sc[3] = {s1, s2, s3}, iv[3] = {i1, i2, i3};
        int q[3];
        float r = v;
#pragma unroll
        for (int e = 0; e < 3; ++e) {
            const float f = rintf(r * iv[e]);
            q[e] = (int)fminf(fmaxf(f, -127.f), 127.f);
            r = fmaf(-(float)q[e], sc[e], r);
        }
        // digits in the codes' own (natural) order: A and B fragments are both loaded by byte
        // position, so the MMA sees the same permutation of k on both sides
        int qs[3];
#pragma unroll
        for (int e = 0; e < 3; ++e) {
            xq[j * 96 + e * 32 + lane] = (int8_t)q[e];
            qs[e] = __reduce_add_sync(0xffffffffu, q[e]);
        }
        if (lane == 0) {
            xsc[j] = make_float4(s1, s2, s3, 0.f);
            xsum[j] = make_int4(BIAS * qs[0], BIAS * qs[1], BIAS * qs[2], 0);
        }
    }
    __syncthreads();
    pdl_launch_dependents();

    // ---------------------------------------------------------------- this warp's blocks
    float acc_a = 0.f, acc_b = 0.f;
    auto consume = [&](const uint2 (&va)[kQUnroll], const uint2 (&vb)[kQUnroll], const __half2 (&dv)[kQUnroll], int bb) {
#pragma unroll
        for (int u = 0; u < kQUnroll; ++u) {
            const int b = bb + u;
            if (b >= wb1) break;
            const int j = b - pb0;
            uint32_t af[4];
            if constexpr (BITS == 8) {
                af[0] = va[u].x;
                af[1] = vb[u].x;
                af[2] = va[u].y;
                af[3] = vb[u].y;
            } else {  // byte i of the word: code 8t + i (low nibble), 8t + 4 + i (high nibble)
                af[0] = va[u].x & 0x0F0F0F0Fu;
                af[1] = vb[u].x & 0x0F0F0F0Fu;
                af[2] = (va[u].x >> 4) & 0x0F0F0F0Fu;
                af[3] = (vb[u].x >> 4) & 0x0F0F0F0Fu;
            }
            uint2 bf = make_uint2(0u, 0u);
            if (g < 3) bf = *reinterpret_cast<const uint2*>(xq + j * 96 + g * 32 + 8 * t);
            int d[4] = {0, 0, 0, 0};
            mma_u8s8(d, af, bf.x, bf.y);
            // lane t = 0 holds the digit-1 and digit-2 products of rows g, g + 8; lane t = 1 digit 3
            const int d3a = __shfl_down_sync(0xffffffffu, d[0], 1);
            const int d3b = __shfl_down_sync(0xffffffffu, d[2], 1);
            if (t == 0) {
                const float4 sc = xsc[j];
                const int4 qb = xsum[j];
                float va_ = sc.z * (float)(d3a - qb.z);
                va_ = fmaf(sc.y, (float)(d[1] - qb.y), va_);
                va_ = fmaf(sc.x, (float)(d[0] - qb.x), va_);
                float vb_ = sc.z * (float)(d3b - qb.z);
                vb_ = fmaf(sc.y, (float)(d[3] - qb.y), vb_);
                vb_ = fmaf(sc.x, (float)(d[2] - qb.x), vb_);
                const float2 ds = __half22float2(dv[u]);
                acc_a = fmaf(ds.x, va_, acc_a);
                acc_b = fmaf(ds.y, vb_, acc_b);
            }
        }
    };
    for (int bb = wb0; bb < wb1; bb += 2 * kQUnroll) {
        consume(pa[0], pb[0], pd[0], bb);
        load(pa[0], pb[0], pd[0], bb + 2 * kQUnroll);
        if (bb + kQUnroll < wb1) {
            consume(pa[1], pb[1], pd[1], bb + kQUnroll);
            load(pa[1], pb[1], pd[1], bb + 3 * kQUnroll);
        }
    }
    if (t == 0) {
        rsum[warp][g] = acc_a;
        rsum[warp][g + 8] = acc_b;
    }
    __syncthreads();
    if (tid < kQRows) rows_sum[tid] = rsum[tid >> 4][tid & 15] + rsum[4 + (tid >> 4)][tid & 15];  // halves in order

    // ---------------------------------------------------------------- parts of the cluster
    if (parts > 1) cluster_sync();  // every part's row sums are in its shared memory
    else __syncthreads();
    float tv = 0.f;
    const int r = tid, row = (int)blockIdx.y * kQRows + r;
    if (part == 0 && tid < kQRows) {
        for (int p = 0; p < parts; ++p) tv += p == 0 ? rows_sum[r] : dsmem_ld(dsmem_addr(&rows_sum[r], (uint32_t)p));
        rows_sum[r] = tv;
    }
    if (parts > 1) cluster_sync();  // rank 0 has read the others' sums (they may leave), and its own are final
    else __syncthreads();
    if (part != 0 || tid >= kQRows || row >= W.rows) return;

    // ---------------------------------------------------------------- epilogue (row pairs)
    if constexpr (EPI == kEpiPlain) {
        a.out[row] = tv;
    } else if ((r & 1) == 0 && row + 1 < W.rows) {
        const float t_odd = rows_sum[r + 1];
        if constexpr (EPI == kEpiSwiglu) {
            a.out[row >> 1] = silu(tv) * t_odd;
        } else {  // kEpiQkvRope: rows (row, row + 1) are the RoPE pair (i, i + dh / 2)
            const int p = *a.len;
            const bool ok = p >= 0 && p < a.cap;
            if (!ok && row == 0) set_status(a.status, VT_DEV_KV_OVERFLOW);
            const int hd = a.dh >> 1;
            const int blk = row / a.dh, i = (row - blk * a.dh) >> 1;
            if (blk < a.hq + a.hk) {
                const float2 cs2 = ok ? a.rope[(int64_t)p * hd + i] : make_float2(1.f, 0.f);
                const float re = tv * cs2.x - t_odd * cs2.y;
                const float ro = tv * cs2.y + t_odd * cs2.x;
                if (blk < a.hq) {
                    a.out[blk * a.dh + i] = re;
                    a.out[blk * a.dh + i + hd] = ro;
                } else if (ok) {
                    __half* kd = a.kcache + ((int64_t)(blk - a.hq) * a.cap + p) * a.dh;
                    kd[i] = __float2half_rn(re);
                    kd[i + hd] = __float2half_rn(ro);
                }
            } else if (ok) {
                __half* vd = a.vcache + ((int64_t)(blk - a.hq - a.hk) * a.cap + p) * a.dh;
                vd[i] = __float2half_rn(tv);
                vd[i + hd] = __float2half_rn(t_odd);
            }
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

// Parts per row tile: enough CTAs for about 2.5 per SM, each part at least 4 blocks, at most 8
// (the portable cluster size).
static int gemv_q_parts(int rows, int nb) {
    const int tiles = (rows + kQRows - 1) / kQRows;
    const int want = (int)std::lround(2.5 * (g_num_sms > 0 ? g_num_sms : 148) / std::max(tiles, 1));
    return std::max(1, std::min({kQMaxParts, want, std::max(1, nb / 4)}));
}

template <int EPI>
static cudaError_t launch_q_epi(const QGemvArgs& a, cudaStream_t st) {
    const int parts = gemv_q_parts(a.w.rows, a.w.nb);
    const int pb = (a.w.nb + parts - 1) / parts;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)parts, (unsigned)((a.w.rows + kQRows - 1) / kQRows));
    cfg.blockDim = dim3(kQThreads);
    cfg.dynamicSmemBytes = gemv_q_smem(pb);
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    int na = 0;
    attr[na].id = cudaLaunchAttributeClusterDimension;
    attr[na].val.clusterDim.x = (unsigned)parts;
    attr[na].val.clusterDim.y = 1;
    attr[na].val.clusterDim.z = 1;
    ++na;
    if (g_use_pdl) {
        attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[na].val.programmaticStreamSerializationAllowed = 1;
        ++na;
    }
    cfg.attrs = attr;
    cfg.numAttrs = (unsigned)na;
    if (a.w.bits == 8) return cudaLaunchKernelEx(&cfg, k_gemv_q<EPI, 8>, a);
    if (a.w.bits == 4) return cudaLaunchKernelEx(&cfg, k_gemv_q<EPI, 4>, a);
    return cudaErrorInvalidValue;
}

cudaError_t launch_gemv_q(int epi, const QGemvArgs& a, cudaStream_t st) {
    if (a.w.rows <= 0) return cudaSuccess;
    const int parts = gemv_q_parts(a.w.rows, a.w.nb);
    if (gemv_q_smem((a.w.nb + parts - 1) / parts) > 200 * 1024) return cudaErrorInvalidValue;
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
