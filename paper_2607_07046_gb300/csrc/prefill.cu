// Prefill-path kernels for one tensor-parallel shard (n prompt rows), sm_103a.
//
// What they compute (Voltron Section 2.1, prefill phase, per shard as in Section 3.2.1): the same
// steps as decode, for n rows at positions p0 .. p0 + n - 1 (p0 = cached length of the layer):
//   ATTN shard: X^ = RMSNorm(X); [Q;K;V] = X^ . Wqkv_s^T; RoPE on Q and K; K, V appended to the
//               cache; causal attention (row i sees positions 0 .. p0 + i); partial = A . Wo_s^T.
//   FFN shard:  X^ = RMSNorm(X); U = silu(X^ Wg_s^T) * (X^ Wu_s^T); partial = U . Wd_s^T.
// The projections are dense contractions and run on the tensor cores (tcgen05.mma, accumulator
// in tensor memory, operands staged by TMA); X^, Q, the attention output and U are fp16 operands,
// accumulation and partials are fp32.
//
//   k_rmsnorm_rows   one CTA per row (also the fp16 hi / lo split of the ATTN input)
//   k_combine_norm   residual + shard partials in shard order, then the next block's RMSNorm
//   k_gemm_p         C = A . B^T, A [M][K] and B [N][K] fp16 (K contiguous), persistent over the
//                    output tiles of every shard's GEMM of a block: CTA pairs (tcgen05 cta_group::2,
//                    256 x BN tiles) or single CTAs (128 x 256); epilogues: fp32 store, RoPE + q
//                    store + KV append, SwiGLU
//   k_gemm           the same MMA and copies, one 128 x 256 tile per CTA with an optional
//                    cluster split-K, for groups too small to fill the GPU
//   k_prefill_attn_tc causal flash attention on tcgen05 (S and O in tensor memory, K / V by TMA),
//                    128 query rows of one head per CTA, one launch over every shard's heads
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include <climits>
#include <cstdlib>
#include <string>

#include "device.cuh"
#include "internal.h"

namespace vt {

// ================================================================== tcgen05 / TMA primitives

namespace tc {

// 2-D tiled TMA load of box (x = inner coordinate in elements, y = row) into shared memory,
// completing as transaction bytes on `bar`.
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int x, int y, uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
            smem_u32(dst)),
        "l"(map), "r"(x), "r"(y), "r"(smem_u32(bar))
        : "memory");
}

// 3-D tiled TMA load: box (0, y, z) of a map whose third dimension steps one 64-column k-tile, so
// one box brings several consecutive k-tiles of the same rows (one swizzled tile after the other).
__device__ __forceinline__ void tma_load_3d(void* dst, const CUtensorMap* map, int y, int z, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(
            smem_u32(dst)),
        "l"(map), "r"(0), "r"(y), "r"(z), "r"(bar)
        : "memory");
}
__device__ __forceinline__ void tma_load_3d_pair(void* dst, const CUtensorMap* map, int y, int z, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.3d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, "
        "%4}], [%5];" ::"r"(smem_u32(dst)),
        "l"(map), "r"(0), "r"(y), "r"(z), "r"(bar)
        : "memory");
}

// The same load issued by either CTA of a pair that shares one MMA (cta_group::2): the box lands in
// this CTA's shared memory and its bytes complete on the mbarrier at cluster address `bar`, which
// may be in the peer CTA.
__device__ __forceinline__ void tma_load_2d_pair(void* dst, const CUtensorMap* map, int x, int y, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], "
        "[%4];" ::"r"(smem_u32(dst)),
        "l"(map), "r"(x), "r"(y), "r"(bar)
        : "memory");
}

// 2-D tiled TMA store of a shared-memory box to (x, y) of the map's tensor (rows past the
// tensor's end are not written); completion is tracked by the bulk async-group of this thread.
__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, int x, int y, const void* src) {
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];" ::"l"(map), "r"(x),
                 "r"(y), "r"(smem_u32(src))
                 : "memory");
}

// 16-byte store into the shared memory of a CTA of the cluster (address from mapa).
__device__ __forceinline__ void dsmem_st4(uint32_t addr, float a, float b, float c, float d) {
    asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "f"(a), "f"(b), "f"(c), "f"(d)
                 : "memory");
}

__device__ __forceinline__ void tmem_alloc(uint32_t* slot, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(slot)), "r"(ncols)
                 : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
// Pair forms (cta_group::2): one warp of each CTA of the pair takes part; both get the same address.
__device__ __forceinline__ void tmem_alloc_pair(uint32_t* slot, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(slot)), "r"(ncols)
                 : "memory");
}
__device__ __forceinline__ void tmem_relinquish_pair() {
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// D (tensor memory) (+)= A (shared, descriptor) . B (shared, descriptor), fp16 inputs, fp32 accumulate
__device__ __forceinline__ void mma_f16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                        uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}
// One MMA over a CTA pair (issued by the even CTA): A rows [0, M/2) from this CTA's shared memory
// and [M/2, M) from the peer's, B rows [0, N/2) here and [N/2, N) in the peer, both at the same
// offsets; each CTA's tensor memory receives its M/2 rows of D.
__device__ __forceinline__ void mma_f16_pair(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                             uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}
// Arrives once on the mbarrier at `bar`'s offset in both CTAs of the pair when every pair MMA
// issued so far has completed.
__device__ __forceinline__ void mma_commit_pair_both(uint64_t* bar) {
    asm volatile(
        "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(
            smem_u32(bar)),
        "h"((uint16_t)3)
        : "memory");
}
// Arrives once on this CTA's `bar` when every pair MMA issued so far has completed.
__device__ __forceinline__ void mma_commit_pair(uint64_t* bar) {
    asm volatile("tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
                 : "memory");
}

// Arrives once on `bar` when every MMA this thread issued so far has completed.
__device__ __forceinline__ void mma_commit(uint64_t* bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
                 : "memory");
}

// 32 lanes x 32 consecutive columns of 32-bit data: thread t of the warp gets lane (base + t).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
// The wait with the loaded registers as operands, so that no use of them is scheduled before it.
__device__ __forceinline__ void tmem_ld_wait_on(uint32_t (&r)[32]) {
    asm volatile("tcgen05.wait::ld.sync.aligned;"
                 : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7]),
                   "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]), "+r"(r[14]),
                   "+r"(r[15]), "+r"(r[16]), "+r"(r[17]), "+r"(r[18]), "+r"(r[19]), "+r"(r[20]), "+r"(r[21]),
                   "+r"(r[22]), "+r"(r[23]), "+r"(r[24]), "+r"(r[25]), "+r"(r[26]), "+r"(r[27]), "+r"(r[28]),
                   "+r"(r[29]), "+r"(r[30]), "+r"(r[31])
                 :
                 : "memory");
}
// The store counterpart: thread t writes 32 consecutive columns of lane (base + t).
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
        "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
        "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
        "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
        "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]),
        "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]),
        "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
        : "memory");
}
__device__ __forceinline__ void tmem_st_wait() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// Shared-memory matrix descriptor of a K-major operand tile written by TMA with the 128-byte
// swizzle: rows of 64 fp16 (128 bytes), 8-row groups 1024 bytes apart.  The tile base is 1024-byte
// aligned; stepping K by 16 elements inside the 128-byte row advances the start address by 32 bytes.
__device__ __forceinline__ uint64_t desc_sw128(uint32_t saddr) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);  // start address
    d |= (uint64_t)1 << 16;                    // leading-dimension offset (unused with this swizzle)
    d |= (uint64_t)(1024 >> 4) << 32;          // stride between 8-row groups
    d |= (uint64_t)1 << 46;                    // descriptor version
    d |= (uint64_t)2 << 61;                    // 128-byte swizzle
    return d;
}

// Descriptor of an MN-major operand (the N index contiguous) written by TMA with the 128-byte
// swizzle: each K index is one 128-byte row of 64 consecutive N elements, 8-row groups are 1024
// bytes apart, and the next 64 N elements sit `lbo` bytes further (the next TMA box).  Stepping K
// by 16 advances the start address by 16 rows (2048 bytes).
__device__ __forceinline__ uint64_t desc_sw128_mn(uint32_t saddr, uint32_t lbo) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);  // start address
    d |= (uint64_t)(lbo >> 4) << 16;           // offset between 64-element groups of N
    d |= (uint64_t)(1024 >> 4) << 32;          // stride between 8-row groups of K
    d |= (uint64_t)1 << 46;                    // descriptor version
    d |= (uint64_t)2 << 61;                    // 128-byte swizzle
    return d;
}

// Instruction descriptor: fp16 A and B (both K-major), fp32 accumulator, M x N.
__host__ __device__ constexpr uint32_t idesc_f16(int m, int n) {
    return (1u << 4) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(m >> 4) << 24);
}
// The same with B MN-major (transposed B).
__host__ __device__ constexpr uint32_t idesc_f16_bmn(int m, int n) { return idesc_f16(m, n) | (1u << 16); }

}  // namespace tc

// ================================================================== RMSNorm rows

// One CTA per row: y = fp16(RMSNorm(x) * gain).  split != 0: the row of y is 2d long and holds
// the fp16 value in [0, d) and the fp16 rounding of the remainder in [d, 2d), so that a GEMM over
// the 2d columns (the weights read twice) multiplies the normalised input at fp32 precision.
__device__ __forceinline__ void store_hl8(__half* row, int d, int c, const float (&v)[8], bool split) {
    uint32_t hi[4], lo[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const __half2 h = __floats2half2_rn(v[2 * e], v[2 * e + 1]);
        hi[e] = *reinterpret_cast<const uint32_t*>(&h);
        const float2 hf = __half22float2(h);
        const __half2 l = __floats2half2_rn(v[2 * e] - hf.x, v[2 * e + 1] - hf.y);
        lo[e] = *reinterpret_cast<const uint32_t*>(&l);
    }
    *reinterpret_cast<uint4*>(row + (size_t)c * 8) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
    if (split) *reinterpret_cast<uint4*>(row + d + (size_t)c * 8) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
}

__global__ void __launch_bounds__(256) k_rmsnorm_rows(const __half* __restrict__ x, const __half* __restrict__ gain,
                                                      float eps, int d, __half* __restrict__ y, int split) {
    __shared__ float red[8];
    pdl_wait();
    const __half* xr = x + (size_t)blockIdx.x * d;
    __half* yr = y + (size_t)blockIdx.x * d * (split ? 2 : 1);
    float ss = 0.f;
    for (int c = threadIdx.x; c < d / 8; c += blockDim.x) {
        const uint4 v = *reinterpret_cast<const uint4*>(xr + c * 8);
        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float2 f = h2_to_f2(w[e]);
            ss = fmaf(f.x, f.x, ss);
            ss = fmaf(f.y, f.y, ss);
        }
    }
    ss = warp_sum(ss);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
    __syncthreads();
    float tot = 0.f;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) tot += red[w];
    const float r = 1.0f / sqrtf(tot / (float)d + eps);
    for (int c = threadIdx.x; c < d / 8; c += blockDim.x) {
        const uint4 v = *reinterpret_cast<const uint4*>(xr + c * 8);
        const uint4 g = *reinterpret_cast<const uint4*>(gain + c * 8);
        const uint32_t w[4] = {v.x, v.y, v.z, v.w}, gw[4] = {g.x, g.y, g.z, g.w};
        float o[8];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float2 f = h2_to_f2(w[e]), gg = h2_to_f2(gw[e]);
            o[2 * e] = f.x * r * gg.x;
            o[2 * e + 1] = f.y * r * gg.y;
        }
        store_hl8(yr, d, c, o, split != 0);
    }
}

// ================================================================== combine + RMSNorm rows

// One CTA per row: out = fp16(residual + sum_s parts[s]) (fp32, shards in order, as k_combine),
// and, when gain is set, xhat = fp16(RMSNorm(out) * gain) computed from the rounded row: the input
// every shard of the next block would normalise for itself.
__global__ void __launch_bounds__(256) k_combine_norm(const __grid_constant__ CombineArgs a, int d,
                                                      const __half* __restrict__ gain, float eps,
                                                      __half* __restrict__ xhat, int split) {
    __shared__ float red[8];
    pdl_wait();
    const size_t row = blockIdx.x;
    float ss = 0.f;
    for (int c = threadIdx.x; c < d / 8; c += blockDim.x) {
        const size_t e0 = row * d + (size_t)c * 8;
        float acc[8];
        if (a.residual) {
            const uint4 r = *reinterpret_cast<const uint4*>(a.residual + e0);
            const uint32_t w[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const float2 f = h2_to_f2(w[j]);
                acc[2 * j] = f.x;
                acc[2 * j + 1] = f.y;
            }
        } else {
#pragma unroll
            for (int j = 0; j < 8; ++j) acc[j] = 0.f;
        }
        for (int sh = 0; sh < a.n; ++sh) {
            if (!a.parts[sh]) continue;
            const float4 p0 = __ldcg(reinterpret_cast<const float4*>(a.parts[sh] + e0));
            const float4 p1 = __ldcg(reinterpret_cast<const float4*>(a.parts[sh] + e0 + 4));
            acc[0] += p0.x; acc[1] += p0.y; acc[2] += p0.z; acc[3] += p0.w;
            acc[4] += p1.x; acc[5] += p1.y; acc[6] += p1.z; acc[7] += p1.w;
        }
        uint32_t o[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const __half2 h = __floats2half2_rn(acc[2 * j], acc[2 * j + 1]);
            o[j] = *reinterpret_cast<const uint32_t*>(&h);
            const float2 f = __half22float2(h);
            ss = fmaf(f.x, f.x, ss);
            ss = fmaf(f.y, f.y, ss);
        }
        *reinterpret_cast<uint4*>(a.out + e0) = make_uint4(o[0], o[1], o[2], o[3]);
    }
    if (!gain) return;
    ss = warp_sum(ss);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
    __syncthreads();
    float tot = 0.f;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) tot += red[w];
    const float r = 1.0f / sqrtf(tot / (float)d + eps);
    for (int c = threadIdx.x; c < d / 8; c += blockDim.x) {
        // this thread's own row elements, written above
        const uint4 hv = *reinterpret_cast<const uint4*>(a.out + row * d + (size_t)c * 8);
        const uint4 g = *reinterpret_cast<const uint4*>(gain + c * 8);
        const uint32_t w[4] = {hv.x, hv.y, hv.z, hv.w}, gw[4] = {g.x, g.y, g.z, g.w};
        float o[8];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const float2 f = h2_to_f2(w[j]), gg = h2_to_f2(gw[j]);
            o[2 * j] = f.x * r * gg.x;
            o[2 * j + 1] = f.y * r * gg.y;
        }
        store_hl8(xhat + row * d * (split ? 2 : 1), d, c, o, split != 0);
    }
}

cudaError_t launch_combine_norm(const CombineArgs& a, int rows, int d, const __half* gain, float eps, __half* xhat,
                                int split, cudaStream_t st) {
    if (rows <= 0) return cudaSuccess;
    if (d % 8 != 0 || d > 16384) return cudaErrorInvalidValue;
    k_combine_norm<<<rows, 256, 0, st>>>(a, d, gain, eps, xhat, split);
    return cudaGetLastError();
}

// ================================================================== tensor-core GEMM

constexpr int kBM = 128, kBK = 64, kBN = 256, kStages = 4;
constexpr int kGemmThreads = 192;  // warp 0: TMA, warp 1: MMA + tensor memory, warps 2-5: epilogue
constexpr int kABytes = kBM * kBK * 2, kBBytes = kBN * kBK * 2, kStageBytes = kABytes + kBBytes;
constexpr size_t kGemmSmem = (size_t)kStages * kStageBytes + 1024 /* alignment */ + 256 /* barriers */;

enum GemmEpi : int { kGemmF32 = 0, kGemmQkv = 1, kGemmSwiglu = 2 };

struct GemmArgs {
    int m, n, k_tiles;
    int kb_wrap;  // > 0: A's k-tile kt multiplies B's k-tile kt mod kb_wrap (B read twice: hi / lo A halves)
    const __half* b;  // B [n][ldb] (prefetched into L2 by the epilogue warps while they wait)
    int64_t ldb;
    // kGemmF32: c[row][col], row stride ldc
    float* c;
    int ldc;
    // kGemmQkv: columns are head blocks of dh in RoPE-pair order (q heads, k heads, v heads)
    __half* q;  // [m][hq][dh]
    __half* kcache;
    __half* vcache;
    int hq, hk, dh, cap;
    const int32_t* len;  // rows sit at positions *len + row_offset + row
    int row_offset;
    const float2* rope;
    // kGemmSwiglu: columns (gate j, up j) interleaved; u[row][ushift + j], zeros in [0, ushift)
    __half* u;
    int ldu, ushift;
    uint32_t* status;
};

// Up to kGemmGroups independent GEMMs of the same row count in one launch (the shards of one
// block, which share M and often A): group g owns the CTAs with blockIdx.x in
// [tile_end[g - 1], tile_end[g]), one per 256-column tile of its N.
constexpr int kGemmGroups = 8;
struct GemmGroup {
    int n_groups;
    int tile_end[kGemmGroups];
    CUtensorMap ta[kGemmGroups], tb[kGemmGroups];
    GemmArgs a[kGemmGroups];
};
static_assert(sizeof(GemmGroup) <= 4096, "the GEMM launch's parameters must fit in 4 KB");

// 16-byte slot of the split-K receive buffer that holds floats [4e, 4e + 4) of 32-column chunk
// `chunk` of local row `lr`.  128-bit shared accesses are served 8 threads at a time; the slot
// permutation keeps those 8 threads on distinct banks both for the writer (8 consecutive rows, one
// chunk) and for the reader (one row, 8 consecutive chunks).
__device__ __forceinline__ int recv_slot(int chunk, int e, int lr) { return chunk * 8 + (e ^ ((chunk + lr) & 7)); }

// B's k-tile for A's k-tile kt.
__device__ __forceinline__ int bk_tile(const GemmArgs& a, int kt) {
    return a.kb_wrap > 0 && kt >= a.kb_wrap ? kt - a.kb_wrap : kt;
}

// Epilogue of 4 consecutive columns [col, col + 4) of one output row (col a multiple of 4).
template <int EPI>
__device__ __forceinline__ void gemm_epilogue_quad(const GemmArgs& a, int row, int col, float4 v, int pos) {
    if constexpr (EPI == kGemmF32) {
        float* dst = a.c + (size_t)row * a.ldc + col;
        if (col + 4 <= a.n) {
            *reinterpret_cast<float4*>(dst) = v;
        } else {
            const float f[4] = {v.x, v.y, v.z, v.w};
            for (int j = 0; j < 4 && col + j < a.n; ++j) dst[j] = f[j];
        }
    } else if constexpr (EPI == kGemmQkv) {
        // columns (col, col + 1) and (col + 2, col + 3): RoPE pairs (i, i + dh/2) and (i + 1, ...)
        const int dh = a.dh, half = dh / 2;
        const int b = col / dh, i = (col % dh) / 2;
        float l0 = v.x, h0 = v.y, l1 = v.z, h1 = v.w;
        if (b < a.hq + a.hk) {
            const float4 cs = *reinterpret_cast<const float4*>(a.rope + (size_t)pos * half + i);
            l0 = v.x * cs.x - v.y * cs.y;
            h0 = v.x * cs.y + v.y * cs.x;
            l1 = v.z * cs.z - v.w * cs.w;
            h1 = v.z * cs.w + v.w * cs.z;
        }
        __half* dst;
        if (b < a.hq) dst = a.q + ((size_t)row * a.hq + b) * dh;
        else if (b < a.hq + a.hk) dst = a.kcache + ((size_t)(b - a.hq) * a.cap + pos) * dh;
        else dst = a.vcache + ((size_t)(b - a.hq - a.hk) * a.cap + pos) * dh;
        *reinterpret_cast<__half2*>(dst + i) = __floats2half2_rn(l0, l1);
        *reinterpret_cast<__half2*>(dst + i + half) = __floats2half2_rn(h0, h1);
    } else {
        // columns (gate, up) of intermediate columns col / 2 and col / 2 + 1
        __half* dst = a.u + (size_t)row * a.ldu + a.ushift + col / 2;
        if (col == 0)
            for (int j = 0; j < a.ushift; ++j) dst[j - a.ushift] = __float2half_rn(0.f);
        dst[0] = __float2half_rn(silu(v.x) * v.y);
        if (col + 2 < a.n) dst[1] = __float2half_rn(silu(v.z) * v.w);
    }
}

// One 128 x 256 tile of C = A . B^T per CTA, or per cluster of S CTAs that split K.
// A k-tile is 64 columns of K: TMA brings the A and B boxes (128-byte swizzle) into one of kStages
// stages; the MMA thread issues four 128 x 256 x 16 MMAs per stage into one tensor-memory
// accumulator (256 columns) and releases the stage through tcgen05.commit.  The CTA's B boxes are
// first requested into L2 with TMA prefetches (the weights do not depend on the preceding kernel,
// so this starts before griddepcontrol.wait), which hides the HBM latency the 4-stage ring cannot.
//
// Split K (gridDim.z = S > 1, one thread-block cluster per output tile): every CTA accumulates
// k-tiles [k_tiles z / S, k_tiles (z + 1) / S).  After the last MMA of every CTA (cluster barrier),
// the accumulators are reduce-scattered through distributed shared memory: tile row r belongs to
// CTA r / ceil(128 / S), which receives every CTA's fp32 values of its rows into its (now free)
// stage memory, adds the S contributions in rank order (so results do not depend on timing) and
// runs the epilogue.  Rows >= m and columns >= n come from TMA's zero fill and are not stored.
// Every wait is bounded; on a timeout the kernel sets VT_DEV_WAIT_TIMEOUT, stops issuing, waits
// for the copies it issued, still reaches both cluster barriers, frees tensor memory and ends.
template <int EPI>
__global__ void __launch_bounds__(kGemmThreads, 1) k_gemm(const __grid_constant__ GemmGroup G) {
    int g = 0;
    while (g + 1 < G.n_groups && (int)blockIdx.x >= G.tile_end[g]) ++g;
    const CUtensorMap& ta = G.ta[g];
    const CUtensorMap& tb = G.tb[g];
    const GemmArgs& a = G.a[g];
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + kStages * kStageBytes);
    uint64_t* empty = full + kStages;
    uint64_t* done = empty + kStages;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);
    __shared__ int s_err;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n0 = ((int)blockIdx.x - (g > 0 ? G.tile_end[g - 1] : 0)) * kBN, m0 = blockIdx.y * kBM;
    const int S = gridDim.z, z = blockIdx.z;
    const int kt0 = (int)((int64_t)a.k_tiles * z / S), kt1 = (int)((int64_t)a.k_tiles * (z + 1) / S);
    const int nk = kt1 - kt0;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_init(done, 1);
        s_err = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tc::tmem_alloc(tmem_slot, kBN);
        tc::tmem_relinquish();
    }
    tc::fence_before();
    __syncthreads();
    tc::fence_after();
    const uint32_t tmem = *tmem_slot;
    // B (the weights) does not depend on the preceding kernel: the B halves of the first stages
    // and the L2 prefetch of the CTA's remaining B tiles are issued before griddepcontrol.wait, so
    // they stream while the preceding kernel finishes; A, which it wrote, is loaded after the wait.
    const int pre = nk < kStages ? nk : kStages;
    if (warp == 0 && lane == 0) {
        for (int i = 0; i < pre; ++i) {
            mbar_arrive_expect_tx(&full[i], kStageBytes);
            tc::tma_load_2d(smem + i * kStageBytes + kABytes, &tb, bk_tile(a, kt0 + i) * kBK, n0, &full[i]);
        }
    } else if (warp >= 2) {
        const int t = threadIdx.x - 64;
        for (int i = kt0 + pre; i < kt1; ++i) {
            if (a.kb_wrap > 0 && i >= a.kb_wrap && kt0 < a.kb_wrap) break;  // the second pass reads the same B again
            for (int r = t; r < kBN; r += kGemmThreads - 64)
                if (n0 + r < a.n)
                    asm volatile("prefetch.global.L2 [%0];" ::"l"(a.b + (size_t)(n0 + r) * a.ldb + (size_t)bk_tile(a, i) * kBK));
        }
    }
    pdl_wait();  // A was written by the preceding kernel

    bool ok = true;
    if (warp == 0) {
        if (lane == 0) {
            int issued = 0;
            for (int i = 0; i < nk; ++i) {
                const int s = i % kStages;
                if (i >= kStages && !mbar_wait(&empty[s], ((i / kStages) - 1) & 1)) {
                    s_err = 1;
                    set_status(a.status, VT_DEV_WAIT_TIMEOUT);
                    break;
                }
                if (*(volatile int*)&s_err) break;
                uint8_t* st = smem + s * kStageBytes;
                if (i < pre) {  // B of this stage is already on its way
                    tc::tma_load_2d(st, &ta, (kt0 + i) * kBK, m0, &full[s]);
                } else {
                    mbar_arrive_expect_tx(&full[s], kStageBytes);
                    tc::tma_load_2d(st, &ta, (kt0 + i) * kBK, m0, &full[s]);
                    tc::tma_load_2d(st + kABytes, &tb, bk_tile(a, kt0 + i) * kBK, n0, &full[s]);
                }
                issued = i + 1;
            }
            // no copy may still be in flight when the stage memory is reused or the CTA ends (after an
            // early stop this includes the B halves issued before griddepcontrol.wait: their stages
            // never complete, and the bounded wait outlasts the copies)
            if (issued < pre) issued = pre;
            for (int i = issued > kStages ? issued - kStages : 0; i < issued; ++i)
                if (!mbar_wait(&full[i % kStages], (i / kStages) & 1)) set_status(a.status, VT_DEV_WAIT_TIMEOUT);
        }
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t idesc = tc::idesc_f16(kBM, kBN);
            for (int i = 0; i < nk; ++i) {
                const int s = i % kStages;
                if (!mbar_wait(&full[s], (i / kStages) & 1)) {
                    s_err = 1;
                    set_status(a.status, VT_DEV_WAIT_TIMEOUT);
                    break;
                }
                tc::fence_after();
                const uint32_t sa = smem_u32(smem + s * kStageBytes), sb = sa + kABytes;
#pragma unroll
                for (int k = 0; k < kBK / 16; ++k)
                    tc::mma_f16(tmem, tc::desc_sw128(sa + k * 32), tc::desc_sw128(sb + k * 32), idesc,
                                (i | k) != 0);
                tc::mma_commit(&empty[s]);
            }
            tc::mma_commit(done);
        }
    } else {
        // one lane per warp polls the barrier (128 pollers would compete with the TMA and MMA
        // threads for issue slots and shared-memory bandwidth during the whole main loop)
        if (lane == 0) {
            ok = mbar_wait(done, 0);
            if (!ok) set_status(a.status, VT_DEV_WAIT_TIMEOUT);
            ok = ok && !*(volatile int*)&s_err;
        }
        __syncwarp();
        // tcgen05.ld is warp-collective: the whole warp reads the accumulator or none of it
        ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
        tc::fence_after();
    }

    // Epilogue.  recv[slot][local row][256] (fp32, 16-byte groups permuted by recv_slot) lives in
    // the stage memory, free once the accumulator is complete (and, with split K, once every CTA
    // of the cluster has passed the first cluster barrier).  Tile row r belongs to CTA
    // r / rows_per of the cluster; every CTA sends each row of its accumulator to the owner's
    // slot `z` (its own rank), the owner adds the S slots in rank order, and each warp then writes
    // whole rows (lane = 4 consecutive columns) so every store instruction covers 512 bytes.
    float* recv = reinterpret_cast<float*>(smem);
    const int rows_per = (kBM + S - 1) / S;
    if (S > 1) cluster_sync();  // every CTA's MMAs have completed; stage memory is free everywhere
    if (warp >= 2 && ok) {
        const int sub = warp & 3, tr = sub * 32 + lane;  // tile row held by this thread
        const int owner = tr / rows_per, lr = tr - owner * rows_per;
        float* row_dst = recv + (size_t)(z * rows_per + lr) * kBN;
        const uint32_t dst = S > 1 ? dsmem_addr(row_dst, (uint32_t)owner) : smem_u32(row_dst);
        for (int c = 0; c < kBN; c += 32) {
            uint32_t r[32];
            tc::tmem_ld32(tmem + ((uint32_t)(sub * 32) << 16) + (uint32_t)c, r);
            tc::tmem_ld_wait();
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                const uint32_t at = dst + (uint32_t)recv_slot(c / 32, e, lr) * 16;
                if (S > 1)
                    tc::dsmem_st4(at, __uint_as_float(r[4 * e]), __uint_as_float(r[4 * e + 1]),
                                  __uint_as_float(r[4 * e + 2]), __uint_as_float(r[4 * e + 3]));
                else
                    asm volatile("st.shared.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(at), "f"(__uint_as_float(r[4 * e])),
                                 "f"(__uint_as_float(r[4 * e + 1])), "f"(__uint_as_float(r[4 * e + 2])),
                                 "f"(__uint_as_float(r[4 * e + 3]))
                                 : "memory");
            }
        }
    }
    if (S > 1) cluster_sync();  // every contribution has landed (all threads of every CTA)
    else if (warp >= 2) asm volatile("bar.sync 1, %0;" ::"n"(kGemmThreads - 64) : "memory");  // the 4 epilogue warps
    if (warp >= 2) {
        const int r0 = z * rows_per, nr = min(kBM, r0 + rows_per) - r0;
        int len0 = 0;
        if constexpr (EPI == kGemmQkv) len0 = *a.len + a.row_offset;
        for (int lr = warp - 2; lr < nr; lr += (kGemmThreads - 64) / 32) {
            const int row = m0 + r0 + lr;
            if (row >= a.m) break;
            const int pos = len0 + row;
            if constexpr (EPI == kGemmQkv) {
                if (pos < 0 || pos >= a.cap) {
                    if (lane == 0) set_status(a.status, VT_DEV_KV_OVERFLOW);
                    continue;
                }
            }
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int f = h * 32 + lane;  // float4 index in the row
                const int col = n0 + 4 * f;
                float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
                for (int sl = 0; sl < S; ++sl) {
                    const uint4 x = lds128(recv + (size_t)(sl * rows_per + lr) * kBN + recv_slot(f / 8, f % 8, lr) * 4);
                    v.x += __uint_as_float(x.x);
                    v.y += __uint_as_float(x.y);
                    v.z += __uint_as_float(x.z);
                    v.w += __uint_as_float(x.w);
                }
                if (col < a.n) gemm_epilogue_quad<EPI>(a, row, col, v, pos);
            }
        }
    }
    tc::fence_before();
    __syncthreads();
    if (warp == 1) {
        tc::fence_after();
        tc::tmem_dealloc(tmem, kBN);
    }
}

// ================================================================== persistent tensor-core GEMM
//
// The grouped projections of a block (every shard's GEMM of one kind) as one persistent launch.
// Each worker walks output tiles t = w, w + workers, ... of the group in an order where the row
// tile is the fastest index, so the tiles that share a weight tile run at the same time and the
// weights leave DRAM once.  A worker is a pair of CTAs on two SMs (CG = 2: 256 x BN tiles, one
// tcgen05.mma cta_group::2 over both CTAs' shared memory, each CTA holding 128 rows of A, half of
// B and its 128 rows of the accumulator) or a single CTA (CG = 1: 128 x 256 tiles).
//   warp 0   TMA producer: per stage, one box of A rows and one of B rows, each bringing two
//            consecutive k-tiles (3-D tensor maps) or one, into a ring of stages as deep as shared
//            memory allows, continuing across tiles.  The copy engine's cost is per box, so two
//            k-tiles per box nearly halve it;
//   warp 1   tensor memory (512 columns: two accumulators of up to 256) and, in the CTA of rank 0,
//            the MMA thread: the tile's k-tiles into accumulator (tile index & 1), a commit per
//            stage that frees it in both CTAs, and a commit that releases the accumulator to both
//            CTAs' epilogues;
//   warps 2-5 epilogue: each warp reads its 32 accumulator lanes (rows) in chunks of 32 columns
//            and writes the tile's outputs (fp32 partials through a shared-memory turn so each
//            store writes whole rows); after the last chunk it hands the accumulator back, so the
//            epilogue of one tile overlaps the MMAs of the next.
// Every wait is bounded; on a timeout the CTA sets VT_DEV_WAIT_TIMEOUT and an abort flag, every
// role stops at its next wait, copies and MMAs in flight are waited for (bounded), and tensor
// memory is freed.

constexpr int kPStages = 8;     // most ring stages
constexpr int kPTmemCols = 512;  // two accumulators
constexpr size_t kPGemmSmem = 227 * 1024;
constexpr size_t kPBarBytes = 256;                    // barriers and the tensor-memory slot
constexpr size_t kPEpiBytes = 4 * 32 * 33 * 4;        // fp32 epilogue staging, one 32 x 33 block per warp

struct PGemmGroup {
    int n_groups, tiles_m, tm, bn, total_tiles, stages;
    int kts;  // k-tiles per stage: 2 (one 3-D box per operand brings two) or 1
    int tile_end[kGemmGroups];  // cumulative tiles (tiles_m x column tiles of each group)
    CUtensorMap ta[kGemmGroups], tb[kGemmGroups];
    GemmArgs a[kGemmGroups];
};

static_assert(sizeof(PGemmGroup) <= 4096, "the GEMM launch's parameters must fit in 4 KB");

// Tile t of the group: the row tile (tm rows: 128, or 256 for a CTA pair) is the fastest index.
__device__ __forceinline__ void ptile(const PGemmGroup& G, int t, int& g, int& m0, int& n0) {
    g = 0;
    while (g + 1 < G.n_groups && t >= G.tile_end[g]) ++g;
    const int u = t - (g > 0 ? G.tile_end[g - 1] : 0);
    m0 = (u % G.tiles_m) * G.tm;
    n0 = (u / G.tiles_m) * G.bn;
}

// Epilogue of 32 consecutive columns [col0, col0 + 32) of row `row` (col0 a multiple of 32).
template <int EPI>
__device__ __forceinline__ void pepi_chunk(const GemmArgs& a, int row, int col0, const uint32_t (&r)[32], int pos) {
    if constexpr (EPI == kGemmF32) {
        float* dst = a.c + (size_t)row * a.ldc + col0;
        if (col0 + 32 <= a.n) {
#pragma unroll
            for (int j = 0; j < 8; ++j)
                reinterpret_cast<float4*>(dst)[j] = make_float4(__uint_as_float(r[4 * j]), __uint_as_float(r[4 * j + 1]),
                                                                __uint_as_float(r[4 * j + 2]), __uint_as_float(r[4 * j + 3]));
        } else {
#pragma unroll
            for (int j = 0; j < 32; ++j)
                if (col0 + j < a.n) dst[j] = __uint_as_float(r[j]);
        }
    } else if constexpr (EPI == kGemmQkv) {
        // 16 RoPE pairs (columns 2p, 2p + 1 = dims i0 + p and i0 + p + dh / 2 of one head block)
        if (col0 >= a.n) return;
        const int dh = a.dh, half = dh / 2;
        const int b = col0 / dh, i0 = (col0 % dh) / 2;
        float lo[16], hi[16];
        if (b < a.hq + a.hk) {
            const float2* cs = a.rope + (size_t)pos * half + i0;
#pragma unroll
            for (int p = 0; p < 16; ++p) {
                const float2 c = cs[p];
                const float x0 = __uint_as_float(r[2 * p]), x1 = __uint_as_float(r[2 * p + 1]);
                lo[p] = x0 * c.x - x1 * c.y;
                hi[p] = x0 * c.y + x1 * c.x;
            }
        } else {
#pragma unroll
            for (int p = 0; p < 16; ++p) {
                lo[p] = __uint_as_float(r[2 * p]);
                hi[p] = __uint_as_float(r[2 * p + 1]);
            }
        }
        __half* dst;
        if (b < a.hq) dst = a.q + ((size_t)row * a.hq + b) * dh;
        else if (b < a.hq + a.hk) dst = a.kcache + ((size_t)(b - a.hq) * a.cap + pos) * dh;
        else dst = a.vcache + ((size_t)(b - a.hq - a.hk) * a.cap + pos) * dh;
        uint32_t wl[8], wh[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const __half2 l2 = __floats2half2_rn(lo[2 * j], lo[2 * j + 1]), h2 = __floats2half2_rn(hi[2 * j], hi[2 * j + 1]);
            wl[j] = *reinterpret_cast<const uint32_t*>(&l2);
            wh[j] = *reinterpret_cast<const uint32_t*>(&h2);
        }
        uint4* dl = reinterpret_cast<uint4*>(dst + i0);
        uint4* dhp = reinterpret_cast<uint4*>(dst + i0 + half);
        dl[0] = make_uint4(wl[0], wl[1], wl[2], wl[3]);
        dl[1] = make_uint4(wl[4], wl[5], wl[6], wl[7]);
        dhp[0] = make_uint4(wh[0], wh[1], wh[2], wh[3]);
        dhp[1] = make_uint4(wh[4], wh[5], wh[6], wh[7]);
    } else {
        // (gate, up) pairs of intermediate columns col0 / 2 + p
        __half* dst = a.u + (size_t)row * a.ldu + a.ushift + col0 / 2;
        if (col0 == 0)
            for (int j = 0; j < a.ushift; ++j) dst[j - a.ushift] = __float2half_rn(0.f);
        if (col0 + 32 <= a.n && ((uintptr_t)dst & 15) == 0) {
            uint32_t w[8];
#pragma unroll
            for (int p = 0; p < 8; ++p) {
                const __half2 h = __floats2half2_rn(silu(__uint_as_float(r[4 * p])) * __uint_as_float(r[4 * p + 1]),
                                                    silu(__uint_as_float(r[4 * p + 2])) * __uint_as_float(r[4 * p + 3]));
                w[p] = *reinterpret_cast<const uint32_t*>(&h);
            }
            reinterpret_cast<uint4*>(dst)[0] = make_uint4(w[0], w[1], w[2], w[3]);
            reinterpret_cast<uint4*>(dst)[1] = make_uint4(w[4], w[5], w[6], w[7]);
        } else {
#pragma unroll
            for (int p = 0; p < 16; ++p)
                if (col0 + 2 * p < a.n)
                    dst[p] = __float2half_rn(silu(__uint_as_float(r[2 * p])) * __uint_as_float(r[2 * p + 1]));
        }
    }
}

// fp32 epilogue of a warp's 32 rows [row0, row0 + 32) x 32 columns [col0, col0 + 32): lane l holds
// row row0 + l.  The chunk is turned around in shared memory (`stg`, 32 x 33 floats, padded so
// both the row-wise writes and the column-wise reads hit 32 distinct banks), then each store
// instruction writes one row's 32 consecutive floats (one 128-byte line) instead of 32 scattered
// 16-byte pieces.
__device__ __forceinline__ void pepi_f32_rows(const GemmArgs& a, float* stg, int row0, int col0, const uint32_t (&r)[32]) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int j = 0; j < 32; ++j) stg[lane * 33 + j] = __uint_as_float(r[j]);
    __syncwarp();
    const int col = col0 + lane;
    const int rows = min(32, a.m - row0);
    if (col < a.n)
        for (int i = 0; i < rows; ++i) a.c[(size_t)(row0 + i) * a.ldc + col] = stg[i * 33 + lane];
    __syncwarp();
}

template <int EPI, int CG>
__global__ void __launch_bounds__(kGemmThreads, 1) k_gemm_p(const __grid_constant__ PGemmGroup G) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    const int S = G.stages, BN = G.bn, BNc = BN / CG;  // BNc: rows of each B tile this CTA holds
    const int T = G.kts;
    // stage: T A tiles (128 x 64) then T B tiles (BNc x 64), each a 128-byte-swizzled K-major tile
    const uint32_t a_bytes = (uint32_t)(T * kABytes), b_tile = (uint32_t)BNc * kBK * 2;
    const uint32_t stage_bytes = a_bytes + (uint32_t)T * b_tile;
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + (size_t)S * stage_bytes);
    uint64_t* empty = full + kPStages;
    uint64_t* tfull = empty + kPStages;  // [2] accumulator b holds a finished tile
    uint64_t* tempty = tfull + 2;        // [2] accumulator b was read by the epilogue
    uint64_t* done = tempty + 2;         // every MMA issued by this CTA has completed
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);
    float* epi_stage = reinterpret_cast<float*>(smem + (size_t)S * stage_bytes + kPBarBytes);  // [4][32][33]
    __shared__ int s_err;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // CG = 2: the two CTAs of a cluster share each tile; rank 0 issues the MMAs.  Its `full`
    // barriers count both CTAs' bytes and its `tempty` barriers both CTAs' epilogue warps; the
    // commits that release a stage or a finished accumulator arrive in both CTAs.
    const int rank = CG == 2 ? (int)cluster_rank() : 0;
    const int cid = (int)blockIdx.x / CG, nctas = (int)gridDim.x / CG;
    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&tfull[b], 1);
            mbar_init(&tempty[b], 4 * CG);
        }
        mbar_init(done, 1);
        s_err = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        if constexpr (CG == 2) {
            tc::tmem_alloc_pair(tmem_slot, kPTmemCols);
            tc::tmem_relinquish_pair();
        } else {
            tc::tmem_alloc(tmem_slot, kPTmemCols);
            tc::tmem_relinquish();
        }
    }
    tc::fence_before();
    if constexpr (CG == 2) cluster_sync();  // the peer's barriers exist before any copy or commit reaches them
    else __syncthreads();
    tc::fence_after();
    const uint32_t tmem = *tmem_slot;
    uint32_t* status = G.a[0].status;
    auto abort_cta = [&]() {
        s_err = 1;
        set_status(status, VT_DEV_WAIT_TIMEOUT);
    };
    // cluster addresses of rank 0's barriers (this CTA's own when CG = 1)
    const uint32_t full0 = CG == 2 ? dsmem_addr(full, 0) : smem_u32(full);
    const uint32_t tempty0 = CG == 2 ? dsmem_addr(tempty, 0) : smem_u32(tempty);

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            pdl_wait();  // A was written by the preceding kernel
            uint32_t k = 0;  // stages filled so far
            for (int t = cid; t < G.total_tiles && !*(volatile int*)&s_err; t += nctas) {
                int g, m0, n0;
                ptile(G, t, g, m0, n0);
                const GemmArgs& a = G.a[g];
                for (int kt = 0; kt < a.k_tiles; kt += T, ++k) {
                    const int s = (int)(k % (uint32_t)S);
                    if (k >= (uint32_t)S && !mbar_wait(&empty[s], ((k / S) - 1) & 1)) {
                        abort_cta();
                        break;
                    }
                    if (*(volatile int*)&s_err) break;
                    uint8_t* st = smem + (size_t)s * stage_bytes;
                    // a 3-D box past the last k-tile is filled with zeros and still counts its bytes
                    const uint32_t fb = full0 + (uint32_t)s * 8;
                    const int ya = m0 + rank * kBM, yb = n0 + rank * BNc, kb = bk_tile(a, kt);
                    if constexpr (CG == 2) {
                        // rank 0 expects both CTAs' bytes; each CTA loads its own A rows and B half
                        if (rank == 0) mbar_arrive_expect_tx(&full[s], 2 * stage_bytes);
                        if (T == 2) {
                            tc::tma_load_3d_pair(st, &G.ta[g], ya, kt, fb);
                            tc::tma_load_3d_pair(st + a_bytes, &G.tb[g], yb, kb, fb);
                        } else {
                            tc::tma_load_2d_pair(st, &G.ta[g], kt * kBK, ya, fb);
                            tc::tma_load_2d_pair(st + a_bytes, &G.tb[g], kb * kBK, yb, fb);
                        }
                    } else {
                        mbar_arrive_expect_tx(&full[s], stage_bytes);
                        if (T == 2) {
                            tc::tma_load_3d(st, &G.ta[g], ya, kt, fb);
                            tc::tma_load_3d(st + a_bytes, &G.tb[g], yb, kb, fb);
                        } else {
                            tc::tma_load_2d(st, &G.ta[g], kt * kBK, ya, &full[s]);
                            tc::tma_load_2d(st + a_bytes, &G.tb[g], kb * kBK, yb, &full[s]);
                        }
                    }
                }
            }
            // no copy may be in flight when the CTA ends (rank 0's barriers count both CTAs' copies;
            // the final cluster barrier keeps the peer until then)
            if (rank == 0)
                for (uint32_t i = k > (uint32_t)S ? k - S : 0; i < k; ++i)
                    if (!mbar_wait(&full[i % S], (i / S) & 1)) set_status(status, VT_DEV_WAIT_TIMEOUT);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer (rank 0)
        if (lane == 0 && rank == 0) {
            uint32_t k = 0;
            int it = 0;
            for (int t = cid; t < G.total_tiles && !*(volatile int*)&s_err; t += nctas, ++it) {
                int g, m0, n0;
                ptile(G, t, g, m0, n0);
                const GemmArgs& a = G.a[g];
                const int buf = it & 1;
                if (it >= 2 && !(CG == 2 ? mbar_wait_cluster(&tempty[buf], ((it >> 1) - 1) & 1)
                                         : mbar_wait(&tempty[buf], ((it >> 1) - 1) & 1))) {
                    abort_cta();
                    break;
                }
                tc::fence_after();
                const uint32_t d_tmem = tmem + (uint32_t)(buf * 256);
                const uint32_t idesc = tc::idesc_f16(kBM * CG, BN);
                bool ok = true;
                for (int kt = 0; kt < a.k_tiles; kt += T, ++k) {
                    const int s = (int)(k % (uint32_t)S);
                    if (!mbar_wait(&full[s], (k / S) & 1)) {
                        ok = false;
                        break;
                    }
                    tc::fence_after();
                    const uint32_t s0 = smem_u32(smem + (size_t)s * stage_bytes);
                    for (int j = 0; j < T && kt + j < a.k_tiles; ++j) {
                        const uint32_t sa = s0 + (uint32_t)j * kABytes, sb = s0 + a_bytes + (uint32_t)j * b_tile;
#pragma unroll
                        for (int kk = 0; kk < kBK / 16; ++kk) {
                            if constexpr (CG == 2)
                                tc::mma_f16_pair(d_tmem, tc::desc_sw128(sa + kk * 32), tc::desc_sw128(sb + kk * 32), idesc,
                                                 (kt + j | kk) != 0);
                            else
                                tc::mma_f16(d_tmem, tc::desc_sw128(sa + kk * 32), tc::desc_sw128(sb + kk * 32), idesc,
                                            (kt + j | kk) != 0);
                        }
                    }
                    if constexpr (CG == 2) tc::mma_commit_pair_both(&empty[s]);
                    else tc::mma_commit(&empty[s]);
                }
                if (!ok) {
                    abort_cta();
                    break;
                }
                if constexpr (CG == 2) tc::mma_commit_pair_both(&tfull[buf]);
                else tc::mma_commit(&tfull[buf]);
            }
            if constexpr (CG == 2) tc::mma_commit_pair(done);
            else tc::mma_commit(done);
            if (!mbar_wait(done, 0)) set_status(status, VT_DEV_WAIT_TIMEOUT);
        }
    } else {
        // ------------------------------------------------------------ epilogue (warps 2-5)
        const int sub = warp & 3;  // accumulator lanes [32 sub, 32 sub + 32)
        int it = 0;
        for (int t = cid; t < G.total_tiles; t += nctas, ++it) {
            int g, m0, n0;
            ptile(G, t, g, m0, n0);
            const GemmArgs& a = G.a[g];
            const int buf = it & 1;
            int ok = 1;
            if (lane == 0) ok = mbar_wait(&tfull[buf], (it >> 1) & 1) && !*(volatile int*)&s_err;
            ok = __shfl_sync(0xffffffffu, ok, 0);
            if (!ok) {
                if (lane == 0) abort_cta();
                break;
            }
            tc::fence_after();
            const int row = m0 + rank * kBM + sub * 32 + lane;
            int pos = 0;
            bool row_ok = row < a.m;
            if constexpr (EPI == kGemmQkv) {
                pos = *a.len + a.row_offset + row;
                if (row_ok && (pos < 0 || pos >= a.cap)) {
                    set_status(a.status, VT_DEV_KV_OVERFLOW);
                    row_ok = false;
                }
            }
            const uint32_t base = tmem + ((uint32_t)(sub * 32) << 16) + (uint32_t)(buf * 256);
            for (int c = 0; c < BN; c += 32) {
                uint32_t r[32];
                tc::tmem_ld32(base + (uint32_t)c, r);  // warp-collective: every lane takes part
                tc::tmem_ld_wait();
                if constexpr (EPI == kGemmF32) {
                    if (n0 + c < a.n) pepi_f32_rows(a, epi_stage + sub * (32 * 33), row - lane, n0 + c, r);
                } else {
                    if (row_ok && n0 + c < a.n) pepi_chunk<EPI>(a, row, n0 + c, r, pos);
                }
            }
            tc::fence_before();
            __syncwarp();
            if (lane == 0) {
                if constexpr (CG == 2) mbar_arrive_cluster(tempty0 + (uint32_t)buf * 8);
                else mbar_arrive(&tempty[buf]);
            }
        }
    }
    tc::fence_before();
    // no CTA of a pair leaves while the other may still copy into its barriers or write its accumulators
    if constexpr (CG == 2) cluster_sync();
    else __syncthreads();
    if (warp == 1) {
        tc::fence_after();
        if constexpr (CG == 2) tc::tmem_dealloc_pair(tmem, kPTmemCols);
        else tc::tmem_dealloc(tmem, kPTmemCols);
    }
}

// Tile width of the single-CTA persistent GEMM: 128 x 256.  Its ring moves 384 lines of 128 bytes
// (A 128 + B 256) per k-tile through shared memory, which the copy engine delivers at about half a
// line per cycle (measured: a stage of that size fills in 600-700 cycles), against 512 cycles of
// MMA; narrower tiles do less MMA work per line, so the widest is the fastest (measured against
// 128, 160 and 192 on the 7B prefill).
constexpr int kPBn = 256;

// bn_cta: rows of the B tile one CTA holds (the tile width, or half of it for a CTA pair);
// kts: k-tiles per stage
static size_t pgemm_stage_bytes(int bn_cta, int kts) { return (size_t)kts * ((size_t)kABytes + (size_t)bn_cta * kBK * 2); }
static int pgemm_stages(int bn_cta, int kts) {
    // the launch may use kPGemmSmem - 1024 bytes, 1024 of them lost to aligning the ring
    const size_t room = kPGemmSmem - 2048 - kPBarBytes - kPEpiBytes;
    int s = (int)(room / pgemm_stage_bytes(bn_cta, kts));
    return s > kPStages ? kPStages : s;
}

__device__ __forceinline__ uint32_t pack_h2(float lo, float hi) {
    const __half2 h = __floats2half2_rn(lo, hi);
    return *reinterpret_cast<const uint32_t*>(&h);
}

// ================================================================== causal attention on tcgen05
//
// One CTA per (query head, 128-row tile); the launch covers every shard's heads (up to kFaGroups
// shards).  The attended positions [kbeg, kend) of the tile are walked in blocks of 128 keys:
//   S_j = Q . K_j^T           (tcgen05, M 128, N 128, K dh; fp32 in tensor memory)
//   P_j = 2^(S_j log2(e)/sqrt(dh) - m), masked (causal, window), fp16 into shared memory
//   O  += P_j . V_j           (tcgen05, M 128, N dh, K 128, one accumulator in tensor memory; V
//                              read MN-major as it lies in the cache, so it needs no transpose)
//   warp 0      TMA: one thread loads Q, then serves the K and V rings (two slots each), filling
//               each slot as soon as the MMA that read it has completed;
//   warp 1      tensor memory (S of even / odd blocks, O) and the MMA thread: S_0, S_1, then per
//               block O += P_j V_j and S_{j+2} (S_{j+2} first when its operands are already there);
//   warps 2-9   softmax: warp (g, q) holds query rows 32q .. 32q + 31 (its quarter of the tensor
//               memory lanes) and key columns 64g .. 64g + 63 of every block; the two warps of a
//               quarter exchange row maxima through shared memory.  m is a reference maximum: O
//               (in tensor memory) and l are rescaled only when a row's block maximum exceeds it
//               by more than 8 (log2 units), so P stays below 2^8.
// Keys past the window or the causal bound, and rows past n (zero Q from TMA's fill), take no
// part in any stored result; V rows outside [kbeg, kend) meet zero weights (the cache holds finite
// values: zeroed at creation, written by the QKV epilogues).  Every wait is bounded; on a timeout
// the CTA sets VT_DEV_WAIT_TIMEOUT and stops issuing, waits for what it issued and frees tensor
// memory; the softmax warps still pass every named barrier, so no partner waits on them.
constexpr int kFaRows = 128, kFaKeys = 128;
constexpr int kFaThreads = 320;
constexpr int kFaGroups = 6;  // four tensor maps a shard: 6 keep the parameters under 4 KB

struct FaShard {
    int n, hq, group, cap, row_offset, window;
    const int32_t* len;  // rows sit at positions *len + row_offset + i
    float scale_log2;
    __half* out;         // [n][hq * dh]
    uint32_t* status;
};
struct FaGroup {
    int n_groups;
    int head_end[kFaGroups];
    CUtensorMap tq[kFaGroups], tk[kFaGroups], tv[kFaGroups];  // q [n][hq dh], K / V [hk cap][dh]
    CUtensorMap to[kFaGroups];                                 // the output [n][hq dh]
    FaShard a[kFaGroups];
};

static_assert(sizeof(FaGroup) <= 4096, "the attention launch's parameters must fit in 4 KB");

// Q, two K and two V slots, two P slots, the max exchange (2 x 128 floats), barriers
template <int DH>
constexpr size_t fa_smem() {
    return 1024 + (size_t)kFaRows * DH * 2 + 4 * (size_t)kFaKeys * DH * 2 + 2 * (size_t)kFaRows * kFaKeys * 2 +
           2 * kFaRows * 4 + 256;
}

// bounded wait polled by lane 0, result broadcast to the warp
__device__ __forceinline__ bool fa_wait_warp(uint64_t* bar, uint32_t parity) {
    int ok = 1;
    if ((threadIdx.x & 31) == 0) ok = mbar_wait(bar, parity) ? 1 : 0;
    return __shfl_sync(0xffffffffu, ok, 0) != 0;
}
// one non-blocking test of a phase
__device__ __forceinline__ bool fa_test(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\tselp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}
__device__ __forceinline__ void fa_pair_sync(uint32_t id) { asm volatile("bar.sync %0, 64;" ::"r"(id) : "memory"); }

// 2^x on the special-function unit (inputs far below -126 and -inf give 0)
__device__ __forceinline__ float fa_ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
__device__ __forceinline__ float fa_max3(float a, float b, float c) {
    float d;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}

// bits [b, e) of a 32-bit word, b and e clamped to [0, 32]
__device__ __forceinline__ uint32_t fa_range_bits(int b, int e) {
    b = max(0, min(32, b));
    e = max(0, min(32, e));
    if (e <= b) return 0u;
    const uint32_t below_e = e == 32 ? 0xffffffffu : ((1u << e) - 1u);
    return below_e & ~((1u << b) - 1u);
}

template <int DH>
__global__ void __launch_bounds__(kFaThreads, 1) k_prefill_attn_tc(const __grid_constant__ FaGroup G) {
    constexpr uint32_t kQBytes = kFaRows * DH * 2, kKVBytes = kFaKeys * DH * 2, kPBytes = kFaRows * kFaKeys * 2;
    constexpr uint32_t kAtom = kFaRows * 128;  // one 64-column box of 128 rows
    constexpr uint32_t kOCol = 2 * kFaKeys;    // O's first tensor-memory column (after the two S)
    const int hg = (int)blockIdx.x;
    int gi = 0;
    while (gi + 1 < G.n_groups && hg >= G.head_end[gi]) ++gi;
    const FaShard& a = G.a[gi];
    const int h = hg - (gi > 0 ? G.head_end[gi - 1] : 0), kvh = h / a.group;
    const int r0 = ((int)gridDim.y - 1 - (int)blockIdx.y) * kFaRows;  // heaviest tiles first

    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    uint8_t* Qs = smem;
    uint8_t* Ks = Qs + kQBytes;       // [2][kKVBytes]
    uint8_t* Vs = Ks + 2 * kKVBytes;  // [2][kKVBytes]
    uint8_t* Ps = Vs + 2 * kKVBytes;  // [2][kPBytes]
    float* red = reinterpret_cast<float*>(Ps + 2 * kPBytes);  // [2 column halves][128 rows]
    uint64_t* bars = reinterpret_cast<uint64_t*>(red + 2 * kFaRows);
    uint64_t* q_full = bars;
    uint64_t* k_full = bars + 1;   // [2]
    uint64_t* v_full = bars + 3;   // [2]
    uint64_t* k_empty = bars + 5;  // [2]
    uint64_t* v_empty = bars + 7;  // [2]
    uint64_t* s_full = bars + 9;   // [2]
    uint64_t* s_free = bars + 11;  // [2]
    uint64_t* p_full = bars + 13;  // [2]
    uint64_t* o_full = bars + 15;  // [2]: O += P_j V_j has completed, j even / odd
    uint64_t* done = bars + 17;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 18);
    volatile int* s_err = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        mbar_init(q_full, 1);
        for (int s = 0; s < 2; ++s) {
            mbar_init(&k_full[s], 1);
            mbar_init(&v_full[s], 1);
            mbar_init(&k_empty[s], 1);
            mbar_init(&v_empty[s], 1);
            mbar_init(&s_full[s], 1);
            mbar_init(&s_free[s], 8);  // one arrival per softmax warp
            mbar_init(&p_full[s], 8);
            mbar_init(&o_full[s], 1);
        }
        mbar_init(done, 1);
        *s_err = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tc::tmem_alloc(tmem_slot, 512);
        tc::tmem_relinquish();
    }
    tc::fence_before();
    __syncthreads();
    tc::fence_after();
    const uint32_t tmem = *tmem_slot;

    pdl_wait();  // q and the cache rows were written by the preceding kernel
    // Q does not depend on the KV length: its load goes out first
    if (warp == 0 && lane == 0 && r0 < a.n) {
        mbar_arrive_expect_tx(q_full, kQBytes);
        for (int c = 0; c < DH / 64; ++c) tc::tma_load_2d(Qs + c * kAtom, &G.tq[gi], h * DH + 64 * c, r0, q_full);
    }
    const int P0 = *a.len + a.row_offset;
    const int rlast = min(r0 + kFaRows - 1, a.n - 1);
    const int kend = min(P0 + rlast + 1, a.cap);
    const int kbeg = a.window > 0 ? max(0, P0 + r0 - a.window + 1) : 0;
    const int nb = kend > kbeg ? (kend - kbeg + kFaKeys - 1) / kFaKeys : 0;

    if (warp == 0) {
        if (lane == 0 && nb == 0) mbar_wait(q_full, 0);  // no copy may be in flight when the CTA ends
        if (lane == 0 && nb > 0) {
            // one thread serves both rings, each load as soon as its slot is free (a blocked wait on
            // one ring would hold up the other); V_j goes out after K_{j+1}, so that the copies the
            // first MMAs need (Q, K_0, K_1) are ahead of V in the copy engine
            const int krow0 = kvh * a.cap + kbeg;
            auto load = [&](bool is_v, int j) {
                const int s = j & 1;
                uint64_t* full = is_v ? &v_full[s] : &k_full[s];
                mbar_arrive_expect_tx(full, kKVBytes);
                for (int c = 0; c < DH / 64; ++c)
                    tc::tma_load_2d((is_v ? Vs : Ks) + s * kKVBytes + c * kAtom, is_v ? &G.tv[gi] : &G.tk[gi], 64 * c,
                                    krow0 + j * kFaKeys, full);
            };
            int jk = 0, jv = 0;
            uint32_t idle = 0;
            bool ok = true;
            while (jk < nb || jv < nb) {
                bool moved = false;
                if (jk < nb && (jk < 2 || fa_test(&k_empty[jk & 1], ((jk - 2) >> 1) & 1))) {
                    load(false, jk++);
                    moved = true;
                }
                if (jv < nb && (jk > jv + 1 || jk == nb) && (jv < 2 || fa_test(&v_empty[jv & 1], ((jv - 2) >> 1) & 1))) {
                    load(true, jv++);
                    moved = true;
                }
                if (moved) {
                    idle = 0;
                } else if (++idle > (kSpinLimit << 2) || *s_err) {
                    ok = false;
                    break;
                }
            }
            if (!ok) {
                *s_err = 1;
                set_status(a.status, VT_DEV_WAIT_TIMEOUT);
                // no copy may still be in flight when the CTA ends
                mbar_wait(q_full, 0);
                for (int j = jk > 2 ? jk - 2 : 0; j < jk; ++j) mbar_wait(&k_full[j & 1], (j >> 1) & 1);
                for (int j = jv > 2 ? jv - 2 : 0; j < jv; ++j) mbar_wait(&v_full[j & 1], (j >> 1) & 1);
            }
        }
    } else if (warp == 1) {
        if (lane == 0 && nb > 0) {
            constexpr uint32_t idesc_s = tc::idesc_f16(kFaRows, kFaKeys);
            constexpr uint32_t idesc_o = tc::idesc_f16_bmn(kFaRows, DH);
            const uint32_t qa = smem_u32(Qs), ka = smem_u32(Ks), va = smem_u32(Vs), pa = smem_u32(Ps);
            auto qk = [&](int j) -> bool {
                const int s = j & 1;
                if (!mbar_wait(&k_full[s], (j >> 1) & 1)) return false;
                if (j >= 2 && !mbar_wait(&s_free[s], ((j - 2) >> 1) & 1)) return false;
                if (*s_err) return false;
                tc::fence_after();
#pragma unroll
                for (int kk = 0; kk < DH / 16; ++kk) {
                    const uint32_t off = (uint32_t)(kk >> 2) * kAtom + (uint32_t)(kk & 3) * 32;
                    tc::mma_f16(tmem + (uint32_t)(s * kFaKeys), tc::desc_sw128(qa + off),
                                tc::desc_sw128(ka + s * kKVBytes + off), idesc_s, kk > 0);
                }
                tc::mma_commit(&k_empty[s]);
                tc::mma_commit(&s_full[s]);
                return true;
            };
            auto qk_ready = [&](int j) -> bool {
                return fa_test(&k_full[j & 1], (j >> 1) & 1) && (j < 2 || fa_test(&s_free[j & 1], ((j - 2) >> 1) & 1));
            };
            auto pv = [&](int j) -> bool {
                const int s = j & 1;
                if (!mbar_wait(&v_full[s], (j >> 1) & 1)) return false;
                if (!mbar_wait(&p_full[s], (j >> 1) & 1)) return false;
                if (*s_err) return false;
                tc::fence_after();
#pragma unroll
                for (int kk = 0; kk < kFaKeys / 16; ++kk)
                    tc::mma_f16(tmem + kOCol,
                                tc::desc_sw128(pa + s * kPBytes + (uint32_t)(kk >> 2) * kAtom + (uint32_t)(kk & 3) * 32),
                                tc::desc_sw128_mn(va + s * kKVBytes + (uint32_t)kk * 2048, kAtom), idesc_o,
                                (j > 0 || kk > 0) ? 1u : 0u);
                tc::mma_commit(&v_empty[s]);
                tc::mma_commit(&o_full[s]);
                return true;
            };
            bool ok = mbar_wait(q_full, 0);
            ok = ok && qk(0);
            if (ok && nb > 1) ok = qk(1);
            for (int j = 0; ok && j < nb; ++j) {
                bool issued = false;
                if (j + 2 < nb && qk_ready(j + 2)) {
                    ok = qk(j + 2);
                    issued = true;
                }
                ok = ok && pv(j);
                if (ok && j + 2 < nb && !issued) ok = qk(j + 2);
            }
            if (!ok) {
                *s_err = 1;
                set_status(a.status, VT_DEV_WAIT_TIMEOUT);
            }
            // tensor memory is freed only after every MMA issued has completed
            tc::mma_commit(done);
            if (!mbar_wait(done, 0)) set_status(a.status, VT_DEV_WAIT_TIMEOUT);
        }
    } else {
        const int g = (warp - 2) >> 2, quad = warp & 3, row = quad * 32 + lane;
        const uint32_t lane_off = (uint32_t)(quad * 32) << 16, pair = 1u + (uint32_t)quad;
        const int qp = P0 + r0 + row;
        const int lo = a.window > 0 ? qp - a.window + 1 : INT_MIN;
        const float sl2 = a.scale_log2;
        float m_use = -INFINITY, l = 0.f;
        bool ok = true;
        for (int j = 0; j < nb; ++j) {
            const int s = j & 1;
            if (ok && *s_err) ok = false;
            if (ok) ok = fa_wait_warp(&s_full[s], (j >> 1) & 1);
            // this warp's 64 columns of S_j and their attended range [cb, ce)
            const int kp0 = kbeg + j * kFaKeys + 64 * g;
            const int cb = a.window > 0 ? max(0, min(64, lo - kp0)) : 0;
            const int ce = max(0, min(64, qp - kp0 + 1));
            uint32_t sv[2][32];
            float pm = -INFINITY;
            if (ok) {
                tc::fence_after();
                const uint32_t at = tmem + lane_off + (uint32_t)(s * kFaKeys + 64 * g);
                tc::tmem_ld32(at, sv[0]);
                tc::tmem_ld32(at + 32, sv[1]);
                tc::tmem_ld_wait_on(sv[0]);
                tc::tmem_ld_wait_on(sv[1]);
                tc::fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&s_free[s]);  // S is in registers: the slot may take S_{j+2}
#pragma unroll
                for (int c = 0; c < 2; ++c) {
                    const uint32_t mw = fa_range_bits(cb - 32 * c, ce - 32 * c);
                    if (__all_sync(0xffffffffu, mw == 0xffffffffu)) {
#pragma unroll
                        for (int e = 0; e < 32; e += 2)
                            pm = fa_max3(pm, __uint_as_float(sv[c][e]), __uint_as_float(sv[c][e + 1]));
                    } else {
#pragma unroll
                        for (int e = 0; e < 32; ++e)
                            if ((mw >> e) & 1u) pm = fmaxf(pm, __uint_as_float(sv[c][e]));
                    }
                }
            }
            // the row maximum over both column halves (every warp passes both barriers)
            red[g * kFaRows + row] = pm;
            fa_pair_sync(pair);
            const float bms = fmaxf(pm, red[(1 - g) * kFaRows + row]) * sl2;
            fa_pair_sync(pair);
            // O += P_{j-2} V_{j-2} has completed: P_j's slot is free
            if (ok && j >= 2) ok = fa_wait_warp(&o_full[s], ((j - 2) >> 1) & 1);
            if (!ok) continue;
            float alpha = 1.f;
            bool resc = false;
            if (bms > m_use + 8.f) {
                if (m_use != -INFINITY) {
                    alpha = fa_ex2(m_use - bms);
                    resc = true;
                }
                m_use = bms;
            }
            if (__any_sync(0xffffffffu, resc)) {
                // O holds every earlier block once O += P_{j-1} V_{j-1} has completed
                if (j >= 1 && !fa_wait_warp(&o_full[(j - 1) & 1], ((j - 1) >> 1) & 1)) {
                    ok = false;
                    continue;
                }
                tc::fence_after();
#pragma unroll
                for (int c = 0; c < DH / 64; ++c) {
                    const uint32_t at = tmem + lane_off + kOCol + (uint32_t)(g * (DH / 2) + 32 * c);
                    uint32_t o[32];
                    tc::tmem_ld32(at, o);
                    tc::tmem_ld_wait_on(o);
#pragma unroll
                    for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
                    tc::tmem_st32(at, o);
                }
                tc::tmem_st_wait();
            }
            l *= alpha;
            // P_j: this warp's 64 keys are box g of the slot (row `row`, 128-byte swizzle)
            uint8_t* prow = Ps + s * kPBytes + g * kAtom + row * 128;
            const float nm = -m_use;
            float ls0 = 0.f, ls1 = 0.f;
#pragma unroll
            for (int c = 0; c < 2; ++c) {
                const uint32_t mw = fa_range_bits(cb - 32 * c, ce - 32 * c);
                uint32_t w[16];
                if (__all_sync(0xffffffffu, mw == 0xffffffffu)) {
#pragma unroll
                    for (int e = 0; e < 16; ++e) {
                        const float p0 = fa_ex2(fmaf(__uint_as_float(sv[c][2 * e]), sl2, nm));
                        const float p1 = fa_ex2(fmaf(__uint_as_float(sv[c][2 * e + 1]), sl2, nm));
                        ls0 += p0;
                        ls1 += p1;
                        w[e] = pack_h2(p0, p1);
                    }
                } else {
#pragma unroll
                    for (int e = 0; e < 16; ++e) {
                        const float x0 = ((mw >> (2 * e)) & 1u) ? fmaf(__uint_as_float(sv[c][2 * e]), sl2, nm) : -INFINITY;
                        const float x1 =
                            ((mw >> (2 * e + 1)) & 1u) ? fmaf(__uint_as_float(sv[c][2 * e + 1]), sl2, nm) : -INFINITY;
                        const float p0 = fa_ex2(x0), p1 = fa_ex2(x1);
                        ls0 += p0;
                        ls1 += p1;
                        w[e] = pack_h2(p0, p1);
                    }
                }
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int chunk = c * 4 + u;
                    *reinterpret_cast<uint4*>(prow + ((chunk ^ (row & 7)) << 4)) =
                        make_uint4(w[4 * u], w[4 * u + 1], w[4 * u + 2], w[4 * u + 3]);
                }
            }
            l += ls0 + ls1;
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            tc::fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&p_full[s]);
        }
        if (ok && nb > 0) ok = fa_wait_warp(done, 0);  // every MMA has completed
        if (!ok && lane == 0) {
            *s_err = 1;
            set_status(a.status, VT_DEV_WAIT_TIMEOUT);
        }
        tc::fence_after();
        // l over both column halves (the same reference maximum)
        red[g * kFaRows + row] = l;
        fa_pair_sync(pair);
        const float lt = l + red[(1 - g) * kFaRows + row];
        const float inv = lt > 0.f ? 1.f / lt : 0.f;
        if (ok) {
            // this warp's half of the row, O columns [g dh/2, (g + 1) dh/2), as fp16 into Q's slot
            // (free once every MMA is done) in the output's 64-column boxes, 128-byte swizzle
            uint32_t o[DH / 64][32];
#pragma unroll
            for (int c = 0; c < DH / 64; ++c) {
                if (nb > 0) tc::tmem_ld32(tmem + lane_off + kOCol + (uint32_t)(g * (DH / 2) + 32 * c), o[c]);
                else
#pragma unroll
                    for (int e = 0; e < 32; ++e) o[c][e] = 0u;
            }
#pragma unroll
            for (int c = 0; c < DH / 64; ++c) tc::tmem_ld_wait_on(o[c]);
#pragma unroll
            for (int c = 0; c < DH / 64; ++c)
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    uint32_t w[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e)
                        w[e] = pack_h2(__uint_as_float(o[c][8 * u + 2 * e]) * inv, __uint_as_float(o[c][8 * u + 2 * e + 1]) * inv);
                    const int col = g * (DH / 2) + 32 * c + 8 * u, box = col >> 6, chunk = (col & 63) >> 3;
                    *reinterpret_cast<uint4*>(Qs + box * kAtom + row * 128 + ((chunk ^ (row & 7)) << 4)) =
                        make_uint4(w[0], w[1], w[2], w[3]);
                }
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        }
        // every softmax warp has staged its part (or has given up): one thread stores the boxes
        asm volatile("bar.sync 5, %0;" ::"n"(kFaThreads - 64) : "memory");
        if (warp == 2 && lane == 0 && !*s_err) {
            for (int c = 0; c < DH / 64; ++c) tc::tma_store_2d(&G.to[gi], h * DH + 64 * c, r0, Qs + c * kAtom);
            asm volatile("cp.async.bulk.commit_group;" ::: "memory");
            asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");  // the slot has been read
        }
    }
    tc::fence_before();
    __syncthreads();
    if (warp == 1) {
        tc::fence_after();
        tc::tmem_dealloc(tmem, 512);
    }
}

// ================================================================== host side

static PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
static bool g_gemm_persistent = true;  // VT_GEMM_PERSISTENT=0 keeps every GEMM on k_gemm
static int g_pgemm_pairs = 0;          // co-resident CTA pairs of the persistent GEMM (0: single CTAs)
constexpr int kMaxSplit = 4;
static int g_split_clusters[kMaxSplit + 1];  // co-resident clusters of S GEMM CTAs (index S)

cudaError_t init_prefill_kernels() {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q{};
    cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
    if (e != cudaSuccess) return e;
    if (q != cudaDriverEntryPointSuccess || !fn) return cudaErrorNotSupported;
    g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    if ((e = cudaFuncSetAttribute(k_gemm<kGemmF32>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kGemmSmem)) != cudaSuccess)
        return e;
    if ((e = cudaFuncSetAttribute(k_gemm<kGemmQkv>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kGemmSmem)) != cudaSuccess)
        return e;
    if ((e = cudaFuncSetAttribute(k_gemm<kGemmSwiglu>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kGemmSmem)) != cudaSuccess)
        return e;
    // how many clusters of S GEMM CTAs fit at once (the split factor's wave size)
    for (int sp = 2; sp <= kMaxSplit; ++sp) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(1, 1, sp * 64);
        cfg.blockDim = dim3(kGemmThreads);
        cfg.dynamicSmemBytes = kGemmSmem;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = 1;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = sp;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        int nc = 0;
        if (cudaOccupancyMaxActiveClusters(&nc, k_gemm<kGemmF32>, &cfg) != cudaSuccess) {
            cudaGetLastError();
            nc = 0;
        }
        g_split_clusters[sp] = nc;
    }
    for (auto f : {k_gemm_p<kGemmF32, 1>, k_gemm_p<kGemmQkv, 1>, k_gemm_p<kGemmSwiglu, 1>, k_gemm_p<kGemmF32, 2>,
                   k_gemm_p<kGemmQkv, 2>, k_gemm_p<kGemmSwiglu, 2>})
        if ((e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)(kPGemmSmem - 1024))) != cudaSuccess)
            return e;
    {
        const char* v = getenv("VT_GEMM_PERSISTENT");
        g_gemm_persistent = !(v && v[0] == '0');
        // VT_GEMM_PAIR=0 keeps the persistent GEMM on single CTAs
        const char* pv = getenv("VT_GEMM_PAIR");
        g_pgemm_pairs = 0;
        if (!(pv && pv[0] == '0')) {
            cudaLaunchConfig_t cfg = {};
            cfg.gridDim = dim3(2 * 64);
            cfg.blockDim = dim3(kGemmThreads);
            cfg.dynamicSmemBytes = kPGemmSmem - 1024;
            cudaLaunchAttribute attr[1];
            attr[0].id = cudaLaunchAttributeClusterDimension;
            attr[0].val.clusterDim.x = 2;
            attr[0].val.clusterDim.y = 1;
            attr[0].val.clusterDim.z = 1;
            cfg.attrs = attr;
            cfg.numAttrs = 1;
            int nc = 0;
            if (cudaOccupancyMaxActiveClusters(&nc, k_gemm_p<kGemmF32, 2>, &cfg) != cudaSuccess) {
                cudaGetLastError();
                nc = 0;
            }
            g_pgemm_pairs = nc;
        }
    }
    if ((e = cudaFuncSetAttribute(k_prefill_attn_tc<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)fa_smem<128>())) != cudaSuccess)
        return e;
    if ((e = cudaFuncSetAttribute(k_prefill_attn_tc<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)fa_smem<64>())) != cudaSuccess)
        return e;
    return cudaSuccess;
}

// K-major fp16 operand [rows][inner] with row stride `ld` elements, read in boxes of 64 x box_rows.
static bool make_map(CUtensorMap* map, const void* base, int64_t inner, int64_t rows, int64_t ld, int box_rows,
                     std::string* err) {
    if (!g_encode) {
        *err = "the tensor-map encoder is not available";
        return false;
    }
    if (((uintptr_t)base & 15) != 0 || (ld * 2) % 16 != 0) {
        *err = "a GEMM operand is not 16-byte aligned (base and row stride)";
        return false;
    }
    const cuuint64_t dims[2] = {(cuuint64_t)inner, (cuuint64_t)rows};
    const cuuint64_t strides[1] = {(cuuint64_t)ld * 2};
    const cuuint32_t box[2] = {(cuuint32_t)kBK, (cuuint32_t)box_rows};
    const cuuint32_t estr[2] = {1, 1};
    const CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(base), dims, strides, box,
                                estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                                CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
        *err = "cuTensorMapEncodeTiled failed (" + std::to_string((int)r) + ")";
        return false;
    }
    return true;
}

// The same operand as a 3-D map {64, rows, inner / 64} whose third dimension steps one k-tile
// (128 bytes), read in boxes of 64 x box_rows x 2: two consecutive k-tiles per copy.  inner must
// be a multiple of 64 (the box does not stop at the row's end).
static bool make_map_k2(CUtensorMap* map, const void* base, int64_t inner, int64_t rows, int64_t ld, int box_rows,
                        std::string* err) {
    if (!g_encode) {
        *err = "the tensor-map encoder is not available";
        return false;
    }
    if (((uintptr_t)base & 15) != 0 || (ld * 2) % 16 != 0 || inner % kBK != 0) {
        *err = "a GEMM operand is not 16-byte aligned or its K is not a multiple of 64";
        return false;
    }
    const cuuint64_t dims[3] = {(cuuint64_t)kBK, (cuuint64_t)rows, (cuuint64_t)(inner / kBK)};
    const cuuint64_t strides[2] = {(cuuint64_t)ld * 2, (cuuint64_t)kBK * 2};
    const cuuint32_t box[3] = {(cuuint32_t)kBK, (cuuint32_t)box_rows, 2};
    const cuuint32_t estr[3] = {1, 1, 1};
    const CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 3, const_cast<void*>(base), dims, strides, box,
                                estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                                CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
        *err = "cuTensorMapEncodeTiled (3-D) failed (" + std::to_string((int)r) + ")";
        return false;
    }
    return true;
}

// Split factor for `tiles` output tiles of `k_tiles` k-tiles, from a time model of one launch:
// per wave, a fixed cost (first loads, epilogue) plus the k-tiles of one split; with S > 1, the
// cluster reduction of the accumulators.  The constants are measured on GB300 (microseconds).
// k_tiles: the longest GEMM of the launch (its time); min_k_tiles: the shortest, which must still
// give every CTA of a split at least 4 k-tiles (a CTA without k-tiles has no accumulator).
static int choose_split(int tiles, int k_tiles, int min_k_tiles) {
    constexpr double kTile = 0.33, kFixed = 4.0, kReduce = 3.5;
    int best = 1;
    double best_t = 1e30;
    for (int s = 1; s <= kMaxSplit; ++s) {
        if (s > 1 && min_k_tiles / s < 4) break;
        const int per_wave = s == 1 ? g_num_sms : g_split_clusters[s];
        if (per_wave < 1) continue;
        const int waves = (tiles + per_wave - 1) / per_wave;
        const double t = waves * (kFixed + kTile * k_tiles / s) + (s > 1 ? kReduce : 0.0);
        if (t < best_t - 1e-9) {
            best = s;
            best_t = t;
        }
    }
    return best;
}

// One GEMM of a grouped launch: C_g = A_g . B_g^T with m rows (shared by the group), n_g columns
// and k_g inner elements; `base` carries the epilogue's pointers.
struct GemmSpec {
    const void* A;
    int64_t lda;
    const void* B;
    int64_t ldb;
    int n, k;
    GemmArgs base;
    int kb = 0;  // > 0: B has kb columns and A's k = 2 kb columns hold the hi and lo halves of the input
};


// Width of a CTA-pair tile (256 rows).  The copy engine's cost is per box rather than per byte
// (measured on GB300: a ring stage of one A box and one B box turns over in about 1000 cycles
// whether the boxes carry one k-tile or two), so a k-tile costs about 500 cycles of copying with
// two k-tiles per box, 900 with one, against 2w cycles of MMA; the width is the one whose rounds
// of tiles over the co-resident pairs cost least (ties to the wider).
static int choose_pair_bn(const GemmSpec* specs, int ng, int tiles_m, int pairs, int kts) {
    int best = 256;
    long best_cost = -1;
    for (int w = 256; w >= 128; w -= 32) {
        int tiles = 0;
        for (int g = 0; g < ng; ++g) tiles += tiles_m * ((specs[g].n + w - 1) / w);
        const long rounds = (tiles + pairs - 1) / pairs;
        const long cost = rounds * (long)std::max(2 * w, kts == 2 ? 500 : 900);
        if (best_cost < 0 || cost < best_cost) {
            best_cost = cost;
            best = w;
        }
    }
    return best;
}

// The grouped GEMMs of `specs` (all with m rows) as one persistent launch: one CTA (CG = 1) or
// one CTA pair (CG = 2, 256-row tiles) per SM or SM pair, or one per tile when there are fewer.
template <int EPI, int CG>
static vt_status run_gemm_persistent(const GemmSpec* specs, int ng, int m, cudaStream_t st, std::string* err) {
    PGemmGroup G{};
    G.n_groups = ng;
    G.tm = kBM * CG;
    G.tiles_m = (m + G.tm - 1) / G.tm;
    const int slots = CG == 2 ? g_pgemm_pairs : (g_num_sms > 0 ? g_num_sms : 148);
    // two k-tiles per box needs every K (and the wrap of a split GEMM) in whole pairs of k-tiles'
    // worth of columns: a 3-D box past K would read the next row instead of zeros
    G.kts = 2;
    for (int g = 0; g < ng; ++g)
        if (specs[g].k % kBK != 0 || (specs[g].kb > 0 && specs[g].kb % (2 * kBK) != 0)) G.kts = 1;
    G.bn = CG == 2 ? choose_pair_bn(specs, ng, G.tiles_m, slots, G.kts) : kPBn;
    G.stages = pgemm_stages(G.bn / CG, G.kts);
    int acc = 0;
    for (int g = 0; g < ng; ++g) {
        const GemmSpec& sp = specs[g];
        if (sp.kb > 0 && (sp.kb % kBK != 0 || sp.k != 2 * sp.kb)) {
            *err = "a split GEMM needs k = 2 kb with kb a multiple of 64";
            return VT_ERR_INVALID_ARG;
        }
        const bool ok = G.kts == 2
                            ? make_map_k2(&G.ta[g], sp.A, sp.k, m, sp.lda, kBM, err) &&
                                  make_map_k2(&G.tb[g], sp.B, sp.kb > 0 ? sp.kb : sp.k, sp.n, sp.ldb, G.bn / CG, err)
                            : make_map(&G.ta[g], sp.A, sp.k, m, sp.lda, kBM, err) &&
                                  make_map(&G.tb[g], sp.B, sp.kb > 0 ? sp.kb : sp.k, sp.n, sp.ldb, G.bn / CG, err);
        if (!ok) return VT_ERR_INVALID_ARG;
        GemmArgs& a = G.a[g];
        a = sp.base;
        a.m = m;
        a.n = sp.n;
        a.b = static_cast<const __half*>(sp.B);
        a.ldb = sp.ldb;
        a.k_tiles = (sp.k + kBK - 1) / kBK;
        a.kb_wrap = sp.kb > 0 ? sp.kb / kBK : 0;
        acc += G.tiles_m * ((sp.n + G.bn - 1) / G.bn);
        G.tile_end[g] = acc;
    }
    G.total_tiles = acc;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(CG * std::min(acc, slots)));
    cfg.blockDim = dim3(kGemmThreads);
    cfg.dynamicSmemBytes = 1024 + (size_t)G.stages * pgemm_stage_bytes(G.bn / CG, G.kts) + kPBarBytes + kPEpiBytes;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = CG;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = CG == 2 ? 1 : 0;
    const cudaError_t e = cudaLaunchKernelEx(&cfg, k_gemm_p<EPI, CG>, G);
    if (e != cudaSuccess) {
        *err = std::string("persistent GEMM launch failed: ") + cudaGetErrorString(e);
        return VT_ERR_CUDA;
    }
    return VT_OK;
}

// Launches the GEMMs of `specs` (all with m rows) kGemmGroups at a time.  A group with at least
// as many 128 x 256 tiles as half the SMs runs as one persistent launch (k_gemm_p); a smaller one
// (short prompts, a single shard) as one CTA, or split-K cluster, per output tile (k_gemm), so
// that its few tiles still spread over the GPU.
template <int EPI>
static vt_status run_gemm_group(const GemmSpec* specs, int n_specs, int m, cudaStream_t st, std::string* err) {
    for (int g0 = 0; g0 < n_specs; g0 += kGemmGroups) {
        const int ng = std::min(kGemmGroups, n_specs - g0);
        {
            int tiles = 0;
            for (int g = 0; g < ng; ++g) tiles += ((m + kBM - 1) / kBM) * ((specs[g0 + g].n + kBN - 1) / kBN);
            if (g_gemm_persistent && 2 * tiles >= (g_num_sms > 0 ? g_num_sms : 148)) {
                const vt_status r = g_pgemm_pairs > 0 ? run_gemm_persistent<EPI, 2>(specs + g0, ng, m, st, err)
                                                      : run_gemm_persistent<EPI, 1>(specs + g0, ng, m, st, err);
                if (r != VT_OK) return r;
                continue;
            }
        }
        GemmGroup G{};
        G.n_groups = ng;
        int tiles_n = 0, max_k_tiles = 1, min_k_tiles = 1 << 30;
        for (int g = 0; g < ng; ++g) {
            const GemmSpec& sp = specs[g0 + g];
            if (sp.kb > 0 && (sp.kb % kBK != 0 || sp.k != 2 * sp.kb)) {
                *err = "a split GEMM needs k = 2 kb with kb a multiple of 64";
                return VT_ERR_INVALID_ARG;
            }
            if (!make_map(&G.ta[g], sp.A, sp.k, m, sp.lda, kBM, err) ||
                !make_map(&G.tb[g], sp.B, sp.kb > 0 ? sp.kb : sp.k, sp.n, sp.ldb, kBN, err))
                return VT_ERR_INVALID_ARG;
            GemmArgs& a = G.a[g];
            a = sp.base;
            a.m = m;
            a.n = sp.n;
            a.b = static_cast<const __half*>(sp.B);
            a.ldb = sp.ldb;
            a.k_tiles = (sp.k + kBK - 1) / kBK;
            a.kb_wrap = sp.kb > 0 ? sp.kb / kBK : 0;
            max_k_tiles = std::max(max_k_tiles, a.k_tiles);
            min_k_tiles = std::min(min_k_tiles, a.k_tiles);
            tiles_n += (sp.n + kBN - 1) / kBN;
            G.tile_end[g] = tiles_n;
        }
        const int tiles_m = (m + kBM - 1) / kBM;
        const int split = choose_split(tiles_n * tiles_m, max_k_tiles, min_k_tiles);
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(tiles_n, tiles_m, split);
        cfg.blockDim = dim3(kGemmThreads);
        cfg.dynamicSmemBytes = kGemmSmem;
        cfg.stream = st;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = 1;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = split;
        cfg.attrs = attr;
        cfg.numAttrs = split > 1 ? 1 : 0;
        const cudaError_t e = cudaLaunchKernelEx(&cfg, k_gemm<EPI>, G);
        if (e != cudaSuccess) {
            *err = std::string("GEMM launch failed: ") + cudaGetErrorString(e);
            return VT_ERR_CUDA;
        }
    }
    return VT_OK;
}

template <int EPI>
static vt_status run_gemm(const void* A, int64_t lda, const void* B, int64_t ldb, int m, int n, int k,
                          const GemmArgs& base, cudaStream_t st, std::string* err) {
    const GemmSpec sp{A, lda, B, ldb, n, k, base};
    return run_gemm_group<EPI>(&sp, 1, m, st, err);
}

cudaError_t launch_rmsnorm_rows(const __half* x, const __half* gain, float eps, int rows, int d, __half* y,
                                int split, cudaStream_t st) {
    if (rows <= 0) return cudaSuccess;
    if (d % 8 != 0) return cudaErrorInvalidValue;
    k_rmsnorm_rows<<<rows, 256, 0, st>>>(x, gain, eps, d, y, split);
    return cudaGetLastError();
}

static vt_status run_rmsnorm(const __half* x, const __half* gain, float eps, int n, int d, __half* y, int split,
                             cudaStream_t st, std::string* err) {
    const cudaError_t e = launch_rmsnorm_rows(x, gain, eps, n, d, y, split, st);
    if (e != cudaSuccess) {
        *err = std::string("RMSNorm launch failed: ") + cudaGetErrorString(e);
        return VT_ERR_CUDA;
    }
    return VT_OK;
}

static GemmSpec qkv_spec(const PrefillAttnArgs& a) {
    GemmArgs g{};
    g.q = a.q;
    g.kcache = a.kcache;
    g.vcache = a.vcache;
    g.hq = a.hq;
    g.hk = a.hk;
    g.dh = a.dh;
    g.cap = a.cap;
    g.len = a.len;
    g.row_offset = a.row_offset;
    g.rope = a.rope;
    g.status = a.status;
    // A = [hi | lo] halves of the normalised input (2d columns), B = Wqkv read once per half
    return GemmSpec{a.xhat, 2 * a.d, a.wqkv, a.d, (a.hq + 2 * a.hk) * a.dh, 2 * a.d, g, a.d};
}

static GemmSpec o_spec(const PrefillAttnArgs& a) {
    GemmArgs o{};
    o.c = a.out;
    o.ldc = a.d;
    o.status = a.status;
    const int K = a.hq * a.dh;
    return GemmSpec{a.attn, K, a.wo, K, a.d, K, o};
}

// Causal attention of every shard of an ATTN block on tcgen05: one launch per kFaGroups shards.
static vt_status prefill_attention_tc(const PrefillAttnArgs* as, int n, cudaStream_t st, std::string* err) {
    for (int g0 = 0; g0 < n; g0 += kFaGroups) {
        const int ng = std::min(kFaGroups, n - g0);
        FaGroup G{};
        int heads = 0;
        for (int i = 0; i < ng; ++i) {
            const PrefillAttnArgs& a = as[g0 + i];
            FaShard& t = G.a[i];
            t.n = a.n;
            t.hq = a.hq;
            t.group = a.hq / a.hk;
            t.cap = a.cap;
            t.row_offset = a.row_offset;
            t.window = a.window;
            t.len = a.len;
            t.scale_log2 = a.scale_log2;
            t.out = a.attn;
            t.status = a.status;
            if (!make_map(&G.tq[i], a.q, (int64_t)a.hq * a.dh, a.n, (int64_t)a.hq * a.dh, kFaRows, err) ||
                !make_map(&G.tk[i], a.kcache, a.dh, (int64_t)a.hk * a.cap, a.dh, kFaKeys, err) ||
                !make_map(&G.tv[i], a.vcache, a.dh, (int64_t)a.hk * a.cap, a.dh, kFaKeys, err) ||
                !make_map(&G.to[i], a.attn, (int64_t)a.hq * a.dh, a.n, (int64_t)a.hq * a.dh, kFaRows, err))
                return VT_ERR_CUDA;
            heads += a.hq;
            G.head_end[i] = heads;
        }
        G.n_groups = ng;
        if (heads < 1 || as[0].n < 1) continue;
        const dim3 grid(heads, (as[0].n + kFaRows - 1) / kFaRows);
        if (as[0].dh == 128) k_prefill_attn_tc<128><<<grid, kFaThreads, fa_smem<128>(), st>>>(G);
        else k_prefill_attn_tc<64><<<grid, kFaThreads, fa_smem<64>(), st>>>(G);
        const cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) {
            *err = std::string("prefill attention launch failed: ") + cudaGetErrorString(e);
            return VT_ERR_CUDA;
        }
    }
    return VT_OK;
}

// Causal attention of every shard of an ATTN block (all with the same rows).
static vt_status prefill_attention(const PrefillAttnArgs* as, int n, cudaStream_t st, std::string* err) {
    return prefill_attention_tc(as, n, st, err);
}

vt_status prefill_attn_shard(const PrefillAttnArgs& a, cudaStream_t st, std::string* err) {
    return prefill_attn_group(&a, 1, st, err);
}

// The shards of one ATTN block: one QKV launch for all of them, their attention, one O launch.
// Every shard has its own q, attention and output buffers; they share the normalised input.
vt_status prefill_attn_group(const PrefillAttnArgs* a, int n, cudaStream_t st, std::string* err) {
    if (n < 1) return VT_OK;
    vt_status r;
    if (!a[0].xhat_ready && (r = run_rmsnorm(a[0].x, a[0].gain, a[0].eps, a[0].n, a[0].d, a[0].xhat, 1, st, err)) != VT_OK)
        return r;
    GemmSpec specs[VT_MAX_DEVICES];
    for (int i = 0; i < n; ++i) specs[i] = qkv_spec(a[i]);
    if ((r = run_gemm_group<kGemmQkv>(specs, n, a[0].n, st, err)) != VT_OK) return r;
    if ((r = prefill_attention(a, n, st, err)) != VT_OK) return r;
    for (int i = 0; i < n; ++i) specs[i] = o_spec(a[i]);
    return run_gemm_group<kGemmF32>(specs, n, a[0].n, st, err);
}

vt_status prefill_ffn_shard(const PrefillFfnArgs& a, cudaStream_t st, std::string* err) {
    return prefill_ffn_group(&a, 1, st, err);
}

// The shards of one FFN block: one gate/up (+ SwiGLU) launch and one down launch for all of them.
vt_status prefill_ffn_group(const PrefillFfnArgs* a, int n, cudaStream_t st, std::string* err) {
    if (n < 1) return VT_OK;
    vt_status r;
    if (!a[0].xhat_ready && (r = run_rmsnorm(a[0].x, a[0].gain, a[0].eps, a[0].n, a[0].d, a[0].xhat, 0, st, err)) != VT_OK)
        return r;
    GemmSpec specs[VT_MAX_DEVICES];
    for (int i = 0; i < n; ++i) {
        GemmArgs g{};
        g.u = a[i].u;
        g.ldu = a[i].ldu;
        g.ushift = a[i].ushift;
        g.status = a[i].status;
        specs[i] = GemmSpec{a[i].xhat, a[i].d, a[i].wgu, a[i].d, 2 * a[i].c, a[i].d, g};
    }
    if ((r = run_gemm_group<kGemmSwiglu>(specs, n, a[0].n, st, err)) != VT_OK) return r;
    for (int i = 0; i < n; ++i) {
        GemmArgs o{};
        o.c = a[i].out;
        o.ldc = a[i].d;
        o.status = a[i].status;
        // K runs over the shifted columns [0, ushift + c) of U and the same columns of Wd from wd
        specs[i] = GemmSpec{a[i].u, a[i].ldu, a[i].wd, a[i].wd_ld, a[i].d, a[i].ushift + a[i].c, o};
    }
    return run_gemm_group<kGemmF32>(specs, n, a[0].n, st, err);
}

}  // namespace vt
