// Device-side helpers shared by the library's kernels (sm_103a): programmatic dependent launch,
// mbarriers with bounded waits, bulk asynchronous copies, warp reductions.
#pragma once

#include <cuda_fp16.h>
#include <stdint.h>

#include "internal.h"

namespace vt {

// ------------------------------------------------------------------ programmatic dependent launch
// Every kernel of the library follows one discipline, which keeps PDL chains correct:
//   * before pdl_wait() it reads only data that no kernel of the same graph writes (weights, the
//     RoPE table, KV entries of earlier tokens) and writes nothing to global memory;
//   * it calls pdl_wait() on every thread that later touches dependent data, and
//     pdl_launch_dependents() only after its own wait, so that when a kernel starts, every kernel
//     two or more launches earlier has completed.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_launch_dependents() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// ------------------------------------------------------------------ shared-memory addresses
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// ------------------------------------------------------------------ mbarrier
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
                 : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
    asm volatile(
        "{\n\t.reg .b64 st;\n\tmbarrier.arrive.shared::cta.b64 st, [%0];\n\t}" ::"r"(smem_u32(bar))
        : "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
    asm volatile(
        "{\n\t.reg .b64 st;\n\tmbarrier.arrive.expect_tx.shared::cta.b64 st, [%0], %1;\n\t}" ::"r"(
            smem_u32(bar)),
        "r"(bytes)
        : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}
// Waits for the phase with the given parity to complete, giving up after kSpinLimit polls
// (each poll may itself suspend the thread for a short, hardware-chosen time).  Returns false on
// timeout; the caller records VT_DEV_WAIT_TIMEOUT and stops using the stage.
constexpr uint32_t kSpinLimit = 1u << 24;
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity) {
    for (uint32_t i = 0; i < kSpinLimit; ++i)
        if (mbar_try_wait(bar, parity)) return true;
    return false;
}

// Cluster forms: an arrival on the mbarrier at cluster address `bar` (this CTA's or a peer's),
// releasing this thread's prior writes at cluster scope, and a bounded wait on this CTA's
// barrier that acquires at cluster scope (for arrivals that come from a peer).
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t bar) {
    asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_wait_cluster(uint64_t* bar, uint32_t parity) {
    for (uint32_t i = 0; i < kSpinLimit; ++i) {
        uint32_t ok;
        asm volatile(
            "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
            "selp.u32 %0, 1, 0, p;\n\t}"
            : "=r"(ok)
            : "r"(smem_u32(bar)), "r"(parity)
            : "memory");
        if (ok) return true;
    }
    return false;
}

// ------------------------------------------------------------------ bulk asynchronous copies
// Global -> shared copy of `bytes` (multiple of 16, both addresses 16-byte aligned) completing
// as transaction bytes on `bar` (the CTA's own shared memory, addressed in the cluster window).
__device__ __forceinline__ void bulk_g2s(void* smem_dst, const void* gmem_src, uint32_t bytes,
                                         uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
            smem_u32(smem_dst)),
        "l"(gmem_src), "r"(bytes), "r"(smem_u32(bar))
        : "memory");
}

// ------------------------------------------------------------------ thread-block clusters
__device__ __forceinline__ uint32_t cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
__device__ __forceinline__ uint32_t cluster_size() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(r));
    return r;
}
// Hardware cluster barrier: every thread of every CTA of the cluster arrives (release) and
// waits (acquire).  Warps must be converged.
__device__ __forceinline__ void cluster_sync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::
                     : "memory");
}
// Split form of the barrier: arrive early (relaxed: orders nothing), wait later.  Used at kernel
// start so that no CTA writes into the shared memory of a cluster peer that has not started.
__device__ __forceinline__ void cluster_arrive_relaxed() {
    asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() {
    asm volatile("barrier.cluster.wait.aligned;" ::: "memory");
}
// Address of the same shared-memory location in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t dsmem_addr(const void* local, uint32_t rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_u32(local)), "r"(rank));
    return r;
}
__device__ __forceinline__ void dsmem_st(uint32_t addr, float v) {
    asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(addr), "f"(v) : "memory");
}
__device__ __forceinline__ float dsmem_ld(uint32_t addr) {
    float v;
    asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(addr) : "memory");
    return v;
}

// ------------------------------------------------------------------ bulk reductions
// Adds `bytes` of fp32 from shared memory into global memory (element-wise atomic add performed
// by the memory system) and waits until the operation has completed.
__device__ __forceinline__ void bulk_reduce_add_f32(float* gdst, const float* ssrc, uint32_t bytes) {
    asm volatile(
        "cp.reduce.async.bulk.global.shared::cta.bulk_group.add.f32 [%0], [%1], %2;\n\t"
        "cp.async.bulk.commit_group;\n\t"
        "cp.async.bulk.wait_group 0;" ::"l"(gdst),
        "r"(smem_u32(ssrc)), "r"(bytes)
        : "memory");
}
// The same addition, waiting only until the source has been read (the shared memory may then be
// reused); bulk_wait_all() later waits until every such addition of the thread has completed.
__device__ __forceinline__ void bulk_reduce_add_f32_issue(float* gdst, const float* ssrc, uint32_t bytes) {
    asm volatile(
        "cp.reduce.async.bulk.global.shared::cta.bulk_group.add.f32 [%0], [%1], %2;\n\t"
        "cp.async.bulk.commit_group;\n\t"
        "cp.async.bulk.wait_group.read 0;" ::"l"(gdst),
        "r"(smem_u32(ssrc)), "r"(bytes)
        : "memory");
}
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// ------------------------------------------------------------------ loads
// 8- and 4-byte loads of read-only data streamed once (weights), no L1 allocation.
__device__ __forceinline__ uint2 ldg_stream_u2(const void* p) {
    uint2 v;
    asm volatile("ld.global.nc.L1::no_allocate.v2.u32 {%0, %1}, [%2];" : "=r"(v.x), "=r"(v.y) : "l"(p));
    return v;
}
__device__ __forceinline__ uint32_t ldg_stream_u1(const void* p) {
    uint32_t v;
    asm volatile("ld.global.nc.L1::no_allocate.u32 %0, [%1];" : "=r"(v) : "l"(p));
    return v;
}
// 16-byte load of read-only data that is streamed once (weights): no L1 allocation.
__device__ __forceinline__ uint4 ldg_stream(const void* p) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}
__device__ __forceinline__ uint4 lds128(const void* p) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "r"(smem_u32(p)));
    return v;
}

__device__ __forceinline__ float2 h2_to_f2(uint32_t u) {
    __half2 h = *reinterpret_cast<__half2*>(&u);
    return __half22float2(h);
}

// dot of 8 fp16 weights (one 16-byte chunk) with 8 fp32 values
__device__ __forceinline__ float dot8(uint4 w, const float* x) {
    float2 a = h2_to_f2(w.x), b = h2_to_f2(w.y), c = h2_to_f2(w.z), d = h2_to_f2(w.w);
    float acc = a.x * x[0];
    acc = fmaf(a.y, x[1], acc);
    acc = fmaf(b.x, x[2], acc);
    acc = fmaf(b.y, x[3], acc);
    acc = fmaf(c.x, x[4], acc);
    acc = fmaf(c.y, x[5], acc);
    acc = fmaf(d.x, x[6], acc);
    acc = fmaf(d.y, x[7], acc);
    return acc;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

// Named barrier over `nthreads` threads (a multiple of 32) of the CTA.
__device__ __forceinline__ void consumer_bar(int id, int nthreads) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
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

__device__ __forceinline__ void set_status(uint32_t* status, uint32_t bits) {
    if (status) atomicOr(status, bits);
}

__device__ __forceinline__ float silu(float z) { return z / (1.0f + expf(-z)); }

}  // namespace vt
