// Device code of the persistent decode-token kernel; included by the translation units that
// instantiate its variants (token_v*.cu).  See token.cu for what it computes.
#pragma once

#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "device.cuh"
#include "internal.h"

namespace vt {
namespace {


constexpr uint32_t kTokSpin = 1u << 22;  // polls before a wait gives up

__device__ __forceinline__ uint32_t ld_acquire(const uint32_t* p) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void st_release(uint32_t* p, uint32_t v) {
    asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ uint32_t ld_volatile(const uint32_t* p) { return *(volatile const uint32_t*)p; }

__device__ __forceinline__ void abort_token(const TokArgs& a) {
    atomicExch(a.sync + kTokSyncAbort, 1u);
    set_status(a.status, VT_DEV_WAIT_TIMEOUT);
}

// Index arithmetic is 32-bit: every total (QKV row pairs, (KV head, position) pairs, O rows,
// FFN columns) is below 2^31, and 64-bit divisions would expand into long instruction sequences
// that crowd the instruction cache.
struct Span {
    int a, b;
};
// floor(t c / nc) without a 64-bit product: t = q nc + r gives q c + floor(r c / nc) (r c < 2^20)
__device__ __forceinline__ int span_at(int t, int c, int nc) {
    const int q = t / nc, r = t - q * nc;
    return q * c + (r * c) / nc;
}
__device__ __forceinline__ Span cta_span(int total, int c, int nc) { return {span_at(total, c, nc), span_at(total, c + 1, nc)}; }

// The CTA whose slice of T (KV head, position) pairs holds pair x: the largest c with
// start(c) <= x (start(c) = floor(c T / nc)), found from an estimate and a short correction.
__device__ __forceinline__ int cta_of(int T, int x, int nc) {
    int c = (int)(((float)x + 0.5f) * (float)nc / (float)T);
    c = c < 0 ? 0 : (c >= nc ? nc - 1 : c);
    while (c > 0 && span_at(T, c, nc) > x) --c;
    while (c < nc - 1 && span_at(T, c + 1, nc) <= x) ++c;
    return c;
}
// The CTAs holding the first and the last position of KV head j.
__device__ __forceinline__ void head_ctas(int T, int j, int n_pos, int nc, int& first, int& last) {
    first = cta_of(T, j * n_pos, nc);
    last = cta_of(T, j * n_pos + n_pos - 1, nc);
}

// dot of 8 fp16 weights with 8 fp32 values held in shared memory (16-byte aligned)
__device__ __forceinline__ float dot8_smem(uint4 w, const float* x) {
    const float4 x0 = *reinterpret_cast<const float4*>(x), x1 = *reinterpret_cast<const float4*>(x + 4);
    const float2 a = h2_to_f2(w.x), b = h2_to_f2(w.y), c = h2_to_f2(w.z), d = h2_to_f2(w.w);
    float acc = a.x * x0.x;
    acc = fmaf(a.y, x0.y, acc);
    acc = fmaf(b.x, x0.z, acc);
    acc = fmaf(b.y, x0.w, acc);
    acc = fmaf(c.x, x1.x, acc);
    acc = fmaf(c.y, x1.y, acc);
    acc = fmaf(d.x, x1.z, acc);
    acc = fmaf(d.y, x1.w, acc);
    return acc;
}

__device__ __forceinline__ void unpack8(uint4 u, float (&v)[8]) {
    const float2 a = h2_to_f2(u.x), b = h2_to_f2(u.y), c = h2_to_f2(u.z), d = h2_to_f2(u.w);
    v[0] = a.x; v[1] = a.y; v[2] = b.x; v[3] = b.y; v[4] = c.x; v[5] = c.y; v[6] = d.x; v[7] = d.y;
}
__device__ __forceinline__ uint4 pack8(const float (&v)[8]) {
    uint4 u;
    __half2 h;
    h = __floats2half2_rn(v[0], v[1]); u.x = *reinterpret_cast<uint32_t*>(&h);
    h = __floats2half2_rn(v[2], v[3]); u.y = *reinterpret_cast<uint32_t*>(&h);
    h = __floats2half2_rn(v[4], v[5]); u.z = *reinterpret_cast<uint32_t*>(&h);
    h = __floats2half2_rn(v[6], v[7]); u.w = *reinterpret_cast<uint32_t*>(&h);
    return u;
}
// v[0..8) += fp32 values p[0..8) read through L2 (written by other CTAs during this launch)
__device__ __forceinline__ void add8_cg(float (&v)[8], const float* p) {
    const float4 a = __ldcg(reinterpret_cast<const float4*>(p)), b = __ldcg(reinterpret_cast<const float4*>(p + 4));
    v[0] += a.x; v[1] += a.y; v[2] += a.z; v[3] += a.w; v[4] += b.x; v[5] += b.y; v[6] += b.z; v[7] += b.w;
}

// ------------------------------------------------------------------ schedule
// The producer and the consumers walk the same enumerations, so they agree on the content of
// every stage.  Ranges are near-equal contiguous slices of a flattened index space.

__device__ __forceinline__ int qkv_pairs(const TokArgs& a, int s) { return (a.hq[s] + 2 * a.hk[s]) * a.dh / 2; }

// f(shard, first local row, end local row) for this CTA's slice of the QKV row pairs
template <class F>
__device__ __forceinline__ void for_qkv_pieces(const TokArgs& a, int c, int nc, F&& f) {
    int tot = 0;
    for (int s = 0; s < a.n_dev; ++s) tot += qkv_pairs(a, s);
    const Span sp = cta_span(tot, c, nc);
    int pre = 0;
    for (int s = 0; s < a.n_dev; ++s) {
        const int ps = qkv_pairs(a, s);
        const int lo = sp.a > pre ? sp.a : pre, hi = sp.b < pre + ps ? sp.b : pre + ps;
        if (lo < hi) f(s, 2 * (lo - pre), 2 * (hi - pre));
        pre += ps;
    }
}

// f(global KV head, first position, end position, segment index) for this CTA's slice of the
// (KV head, position) pairs
template <class F>
__device__ __forceinline__ void for_kv_pieces(const TokArgs& a, int n_pos, int c, int nc, F&& f) {
    const int tot = a.n_kv * n_pos;
    if (tot <= 0) return;
    const Span sp = cta_span(tot, c, nc);
    if (sp.a >= sp.b) return;
    const int j0 = sp.a / n_pos, j1 = (sp.b - 1) / n_pos;
    for (int j = j0; j <= j1; ++j) {
        const int base = j * n_pos;
        const int lo = sp.a > base ? sp.a : base, hi = sp.b < base + n_pos ? sp.b : base + n_pos;
        f(j, lo - base, hi - base, j - j0);
    }
}

// f(shard, first row, end row) for this CTA's slice of the rows of every non-empty Wo
template <class F>
__device__ __forceinline__ void for_o_pieces(const TokArgs& a, int c, int nc, F&& f) {
    int tot = 0;
    for (int s = 0; s < a.n_dev; ++s) tot += a.hq[s] > 0 ? a.d : 0;
    const Span sp = cta_span(tot, c, nc);
    int pre = 0;
    for (int s = 0; s < a.n_dev; ++s) {
        if (a.hq[s] == 0) continue;
        const int lo = sp.a > pre ? sp.a : pre, hi = sp.b < pre + a.d ? sp.b : pre + a.d;
        if (lo < hi) f(s, lo - pre, hi - pre);
        pre += a.d;
    }
}

// f(shard, first column, end column) for this CTA's slice of all shards' FFN columns
template <class F>
__device__ __forceinline__ void for_ffn_pieces(const TokArgs& a, int c, int nc, F&& f) {
    int tot = 0;
    for (int s = 0; s < a.n_dev; ++s) tot += a.cols[s];
    const Span sp = cta_span(tot, c, nc);
    int pre = 0;
    for (int s = 0; s < a.n_dev; ++s) {
        const int lo = sp.a > pre ? sp.a : pre, hi = sp.b < pre + a.cols[s] ? sp.b : pre + a.cols[s];
        if (lo < hi) f(s, lo - pre, hi - pre);
        pre += a.cols[s];
    }
}

__device__ __forceinline__ int shard_of_kv(const TokArgs& a, int j) {
    int s = 0;
    while (s < a.n_dev - 1 && j >= a.kv0[s] + a.hk[s]) ++s;
    return s;
}

__device__ __forceinline__ void kv_geom(int len, int cap, int& n_pos, int& pnew, bool& ok) {
    ok = len >= 0 && len < cap;
    n_pos = ok ? len + 1 : min(max(len, 0), cap);
    pnew = ok ? len : -1;
}
// First attended position of a layer with sliding window `win` (0: every cached position).
__device__ __forceinline__ int window_start(int n_pos, int win) { return (win > 0 && n_pos > win) ? n_pos - win : 0; }

// ------------------------------------------------------------------ ring of stages

struct Ring {
    uint8_t* base;
    uint64_t* full;
    uint64_t* empty;
    int S;
    uint32_t k;      // stages consumed (consumer) or issued (producer) so far
    int slot;        // k mod S
    uint32_t phase;  // (k / S) mod 2
    bool live;       // consumer: false once the token is aborted (set around out-of-line calls)
    __device__ __forceinline__ void advance() {
        ++k;
        if (++slot == S) {
            slot = 0;
            phase ^= 1u;
        }
    }
};

// Bounded wait on an mbarrier phase; gives up early once the token is aborted.  Each try_wait may
// suspend the thread for up to kTokSuspendNs in hardware (it wakes as soon as the phase
// completes), so waiting threads take no issue slots from the warps that compute.
constexpr uint32_t kTokSuspendNs = 1000;
constexpr uint32_t kTokWaitPolls = 1u << 20;
__device__ __forceinline__ bool mbar_try_wait_suspend(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity), "r"(kTokSuspendNs)
        : "memory");
    return ok != 0;
}
__device__ __forceinline__ bool wait_phase(uint64_t* bar, uint32_t parity, const uint32_t* abort_word) {
    for (uint32_t i = 0; i < kTokWaitPolls; ++i) {
        if (mbar_try_wait_suspend(bar, parity)) return true;
        if ((i & 63) == 63 && ld_volatile(abort_word)) return false;  // rare: an L2 round trip
    }
    return false;
}

// Consumer side: returns the next stage, or nullptr once the token is aborted.
__device__ __forceinline__ const uint8_t* ring_acquire(Ring& r, bool& live, const TokArgs& a) {
    if (!live) return nullptr;
    if (!wait_phase(&r.full[r.slot], r.phase, a.sync + kTokSyncAbort)) {
        live = false;
        abort_token(a);
        return nullptr;
    }
    return r.base + (size_t)r.slot * kTokStageBytes;
}
__device__ __forceinline__ void ring_release(Ring& r, int lane) {
    __syncwarp();
    if (lane == 0) mbar_arrive(&r.empty[r.slot]);
    r.advance();
}

// ------------------------------------------------------------------ grid barrier
// Barrier over the CTAs of the (cooperative) launch.  Barrier i of a launch has epoch
// base + i + 1, base being the count of barriers of all earlier launches (sync[kTokSyncEpoch]).
// A CTA arrives by publishing the epoch in its own flag (release) and waits until every CTA's
// flag has reached it: warp 0 polls all flags with acquire loads (a few per lane), and the CTA
// barrier that follows orders every consumer thread's later reads after the other CTAs' writes
// (no full fence: under the weight stream one costs about a microsecond per barrier).  No two CTAs write one word, so
// arrivals do not queue behind each other.  Called by all consumer threads; returns false when
// the token is aborted (then it does not wait).  Out of line, like the other helpers called from
// several places: the kernel is larger than the instruction cache, and every miss waits behind
// the weight stream for its L2 round trip (one copy of the barrier instead of four measured 7%
// of the token time).

// spin: polls before the wait gives up; skip_epoch: the barrier (epoch) at which this CTA does
// not publish its arrival (0: none) -- both from the test words of the sync area, which a status
// clear zeroes, so outside a test every CTA arrives and waits up to kTokSpin polls.
__device__ __noinline__ bool grid_sync(const TokArgs& a, int* s_flag, bool live, uint32_t epoch, uint32_t spin,
                                       uint32_t skip_epoch) {
    consumer_bar(1, kTokConsumers);
    const int lane = threadIdx.x & 31;
    if (threadIdx.x < 32) {
        int ok = live ? 1 : 0;
        uint32_t* flags = a.sync + kTokSyncFlags;
        if (ok) {
            // the CTA's writes precede this store through the CTA barrier above, and a release
            // store makes them visible to every thread that acquires the flag
            if (lane == 0 && epoch != skip_epoch) st_release(flags + blockIdx.x, epoch);
            // each poll is one round of independent loads; the abort word is read only every 64
            // polls, so a poll costs one L2 round trip
            for (uint32_t i = 1;; ++i) {
                bool mine = true;
                for (int x = lane; x < (int)gridDim.x; x += 32) mine &= (int32_t)(ld_acquire(flags + x) - epoch) >= 0;
                if (__all_sync(0xffffffffu, mine)) break;
                if ((i & 63) == 0) {
                    int stop = 0;
                    if (lane == 0) {
                        if (ld_volatile(a.sync + kTokSyncAbort)) stop = 1;
                        else if (i > spin) {
                            stop = 1;
                            abort_token(a);
                        }
                    }
                    if (__shfl_sync(0xffffffffu, stop, 0)) {
                        ok = 0;
                        break;
                    }
                }
            }
            // no second look at the abort word here: it costs an L2 round trip on every barrier,
            // and a CTA that aborts after arriving is seen at the next wait
        }
        if (lane == 0) *s_flag = ok;
    }
    consumer_bar(1, kTokConsumers);
    return *s_flag != 0;
}

// ------------------------------------------------------------------ tensor-core GEMV over a stage
// A stage holds R rows of K fp16 weights (row-major, rows K*2 bytes apart, so every row starts on
// the same shared-memory bank).  The products W . x run on mma.sync m16n8k16 (fp16 in, fp32
// accumulate): the 16 rows of an MMA are 2 weight rows (h) x 8 segments (j) of the row's K range
// (segment length L), and B column j holds the input values of segment j, so the useful results
// are D[8 h + j][j].  At step i, virtual row (h, j) reads the 16 elements
// (16 i + 8 j + [0, 16)) mod L of its segment: the 8 row addresses of each 8x8 block then sit 16
// bytes apart and the ldmatrix loads are free of bank conflicts.  The fp32 input is split into
// hi = fp16(x) and lo = fp16(x - hi) and both are multiplied (two MMAs), which keeps the input's
// fp32 precision; the weights are exact fp16.  Each warp covers one row pair over WP-th of the
// row (8 segments), and the 8 segment results of a row go to shared-memory slots that are summed
// in a fixed order after the phase, so no shuffles are needed.

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}
__device__ __forceinline__ void mma16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3, uint32_t b0,
                                         uint32_t b1) {
    asm("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
// (x0, x1) -> fp16 pairs hi = (fp16(x0), fp16(x1)) and lo = (fp16(x0 - hi0), fp16(x1 - hi1))
__device__ __forceinline__ void split2(float x0, float x1, uint32_t& hi, uint32_t& lo) {
    const __half h0 = __float2half_rn(x0), h1 = __float2half_rn(x1);
    const __half l0 = __float2half_rn(x0 - __half2float(h0)), l1 = __float2half_rn(x1 - __half2float(h1));
    __half2 a = __halves2half2(h0, h1), b = __halves2half2(l0, l1);
    hi = *reinterpret_cast<uint32_t*>(&a);
    lo = *reinterpret_cast<uint32_t*>(&b);
}

// Per-lane constants of the tensor-core GEMV for rows of length K, computed once per phase.
struct MmaLane {
    int q;            // segment group (WP-th of the row) of the warp
    int p0, pstep;    // first row pair of the warp and the stride between its pairs
    int lr, hh;       // ldmatrix: row of the 8x8 block this lane addresses, and which row of the pair
    uint32_t aseg;    // byte offset of the lane's A segment in a row
    int aoff0;        // A window start (elements) at step 0
    int bseg, boff0;  // B: element index of the lane's segment, window start at step 0
    bool holder;      // this lane holds D[g][g] and D[g + 8][g]
    int cc;           // accumulator component of those results
    int slot;         // q * 8 + g
};

__device__ __forceinline__ MmaLane mma_lane(const MmaGeom& gm, int warp, int lane) {
    MmaLane m;
    const int g = lane >> 2, t = lane & 3, kb = lane >> 4, L = gm.L;
    m.q = warp % gm.WP;
    m.p0 = warp / gm.WP;
    m.pstep = 8 / gm.WP;
    m.lr = lane & 7;
    m.hh = (lane >> 3) & 1;
    m.aseg = (uint32_t)((m.q * 8 + m.lr) * L) * 2u;
    m.aoff0 = (8 * m.lr + 8 * kb) % L;
    m.bseg = (m.q * 8 + g) * L;
    m.boff0 = (8 * g + 2 * t) % L;
    m.holder = t == (g >> 1);
    m.cc = g & 1;
    m.slot = m.q * 8 + g;
    return m;
}

// B fragments of this lane for every step: x^ = x16 * rinv * gain at the lane's positions, split
// into hi / lo halves (x16 in shared memory, the gains prefetched as half2 pairs).
template <int STEPS>
__device__ __forceinline__ void make_bfrags(const __half* x16, float rinv, const uint32_t (&gf)[STEPS][2],
                                            const MmaLane& ml, int L, uint32_t (&bh)[STEPS][2],
                                            uint32_t (&bl)[STEPS][2]) {
    int off = ml.boff0;
#pragma unroll
    for (int i = 0; i < STEPS; ++i) {
        int o2 = off + 8;
        if (o2 >= L) o2 -= L;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int e = ml.bseg + (h ? o2 : off);
            const float2 xv = __half22float2(*reinterpret_cast<const __half2*>(x16 + e));
            uint32_t gw = gf[i][h];
            const float2 gv = __half22float2(*reinterpret_cast<__half2*>(&gw));
            split2(xv.x * rinv * gv.x, xv.y * rinv * gv.y, bh[i][h], bl[i][h]);
        }
        off += 16;
        if (off >= L) off -= L;
    }
}

// The gains at this lane's B positions (loaded before the barrier that precedes the norm).
template <int STEPS>
__device__ __forceinline__ void prefetch_bgain(const __half* gain, const MmaLane& ml, int L, uint32_t (&gf)[STEPS][2]) {
    int off = ml.boff0;
#pragma unroll
    for (int i = 0; i < STEPS; ++i) {
        int o2 = off + 8;
        if (o2 >= L) o2 -= L;
        gf[i][0] = *reinterpret_cast<const uint32_t*>(gain + ml.bseg + off);
        gf[i][1] = *reinterpret_cast<const uint32_t*>(gain + ml.bseg + o2);
        off += 16;
        if (off >= L) off -= L;
    }
}

// B fragments of this lane from hi / lo fp16 copies of the input in shared memory.
template <int STEPS>
__device__ __forceinline__ void load_bfrags_h(const __half* xh, const __half* xl, const MmaLane& ml, int L,
                                              uint32_t (&bh)[STEPS][2], uint32_t (&bl)[STEPS][2]) {
    int off = ml.boff0;
#pragma unroll
    for (int i = 0; i < STEPS; ++i) {
        int o2 = off + 8;
        if (o2 >= L) o2 -= L;
        bh[i][0] = *reinterpret_cast<const uint32_t*>(xh + ml.bseg + off);
        bh[i][1] = *reinterpret_cast<const uint32_t*>(xh + ml.bseg + o2);
        bl[i][0] = *reinterpret_cast<const uint32_t*>(xl + ml.bseg + off);
        bl[i][1] = *reinterpret_cast<const uint32_t*>(xl + ml.bseg + o2);
        off += 16;
        if (off >= L) off -= L;
    }
}

// One stage of nrows rows of length K against B fragments held in registers: per row, 8 WP
// partial sums go to slots[(rowbase + row) * spr + ...].
template <int STEPS>
__device__ __forceinline__ void stage_mma_regs(uint32_t st, int nrows, int K, const MmaGeom& gm, const MmaLane& ml,
                                               int rowbase, const uint32_t (&bh)[STEPS][2],
                                               const uint32_t (&bl)[STEPS][2], float* slots) {
    const int NP = (nrows + 1) >> 1, L = gm.L;
    for (int p = ml.p0; p < NP; p += ml.pstep) {
        int row = 2 * p + ml.hh;
        if (row >= nrows) row = 2 * p;  // the missing second row of an odd stage: results unused
        const uint32_t rb = st + (uint32_t)row * (uint32_t)K * 2u + ml.aseg;
        float d0[4] = {0.f, 0.f, 0.f, 0.f}, d1[4] = {0.f, 0.f, 0.f, 0.f};
        float e0[4] = {0.f, 0.f, 0.f, 0.f}, e1[4] = {0.f, 0.f, 0.f, 0.f};
        int off = ml.aoff0;
#pragma unroll
        for (int i = 0; i < STEPS; ++i) {
            uint32_t a0, a1, a2, a3;
            ldsm_x4(rb + (uint32_t)off * 2u, a0, a1, a2, a3);
            if (i & 1) {
                mma16816(d1, a0, a1, a2, a3, bh[i][0], bh[i][1]);
                mma16816(e1, a0, a1, a2, a3, bl[i][0], bl[i][1]);
            } else {
                mma16816(d0, a0, a1, a2, a3, bh[i][0], bh[i][1]);
                mma16816(e0, a0, a1, a2, a3, bl[i][0], bl[i][1]);
            }
            off += 16;
            if (off >= L) off -= L;
        }
        if (ml.holder) {
            // component cc of each accumulator, selected with constant indices (a runtime index
            // would put the accumulators in local memory)
            const bool c1 = ml.cc != 0;
            const float r0 = c1 ? (d0[1] + d1[1]) + (e0[1] + e1[1]) : (d0[0] + d1[0]) + (e0[0] + e1[0]);
            const float r1 = c1 ? (d0[3] + d1[3]) + (e0[3] + e1[3]) : (d0[2] + d1[2]) + (e0[2] + e1[2]);
            slots[(rowbase + 2 * p) * gm.spr + ml.slot] = r0;
            if (2 * p + 1 < nrows) slots[(rowbase + 2 * p + 1) * gm.spr + ml.slot] = r1;
        }
    }
}

// The same for rows whose length varies per call (the O projection): B fragments come from
// hi / lo fp16 copies of the input in shared memory (xh, xl: K halves each).
__device__ __forceinline__ void stage_mma_smem(uint32_t st, int nrows, int K, const MmaGeom& gm, const MmaLane& ml,
                                               int rowbase, const __half* xh, const __half* xl, float* slots) {
    const int L = gm.L, steps = L / 16;
    const int NP = (nrows + 1) >> 1;
    for (int p = ml.p0; p < NP; p += ml.pstep) {
        int row = 2 * p + ml.hh;
        if (row >= nrows) row = 2 * p;
        const uint32_t rb = st + (uint32_t)row * (uint32_t)K * 2u + ml.aseg;
        float d0[4] = {0.f, 0.f, 0.f, 0.f}, d1[4] = {0.f, 0.f, 0.f, 0.f};
        int off = ml.aoff0, bo = ml.boff0;
        for (int i = 0; i < steps; ++i) {
            uint32_t a0, a1, a2, a3;
            ldsm_x4(rb + (uint32_t)off * 2u, a0, a1, a2, a3);
            int bo2 = bo + 8;
            if (bo2 >= L) bo2 -= L;
            const uint32_t h0 = *reinterpret_cast<const uint32_t*>(xh + ml.bseg + bo);
            const uint32_t h1 = *reinterpret_cast<const uint32_t*>(xh + ml.bseg + bo2);
            const uint32_t l0 = *reinterpret_cast<const uint32_t*>(xl + ml.bseg + bo);
            const uint32_t l1 = *reinterpret_cast<const uint32_t*>(xl + ml.bseg + bo2);
            mma16816(d0, a0, a1, a2, a3, h0, h1);
            mma16816(d1, a0, a1, a2, a3, l0, l1);
            off += 16;
            if (off >= L) off -= L;
            bo += 16;
            if (bo >= L) bo -= L;
        }
        if (ml.holder) {
            const bool c1 = ml.cc != 0;
            const float r0 = c1 ? d0[1] + d1[1] : d0[0] + d1[0];
            const float r1 = c1 ? d0[3] + d1[3] : d0[2] + d1[2];
            slots[(rowbase + 2 * p) * gm.spr + ml.slot] = r0;
            if (2 * p + 1 < nrows) slots[(rowbase + 2 * p + 1) * gm.spr + ml.slot] = r1;
        }
    }
}

// Sum of the spr partial sums of a row, in slot order.
// (spr is a multiple of 8; four interleaved partial sums, added in a fixed order)
__device__ __noinline__ float row_total(const float* slots, int row, int spr) {
    const float* r = slots + row * spr;
    float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
    for (int i = 0; i < spr; i += 4) {
        const float4 v = *reinterpret_cast<const float4*>(r + i);
        a0 += v.x;
        a1 += v.y;
        a2 += v.z;
        a3 += v.w;
    }
    return (a0 + a1) + (a2 + a3);
}

// Online-softmax attention of one KV head over positions [t0, t1) (EPL = dh / 32 elements per
// lane, G query heads per KV head), then the warps' states merged into one slice state.
// The ring state goes in and comes back by value.
template <int EPL, int G>
__device__ __forceinline__ Ring attn_slice(const TokArgs& a, const TokShardPtrs* sp, Ring ring, int j, int t0, int t1,
                                        int seg, int pnew, float* wst, int tid, int warp, int lane) {
    bool live = ring.live;
    constexpr int DH = EPL * 32;
    constexpr int P = 8 / G;  // positions per batch (G x P scores reduced together)
    const int s = shard_of_kv(a, j), jl = j - a.kv0[s];
    const __half* kb = sp[s].kc + (int64_t)jl * a.cap * DH;
    const __half* vb = sp[s].vc + (int64_t)jl * a.cap * DH;
    const int np_stage = kTokStageBytes / (4 * DH);
    const int old_end = pnew >= 0 ? min(t1, pnew) : t1;
    const bool has_new = pnew >= t0 && pnew < t1;

    float q[G][EPL];
#pragma unroll
    for (int g = 0; g < G; ++g)
#pragma unroll
        for (int e = 0; e < EPL; ++e) q[g][e] = __ldcg(a.q_all + (j * G + g) * DH + lane * EPL + e);
    float m[G], l[G], o[G][EPL];
#pragma unroll
    for (int g = 0; g < G; ++g) {
        m[g] = -INFINITY;
        l[g] = 0.f;
#pragma unroll
        for (int e = 0; e < EPL; ++e) o[g][e] = 0.f;
    }
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
    for (int t = t0; t < old_end; t += np_stage) {
        const int n = min(np_stage, old_end - t);
        const uint8_t* st = ring_acquire(ring, live, a);
        if (!st) continue;
        const __half* kt = reinterpret_cast<const __half*>(st);
        const __half* vt = reinterpret_cast<const __half*>(st + kTokStageBytes / 2);
        for (int b0 = warp * P; b0 < n; b0 += kTokWarps * P) {
            float kv[P][EPL], vv[P][EPL];
#pragma unroll
            for (int i = 0; i < P; ++i) {
                if (b0 + i < n) {
                    load_lane(kt + (b0 + i) * DH, kv[i]);
                    load_lane(vt + (b0 + i) * DH, vv[i]);
                } else {
#pragma unroll
                    for (int e = 0; e < EPL; ++e) kv[i][e] = vv[i][e] = 0.f;
                }
            }
            float part[8];
#pragma unroll
            for (int g = 0; g < G; ++g)
#pragma unroll
                for (int i = 0; i < P; ++i) {
                    float sc = 0.f;
#pragma unroll
                    for (int e = 0; e < EPL; ++e) sc = fmaf(q[g][e], kv[i][e], sc);
                    part[g * P + i] = sc;
                }
            const float mine = multi_row_sum<8>(part, lane);  // lane 4 r holds row r = g P + i
            float sc[G][P];
#pragma unroll
            for (int r = 0; r < 8; ++r) sc[r / P][r % P] = __shfl_sync(0xffffffffu, mine, 4 * r) * a.scale_log2;
#pragma unroll
            for (int g = 0; g < G; ++g) {
                float mb = m[g];
#pragma unroll
                for (int i = 0; i < P; ++i)
                    if (b0 + i < n) mb = fmaxf(mb, sc[g][i]);
                const float corr = exp2f(m[g] - mb);
                float lsum = l[g] * corr;
                float acc[EPL];
#pragma unroll
                for (int e = 0; e < EPL; ++e) acc[e] = o[g][e] * corr;
#pragma unroll
                for (int i = 0; i < P; ++i) {
                    const float pw = (b0 + i < n) ? exp2f(sc[g][i] - mb) : 0.f;
                    lsum += pw;
#pragma unroll
                    for (int e = 0; e < EPL; ++e) acc[e] = fmaf(pw, vv[i][e], acc[e]);
                }
                l[g] = lsum;
#pragma unroll
                for (int e = 0; e < EPL; ++e) o[g][e] = acc[e];
                m[g] = mb;
            }
        }
        ring_release(ring, lane);
    }
    if (has_new && warp == 0 && live) {
        // the token's own K/V row, appended by the QKV phase of this launch: read through L2
        float kn[EPL], vn[EPL];
#pragma unroll
        for (int e = 0; e < EPL; ++e) {
            kn[e] = __half2float(__ldcg(kb + (int64_t)pnew * DH + lane * EPL + e));
            vn[e] = __half2float(__ldcg(vb + (int64_t)pnew * DH + lane * EPL + e));
        }
#pragma unroll
        for (int g = 0; g < G; ++g) {
            float sc = 0.f;
#pragma unroll
            for (int e = 0; e < EPL; ++e) sc = fmaf(q[g][e], kn[e], sc);
            sc = warp_sum(sc) * a.scale_log2;
            const float mn = fmaxf(m[g], sc);
            const float corr = exp2f(m[g] - mn);
            const float pw = exp2f(sc - mn);
            l[g] = l[g] * corr + pw;
#pragma unroll
            for (int e = 0; e < EPL; ++e) o[g][e] = fmaf(o[g][e], corr, pw * vn[e]);
            m[g] = mn;
        }
    }
    // per-warp states -> one slice state (warps merged in fixed order)
    float* wm = wst;                          // [warps][G]
    float* wl = wm + kTokWarps * G;           // [warps][G]
    float* wo = wl + kTokWarps * G;           // [warps][G][DH]
#pragma unroll
    for (int g = 0; g < G; ++g) {
        if (lane == 0) {
            wm[warp * G + g] = m[g];
            wl[warp * G + g] = l[g];
        }
#pragma unroll
        for (int e = 0; e < EPL; ++e) wo[(warp * G + g) * DH + lane * EPL + e] = o[g][e];
    }
    consumer_bar(1, kTokConsumers);
    float* out = a.states + ((size_t)(blockIdx.x * kTokMaxSeg + seg) * G) * (DH + 4);
    for (int idx = tid; idx < G * DH; idx += kTokConsumers) {
        const int g = idx / DH, d = idx - g * DH;
        float M = -INFINITY;
        for (int w = 0; w < kTokWarps; ++w) M = fmaxf(M, wm[w * G + g]);
        float L = 0.f, O = 0.f;
        if (M != -INFINITY) {
            for (int w = 0; w < kTokWarps; ++w) {
                const float f = exp2f(wm[w * G + g] - M);
                L += wl[w * G + g] * f;
                O += wo[(w * G + g) * DH + d] * f;
            }
        }
        float* so = out + (size_t)g * (DH + 4);
        __stcg(so + 4 + d, O);
        if (d == 0) {
            __stcg(so, M);
            __stcg(so + 1, L);
        }
    }
    consumer_bar(1, kTokConsumers);  // the warp states are reused by the next slice
    ring.live = live;
    return ring;
}

// The attention output of shard s (K = its query heads x dh), merged from the slice states with
// log-sum-exp weights: each thread takes 4 consecutive elements of one query head and issues the
// loads of 8 slices together (heads cut into more slices take further batches of 8); the result
// goes to xh / xl as fp16 hi / lo halves.
__device__ __forceinline__ void merge_heads(const TokArgs& a, int s, int K, const int* mtab, int mstride, int dsh, int gsh,
                                         __half* xh, __half* xl, int tid) {
    const int dh = a.dh, G = a.group;
    for (int f4 = 4 * tid; f4 < K; f4 += 4 * kTokConsumers) {
        const int h = a.h0[s] + (f4 >> dsh), d = f4 & (dh - 1);
        const int j = h >> gsh, g = h & (G - 1);
        const int* tb = mtab + j * mstride;
        float2 ml[8];
        float4 ov[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const int b = k < mstride ? tb[k] : -1;
            if (b >= 0) {
                const float* st = a.states + b + g * (dh + 4);
                ml[k] = __ldcg(reinterpret_cast<const float2*>(st));
                ov[k] = __ldcg(reinterpret_cast<const float4*>(st + 4 + d));
            } else {
                ml[k] = make_float2(-INFINITY, 0.f);
                ov[k] = make_float4(0.f, 0.f, 0.f, 0.f);
            }
        }
        float M = -INFINITY;
#pragma unroll
        for (int k = 0; k < 8; ++k) M = fmaxf(M, ml[k].x);
        float L = 0.f, y0 = 0.f, y1 = 0.f, y2 = 0.f, y3 = 0.f;
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const float w = ml[k].x == -INFINITY ? 0.f : exp2f(ml[k].x - M);
            L = fmaf(ml[k].y, w, L);
            y0 = fmaf(ov[k].x, w, y0);
            y1 = fmaf(ov[k].y, w, y1);
            y2 = fmaf(ov[k].z, w, y2);
            y3 = fmaf(ov[k].w, w, y3);
        }
        // heads split over more than 8 CTAs (long caches): further slices 8 at a time, each
        // batch's loads issued together, the running sums rescaled when a batch raises the maximum
        for (int k0 = 8; k0 < mstride; k0 += 8) {
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                const int b = k0 + k < mstride ? tb[k0 + k] : -1;
                if (b >= 0) {
                    const float* st = a.states + b + g * (dh + 4);
                    ml[k] = __ldcg(reinterpret_cast<const float2*>(st));
                    ov[k] = __ldcg(reinterpret_cast<const float4*>(st + 4 + d));
                } else {
                    ml[k] = make_float2(-INFINITY, 0.f);
                    ov[k] = make_float4(0.f, 0.f, 0.f, 0.f);
                }
            }
            float nm = M;
#pragma unroll
            for (int k = 0; k < 8; ++k) nm = fmaxf(nm, ml[k].x);
            if (M != -INFINITY && nm != M) {
                const float r = exp2f(M - nm);
                L *= r;
                y0 *= r;
                y1 *= r;
                y2 *= r;
                y3 *= r;
            }
            M = nm;
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                const float w = ml[k].x == -INFINITY ? 0.f : exp2f(ml[k].x - M);
                L = fmaf(ml[k].y, w, L);
                y0 = fmaf(ov[k].x, w, y0);
                y1 = fmaf(ov[k].y, w, y1);
                y2 = fmaf(ov[k].z, w, y2);
                y3 = fmaf(ov[k].w, w, y3);
            }
        }
        const float linv = L > 0.f ? 1.0f / L : 0.f;
        const float yv[4] = {y0 * linv, y1 * linv, y2 * linv, y3 * linv};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const __half hy = __float2half_rn(yv[e]);
            xh[f4 + e] = hy;
            xl[f4 + e] = __float2half_rn(yv[e] - __half2float(hy));
        }
    }}

template <int STEPS, int MC, int DH_, int G_, bool OSMEM>
__global__ void __launch_bounds__(kTokThreads, 1) k_decode_token(const __grid_constant__ TokArgs a) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* ring_base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    // head dim and query heads per KV head are compile-time: each variant carries one attention
    // code path, which keeps the kernel small in the instruction cache
    constexpr int dh = DH_, G = G_;
    constexpr int dsh = dh == 128 ? 7 : 6, gsh = G == 4 ? 2 : (G == 2 ? 1 : 0);  // log2 of dh and G
    const int S = a.stages, D = a.d;
    const int nch = D >> 3;
    uint8_t* p = ring_base + (size_t)S * kTokStageBytes;
    // residual stream of the CTA (fp16): the layer input x, replaced in place by h after the
    // ATTN combine and by the next layer's input after the FFN combine (each thread updates the
    // chunks it owns)
    __half* x16 = reinterpret_cast<__half*>(p);
    p += ((size_t)D * 2 + 127) & ~(size_t)127;
    float* uni = reinterpret_cast<float*>(p);    // attention warp states, or hi / lo halves of one shard's attention output
    p += ((size_t)a.uni_floats * 4 + 127) & ~(size_t)127;
    float* slots = reinterpret_cast<float*>(p);  // per-row partial sums; the normalised input during a prologue
    p += ((size_t)a.slot_floats * 4 + 127) & ~(size_t)127;
    float* act = reinterpret_cast<float*>(p);    // SwiGLU activations of one column group
    p += 128 * 4;
    float* red = reinterpret_cast<float*>(p);
    p += 64 * 4;
    int* lens = reinterpret_cast<int*>(p);
    p += kTokMaxLayers * 4;
    uint64_t* full = reinterpret_cast<uint64_t*>(p);
    uint64_t* empty = full + S;
    __shared__ int s_flag;
    __shared__ uint32_t s_epoch, s_test_skip, s_test_spin;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int c = blockIdx.x, NC = gridDim.x;
    if (tid == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], kTokWarps);
        }
        fence_mbar_init();
        s_epoch = a.sync[kTokSyncEpoch];
        s_test_skip = a.sync[kTokSyncTestSkip];
        s_test_spin = a.sync[kTokSyncTestSpin];
    }
    for (int l = tid; l < a.n_layers; l += blockDim.x) lens[l] = a.len[l];
    __syncthreads();

    const MmaGeom gd = mma_geom(D);
    const int rps_d = gd.R;
    // FFN columns per group: all gate/up rows of the group, then its down rows.  A CTA's columns
    // of one shard form one group when they fit the slots (at most 128 columns), which keeps the
    // input fragments and the down-projection accumulators from being live at the same time.
    const int gcol = a.ffn_gcol;
    Ring ring{ring_base, full, empty, S, 0u, 0, 0u, true};

    if (warp >= kTokWarps) {
        // ================================================================ producer
        // the producer warpgroup keeps kTokProducerRegs registers per thread and gives the rest
        // to the two consumer warpgroups (both sides of the split run before any wait)
        asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(kTokProducerRegs));
        if (warp == kTokWarps && lane == 0) {
            bool live = true;
            auto issue = [&](const void* s0, uint32_t b0, const void* s1, uint32_t b1) {
                if (!live) return;
                const int slot = ring.slot;
                // stage k reuses the slot of stage k - S: wait until the consumers released it
                if (ring.k >= (uint32_t)S && !wait_phase(&empty[slot], ring.phase ^ 1u, a.sync + kTokSyncAbort)) {
                    live = false;
                    abort_token(a);
                    return;
                }
                uint8_t* dst = ring_base + (size_t)slot * kTokStageBytes;
                mbar_arrive_expect_tx(&full[slot], b0 + b1);
                bulk_g2s(dst, s0, b0, &full[slot]);
                if (b1) bulk_g2s(dst + kTokStageBytes / 2, s1, b1, &full[slot]);
                ring.advance();
            };
            for (int l = 0; l < a.n_layers && live; ++l) {
                const TokShardPtrs* sp = a.shard + (size_t)l * a.n_dev;
                int n_pos, pnew;
                bool ok;
                kv_geom(lens[l], a.cap, n_pos, pnew, ok);
                for_qkv_pieces(a, c, NC, [&](int s, int r0, int r1) {
                    const __half* w = sp[s].wqkv;
                    for (int r = r0; r < r1; r += rps_d)
                        issue(w + (int64_t)r * D, (uint32_t)(min(rps_d, r1 - r) * D * 2), nullptr, 0);
                });
                const int np_stage = kTokStageBytes / (4 * dh);
                const int t_lo = window_start(n_pos, a.layer[l].window);
                for_kv_pieces(a, n_pos - t_lo, c, NC, [&](int j, int t0, int t1, int) {
                    t0 += t_lo;
                    t1 += t_lo;
                    const int s = shard_of_kv(a, j), jl = j - a.kv0[s];
                    const __half* kb = sp[s].kc + (int64_t)jl * a.cap * dh;
                    const __half* vb = sp[s].vc + (int64_t)jl * a.cap * dh;
                    const int old_end = pnew >= 0 ? min(t1, pnew) : t1;
                    for (int t = t0; t < old_end; t += np_stage) {
                        const uint32_t bytes = (uint32_t)(min(np_stage, old_end - t) * dh * 2);
                        issue(kb + (int64_t)t * dh, bytes, vb + (int64_t)t * dh, bytes);
                    }
                });
                for_o_pieces(a, c, NC, [&](int s, int r0, int r1) {
                    const int K = a.hq[s] * dh, rps = mma_geom(K).R;
                    const __half* w = sp[s].wo;
                    for (int r = r0; r < r1; r += rps)
                        issue(w + (int64_t)r * K, (uint32_t)(min(rps, r1 - r) * K * 2), nullptr, 0);
                });
                for_ffn_pieces(a, c, NC, [&](int s, int j0, int j1) {
                    const __half* wgu = sp[s].wgu;
                    const __half* wdt = sp[s].wdt;
                    for (int g = j0; g < j1; g += gcol) {
                        const int ng = min(gcol, j1 - g);
                        for (int r = 2 * g; r < 2 * (g + ng); r += rps_d)
                            issue(wgu + (int64_t)r * D, (uint32_t)(min(rps_d, 2 * (g + ng) - r) * D * 2), nullptr, 0);
                        for (int r = g; r < g + ng; r += rps_d)
                            issue(wdt + (int64_t)r * D, (uint32_t)(min(rps_d, g + ng - r) * D * 2), nullptr, 0);
                    }
                });
            }
            // never leave with copies in flight: wait for the last fill of every stage
            const uint32_t first = ring.k > (uint32_t)S ? ring.k - (uint32_t)S : 0u;
            for (uint32_t i = first; i < ring.k; ++i) {
                bool done = false;
                for (uint32_t t = 0; t < kTokWaitPolls && !done; ++t)
                    done = mbar_try_wait_suspend(&full[i % (uint32_t)S], (i / (uint32_t)S) & 1);
                if (!done) set_status(a.status, VT_DEV_WAIT_TIMEOUT);
            }
        }
        return;
    }

    // ==================================================================== consumers (256 threads)
    asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(kTokConsumerRegs));
    bool live = ld_volatile(a.sync + kTokSyncAbort) == 0;
    uint32_t epoch = s_epoch;
    const uint32_t spin = s_test_spin ? s_test_spin : kTokSpin;
    const uint32_t skip_epoch = s_test_skip == (uint32_t)c + 1u ? s_epoch + 1u : 0u;
    const uint32_t ring_s = smem_u32(ring_base);
    uint32_t bh[STEPS][2], bl[STEPS][2];  // hi / lo fp16 B fragments of the normalised input
    uint32_t gf[STEPS][2];                // RMSNorm gains at the B positions, loaded before the barrier that precedes the norm
    const MmaLane mld = mma_lane(gd, warp, lane);
    // Combine and RMSNorm over the residual stream (chunk tid + 256 m belongs to this thread):
    //   x16 = fp16(x16 + sum of partials, shards in order)   (layer 0: the token input),
    //   x^ = x16 * rinv * gain, rinv = 1 / sqrt(mean(x16^2) + eps),
    // and every lane builds its B fragments of x^ from x16 (one barrier: after it, every chunk of
    // x16 is final and the sum of squares is complete).
    auto combine_norm = [&](const float* parts, bool attn_parts, bool first) {
        float ss = 0.f;
#pragma unroll
        for (int m = 0; m < MC; ++m) {
            const int ch = tid + kTokConsumers * m;
            if (ch < nch && live) {
                uint4 hv;
                if (first) {
                    hv = *reinterpret_cast<const uint4*>(a.x_in + ch * 8);
                } else {
                    float v[8];
                    unpack8(lds128(x16 + ch * 8), v);
                    for (int s = 0; s < a.n_dev; ++s)
                        if (!attn_parts || a.hq[s] > 0) add8_cg(v, parts + (size_t)s * D + ch * 8);
                    hv = pack8(v);
                }
                *reinterpret_cast<uint4*>(x16 + ch * 8) = hv;
                float xv[8];
                unpack8(hv, xv);
#pragma unroll
                for (int e = 0; e < 8; ++e) ss = fmaf(xv[e], xv[e], ss);
            }
        }
        ss = warp_sum(ss);
        if (lane == 0) red[warp] = ss;
        consumer_bar(1, kTokConsumers);
        float tot = 0.f;
        for (int w = 0; w < kTokWarps; ++w) tot += red[w];
        make_bfrags<STEPS>(x16, 1.0f / sqrtf(tot / (float)D + a.eps), gf, mld, gd.L, bh, bl);
    };

    prefetch_bgain<STEPS>(a.layer[0].attn_norm, mld, gd.L, gf);
    for (int l = 0; l < a.n_layers; ++l) {
        const TokShardPtrs* sp = a.shard + (size_t)l * a.n_dev;
        int n_pos, pnew;
        bool ok;
        kv_geom(lens[l], a.cap, n_pos, pnew, ok);

        // ------------------------------------------------------------ layer input x (fp16)
        // x = h + sum of the previous layer's FFN partials (layer 0: the token input)
        combine_norm(a.ffn_part, false, l == 0);

        // ------------------------------------------------------------ QKV rows
        {
            int rowbase = 0;
            for_qkv_pieces(a, c, NC, [&](int s, int r0, int r1) {
                for (int r = r0; r < r1; r += rps_d) {
                    const int n = min(rps_d, r1 - r);
                    const uint8_t* st = ring_acquire(ring, live, a);
                    if (!st) continue;
                    stage_mma_regs<STEPS>(ring_s + (uint32_t)(st - ring_base), n, D, gd, mld, rowbase + (r - r0), bh,
                                          bl, slots);
                    ring_release(ring, lane);
                }
                rowbase += r1 - r0;
            });
            consumer_bar(1, kTokConsumers);
            // epilogue: row pairs -> RoPE; q to the token's query buffer, k/v appended at pnew
            const int half = dh >> 1;
            rowbase = 0;
            for_qkv_pieces(a, c, NC, [&](int s, int r0, int r1) {
                const int npairs = (r1 - r0) >> 1, hq = a.hq[s], hk = a.hk[s];
                for (int t = tid; t < npairs && live; t += kTokConsumers) {
                    const int lr = rowbase + 2 * t;
                    const float ye = row_total(slots, lr, gd.spr), yo = row_total(slots, lr + 1, gd.spr);
                    const int gr = r0 + 2 * t;
                    const int b = gr / dh, i = (gr - b * dh) >> 1;
                    if (b < hq + hk) {
                        const float2 cs = ok ? a.rope[(int64_t)pnew * half + i] : make_float2(1.f, 0.f);
                        const float re = ye * cs.x - yo * cs.y;
                        const float ro = ye * cs.y + yo * cs.x;
                        if (b < hq) {
                            float* q = a.q_all + (size_t)(a.h0[s] + b) * dh;
                            __stcg(q + i, re);
                            __stcg(q + i + half, ro);
                        } else if (ok) {
                            __half* kd = sp[s].kc + ((int64_t)(b - hq) * a.cap + pnew) * dh;
                            kd[i] = __float2half_rn(re);
                            kd[i + half] = __float2half_rn(ro);
                        }
                    } else if (ok) {
                        __half* vd = sp[s].vc + ((int64_t)(b - hq - hk) * a.cap + pnew) * dh;
                        vd[i] = __float2half_rn(ye);
                        vd[i + half] = __float2half_rn(yo);
                    }
                }
                rowbase += r1 - r0;
            });
            if (!ok && c == 0 && tid == 0) set_status(a.status, VT_DEV_KV_OVERFLOW);
        }
        live = grid_sync(a, &s_flag, live, ++epoch, spin, skip_epoch);

        // ------------------------------------------------------------ attention slices
        if (c == 0 && live)  // nobody reads the previous layer's FFN partials any more
            for (int i = tid; i < a.n_dev * D; i += kTokConsumers) __stcg(a.ffn_part + i, 0.f);
        ring.live = live;
        // sliding window: the layer attends to positions [t_lo, n_pos); slices are cut from those
        const int t_lo = window_start(n_pos, a.layer[l].window), n_att = n_pos - t_lo;
        for_kv_pieces(a, n_att, c, NC, [&](int j, int t0, int t1, int seg) {
            ring = attn_slice<dh / 32, G>(a, sp, ring, j, t_lo + t0, t_lo + t1, seg, pnew, uni, tid, warp, lane);
        });
        live = ring.live;
        // Slice table of every KV head for the O phase: the state offset of each CTA slice of the
        // head (-1: none), mstride entries per head.  Every CTA builds the same table.
        const int T = a.n_kv * n_att;
        const int mstride = NC / a.n_kv + 3;
        int* mtab = reinterpret_cast<int*>(slots + a.slot_floats / 2);
        for (int idx = tid; idx < a.n_kv * mstride; idx += kTokConsumers) {
            const int j = idx / mstride, k = idx - j * mstride;
            int cf = 0, cl = -1, base = -1;
            if (T > 0) head_ctas(T, j, n_att, NC, cf, cl);
            if (cf + k <= cl) {
                const Span sx = cta_span(T, cf + k, NC);
                if (sx.a < sx.b) base = (((cf + k) * kTokMaxSeg + (j - sx.a / n_att)) * G) * (dh + 4);
            }
            mtab[idx] = base;
        }
        live = grid_sync(a, &s_flag, live, ++epoch, spin, skip_epoch);

        // ------------------------------------------------------------ O rows
        {
            for_o_pieces(a, c, NC, [&](int s, int r0, int r1) {
                const int K = a.hq[s] * dh;
                // Attention output of shard s: each thread merges 4 consecutive elements of one query
                // head over the head's slices (log-sum-exp weights), all its loads issued together.
                __half* xh = reinterpret_cast<__half*>(uni);
                __half* xl = xh + K;
                if (live) merge_heads(a, s, K, mtab, mstride, dsh, gsh, xh, xl, tid);
                consumer_bar(1, kTokConsumers);  // xh / xl ready; the merge scratch in the slots is free
                const MmaGeom go = mma_geom(K);
                const MmaLane mlo = mma_lane(go, warp, lane);
                const bool regs = mma_ok(K) && go.L == 16 * STEPS;
                if (!OSMEM || regs) {
                    // the rows' steps match the kernel's: B fragments in registers
                    load_bfrags_h<STEPS>(xh, xl, mlo, go.L, bh, bl);
                    int rowbase = 0;
                    for (int r = r0; r < r1; r += go.R) {
                        const int n = min(go.R, r1 - r);
                        const uint8_t* st = ring_acquire(ring, live, a);
                        if (!st) continue;
                        stage_mma_regs<STEPS>(ring_s + (uint32_t)(st - ring_base), n, K, go, mlo, rowbase, bh, bl, slots);
                        ring_release(ring, lane);
                        rowbase += n;
                    }
                    consumer_bar(1, kTokConsumers);
                    for (int rr = tid; rr < r1 - r0 && live; rr += kTokConsumers)
                        __stcg(a.attn_part + (size_t)s * D + r0 + rr, row_total(slots, rr, go.spr));
                } else if constexpr (OSMEM) {
                    if (mma_ok(K)) {
                        // B fragments from shared memory
                        int rowbase = 0;
                        for (int r = r0; r < r1; r += go.R) {
                            const int n = min(go.R, r1 - r);
                            const uint8_t* st = ring_acquire(ring, live, a);
                            if (!st) continue;
                            stage_mma_smem(ring_s + (uint32_t)(st - ring_base), n, K, go, mlo, rowbase, xh, xl, slots);
                            ring_release(ring, lane);
                            rowbase += n;
                        }
                        consumer_bar(1, kTokConsumers);
                        for (int rr = tid; rr < r1 - r0 && live; rr += kTokConsumers)
                            __stcg(a.attn_part + (size_t)s * D + r0 + rr, row_total(slots, rr, go.spr));
                    } else {
                        // rows too short for whole tensor-core steps: one warp per row on the CUDA cores
                        for (int r = r0; r < r1; r += go.R) {
                            const int n = min(go.R, r1 - r);
                            const uint8_t* st = ring_acquire(ring, live, a);
                            if (!st) continue;
                            for (int rr = warp; rr < n; rr += kTokWarps) {
                                const __half* row = reinterpret_cast<const __half*>(st) + (size_t)rr * K;
                                float acc = 0.f;
                                for (int e = lane; e < K; e += 32)
                                    acc = fmaf(__half2float(row[e]), __half2float(xh[e]) + __half2float(xl[e]), acc);
                                acc = warp_sum(acc);
                                if (lane == 0) __stcg(a.attn_part + (size_t)s * D + r + rr, acc);
                            }
                            ring_release(ring, lane);
                        }
                    }
                }
                consumer_bar(1, kTokConsumers);  // uni and the slots are rewritten by the next piece
            });
        }
        prefetch_bgain<STEPS>(a.layer[l].ffn_norm, mld, gd.L, gf);
        live = grid_sync(a, &s_flag, live, ++epoch, spin, skip_epoch);

        // ------------------------------------------------------------ FFN columns
        // h = x + sum of the ATTN partials (shards in order), rounded to fp16
        combine_norm(a.attn_part, true, false);
        for_ffn_pieces(a, c, NC, [&](int s, int j0, int j1) {
            for (int g = j0; g < j1; g += gcol) {
                const int ng = min(gcol, j1 - g);
                for (int r = 2 * g; r < 2 * (g + ng); r += rps_d) {
                    const int n = min(rps_d, 2 * (g + ng) - r);
                    const uint8_t* st = ring_acquire(ring, live, a);
                    if (!st) continue;
                    stage_mma_regs<STEPS>(ring_s + (uint32_t)(st - ring_base), n, D, gd, mld, r - 2 * g, bh, bl, slots);
                    ring_release(ring, lane);
                }
                consumer_bar(1, kTokConsumers);
                if (tid < ng) act[tid] = silu(row_total(slots, 2 * tid, gd.spr)) * row_total(slots, 2 * tid + 1, gd.spr);
                consumer_bar(1, kTokConsumers);
                float acc[MC][8];
#pragma unroll
                for (int m = 0; m < MC; ++m)
#pragma unroll
                    for (int e = 0; e < 8; ++e) acc[m][e] = 0.f;
                for (int r = g; r < g + ng; r += rps_d) {
                    const int n = min(rps_d, g + ng - r);
                    const uint8_t* st = ring_acquire(ring, live, a);
                    if (!st) continue;
                    for (int rr = 0; rr < n; ++rr) {
                        const float av = act[r - g + rr];
                        const uint8_t* row = st + (size_t)rr * D * 2;
#pragma unroll
                        for (int m = 0; m < MC; ++m) {
                            const int ch = tid + kTokConsumers * m;
                            if (ch < nch) {
                                float w[8];
                                unpack8(lds128(row + ch * 16), w);
#pragma unroll
                                for (int e = 0; e < 8; ++e) acc[m][e] = fmaf(av, w[e], acc[m][e]);
                            }
                        }
                    }
                    ring_release(ring, lane);
                }
                // the group's D-vector goes to the slots (free once the activations are computed) and
                // is added into the shard partial by one bulk reduction: a few hundred line-sized
                // additions in the L2 instead of thousands of vector atomics, which the CTA's barrier
                // arrival would have to wait for
#pragma unroll
                for (int m = 0; m < MC; ++m) {
                    const int ch = tid + kTokConsumers * m;
                    if (ch < nch) {
                        float4* v = reinterpret_cast<float4*>(slots + ch * 8);
                        v[0] = make_float4(acc[m][0], acc[m][1], acc[m][2], acc[m][3]);
                        v[1] = make_float4(acc[m][4], acc[m][5], acc[m][6], acc[m][7]);
                    }
                }
                fence_proxy_async_smem();
                consumer_bar(1, kTokConsumers);
                // (the additions complete before the phase's grid barrier, below)
                if (tid == 0 && live) bulk_reduce_add_f32_issue(a.ffn_part + (size_t)s * D, slots, (uint32_t)D * 4u);
                consumer_bar(1, kTokConsumers);  // the reduction has read the slots
            }
        });
        if (l + 1 < a.n_layers) prefetch_bgain<STEPS>(a.layer[l + 1].attn_norm, mld, gd.L, gf);
        if (tid == 0) {
            // this CTA's FFN partial additions (async proxy) complete before the barrier's release
            // store, which thread 0 makes
            bulk_wait_all();
            asm volatile("fence.proxy.async;" ::: "memory");
        }
        live = grid_sync(a, &s_flag, live, ++epoch, spin, skip_epoch);
    }

    // ---------------------------------------------------------------- output and KV lengths
    if (live) {
        // x16 holds h of the last layer in this thread's chunks; add the FFN partials
#pragma unroll
        for (int m = 0; m < MC; ++m) {
            const int ch = tid + kTokConsumers * m;
            if (ch < nch && (ch % NC) == c) {
                float v[8];
                unpack8(lds128(x16 + ch * 8), v);
                for (int s = 0; s < a.n_dev; ++s) add8_cg(v, a.ffn_part + (size_t)s * D + ch * 8);
                *reinterpret_cast<uint4*>(a.x_out + ch * 8) = pack8(v);
            }
        }
    }
    // every CTA read the lengths and the barrier epoch before its first grid barrier
    if (c == 0 && tid == 0) {
        for (int l = 0; l < a.n_layers; ++l) a.len[l] = lens[l] + 1;
        if (live) a.sync[kTokSyncEpoch] = epoch;
    }
}


// Host side of one kernel variant (instantiated by the token_v*.cu translation units).
template <int STEPS, int MC, int DH, int G, bool OSMEM>
struct TokVariantImpl {
    static cudaError_t init(int optin, size_t* dyn_max) {
        cudaFuncAttributes fa{};
        cudaError_t e = cudaFuncGetAttributes(&fa, k_decode_token<STEPS, MC, DH, G, OSMEM>);
        if (e != cudaSuccess) return e;
        *dyn_max = (size_t)optin > fa.sharedSizeBytes ? (size_t)optin - fa.sharedSizeBytes : 0;
        return cudaFuncSetAttribute(k_decode_token<STEPS, MC, DH, G, OSMEM>,
                                    cudaFuncAttributeMaxDynamicSharedMemorySize, (int)*dyn_max);
    }
    static cudaError_t occupancy(int* per_sm, size_t smem) {
        return cudaOccupancyMaxActiveBlocksPerMultiprocessor(per_sm, k_decode_token<STEPS, MC, DH, G, OSMEM>,
                                                             kTokThreads, smem);
    }
    static cudaError_t launch(const TokArgs& a, const cudaLaunchConfig_t& cfg) {
        return cudaLaunchKernelEx(&cfg, k_decode_token<STEPS, MC, DH, G, OSMEM>, a);
    }
    static TokVariant desc() {
        return TokVariant{STEPS, MC, DH, G, OSMEM, &init, &occupancy, &launch};
    }
};

}  // namespace
}  // namespace vt
