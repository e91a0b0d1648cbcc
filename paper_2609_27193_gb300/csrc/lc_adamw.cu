// lc_adamw.cu -- one AdamW step fused with the Eq. 1 sums of its update
// (§3.4.2: the drift is computed on the optimizer update path, so W(t-1) is
// read once, by the optimizer).  W is fp32 master weights here, so a
// 16-byte vector holds 4 parameters; the work partition, the partial slots
// and the fixed-order finalize are those of the measure scan.
#include "lc_bulk.cuh"
#include "lc_reduce.cuh"

#include <cuda_bf16.h>

namespace lc {
namespace {

#ifndef LC_ADAM_UNROLL
#define LC_ADAM_UNROLL 2
#endif
#ifndef LC_ADAM_MIN_BLOCKS
#define LC_ADAM_MIN_BLOCKS 2
#endif
constexpr int kAdamUnroll = LC_ADAM_UNROLL;      // vectors in flight per thread (5 arrays each)
constexpr int kAdamFlush = 16 / LC_ADAM_UNROLL;  // fp32 chains of 16 terms

__device__ __forceinline__ float adam_elem(float p, float& m, float& v, float g, const AdamConsts& c,
                                           float& p_out) {
    const float p_decayed = __fmul_rn(p, c.decay);
    const float m_new = __fadd_rn(__fmul_rn(c.b1, m), __fmul_rn(c.omb1, g));
    const float v_new = __fadd_rn(__fmul_rn(c.b2, v), __fmul_rn(c.omb2, __fmul_rn(g, g)));
    const float v_hat = __fmul_rn(v_new, c.rbc2);
    const float denom = __fadd_rn(__fsqrt_rn(v_hat), c.eps);
    const float step = __fdiv_rn(__fmul_rn(m_new, c.step_size), denom);
    p_out = __fsub_rn(p_decayed, step);
    m = m_new;
    v = v_new;
    return p_out;
}

__device__ __forceinline__ uint32_t bf16_pair(float lo, float hi) {
    const __nv_bfloat162 b = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<const uint32_t*>(&b);
}

__device__ __forceinline__ uint2 ld_u2(const void* p) {
    uint2 v;
    asm volatile("ld.global.nc.L1::no_allocate.v2.u32 {%0,%1}, [%2];" : "=r"(v.x), "=r"(v.y) : "l"(p));
    return v;
}

// Coherent load of data this kernel rewrites (volatile: kept in program
// order with the stores, which all come after the loads they follow).
__device__ __forceinline__ uint4 ld_rw(const void* p) {
    uint4 v;
    asm volatile("ld.global.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

__device__ __forceinline__ void st_u2(void* p, uint2 v) {
    asm volatile("st.global.v2.u32 [%0], {%1,%2};" : : "l"(p), "r"(v.x), "r"(v.y) : "memory");
}

// kAdamUnroll aligned vectors (4 parameters each) of a fast segment: all
// loads first, then the arithmetic, then all stores.
template <bool GRAD_BF16>
__device__ __forceinline__ void adam_vectors(const SegDev& sd, const OptSegDev& od, int64_t k,
                                             int64_t kend, const AdamConsts& c, float (&ad)[4],
                                             float (&aa)[4]) {
    constexpr int BS = kMeasureThreads;
    constexpr int U = kAdamUnroll;
    uint8_t* wb = const_cast<uint8_t*>(sd.w) - 4 * int64_t(sd.lead);
    uint8_t* mb = reinterpret_cast<uint8_t*>(od.m) - 4 * int64_t(sd.lead);
    uint8_t* vb = reinterpret_cast<uint8_t*>(od.v) - 4 * int64_t(sd.lead);
    const uint8_t* gb = od.grad - (GRAD_BF16 ? 2 : 4) * int64_t(sd.lead);
    uint4 pw[U], mw[U], vw[U];
    uint4 gw[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
        const int64_t kk = k + int64_t(u) * BS;
        if (kk < kend) {
            pw[u] = ld_rw(wb + 16 * kk);
            mw[u] = ld_rw(mb + 16 * kk);
            vw[u] = ld_rw(vb + 16 * kk);
            if (GRAD_BF16) {
                const uint2 g2 = ld_u2(gb + 8 * kk);
                gw[u] = make_uint4(g2.x, g2.y, 0u, 0u);
            } else {
                gw[u] = ld_stream(gb + 16 * kk);
            }
        }
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
        const int64_t kk = k + int64_t(u) * BS;
        if (kk >= kend) continue;
        float g[4];
        if (GRAD_BF16) {
            g[0] = bf16_lo(gw[u].x); g[1] = bf16_hi(gw[u].x); g[2] = bf16_lo(gw[u].y); g[3] = bf16_hi(gw[u].y);
        } else {
            g[0] = __uint_as_float(gw[u].x); g[1] = __uint_as_float(gw[u].y);
            g[2] = __uint_as_float(gw[u].z); g[3] = __uint_as_float(gw[u].w);
        }
        float p[4] = {__uint_as_float(pw[u].x), __uint_as_float(pw[u].y), __uint_as_float(pw[u].z),
                      __uint_as_float(pw[u].w)};
        float m[4] = {__uint_as_float(mw[u].x), __uint_as_float(mw[u].y), __uint_as_float(mw[u].z),
                      __uint_as_float(mw[u].w)};
        float v[4] = {__uint_as_float(vw[u].x), __uint_as_float(vw[u].y), __uint_as_float(vw[u].z),
                      __uint_as_float(vw[u].w)};
        float pn[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            adam_elem(p[j], m[j], v[j], g[j], c, pn[j]);
            ad[j] += fabsf(pn[j] - p[j]);
            aa[j] += fabsf(p[j]);
        }
        st_vec(wb + 16 * kk, make_uint4(__float_as_uint(pn[0]), __float_as_uint(pn[1]),
                                        __float_as_uint(pn[2]), __float_as_uint(pn[3])));
        st_vec(mb + 16 * kk, make_uint4(__float_as_uint(m[0]), __float_as_uint(m[1]),
                                        __float_as_uint(m[2]), __float_as_uint(m[3])));
        st_vec(vb + 16 * kk, make_uint4(__float_as_uint(v[0]), __float_as_uint(v[1]),
                                        __float_as_uint(v[2]), __float_as_uint(v[3])));
        if (od.model)
            st_u2(od.model - 2 * int64_t(sd.lead) + 8 * kk,
                  make_uint2(bf16_pair(pn[0], pn[1]), bf16_pair(pn[2], pn[3])));
    }
}

// Element-wise path: partial edge vectors and segments that do not line up.
__device__ void adam_scalar_vector(const SegDev& sd, const OptSegDev& od, int64_t k,
                                   const AdamConsts& c, double& dd, double& da) {
    float* w = reinterpret_cast<float*>(const_cast<uint8_t*>(sd.w));
    for (int j = 0; j < 4; ++j) {
        const int64_t e = 4 * k - sd.lead + j;
        if (e < 0 || e >= sd.numel) continue;
        const float g = od.grad_bf16
                            ? __uint_as_float(uint32_t(reinterpret_cast<const uint16_t*>(od.grad)[e]) << 16)
                            : reinterpret_cast<const float*>(od.grad)[e];
        const float p = w[e];
        float m = od.m[e], v = od.v[e], pn;
        adam_elem(p, m, v, g, c, pn);
        w[e] = pn;
        od.m[e] = m;
        od.v[e] = v;
        if (od.model) reinterpret_cast<__nv_bfloat16*>(od.model)[e] = __float2bfloat16_rn(pn);
        dd += double(fabsf(pn - p));
        da += double(fabsf(p));
    }
}

__device__ void adam_run(const SegDev& sd, const OptSegDev& od, int64_t lo, int64_t hi,
                         const AdamConsts& c, double& dd, double& da) {
    constexpr int BS = kMeasureThreads;
    const bool head_partial = sd.lead > 0;
    const bool tail_partial = ((int64_t(sd.lead) + sd.numel) % 4) != 0;
    if (!od.fast) {
        for (int64_t k = lo + threadIdx.x; k < hi; k += BS) adam_scalar_vector(sd, od, k, c, dd, da);
        return;
    }
    const int64_t kf0 = head_partial ? 1 : 0;
    const int64_t kf1 = tail_partial ? sd.nvec - 1 : sd.nvec;
    const int64_t a = lo > kf0 ? lo : kf0;
    const int64_t b = hi < kf1 ? hi : kf1;
    int64_t k = a + threadIdx.x;
    while (k < b) {
        float ad[4] = {0.f, 0.f, 0.f, 0.f}, aa[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 1
        for (int f = 0; f < kAdamFlush && k < b; ++f) {
            if (od.grad_bf16) adam_vectors<true>(sd, od, k, b, c, ad, aa);
            else adam_vectors<false>(sd, od, k, b, c, ad, aa);
            k += int64_t(kAdamUnroll) * BS;
        }
        dd += double((ad[0] + ad[1]) + (ad[2] + ad[3]));
        da += double((aa[0] + aa[1]) + (aa[2] + aa[3]));
    }
    if (threadIdx.x == 0) {
        if (head_partial && lo <= 0 && 0 < hi) adam_scalar_vector(sd, od, 0, c, dd, da);
        const int64_t last = sd.nvec - 1;
        if (tail_partial && last >= lo && last < hi && !(head_partial && last == 0))
            adam_scalar_vector(sd, od, last, c, dd, da);
    }
}

__global__ void __launch_bounds__(kMeasureThreads, LC_ADAM_MIN_BLOCKS) adamw_measure_kernel(const MeasureParams p,
                                                                        const OptSegDev* opt,
                                                                        const AdamConsts c) {
    __shared__ double red_d[kMeasureThreads / 32];
    __shared__ double red_a[kMeasureThreads / 32];
    __shared__ unsigned int s_ticket;
    const int b = blockIdx.x;
    int64_t v0 = p.cta_vec_begin[b];
    const int64_t v1 = p.cta_vec_begin[b + 1];
    int s = p.cta_seg0[b];
    int slot = p.cta_slot0[b];
    while (v0 < v1 && s < p.nseg) {
        const SegDev sd = p.segs[s];
        const OptSegDev od = opt[s];
        const int64_t seg_end = sd.vec_begin + sd.nvec;
        const int64_t lo = v0 - sd.vec_begin;
        const int64_t hi = (v1 < seg_end ? v1 : seg_end) - sd.vec_begin;
        double dd = 0.0, da = 0.0;
        adam_run(sd, od, lo, hi, c, dd, da);
        block_sum(dd, da, red_d, red_a);
        if (threadIdx.x == 0) p.partials[slot] = make_double2(dd, da);
        ++slot;
        ++s;
        v0 = sd.vec_begin + hi;
    }
    if (threadIdx.x == 0) {
        __threadfence();
        s_ticket = atomicAdd(p.ticket, 1u);
    }
    __syncthreads();
    if (s_ticket != gridDim.x - 1) return;
    __threadfence();
    finalize(p);
}

// ---------------------------------------------------------------------------
// Bulk-load form.  A per-thread step keeps only a few vectors of each array
// in flight (registers bound it).  Here one producer thread (warp 0) streams
// chunks of kAChunkVec vectors of w, m, v and the gradient into a ring of
// kAStages shared-memory buffers with cp.async.bulk, so the bytes in flight
// no longer cost registers; seven consumer warps take each chunk from
// shared memory, run the same element step, store w, m, v and the bf16
// model copy with ordinary 16- and 8-byte stores, and add the Eq. 1 sums of
// the update.  Edge vectors, segments whose arrays do not line up and
// gradient vectors that would start a bulk copy off a 16-byte boundary go
// element by element.  Partition (with its pool of units), jobs, the run
// box that combines the warps' partial sums, and bounded waits are those of
// the bulk-load measure.
// ---------------------------------------------------------------------------
#ifndef LC_ADAM_BULK_STAGES
#define LC_ADAM_BULK_STAGES 2
#endif
#ifndef LC_ADAM_BULK_VECS
#define LC_ADAM_BULK_VECS 512
#endif
// 1: the updated w, m and v go back into the buffer and one thread (warp 1)
// writes them with bulk stores; 0: the consumers store them themselves.
#ifndef LC_ADAM_BULK_STORE
#define LC_ADAM_BULK_STORE 1
#endif
constexpr bool kABulkStore = LC_ADAM_BULK_STORE != 0;
constexpr int kAStages = LC_ADAM_BULK_STAGES;
constexpr int kAChunkVec = LC_ADAM_BULK_VECS;                 // vectors of 4 parameters per chunk
constexpr uint32_t kAStage = uint32_t(kAChunkVec) * 64u;      // w, m, v and gradient, 16 B each per vector
constexpr size_t kAdamBulkSmem = size_t(kAStages) * kAStage;
constexpr int kAFirstConsumerWarp = kABulkStore ? 2 : 1;
constexpr int kAConsumerWarps = kMeasureThreads / 32 - kAFirstConsumerWarp;
constexpr int kAConsumers = 32 * kAConsumerWarps;
static_assert(kAChunkVec % 2 == 0 && kAStages >= 2, "fused ring shape");

enum : int32_t { kAJobChunk = 0, kAJobScalar = 1, kAJobFlush = 2, kAJobEnd = 3 };

struct AJob {
    int64_t k0, k1;
    int32_t kind;
    int32_t seg;
    int32_t slot;
    int32_t pad;
};

struct ARing {
    uint64_t full[kAStages];
    uint64_t computed[kAStages];   // consumers done with the buffer (bulk-store form)
    uint64_t empty[kAStages];
    AJob jobs[kAStages];
    RunBox<kAStages, kAConsumerWarps> box;
};

__device__ void adam_produce(const MeasureParams& p, const OptSegDev* opt, uint8_t* ring, ARing& r) {
    const uint32_t ring_s = smem_addr(ring);
    const uint32_t full_s = smem_addr(r.full), empty_s = smem_addr(r.empty);
    uint64_t k = 0;
    bool stall = p.stall_first != 0;
    auto post = [&](const AJob& j, const SegDev& sd, const OptSegDev& od) -> bool {
        const int st = int(k % kAStages);
        if (k >= uint64_t(kAStages) &&
            !mbar_wait_bounded(empty_s + 8 * st, uint32_t((k / kAStages - 1) & 1), kWaitNs))
            return false;
        r.jobs[st] = j;
        if (j.kind == kAJobChunk) {
            const uint32_t n = uint32_t(j.k1 - j.k0);
            const int64_t lead = sd.lead;
            const uint32_t gsz = od.grad_bf16 ? 8u : 16u;
            const uint32_t buf = ring_s + uint32_t(st) * kAStage;
            mbar_expect_tx(full_s + 8 * st, n * (48u + gsz) + (stall ? 16u : 0u));
            stall = false;
            bulk_g2s(buf, sd.w - 4 * lead + 16 * j.k0, 16 * n, full_s + 8 * st);
            bulk_g2s(buf + 16 * kAChunkVec, reinterpret_cast<const uint8_t*>(od.m) - 4 * lead + 16 * j.k0,
                     16 * n, full_s + 8 * st);
            bulk_g2s(buf + 32 * kAChunkVec, reinterpret_cast<const uint8_t*>(od.v) - 4 * lead + 16 * j.k0,
                     16 * n, full_s + 8 * st);
            bulk_g2s(buf + 48 * kAChunkVec, od.grad - (od.grad_bf16 ? 2 : 4) * lead + int64_t(gsz) * j.k0,
                     gsz * n, full_s + 8 * st);
        } else {
            mbar_arrive(full_s + 8 * st);
        }
        ++k;
        return true;
    };
    bool ok = true;
    SegDev sd{};
    OptSegDev od{};
    // the CTA's own range, then units of the pool until it is empty
    for (int rng = int(blockIdx.x); ok && rng >= 0; rng = ok ? next_pool_range(p) : -1) {
        int64_t v0 = p.cta_vec_begin[rng];
        const int64_t v1 = p.cta_vec_begin[rng + 1];
        int s = p.cta_seg0[rng];
        int slot = p.cta_slot0[rng];
        while (ok && v0 < v1 && s < p.nseg) {
            sd = p.segs[s];
            od = opt[s];
            const int64_t seg_end = sd.vec_begin + sd.nvec;
            const int64_t lo = v0 - sd.vec_begin;
            const int64_t hi = (v1 < seg_end ? v1 : seg_end) - sd.vec_begin;
            const bool head_partial = sd.lead > 0;
            const bool tail_partial = ((int64_t(sd.lead) + sd.numel) % 4) != 0;
            if (od.fast) {
                if (head_partial && lo <= 0 && 0 < hi) ok = post({0, 1, kAJobScalar, s, slot, 0}, sd, od);
                const int64_t kf0 = head_partial ? 1 : 0;
                const int64_t kf1 = tail_partial ? sd.nvec - 1 : sd.nvec;
                int64_t x = lo > kf0 ? lo : kf0;
                const int64_t e = hi < kf1 ? hi : kf1;
                // a bf16 gradient vector is 8 bytes: a bulk copy must start on 16
                const uintptr_t gb = uintptr_t(od.grad) - 2 * uintptr_t(sd.lead);
                if (ok && od.grad_bf16 && x < e && ((gb + 8 * uintptr_t(x)) & 15)) {
                    ok = post({x, x + 1, kAJobScalar, s, slot, 0}, sd, od);
                    ++x;
                }
                while (ok && x < e) {
                    int64_t n = e - x < kAChunkVec ? e - x : kAChunkVec;
                    if (od.grad_bf16 && (n & 1)) n -= 1;      // the gradient bytes stay a multiple of 16
                    if (n == 0) {
                        ok = post({x, x + 1, kAJobScalar, s, slot, 0}, sd, od);
                        ++x;
                        continue;
                    }
                    ok = post({x, x + n, kAJobChunk, s, slot, 0}, sd, od);
                    x += n;
                }
                const int64_t last = sd.nvec - 1;
                if (ok && tail_partial && last >= lo && last < hi && !(head_partial && last == 0))
                    ok = post({last, last + 1, kAJobScalar, s, slot, 0}, sd, od);
            } else {
                ok = post({lo, hi, kAJobScalar, s, slot, 0}, sd, od);
            }
            if (ok) ok = post({0, 0, kAJobFlush, s, slot, 0}, sd, od);
            slot += kMeasureBulkSlotsPerRun;
            ++s;
            v0 = sd.vec_begin + hi;
        }
    }
    if (ok) ok = post({0, 0, kAJobEnd, 0, 0, 0}, sd, od);
    if (!ok) {
        raise_fault(p.fault);
        const uint64_t first = k > uint64_t(kAStages) ? k - kAStages : 0;
        for (uint64_t c = first; c < k; ++c)
            mbar_wait_bounded(full_s + 8 * int(c % kAStages), uint32_t((c / kAStages) & 1), kDrainNs);
    }
}

__device__ void adam_consume(const MeasureParams& p, const OptSegDev* opt, const AdamConsts& c,
                             uint8_t* ring, ARing& r) {
    const uint32_t full_s = smem_addr(r.full), empty_s = smem_addr(r.empty);
    const uint32_t done_s = smem_addr(r.computed);
    const int tid = int(threadIdx.x) - 32 * kAFirstConsumerWarp;
    const int warp = tid >> 5, lane = tid & 31;
    double dd = 0.0, da = 0.0;
    for (uint64_t k = 0;; ++k) {
        const int st = int(k % kAStages);
        const uint32_t parity = uint32_t((k / kAStages) & 1);
        int ok = 1;
        if (lane == 0) ok = mbar_wait_bounded(full_s + 8 * st, parity, kWaitNs) ? 1 : 0;
        ok = __shfl_sync(0xffffffffu, ok, 0);
        if (!ok) {
            if (lane == 0) raise_fault(p.fault);
            break;
        }
        mbar_try_wait(full_s + 8 * st, parity);
        const AJob j = r.jobs[st];
        if (j.kind == kAJobEnd) {
            if (kABulkStore && lane == 0) mbar_arrive(done_s + 8 * st);   // lets the storer see the end
            break;
        }
        if (j.kind == kAJobChunk) {
            const SegDev sd = p.segs[j.seg];
            const OptSegDev od = opt[j.seg];
            uint8_t* buf = ring + size_t(st) * kAStage;
            uint4* W = reinterpret_cast<uint4*>(buf);
            uint4* M = reinterpret_cast<uint4*>(buf + 16 * kAChunkVec);
            uint4* V = reinterpret_cast<uint4*>(buf + 32 * kAChunkVec);
            const uint8_t* G = buf + 48 * kAChunkVec;
            uint8_t* wb = const_cast<uint8_t*>(sd.w) - 4 * int64_t(sd.lead) + 16 * j.k0;
            uint8_t* mb = reinterpret_cast<uint8_t*>(od.m) - 4 * int64_t(sd.lead) + 16 * j.k0;
            uint8_t* vb = reinterpret_cast<uint8_t*>(od.v) - 4 * int64_t(sd.lead) + 16 * j.k0;
            uint8_t* modb = od.model ? od.model - 2 * int64_t(sd.lead) + 8 * j.k0 : nullptr;
            const int n = int(j.k1 - j.k0);
            float ad[4] = {0.f, 0.f, 0.f, 0.f}, aa[4] = {0.f, 0.f, 0.f, 0.f};
            for (int q = tid; q < n; q += kAConsumers) {
                const uint4 pw = W[q], mw = M[q], vw = V[q];
                float g[4];
                if (od.grad_bf16) {
                    const uint2 g2 = reinterpret_cast<const uint2*>(G)[q];
                    g[0] = bf16_lo(g2.x); g[1] = bf16_hi(g2.x); g[2] = bf16_lo(g2.y); g[3] = bf16_hi(g2.y);
                } else {
                    const uint4 g4 = reinterpret_cast<const uint4*>(G)[q];
                    g[0] = __uint_as_float(g4.x); g[1] = __uint_as_float(g4.y);
                    g[2] = __uint_as_float(g4.z); g[3] = __uint_as_float(g4.w);
                }
                float pv[4] = {__uint_as_float(pw.x), __uint_as_float(pw.y), __uint_as_float(pw.z),
                               __uint_as_float(pw.w)};
                float m[4] = {__uint_as_float(mw.x), __uint_as_float(mw.y), __uint_as_float(mw.z),
                              __uint_as_float(mw.w)};
                float v[4] = {__uint_as_float(vw.x), __uint_as_float(vw.y), __uint_as_float(vw.z),
                              __uint_as_float(vw.w)};
                float pn[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    adam_elem(pv[e], m[e], v[e], g[e], c, pn[e]);
                    ad[e] += fabsf(pn[e] - pv[e]);
                    aa[e] += fabsf(pv[e]);
                }
                const uint4 pnw = make_uint4(__float_as_uint(pn[0]), __float_as_uint(pn[1]),
                                             __float_as_uint(pn[2]), __float_as_uint(pn[3]));
                const uint4 mnw = make_uint4(__float_as_uint(m[0]), __float_as_uint(m[1]),
                                             __float_as_uint(m[2]), __float_as_uint(m[3]));
                const uint4 vnw = make_uint4(__float_as_uint(v[0]), __float_as_uint(v[1]),
                                             __float_as_uint(v[2]), __float_as_uint(v[3]));
                if (kABulkStore) {
                    W[q] = pnw;
                    M[q] = mnw;
                    V[q] = vnw;
                } else {
                    st_vec(wb + 16 * q, pnw);
                    st_vec(mb + 16 * q, mnw);
                    st_vec(vb + 16 * q, vnw);
                }
                if (modb) st_u2(modb + 8 * q, make_uint2(bf16_pair(pn[0], pn[1]), bf16_pair(pn[2], pn[3])));
            }
            dd += double((ad[0] + ad[1]) + (ad[2] + ad[3]));
            da += double((aa[0] + aa[1]) + (aa[2] + aa[3]));
            // the storer's bulk copies read what this thread wrote to the buffer
            if (kABulkStore) asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        } else if (j.kind == kAJobScalar) {
            const SegDev sd = p.segs[j.seg];
            const OptSegDev od = opt[j.seg];
            for (int64_t q = j.k0 + tid; q < j.k1; q += kAConsumers) adam_scalar_vector(sd, od, q, c, dd, da);
        } else {
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) {
                dd += __shfl_down_sync(0xffffffffu, dd, off);
                da += __shfl_down_sync(0xffffffffu, da, off);
            }
            if (lane == 0) run_box_put<kAConsumerWarps>(r.box, st, warp, dd, da, p.partials + j.slot);
            dd = 0.0;
            da = 0.0;
        }
        __syncwarp();
        if (lane == 0) mbar_arrive((kABulkStore ? done_s : empty_s) + 8 * st);
    }
}

// Bulk-store form: once every consumer warp is done with a buffer, write its
// updated w, m and v back with bulk stores, and hand the buffer to the
// producer when those stores have read it.
__device__ void adam_store(const MeasureParams& p, const OptSegDev* opt, const uint8_t* ring, ARing& r) {
    const uint32_t done_s = smem_addr(r.computed), empty_s = smem_addr(r.empty);
    const uint32_t ring_s = smem_addr(ring);
    for (uint64_t k = 0;; ++k) {
        const int st = int(k % kAStages);
        if (!mbar_wait_bounded(done_s + 8 * st, uint32_t((k / kAStages) & 1), kWaitNs)) {
            raise_fault(p.fault);
            break;
        }
        const AJob j = r.jobs[st];
        if (j.kind == kAJobEnd) break;
        if (j.kind == kAJobChunk) {
            const SegDev sd = p.segs[j.seg];
            const OptSegDev od = opt[j.seg];
            const int64_t off = 16 * j.k0 - 4 * int64_t(sd.lead);
            const uint32_t bytes = uint32_t(j.k1 - j.k0) * 16u;
            const uint32_t buf = ring_s + uint32_t(st) * kAStage;
            asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(sd.w + off),
                         "r"(buf), "r"(bytes)
                         : "memory");
            asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(
                             reinterpret_cast<uint8_t*>(od.m) + off),
                         "r"(buf + 16 * kAChunkVec), "r"(bytes)
                         : "memory");
            asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(
                             reinterpret_cast<uint8_t*>(od.v) + off),
                         "r"(buf + 32 * kAChunkVec), "r"(bytes)
                         : "memory");
            asm volatile("cp.async.bulk.commit_group;" ::: "memory");
            asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
        }
        mbar_arrive(empty_s + 8 * st);
    }
    asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
}

__global__ void __launch_bounds__(kMeasureThreads, 1) adamw_bulk_kernel(const MeasureParams p,
                                                                         const OptSegDev* opt,
                                                                         const AdamConsts c) {
    extern __shared__ __align__(128) uint8_t ring[];
    __shared__ __align__(8) ARing r;
    __shared__ unsigned int s_ticket;
    if (threadIdx.x == 0) {
        for (int st = 0; st < kAStages; ++st) {
            mbar_init(smem_addr(&r.full[st]), 1);
            mbar_init(smem_addr(&r.computed[st]), kAConsumerWarps);
            mbar_init(smem_addr(&r.empty[st]), kABulkStore ? 1 : kAConsumerWarps);
            r.box.count[st] = 0u;
        }
        mbar_init_fence();
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        adam_produce(p, opt, ring, r);
    } else if (kABulkStore && threadIdx.x < 64) {
        if (threadIdx.x == 32) adam_store(p, opt, ring, r);
    } else if (threadIdx.x >= 32) {
        adam_consume(p, opt, c, ring, r);
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        s_ticket = atomicAdd(p.ticket, 1u);
    }
    __syncthreads();
    if (s_ticket != gridDim.x - 1) return;
    __threadfence();
    // every load and bulk store of the ring is complete: it stages the combine
    finalize(p, reinterpret_cast<double2*>(ring), int32_t(kAdamBulkSmem / sizeof(double2)));
}

}  // namespace

cudaError_t launch_adamw_measure(const MeasureParams& p, const OptSegDev* opt, const AdamConsts& c,
                                 int grid, cudaStream_t s) {
    cudaGetLastError();
    adamw_measure_kernel<<<grid, kMeasureThreads, 0, s>>>(p, opt, c);
    return cudaGetLastError();
}

cudaError_t launch_adamw_bulk(const MeasureParams& p, const OptSegDev* opt, const AdamConsts& c, int grid,
                              cudaStream_t s) {
    cudaGetLastError();
    adamw_bulk_kernel<<<grid, kMeasureThreads, kAdamBulkSmem, s>>>(p, opt, c);
    return cudaGetLastError();
}

cudaError_t adamw_bulk_prepare(int* blocks_per_sm) {
    const cudaError_t e = cudaFuncSetAttribute(adamw_bulk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               int(kAdamBulkSmem));
    if (e != cudaSuccess) return e;
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks_per_sm, adamw_bulk_kernel, kMeasureThreads,
                                                         kAdamBulkSmem);
}

}  // namespace lc
