// lc_reduce.cuh -- device helpers shared by the kernels that reduce over
// the measure work space (lc_measure.cu: the Eq. 1 scan; lc_adamw.cu: the
// fused optimizer step): streaming loads and stores, bf16 decoding, the
// fixed-order CTA sum and the last-CTA fp64 combine per segment and layer.
#pragma once

#include "lc_internal.cuh"

namespace lc {
namespace {

#ifndef LC_LD_PREFETCH
#define LC_LD_PREFETCH 1
#endif

__device__ __forceinline__ uint4 ld_stream(const void* p) {
    uint4 v;
#if LC_LD_PREFETCH
    asm volatile("ld.global.nc.L1::no_allocate.L2::256B.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
#else
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
#endif
    return v;
}

// Coherent load for R when the kernel also writes R (accumulate mode).
__device__ __forceinline__ uint4 ld_coherent(const void* p) {
    uint4 v;
    asm volatile("ld.global.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p)
                 : "memory");
    return v;
}

__device__ __forceinline__ void st_vec(void* p, uint4 v) {
    asm volatile("st.global.v4.u32 [%0], {%1,%2,%3,%4};"
                 :
                 : "l"(p), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
                 : "memory");
}

__device__ __forceinline__ float bf16_lo(uint32_t x) { return __uint_as_float(x << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t x) { return __uint_as_float(x & 0xffff0000u); }

// Sum over the CTA in a fixed order; the result is valid in thread 0.
__device__ __forceinline__ void block_sum(double& d, double& a, double* sd, double* sa) {
    constexpr int kWarps = kMeasureThreads / 32;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
        d += __shfl_down_sync(0xffffffffu, d, off);
        a += __shfl_down_sync(0xffffffffu, a, off);
    }
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (lane == 0) { sd[warp] = d; sa[warp] = a; }
    __syncthreads();
    if (threadIdx.x == 0) {
        double td = 0.0, ta = 0.0;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) { td += sd[w]; ta += sa[w]; }
        d = td;
        a = ta;
    }
    __syncthreads();
}

// A run's partial from a bulk kernel's consumer warps.  Each warp's lane 0
// leaves its warp-reduced (d, a) in the box of the flush job's ring stage;
// the last of the N contributing warps to arrive adds them in warp order and
// writes the run's one partial slot.  No warp waits for another.  A stage's
// box is used again only once every warp has handed that stage back, so
// warps up to a ring's depth apart never share a box.
template <int NSTAGES, int MAXW>
struct RunBox {
    double d[NSTAGES][MAXW];
    double a[NSTAGES][MAXW];
    unsigned int count[NSTAGES];
};

template <int N, int NSTAGES, int MAXW>
__device__ __forceinline__ void run_box_put(RunBox<NSTAGES, MAXW>& b, int st, int w, double d, double a,
                                            double2* slot) {
    static_assert(N <= MAXW, "run box too small");
    volatile double* vd = b.d[st];
    volatile double* va = b.a[st];
    vd[w] = d;
    va[w] = a;
    __threadfence_block();
    if (atomicAdd(&b.count[st], 1u) == unsigned(N - 1)) {
        __threadfence_block();
        double sd = 0.0, sa = 0.0;
        for (int i = 0; i < N; ++i) {
            sd += vd[i];
            sa += va[i];
        }
        *slot = make_double2(sd, sa);
        *reinterpret_cast<volatile unsigned int*>(&b.count[st]) = 0u;
    }
}

// The next pool range for the calling CTA (its producer thread), or -1 once
// the pool is empty.  Asked for only when the CTA's current range has been
// handed to its consumers, so a unit is claimed by whichever CTA is ready
// first.
__device__ __forceinline__ int next_pool_range(const MeasureParams& p) {
    if (p.units <= 0) return -1;
    const unsigned int u = atomicAdd(p.unit_next, 1u);
    return u < unsigned(p.units) ? int(gridDim.x) + int(u) : -1;
}

// Run by the last CTA: the partial slots of every segment are added, then
// one thread per layer adds its segments in order.  The order of every
// addition is fixed by the layout.  The combine runs while the rest of the
// GPU is idle, so its latency is the kernel's tail, and on this GPU fp64
// arithmetic runs at a few operations per cycle per SM: a warp-wide fp64
// add is expensive whether its lanes hold data or not.  The slot bounds of
// up to kFinBatch segments are staged in shared memory first.
//
// With `stage` (shared memory free for reuse, stage_slots slots of it: the
// bulk kernels' rings) the slots of consecutive segments -- contiguous in
// `partials` -- are first copied there by the whole CTA with kFinLoads
// independent loads in flight per thread.  A segment of at most kFinLane
// slots is then added by one thread in slot order (32 segments per warp
// instruction); a larger one by a warp (lane l takes slots l, l+32, ... in
// order, then a fixed shuffle tree); a segment with more slots than fit in
// the stage is added by a warp from global memory.  Without `stage` the
// same split applies with the slots read from global memory, a thread
// keeping kFinLaneLoads loads in flight.
constexpr int kFinBatch = 512;
constexpr int kFinLaneLoads = 4;
constexpr int kFinLoads = 8;
constexpr int kFinLane = 32;

// Slots [b0, b1) of one segment into (d, a) of lane 0, in the fixed order.
template <typename Slots>
__device__ __forceinline__ void fin_segment(const Slots& slot, int32_t b0, int32_t b1, int lane, double& d,
                                            double& a) {
    d = 0.0;
    a = 0.0;
    for (int32_t j = b0 + lane; j < b1; j += 32) {
        const double2 v = slot(j);
        d += v.x;
        a += v.y;
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
        d += __shfl_down_sync(0xffffffffu, d, off);
        a += __shfl_down_sync(0xffffffffu, a, off);
    }
}

__device__ void finalize(const MeasureParams& p, double2* stage = nullptr, int32_t stage_slots = 0) {
    __shared__ int32_t s_beg[kFinBatch + 1];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    auto global_slot = [&](int32_t j) { return __ldcg(&p.partials[j]); };
    for (int base = 0; base < p.nseg; base += kFinBatch) {
        const int nb = p.nseg - base < kFinBatch ? p.nseg - base : kFinBatch;
        __syncthreads();
        for (int i = threadIdx.x; i <= nb; i += blockDim.x) s_beg[i] = p.seg_slot_begin[base + i];
        __syncthreads();
        if (stage) {
            for (int g0 = 0; g0 < nb;) {
                // the longest run of segments [g0, g1) whose slots fit the stage
                int lo = g0 + 1, hi = nb;
                while (lo < hi) {
                    const int mid = (lo + hi + 1) >> 1;
                    if (s_beg[mid] - s_beg[g0] <= stage_slots) lo = mid;
                    else hi = mid - 1;
                }
                const int g1 = lo;
                const int32_t first = s_beg[g0];
                const int32_t n = s_beg[g1] - first;
                if (n > stage_slots) {          // one segment larger than the stage
                    if (warp == 0) {
                        double d, a;
                        fin_segment(global_slot, s_beg[g0], s_beg[g0 + 1], lane, d, a);
                        if (lane == 0) {
                            p.seg_sums[2 * (base + g0)] = d;
                            p.seg_sums[2 * (base + g0) + 1] = a;
                        }
                    }
                } else {
                    for (int32_t i0 = 0; i0 < n; i0 += int32_t(blockDim.x) * kFinLoads) {
                        double2 v[kFinLoads];
#pragma unroll
                        for (int k = 0; k < kFinLoads; ++k) {
                            const int32_t i = i0 + k * int32_t(blockDim.x) + int32_t(threadIdx.x);
                            if (i < n) v[k] = __ldcg(&p.partials[first + i]);
                        }
#pragma unroll
                        for (int k = 0; k < kFinLoads; ++k) {
                            const int32_t i = i0 + k * int32_t(blockDim.x) + int32_t(threadIdx.x);
                            if (i < n) stage[i] = v[k];
                        }
                    }
                    __syncthreads();
                    auto staged_slot = [&](int32_t j) { return stage[j - first]; };
                    for (int s = g0 + int(threadIdx.x); s < g1; s += int(blockDim.x)) {
                        const int32_t b0 = s_beg[s], b1 = s_beg[s + 1];
                        if (b1 - b0 > kFinLane) continue;
                        double d = 0.0, a = 0.0;
                        for (int32_t j = b0; j < b1; ++j) {
                            const double2 v = stage[j - first];
                            d += v.x;
                            a += v.y;
                        }
                        p.seg_sums[2 * (base + s)] = d;
                        p.seg_sums[2 * (base + s) + 1] = a;
                    }
                    for (int s = g0 + warp; s < g1; s += nw) {
                        if (s_beg[s + 1] - s_beg[s] <= kFinLane) continue;
                        double d, a;
                        fin_segment(staged_slot, s_beg[s], s_beg[s + 1], lane, d, a);
                        if (lane == 0) {
                            p.seg_sums[2 * (base + s)] = d;
                            p.seg_sums[2 * (base + s) + 1] = a;
                        }
                    }
                }
                __syncthreads();
                g0 = g1;
            }
            continue;
        }
        for (int s = int(threadIdx.x); s < nb; s += int(blockDim.x)) {
            const int32_t b0 = s_beg[s], b1 = s_beg[s + 1];
            if (b1 - b0 > kFinLane) continue;
            double d = 0.0, a = 0.0;
            for (int32_t j = b0; j < b1; j += kFinLaneLoads) {
                double2 v[kFinLaneLoads];
#pragma unroll
                for (int k = 0; k < kFinLaneLoads; ++k)
                    if (j + k < b1) v[k] = __ldcg(&p.partials[j + k]);
#pragma unroll
                for (int k = 0; k < kFinLaneLoads; ++k)
                    if (j + k < b1) {
                        d += v[k].x;
                        a += v[k].y;
                    }
            }
            p.seg_sums[2 * (base + s)] = d;
            p.seg_sums[2 * (base + s) + 1] = a;
        }
        for (int s = warp; s < nb; s += nw) {
            if (s_beg[s + 1] - s_beg[s] <= kFinLane) continue;
            double d, a;
            fin_segment(global_slot, s_beg[s], s_beg[s + 1], lane, d, a);
            if (lane == 0) {
                p.seg_sums[2 * (base + s)] = d;
                p.seg_sums[2 * (base + s) + 1] = a;
            }
        }
    }
    __syncthreads();
    for (int l = threadIdx.x; l < p.nlayers; l += blockDim.x) {
        double d = 0.0, a = 0.0;
        int64_t n = 0;
        const int sb = p.layer_seg_begin[l], se = p.layer_seg_begin[l + 1];
#pragma unroll 4
        for (int s = sb; s < se; ++s) {
            d += __ldcg(&p.seg_sums[2 * s]);
            a += __ldcg(&p.seg_sums[2 * s + 1]);
            n += p.segs[s].numel;
        }
        p.sums[3 * l] = d;
        p.sums[3 * l + 1] = a;
        p.sums[3 * l + 2] = double(n);
    }
    if (threadIdx.x == 0) {
        *p.ticket = 0u;
        if (p.unit_next) *p.unit_next = 0u;   // every CTA has left the pool
    }
}

}  // namespace
}  // namespace lc
