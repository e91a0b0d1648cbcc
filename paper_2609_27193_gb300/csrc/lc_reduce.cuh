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

// Run by the last CTA: one warp per segment adds the segment's partial
// slots (lane l takes slots l, l+32, ... in order, then a fixed shuffle
// tree), so a segment that spans many CTAs costs a few dependent loads per
// lane instead of one per slot; then one thread per layer adds its segments.
__device__ void finalize(const MeasureParams& p) {
    const int lane = threadIdx.x & 31;
    for (int s = threadIdx.x >> 5; s < p.nseg; s += blockDim.x >> 5) {
        double d = 0.0, a = 0.0;
        for (int j = p.seg_slot_begin[s] + lane; j < p.seg_slot_begin[s + 1]; j += 32) {
            const double2 v = __ldcg(&p.partials[j]);
            d += v.x;
            a += v.y;
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
            d += __shfl_down_sync(0xffffffffu, d, off);
            a += __shfl_down_sync(0xffffffffu, a, off);
        }
        if (lane == 0) {
            p.seg_sums[2 * s] = d;
            p.seg_sums[2 * s + 1] = a;
        }
    }
    __syncthreads();
    for (int l = threadIdx.x; l < p.nlayers; l += blockDim.x) {
        double d = 0.0, a = 0.0;
        int64_t n = 0;
        for (int s = p.layer_seg_begin[l]; s < p.layer_seg_begin[l + 1]; ++s) {
            d += __ldcg(&p.seg_sums[2 * s]);
            a += __ldcg(&p.seg_sums[2 * s + 1]);
            n += p.segs[s].numel;
        }
        p.sums[3 * l] = d;
        p.sums[3 * l + 1] = a;
        p.sums[3 * l + 2] = double(n);
    }
    if (threadIdx.x == 0) *p.ticket = 0u;
}

}  // namespace
}  // namespace lc
