// lc_measure.cu -- Eq. 1 (§3.2) on sm_103a: per segment sum|W - R| and
// sum|R|, combined per layer with the element count.
//
// Work decomposition: every segment is covered by 16-byte "virtual vectors"
// aligned to absolute addresses (lc_internal.cuh).  All vectors of all
// segments, layers ascending, form one linear work space that is cut into
// G equal contiguous ranges, one per CTA, with G = resident CTAs on the
// device (one wave).  A CTA streams its range with 128-bit non-allocating
// loads of W and R, several in flight per thread, and writes one fp64
// partial per (CTA, segment) run.  The last CTA to finish (atomic ticket, no
// spinning) adds the partials of each segment, then the segments of each
// layer, in a fixed order, so the result is deterministic for a layout.
//
// Precision: per-thread fp32 accumulators take at most kUnroll * kFlush
// terms each before they are added (fixed tree) into per-thread fp64 sums;
// the relative error of a layer sum is below about 2e-6 (all terms >= 0).
#include "lc_internal.cuh"

#include <cuda_bf16.h>

namespace lc {
namespace {

#ifndef LC_MEASURE_UNROLL
#define LC_MEASURE_UNROLL 4
#endif
#ifndef LC_MEASURE_FLUSH
#define LC_MEASURE_FLUSH 4
#endif
#ifndef LC_LD_PREFETCH
#define LC_LD_PREFETCH 1
#endif
constexpr int kUnroll = LC_MEASURE_UNROLL;   // vectors of W (and of R) in flight per thread
constexpr int kFlush = LC_MEASURE_FLUSH;     // unrolled iterations between fp64 flushes
static_assert(kUnroll * kFlush <= 32, "fp32 partial sums are bounded to 32 terms");

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

// Adds one 16-byte vector pair into 8 fp32 lane accumulators.
template <int ESZ_LOG2>
__device__ __forceinline__ void accumulate(const uint4& w, const uint4& r, float (&ad)[8], float (&aa)[8]) {
    const uint32_t wv[4] = {w.x, w.y, w.z, w.w};
    const uint32_t rv[4] = {r.x, r.y, r.z, r.w};
    if constexpr (ESZ_LOG2 == 1) {
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const float w0 = bf16_lo(wv[j]), w1 = bf16_hi(wv[j]);
            const float r0 = bf16_lo(rv[j]), r1 = bf16_hi(rv[j]);
            ad[2 * j] += fabsf(w0 - r0);
            ad[2 * j + 1] += fabsf(w1 - r1);
            aa[2 * j] += fabsf(r0);
            aa[2 * j + 1] += fabsf(r1);
        }
    } else {
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const float w0 = __uint_as_float(wv[j]), r0 = __uint_as_float(rv[j]);
            ad[j] += fabsf(w0 - r0);
            aa[j] += fabsf(r0);
        }
    }
}

__device__ __forceinline__ float tree8(const float (&a)[8]) {
    return ((a[0] + a[1]) + (a[2] + a[3])) + ((a[4] + a[5]) + (a[6] + a[7]));
}

// Full, co-aligned vectors [k0, k1) of one segment.
template <int ESZ_LOG2, bool WRITE_R>
__device__ __forceinline__ void run_vectors(const SegDev& sd, int64_t k0, int64_t k1,
                                            double& dd, double& da) {
    constexpr int BS = kMeasureThreads;
    const uint8_t* wb = sd.w - (int64_t(sd.lead) << ESZ_LOG2);
    uint8_t* rb = sd.r - (int64_t(sd.lead) << ESZ_LOG2);
    int64_t k = k0 + threadIdx.x;
    while (k < k1) {
        float ad[8], aa[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) { ad[j] = 0.f; aa[j] = 0.f; }
#pragma unroll 1
        for (int f = 0; f < kFlush && k < k1; ++f) {
            if (k + int64_t(kUnroll - 1) * BS < k1) {
                uint4 w[kUnroll], r[kUnroll];
#pragma unroll
                for (int u = 0; u < kUnroll; ++u) {
                    w[u] = ld_stream(wb + 16 * (k + int64_t(u) * BS));
                    r[u] = WRITE_R ? ld_coherent(rb + 16 * (k + int64_t(u) * BS))
                                   : ld_stream(rb + 16 * (k + int64_t(u) * BS));
                }
                if constexpr (WRITE_R) {
#pragma unroll
                    for (int u = 0; u < kUnroll; ++u) st_vec(rb + 16 * (k + int64_t(u) * BS), w[u]);
                }
#pragma unroll
                for (int u = 0; u < kUnroll; ++u) accumulate<ESZ_LOG2>(w[u], r[u], ad, aa);
                k += int64_t(kUnroll) * BS;
            } else {
                const uint4 w = ld_stream(wb + 16 * k);
                const uint4 r = WRITE_R ? ld_coherent(rb + 16 * k) : ld_stream(rb + 16 * k);
                if constexpr (WRITE_R) st_vec(rb + 16 * k, w);
                accumulate<ESZ_LOG2>(w, r, ad, aa);
                k += BS;
            }
        }
        dd += double(tree8(ad));
        da += double(tree8(aa));
    }
}

__device__ __forceinline__ float load_elem(const uint8_t* base, int esz_log2, int64_t e) {
    if (esz_log2 == 1) {
        const uint16_t x = *reinterpret_cast<const uint16_t*>(base + 2 * e);
        return __uint_as_float(uint32_t(x) << 16);
    }
    return *reinterpret_cast<const float*>(base + 4 * e);
}

// Vector k of a segment element by element (partial edge vectors, and every
// vector of a segment whose W and R are not co-aligned).
template <bool WRITE_R>
__device__ void scalar_vector(const SegDev& sd, int64_t k, double& dd, double& da) {
    const int ve = 16 >> sd.esz_log2;
    for (int j = 0; j < ve; ++j) {
        const int64_t e = k * ve - sd.lead + j;
        if (e < 0 || e >= sd.numel) continue;
        const float w = load_elem(sd.w, sd.esz_log2, e);
        const float r = load_elem(sd.r, sd.esz_log2, e);
        dd += double(fabsf(w - r));
        da += double(fabsf(r));
        if constexpr (WRITE_R) {
            if (sd.esz_log2 == 1)
                reinterpret_cast<uint16_t*>(sd.r)[e] = reinterpret_cast<const uint16_t*>(sd.w)[e];
            else
                reinterpret_cast<float*>(sd.r)[e] = reinterpret_cast<const float*>(sd.w)[e];
        }
    }
}

// Vectors [lo, hi) of one segment into the calling thread's fp64 sums.
template <bool WRITE_R>
__device__ void process_run(const SegDev& sd, int64_t lo, int64_t hi, double& dd, double& da) {
    const int ve = 16 >> sd.esz_log2;
    const bool head_partial = sd.lead > 0;
    const bool tail_partial = ((int64_t(sd.lead) + sd.numel) % ve) != 0;
    if (sd.coaligned) {
        const int64_t kf0 = head_partial ? 1 : 0;
        const int64_t kf1 = tail_partial ? sd.nvec - 1 : sd.nvec;
        const int64_t a = lo > kf0 ? lo : kf0;
        const int64_t b = hi < kf1 ? hi : kf1;
        if (a < b) {
            if (sd.esz_log2 == 1) run_vectors<1, WRITE_R>(sd, a, b, dd, da);
            else run_vectors<2, WRITE_R>(sd, a, b, dd, da);
        }
        if (threadIdx.x == 0) {
            if (head_partial && lo <= 0 && 0 < hi) scalar_vector<WRITE_R>(sd, 0, dd, da);
            const int64_t last = sd.nvec - 1;
            if (tail_partial && last >= lo && last < hi && !(head_partial && last == 0))
                scalar_vector<WRITE_R>(sd, last, dd, da);
        }
    } else {
        for (int64_t k = lo + threadIdx.x; k < hi; k += kMeasureThreads)
            scalar_vector<WRITE_R>(sd, k, dd, da);
    }
}

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

__device__ void finalize(const MeasureParams& p) {
    for (int s = threadIdx.x; s < p.nseg; s += blockDim.x) {
        double d = 0.0, a = 0.0;
        for (int j = p.seg_slot_begin[s]; j < p.seg_slot_begin[s + 1]; ++j) {
            const double2 v = __ldcg(&p.partials[j]);
            d += v.x;
            a += v.y;
        }
        p.seg_sums[2 * s] = d;
        p.seg_sums[2 * s + 1] = a;
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

template <bool WRITE_R>
__global__ void __launch_bounds__(kMeasureThreads) measure_kernel(const MeasureParams p) {
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
        const int64_t seg_end = sd.vec_begin + sd.nvec;
        const int64_t lo = v0 - sd.vec_begin;
        const int64_t hi = (v1 < seg_end ? v1 : seg_end) - sd.vec_begin;
        double dd = 0.0, da = 0.0;
        process_run<WRITE_R>(sd, lo, hi, dd, da);
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
// Fused AdamW step + Eq. 1 sums of the update (§3.4.2).  W is fp32 here, so
// a 16-byte vector holds 4 parameters; the work partition, the partial
// slots and the finalize are those of the measure kernel.
// ---------------------------------------------------------------------------

constexpr int kAdamUnroll = 2;   // vectors in flight per thread (5 arrays each)
constexpr int kAdamFlush = 8;    // fp32 chains of kAdamUnroll*kAdamFlush = 16 terms

__device__ __forceinline__ float adam_elem(float p, float& m, float& v, float g, const AdamConsts& c,
                                           float& p_out) {
    const float p_decayed = __fmul_rn(p, c.decay);
    const float m_new = __fadd_rn(__fmul_rn(c.b1, m), __fmul_rn(c.omb1, g));
    const float v_new = __fadd_rn(__fmul_rn(c.b2, v), __fmul_rn(c.omb2, __fmul_rn(g, g)));
    const float m_hat = __fdiv_rn(m_new, c.bc1);
    const float v_hat = __fdiv_rn(v_new, c.bc2);
    const float denom = __fadd_rn(__fsqrt_rn(v_hat), c.eps);
    const float step = __fmul_rn(c.lr, __fdiv_rn(m_hat, denom));
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

__global__ void __launch_bounds__(kMeasureThreads) adamw_measure_kernel(const MeasureParams p,
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

}  // namespace

cudaError_t launch_adamw_measure(const MeasureParams& p, const OptSegDev* opt, const AdamConsts& c,
                                 int grid, cudaStream_t s) {
    cudaGetLastError();
    adamw_measure_kernel<<<grid, kMeasureThreads, 0, s>>>(p, opt, c);
    return cudaGetLastError();
}

cudaError_t launch_measure(const MeasureParams& p, int grid, bool write_ref, cudaStream_t s) {
    cudaGetLastError();  // a stale non-sticky status must not be blamed on this launch
    if (write_ref) measure_kernel<true><<<grid, kMeasureThreads, 0, s>>>(p);
    else measure_kernel<false><<<grid, kMeasureThreads, 0, s>>>(p);
    return cudaGetLastError();
}

cudaError_t measure_occupancy(int* blocks_per_sm) {
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks_per_sm, measure_kernel<false>,
                                                         kMeasureThreads, 0);
}

}  // namespace lc
