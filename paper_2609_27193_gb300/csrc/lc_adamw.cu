// lc_adamw.cu -- one AdamW step fused with the Eq. 1 sums of its update
// (§3.4.2: the drift is computed on the optimizer update path, so W(t-1) is
// read once, by the optimizer).  W is fp32 master weights here, so a
// 16-byte vector holds 4 parameters; the work partition, the partial slots
// and the fixed-order finalize are those of the measure scan.
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

}  // namespace

cudaError_t launch_adamw_measure(const MeasureParams& p, const OptSegDev* opt, const AdamConsts& c,
                                 int grid, cudaStream_t s) {
    cudaGetLastError();
    adamw_measure_kernel<<<grid, kMeasureThreads, 0, s>>>(p, opt, c);
    return cudaGetLastError();
}

}  // namespace lc
