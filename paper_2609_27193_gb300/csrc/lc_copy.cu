// lc_copy.cu -- the byte-moving kernel behind the pack (§3.1 full layer
// state into one contiguous stream), the snapshot commit and the restore
// scatter (§3.5).
//
// A launch covers the work range [lo, hi) of a descriptor list whose
// entries tile a linear work space (lc_internal.cuh).  The range is cut into
// G equal 16-byte-aligned pieces, one per CTA; a CTA finds its first entry
// by binary search and walks the entries it overlaps.  Within an entry the
// payload moves in 16-byte vectors when source and destinations are all
// 16-byte aligned (the usual case: torch allocations, 256-byte packed
// sections), else in the widest unit the three addresses share.  In GATHER
// mode the padding of every section is written as zero.
#include "lc_internal.cuh"

namespace lc {
namespace {

constexpr int BS = kCopyThreads;

#ifndef LC_LD_PREFETCH
#define LC_LD_PREFETCH 1
#endif

__device__ __forceinline__ uint4 ld_nc(const void* p) {
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

#ifndef LC_ST_CS
#define LC_ST_CS 1
#endif
#ifndef LC_COPY_UNROLL
#define LC_COPY_UNROLL 8
#endif

__device__ __forceinline__ void st_v4(void* p, uint4 v) {
#if LC_ST_CS
    asm volatile("st.global.cs.v4.u32 [%0], {%1,%2,%3,%4};"
                 :
                 : "l"(p), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
                 : "memory");
#else
    asm volatile("st.global.v4.u32 [%0], {%1,%2,%3,%4};"
                 :
                 : "l"(p), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
                 : "memory");
#endif
}

// 16-byte vectors [v0, v1) of an entry, LC_COPY_UNROLL loads in flight per thread.
__device__ __forceinline__ void copy_vec(const uint8_t* src, uint8_t* dst, uint8_t* dst2,
                                         uint64_t v0, uint64_t v1) {
    constexpr int U = LC_COPY_UNROLL;
    uint64_t v = v0 + threadIdx.x;
    for (; v + (U - 1) * BS < v1; v += U * BS) {
        uint4 x[U];
#pragma unroll
        for (int u = 0; u < U; ++u) x[u] = ld_nc(src + 16 * (v + uint64_t(u) * BS));
#pragma unroll
        for (int u = 0; u < U; ++u) st_v4(dst + 16 * (v + uint64_t(u) * BS), x[u]);
        if (dst2) {
#pragma unroll
            for (int u = 0; u < U; ++u) st_v4(dst2 + 16 * (v + uint64_t(u) * BS), x[u]);
        }
    }
    for (; v < v1; v += BS) {
        const uint4 x = ld_nc(src + 16 * v);
        st_v4(dst + 16 * v, x);
        if (dst2) st_v4(dst2 + 16 * v, x);
    }
}

// Units of T (4, 2 or 1 bytes) [u0, u1) of an entry.
template <typename T>
__device__ __forceinline__ void copy_units(const uint8_t* src, uint8_t* dst, uint8_t* dst2,
                                           uint64_t u0, uint64_t u1) {
    const T* s = reinterpret_cast<const T*>(src);
    T* d = reinterpret_cast<T*>(dst);
    T* d2 = reinterpret_cast<T*>(dst2);
    for (uint64_t u = u0 + threadIdx.x; u < u1; u += BS) {
        const T x = s[u];
        d[u] = x;
        if (d2) d2[u] = x;
    }
}

__device__ __forceinline__ void zero_vec(uint8_t* dst, uint64_t v0, uint64_t v1) {
    const uint4 z = make_uint4(0u, 0u, 0u, 0u);
    for (uint64_t v = v0 + threadIdx.x; v < v1; v += BS) st_v4(dst + 16 * v, z);
}

// Bytes [a, b) of one entry, a and b multiples of 16 within [0, span].
__device__ void copy_entry(const CopyParams& p, const CopyDesc& d, uint64_t a, uint64_t b) {
    const uint8_t* src = p.mode == kScatter ? p.base + (d.woff - p.lo) : d.src;
    uint8_t* dst = p.mode == kGather ? p.base + (d.woff - p.lo) : d.dst;
    uint8_t* dst2 = d.dst2;
    const uint64_t pe = b < d.nbytes ? b : d.nbytes;   // payload end inside [a, b)
    if (a < pe) {
        const uintptr_t al = uintptr_t(src) | uintptr_t(dst) | uintptr_t(dst2);
        uint64_t done;   // payload bytes [a, done) handled by the unit loop
        if ((al & 15) == 0) {
            done = pe & ~uint64_t(15);
            if (a < done) copy_vec(src, dst, dst2, a >> 4, done >> 4);
        } else if ((al & 3) == 0) {
            done = pe & ~uint64_t(3);
            if (a < done) copy_units<uint32_t>(src, dst, dst2, a >> 2, done >> 2);
        } else if ((al & 1) == 0) {
            done = pe & ~uint64_t(1);
            if (a < done) copy_units<uint16_t>(src, dst, dst2, a >> 1, done >> 1);
        } else {
            done = pe;
            copy_units<uint8_t>(src, dst, dst2, a, pe);
        }
        if (threadIdx.x == 0) {
            for (uint64_t q = done > a ? done : a; q < pe; ++q) {
                dst[q] = src[q];
                if (dst2) dst2[q] = src[q];
            }
        }
    }
    if (p.mode == kGather && b > d.nbytes) {
        const uint64_t z0 = a > d.nbytes ? a : d.nbytes;
        const uint64_t zv = (z0 + 15) & ~uint64_t(15);
        if (threadIdx.x == 0)
            for (uint64_t q = z0; q < zv && q < b; ++q) dst[q] = 0;
        if (zv < b) zero_vec(dst, zv >> 4, b >> 4);
    }
}

__global__ void __launch_bounds__(kCopyThreads) copy_kernel(CopyParams p) {
    if (p.ndesc_dev) {           // sizes decided on the device by the select kernel
        p.ndesc = *p.ndesc_dev;
        p.hi = p.lo + *p.hi_dev;
    }
    // CTA ranges in granules of LC_COPY_ALIGN_BYTES (the last one ragged)
    constexpr uint64_t kGran = LC_COPY_ALIGN_BYTES / 16;
    const uint64_t units = (p.hi - p.lo) >> 4;
    const uint64_t grans = (units + kGran - 1) / kGran;
    uint64_t u0 = grans * blockIdx.x / gridDim.x * kGran;
    uint64_t u1 = grans * (blockIdx.x + 1) / gridDim.x * kGran;
    if (u1 > units) u1 = units;
    if (u0 >= u1 || p.ndesc <= 0) return;
    uint64_t x = p.lo + (u0 << 4);
    const uint64_t xe = p.lo + (u1 << 4);
    // last entry with woff <= x
    int lo_i = 0, hi_i = p.ndesc - 1;
    while (lo_i < hi_i) {
        const int mid = (lo_i + hi_i + 1) >> 1;
        if (p.desc[mid].woff <= x) lo_i = mid;
        else hi_i = mid - 1;
    }
    for (int i = lo_i; x < xe && i < p.ndesc; ++i) {
        const CopyDesc d = p.desc[i];
        const uint64_t ent_end = d.woff + d.span;
        if (ent_end <= x) continue;
        const uint64_t end = xe < ent_end ? xe : ent_end;
        copy_entry(p, d, x - d.woff, end - d.woff);
        x = end;
    }
}

}  // namespace

cudaError_t launch_copy(const CopyParams& p, int grid, cudaStream_t s) {
    cudaGetLastError();
    copy_kernel<<<grid, kCopyThreads, 0, s>>>(p);
    return cudaGetLastError();
}

cudaError_t copy_occupancy(int* blocks_per_sm) {
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks_per_sm, copy_kernel, kCopyThreads, 0);
}

}  // namespace lc
