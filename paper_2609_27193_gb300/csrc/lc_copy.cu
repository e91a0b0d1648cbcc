// lc_copy.cu -- the byte-moving kernels behind the pack (§3.1 full layer
// state into one contiguous stream), the snapshot commit and the restore
// scatter (§3.5): copy_bulk_kernel (the payload goes through shared memory
// on the bulk-copy engine; the default whenever every address is device
// memory) and copy_kernel (every thread loads and stores 16-byte vectors;
// used for host memory and on request).
//
// A launch covers the work range [lo, hi) of a descriptor list whose
// entries tile a linear work space (lc_internal.cuh).  The range is cut into
// G equal 16-byte-aligned pieces, one per CTA; a CTA finds its first entry
// by binary search and walks the entries it overlaps.  Within an entry the
// payload moves in 16-byte vectors when source and destinations are all
// 16-byte aligned (the usual case: torch allocations, 256-byte packed
// sections), else in the widest unit the three addresses share.  In GATHER
// mode the padding of every section is written as zero.
#include "lc_bulk.cuh"

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

// 16-byte vectors [v0, v1) of an entry, LC_COPY_UNROLL loads in flight per
// thread; thread tid of NT workers.
template <int NT>
__device__ __forceinline__ void copy_vec(const uint8_t* src, uint8_t* dst, uint8_t* dst2,
                                         uint64_t v0, uint64_t v1, int tid) {
    constexpr int U = LC_COPY_UNROLL;
    uint64_t v = v0 + tid;
    for (; v + (U - 1) * NT < v1; v += U * NT) {
        uint4 x[U];
#pragma unroll
        for (int u = 0; u < U; ++u) x[u] = ld_nc(src + 16 * (v + uint64_t(u) * NT));
#pragma unroll
        for (int u = 0; u < U; ++u) st_v4(dst + 16 * (v + uint64_t(u) * NT), x[u]);
        if (dst2) {
#pragma unroll
            for (int u = 0; u < U; ++u) st_v4(dst2 + 16 * (v + uint64_t(u) * NT), x[u]);
        }
    }
    for (; v < v1; v += NT) {
        const uint4 x = ld_nc(src + 16 * v);
        st_v4(dst + 16 * v, x);
        if (dst2) st_v4(dst2 + 16 * v, x);
    }
}

// Units of T (4, 2 or 1 bytes) [u0, u1) of an entry.
template <typename T, int NT>
__device__ __forceinline__ void copy_units(const uint8_t* src, uint8_t* dst, uint8_t* dst2,
                                           uint64_t u0, uint64_t u1, int tid) {
    const T* s = reinterpret_cast<const T*>(src);
    T* d = reinterpret_cast<T*>(dst);
    T* d2 = reinterpret_cast<T*>(dst2);
    for (uint64_t u = u0 + tid; u < u1; u += NT) {
        const T x = s[u];
        d[u] = x;
        if (d2) d2[u] = x;
    }
}

template <int NT>
__device__ __forceinline__ void zero_vec(uint8_t* dst, uint64_t v0, uint64_t v1, int tid) {
    const uint4 z = make_uint4(0u, 0u, 0u, 0u);
    for (uint64_t v = v0 + tid; v < v1; v += NT) st_v4(dst + 16 * v, z);
}

// Resolved addresses of one entry for the launch's mode.
struct EntryAddr {
    const uint8_t* src;
    uint8_t* dst;
    uint8_t* dst2;
    bool vec;   // src, dst and dst2 all 16-byte aligned
};

__device__ __forceinline__ EntryAddr entry_addr(const CopyParams& p, const CopyDesc& d) {
    EntryAddr e;
    e.src = p.mode == kScatter ? p.base + (d.woff - p.lo) : d.src;
    e.dst = p.mode == kGather ? p.base + (d.woff - p.lo) : d.dst;
    e.dst2 = d.dst2;
    e.vec = ((uintptr_t(e.src) | uintptr_t(e.dst) | uintptr_t(e.dst2)) & 15) == 0;
    return e;
}

// Bytes [a, b) of one entry, a and b multiples of 16 within [0, span], by
// thread tid of NT workers.  With kBulkPayload the 16-byte vectors of the
// payload of a vector-aligned entry are left to the bulk engine
// (bulk_next_chunk takes exactly those); everything else -- sub-vector
// tails, entries with misaligned addresses and the GATHER padding -- is
// written here.
template <int NT, bool kBulkPayload>
__device__ void copy_entry(const CopyParams& p, const CopyDesc& d, uint64_t a, uint64_t b, int tid) {
    const EntryAddr e = entry_addr(p, d);
    const uint64_t pe = b < d.nbytes ? b : d.nbytes;   // payload end inside [a, b)
    if (a < pe) {
        const uintptr_t al = uintptr_t(e.src) | uintptr_t(e.dst) | uintptr_t(e.dst2);
        uint64_t done;   // payload bytes [a, done) handled by the unit loop
        if (e.vec) {
            done = pe & ~uint64_t(15);
            if (!kBulkPayload && a < done) copy_vec<NT>(e.src, e.dst, e.dst2, a >> 4, done >> 4, tid);
        } else if ((al & 3) == 0) {
            done = pe & ~uint64_t(3);
            if (a < done) copy_units<uint32_t, NT>(e.src, e.dst, e.dst2, a >> 2, done >> 2, tid);
        } else if ((al & 1) == 0) {
            done = pe & ~uint64_t(1);
            if (a < done) copy_units<uint16_t, NT>(e.src, e.dst, e.dst2, a >> 1, done >> 1, tid);
        } else {
            done = pe;
            copy_units<uint8_t, NT>(e.src, e.dst, e.dst2, a, pe, tid);
        }
        if (tid == 0) {
            for (uint64_t q = done > a ? done : a; q < pe; ++q) {
                e.dst[q] = e.src[q];
                if (e.dst2) e.dst2[q] = e.src[q];
            }
        }
    }
    if (p.mode == kGather && b > d.nbytes) {
        const uint64_t z0 = a > d.nbytes ? a : d.nbytes;
        const uint64_t zv = (z0 + 15) & ~uint64_t(15);
        if (tid == 0)
            for (uint64_t q = z0; q < zv && q < b; ++q) e.dst[q] = 0;
        if (zv < b) zero_vec<NT>(e.dst, zv >> 4, b >> 4, tid);
    }
}

// The CTA's work range [x, xe) (granules of LC_COPY_ALIGN_BYTES, the last
// one ragged) and the last entry with woff <= x.  Returns false when the
// CTA has nothing to do.
__device__ __forceinline__ bool cta_range(CopyParams& p, uint64_t& x, uint64_t& xe, int& first) {
    if (p.ndesc_dev) {           // sizes decided on the device by the select kernel
        p.ndesc = *p.ndesc_dev;
        p.hi = p.lo + *p.hi_dev;
    }
    constexpr uint64_t kGran = LC_COPY_ALIGN_BYTES / 16;
    const uint64_t units = (p.hi - p.lo) >> 4;
    const uint64_t grans = (units + kGran - 1) / kGran;
    const uint64_t u0 = grans * blockIdx.x / gridDim.x * kGran;
    uint64_t u1 = grans * (blockIdx.x + 1) / gridDim.x * kGran;
    if (u1 > units) u1 = units;
    if (u0 >= u1 || p.ndesc <= 0) return false;
    x = p.lo + (u0 << 4);
    xe = p.lo + (u1 << 4);
    int lo_i = 0, hi_i = p.ndesc - 1;
    while (lo_i < hi_i) {
        const int mid = (lo_i + hi_i + 1) >> 1;
        if (p.desc[mid].woff <= x) lo_i = mid;
        else hi_i = mid - 1;
    }
    first = lo_i;
    return true;
}

// Every entry overlapping [x, xe), clipped to it, through copy_entry.
template <int NT, bool kBulkPayload>
__device__ __forceinline__ void walk_entries(const CopyParams& p, int i, uint64_t x, uint64_t xe, int tid) {
    for (; x < xe && i < p.ndesc; ++i) {
        const CopyDesc d = p.desc[i];
        const uint64_t ent_end = d.woff + d.span;
        if (ent_end <= x) continue;
        const uint64_t end = xe < ent_end ? xe : ent_end;
        copy_entry<NT, kBulkPayload>(p, d, x - d.woff, end - d.woff, tid);
        x = end;
    }
}

__global__ void __launch_bounds__(kCopyThreads) copy_kernel(CopyParams p) {
    uint64_t x, xe;
    int first;
    if (!cta_range(p, x, xe, first)) return;
    walk_entries<BS, false>(p, first, x, xe, threadIdx.x);
}

// ---------------------------------------------------------------------------
// Bulk engine.  The 16-byte-aligned payload streams through a ring of
// kStages shared-memory buffers.  One thread (warp 0) is the producer: it
// issues cp.async.bulk loads global -> shared, each completing on the
// buffer's "full" mbarrier.  Another (warp 1) is the consumer: it waits for
// a full buffer and issues cp.async.bulk stores shared -> global (dst and,
// for the fused commit, dst2), one bulk group per buffer; once the group of
// buffer k has finished reading shared memory (wait_group.read, kLag groups
// behind) it arrives on that buffer's "empty" mbarrier, which the producer
// waits for before it refills the buffer.  A job with zero bytes marks the
// end of the CTA's range.  Warps 2.. walk the same range for the rest
// (tails, misaligned entries, padding) with ordinary loads and stores; the
// two sides write disjoint bytes and never synchronise.
// ---------------------------------------------------------------------------
// Ring shape: 2 buffers of 48 KB, one store group in flight (two CTAs per
// SM).  Measured on the 8B pack against 3 x 32 KB with two groups in flight:
// 6.80 vs 6.88 ms; 4 x 24 KB, 6 x 16 KB, 8 x 12 KB and 2 x 56 KB all fell in
// between, 3 x 48 KB (one CTA per SM) at 8.03 ms.
#ifndef LC_BULK_STAGES
#define LC_BULK_STAGES 2
#endif
#ifndef LC_BULK_CHUNK
#define LC_BULK_CHUNK 49152
#endif
#ifndef LC_BULK_LAG
#define LC_BULK_LAG 1
#endif
constexpr int kStages = LC_BULK_STAGES;
constexpr uint32_t kChunk = LC_BULK_CHUNK;
constexpr int kLag = LC_BULK_LAG;         // store groups still reading shared memory
constexpr int kWorkers = BS - 64;
constexpr size_t kBulkSmem = size_t(kStages) * kChunk;
static_assert(kChunk % 16 == 0 && kStages >= 2 && kLag >= 1 && kLag < kStages, "bulk ring shape");

struct BulkJob {
    const uint8_t* src;
    uint8_t* dst;
    uint8_t* dst2;
    uint32_t bytes;
};

// Every byte is read once and written once.  LC_BULK_L2_HINT asks L2 to
// evict the copies' lines first: 0 never, 1 loads and stores, 2 loads only,
// 3 stores only.
#ifndef LC_BULK_L2_HINT
#define LC_BULK_L2_HINT 0
#endif
#define LC_BULK_HINT_LOADS (LC_BULK_L2_HINT == 1 || LC_BULK_L2_HINT == 2)
#define LC_BULK_HINT_STORES (LC_BULK_L2_HINT == 1 || LC_BULK_L2_HINT == 3)

__device__ __forceinline__ uint64_t evict_first_policy() {
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}

__device__ __forceinline__ void bulk_load(uint32_t dst_smem, const void* src, uint32_t bytes, uint32_t bar,
                                          uint32_t announced, uint64_t pol) {
    mbar_expect_tx(bar, announced);
#if LC_BULK_HINT_LOADS
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;"
        ::"r"(dst_smem), "l"(src), "r"(bytes), "r"(bar), "l"(pol)
        : "memory");
#else
    (void)pol;
    bulk_g2s(dst_smem, src, bytes, bar);
#endif
}

__device__ __forceinline__ void bulk_store(void* dst, uint32_t src_smem, uint32_t bytes, uint64_t pol) {
#if LC_BULK_HINT_STORES
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group.L2::cache_hint [%0], [%1], %2, %3;" ::"l"(dst),
                 "r"(src_smem), "r"(bytes), "l"(pol)
                 : "memory");
#else
    (void)pol;
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst), "r"(src_smem),
                 "r"(bytes)
                 : "memory");
#endif
}

// The producer's position: entry i, work position x, and entry i's
// descriptor and addresses kept in registers (read once per entry, not once
// per chunk).
struct ChunkCursor {
    int i;
    uint64_t x;
    int cached;          // entry whose descriptor is in d and e, or -1
    CopyDesc d;
    EntryAddr e;
};

// Next chunk (at most kChunk bytes) of 16-byte-aligned payload at or after
// the cursor, advancing the cursor past it.  Takes exactly the bytes
// copy_entry<..., true> leaves out.
__device__ bool bulk_next_chunk(const CopyParams& p, ChunkCursor& c, uint64_t xe, BulkJob& j) {
    while (c.x < xe && c.i < p.ndesc) {
        if (c.cached != c.i) {
            c.d = p.desc[c.i];
            c.e = entry_addr(p, c.d);
            c.cached = c.i;
        }
        const uint64_t ent_end = c.d.woff + c.d.span;
        if (ent_end <= c.x) {
            ++c.i;
            continue;
        }
        const uint64_t end = xe < ent_end ? xe : ent_end;
        const uint64_t a = c.x - c.d.woff, b = end - c.d.woff;
        const uint64_t pv = (b < c.d.nbytes ? b : c.d.nbytes) & ~uint64_t(15);
        if (c.e.vec && a < pv) {
            const uint64_t n = pv - a < kChunk ? pv - a : kChunk;
            j.src = c.e.src + a;
            j.dst = c.e.dst + a;
            j.dst2 = c.e.dst2 ? c.e.dst2 + a : nullptr;
            j.bytes = uint32_t(n);
            c.x += n;
            return true;
        }
        c.x = end;
        ++c.i;
    }
    return false;
}

struct BulkRing {
    uint64_t full[kStages];
    uint64_t empty[kStages];
    BulkJob jobs[kStages];
};

// A bounded wait ran out: the host-mapped word tells the host, the device
// copy tells the CTAs that start after this one.
__device__ __forceinline__ void raise_copy_fault(const CopyParams& p) {
    raise_fault(p.fault);
    if (p.fault_dev) {
        *reinterpret_cast<volatile uint32_t*>(p.fault_dev) = 1u;
        __threadfence();
    }
}

__device__ void bulk_produce(const CopyParams& p, int i, uint64_t x, uint64_t xe, uint32_t ring_s, BulkRing& r) {
    const uint32_t full_s = smem_addr(r.full), empty_s = smem_addr(r.empty);
    const uint64_t pol = evict_first_policy();
    ChunkCursor c;
    c.i = i;
    c.x = x;
    c.cached = -1;
    BulkJob j;
    bool have = bulk_next_chunk(p, c, xe, j);   // the next job is found before its buffer is free
    uint64_t k = 0;
    bool ok = true;
    for (;; ++k) {
        const int s = int(k % kStages);
        if (k >= uint64_t(kStages) &&
            !mbar_wait_bounded(empty_s + 8 * s, uint32_t((k / kStages - 1) & 1), kWaitNs)) {
            ok = false;
            break;
        }
        if (!have) {
            r.jobs[s].bytes = 0;            // end of the range
            mbar_arrive(full_s + 8 * s);
            break;
        }
        r.jobs[s] = j;
        const uint32_t announced = j.bytes + (p.stall_first && k == 0 ? 16u : 0u);
        bulk_load(ring_s + uint32_t(s) * kChunk, j.src, j.bytes, full_s + 8 * s, announced, pol);
        have = bulk_next_chunk(p, c, xe, j);
    }
    if (!ok) {
        raise_copy_fault(p);
        // the loads of the last kStages chunks may still be landing in shared memory
        const uint64_t first = k > uint64_t(kStages) ? k - kStages : 0;
        for (uint64_t c = first; c < k; ++c)
            mbar_wait_bounded(full_s + 8 * int(c % kStages), uint32_t((c / kStages) & 1), kDrainNs);
    }
}

__device__ void bulk_consume(const CopyParams& p, uint32_t ring_s, BulkRing& r) {
    const uint32_t full_s = smem_addr(r.full), empty_s = smem_addr(r.empty);
    const uint64_t pol = evict_first_policy();
    for (uint64_t k = 0;; ++k) {
        const int s = int(k % kStages);
        if (!mbar_wait_bounded(full_s + 8 * s, uint32_t((k / kStages) & 1), kWaitNs)) {
            raise_copy_fault(p);
            break;
        }
        const BulkJob j = r.jobs[s];
        if (j.bytes == 0) break;
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        bulk_store(j.dst, ring_s + uint32_t(s) * kChunk, j.bytes, pol);
        if (j.dst2) bulk_store(j.dst2, ring_s + uint32_t(s) * kChunk, j.bytes, pol);
        asm volatile("cp.async.bulk.commit_group;" ::: "memory");
        if (k >= uint64_t(kLag)) {
            // groups up to k - kLag have read their buffers: hand that one back
            asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(kLag) : "memory");
            mbar_arrive(empty_s + 8 * int((k - kLag) % kStages));
        }
    }
    asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
}

__global__ void __launch_bounds__(kCopyThreads, 1) copy_bulk_kernel(CopyParams p) {
    extern __shared__ __align__(128) uint8_t ring[];
    __shared__ __align__(8) BulkRing r;
    __shared__ uint32_t s_abort;
    uint64_t x, xe;
    int first;
    if (!cta_range(p, x, xe, first)) return;
    if (threadIdx.x == 0) {
        // an earlier CTA of this context gave up waiting: the copy's bytes
        // are lost anyway, so this CTA does not start a wait of its own
        s_abort = p.fault_dev ? *reinterpret_cast<volatile const uint32_t*>(p.fault_dev) : 0u;
        for (int s = 0; s < kStages; ++s) {
            mbar_init(smem_addr(&r.full[s]), 1);
            mbar_init(smem_addr(&r.empty[s]), 1);
        }
        mbar_init_fence();
    }
    __syncthreads();
    if (s_abort) return;
    if (threadIdx.x < 64) {
        if (threadIdx.x == 0) bulk_produce(p, first, x, xe, smem_addr(ring), r);
        else if (threadIdx.x == 32) bulk_consume(p, smem_addr(ring), r);
        return;
    }
    walk_entries<kWorkers, true>(p, first, x, xe, int(threadIdx.x) - 64);
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

cudaError_t launch_copy_bulk(const CopyParams& p, int grid, cudaStream_t s) {
    cudaGetLastError();
    copy_bulk_kernel<<<grid, kCopyThreads, kBulkSmem, s>>>(p);
    return cudaGetLastError();
}

cudaError_t copy_bulk_prepare(int* blocks_per_sm) {
    cudaError_t e = cudaFuncSetAttribute(copy_bulk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         int(kBulkSmem));
    if (e != cudaSuccess) return e;
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks_per_sm, copy_bulk_kernel, kCopyThreads,
                                                         kBulkSmem);
}

}  // namespace lc
