// lc_measure.cu -- Eq. 1 (§3.2) on sm_103a: per segment sum|W - R| and
// sum|R|, combined per layer with the element count.
//
// Work decomposition: every segment is covered by 16-byte "virtual vectors"
// aligned to absolute addresses (lc_internal.cuh).  All vectors of all
// segments, layers ascending, form one linear work space that is cut into
// contiguous ranges: G equal ones, one per CTA, with G = resident CTAs on
// the device (one wave), and for the bulk kernel a pool of small ones after
// them.  A CTA streams its range(s) (the thread kernel: 128-bit
// non-allocating loads of W and R, several in flight per thread) and writes
// one fp64 partial per (range, segment) run.  The last CTA to finish (atomic
// ticket, no spinning) adds the partials of each segment, then the segments
// of each layer, in a fixed order, so the result is deterministic for a
// layout.
//
// Precision: per-thread fp32 accumulators take at most kUnroll * kFlush
// terms each before they are added (fixed tree) into per-thread fp64 sums;
// the relative error of a layer sum is below about 2e-6 (all terms >= 0).
#include "lc_bulk.cuh"
#include "lc_reduce.cuh"

namespace lc {
namespace {

#ifndef LC_MEASURE_UNROLL
#define LC_MEASURE_UNROLL 4
#endif
#ifndef LC_MEASURE_FLUSH
#define LC_MEASURE_FLUSH 4
#endif
constexpr int kUnroll = LC_MEASURE_UNROLL;   // vectors of W (and of R) in flight per thread
constexpr int kFlush = LC_MEASURE_FLUSH;     // unrolled iterations between fp64 flushes
static_assert(kUnroll * kFlush <= 32, "fp32 partial sums are bounded to 32 terms");

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
// Bulk-load measure.  The CTA walks its own range of the work space and
// then units of a pool of small ranges, each taken from a counter
// (next_pool_range), so that CTAs streaming faster take more of the work.
// Each range is the same walk over segment runs as above, turned into a
// sequence of jobs by one producer thread (warp 0): for the full co-aligned
// vectors of a run, chunks of up to
// kMChunk bytes of W and the same bytes of R loaded by cp.async.bulk into a
// ring of kMStages buffers (one "full" mbarrier per buffer, completed by the
// loads' byte count); for partial edge vectors and runs whose W and R are
// not co-aligned, a job the consumers read from global memory element by
// element; after each run a flush.  Warps 1..7 consume every job in order:
// each thread adds its 16-byte vectors of the chunk into fp32 lanes (at most
// ceil(chunk vectors / 224) terms before they go to fp64), and at a flush
// each warp reduces its threads' fp64 sums in a fixed order into the run
// box; the last warp to arrive adds the warps' sums in warp order and
// writes the run's partial slot (run_box_put), so no warp waits for another
// and no barrier spans warps.  Each warp hands a buffer back on its "empty"
// mbarrier (7 arrivals).  Every wait is
// bounded; a wait that runs out raises the fault word.  Warp-wide decisions
// (the wait's outcome) are taken by lane 0 and broadcast, so the lanes of a
// warp never part ways.
// ---------------------------------------------------------------------------
#ifndef LC_MEASURE_BULK_STAGES
#define LC_MEASURE_BULK_STAGES 2
#endif
#ifndef LC_MEASURE_BULK_CHUNK
#define LC_MEASURE_BULK_CHUNK 24576
#endif
constexpr int kMStages = LC_MEASURE_BULK_STAGES;
constexpr uint32_t kMChunk = LC_MEASURE_BULK_CHUNK;      // bytes of W (and of R) per buffer
constexpr int kMConsumerWarps = kMeasureThreads / 32 - 1;   // warps 1.. consume (2.. in accumulate mode)
constexpr int kMConsumers = 32 * kMConsumerWarps;
constexpr size_t kMeasureBulkSmem = size_t(kMStages) * 2 * kMChunk;
static_assert(kMChunk % 16 == 0 && kMStages >= 2, "measure ring shape");

enum : int32_t { kJobChunk = 0, kJobScalar = 1, kJobFlush = 2, kJobEnd = 3 };

struct MJob {
    int64_t k0, k1;     // vectors [k0, k1) of the segment (chunk or scalar job)
    int32_t kind;
    int32_t seg;
    int32_t slot;       // first partial slot of the run (flush)
    int32_t esz_log2;   // element size of the segment (chunk)
};

struct MRing {
    uint64_t full[kMStages];
    uint64_t empty[kMStages];
    MJob jobs[kMStages];
    RunBox<kMStages, kMConsumerWarps> box;
};

__device__ void measure_produce(const MeasureParams& p, uint8_t* ring, MRing& r) {
    const uint32_t ring_s = smem_addr(ring);
    const uint32_t full_s = smem_addr(r.full), empty_s = smem_addr(r.empty);
    uint64_t k = 0;
    bool stall = p.stall_first != 0;
    auto post = [&](const MJob& j, const SegDev& sd) -> bool {
        const int st = int(k % kMStages);
        if (k >= uint64_t(kMStages) &&
            !mbar_wait_bounded(empty_s + 8 * st, uint32_t((k / kMStages - 1) & 1), kWaitNs))
            return false;
        r.jobs[st] = j;
        if (j.kind == kJobChunk) {
            const uint32_t bytes = uint32_t(j.k1 - j.k0) * 16u;
            const uint8_t* wb = sd.w - (int64_t(sd.lead) << sd.esz_log2) + 16 * j.k0;
            const uint8_t* rb = sd.r - (int64_t(sd.lead) << sd.esz_log2) + 16 * j.k0;
            mbar_expect_tx(full_s + 8 * st, 2 * bytes + (stall ? 16u : 0u));
            stall = false;
            bulk_g2s(ring_s + uint32_t(st) * 2 * kMChunk, wb, bytes, full_s + 8 * st);
            bulk_g2s(ring_s + uint32_t(st) * 2 * kMChunk + kMChunk, rb, bytes, full_s + 8 * st);
        } else {
            mbar_arrive(full_s + 8 * st);
        }
        ++k;
        return true;
    };
    bool ok = true;
    SegDev sd{};
    // the CTA's own range, then units of the pool until it is empty
    for (int rng = int(blockIdx.x); ok && rng >= 0; rng = ok ? next_pool_range(p) : -1) {
        int64_t v0 = p.cta_vec_begin[rng];
        const int64_t v1 = p.cta_vec_begin[rng + 1];
        int s = p.cta_seg0[rng];
        int slot = p.cta_slot0[rng];
        while (ok && v0 < v1 && s < p.nseg) {
            sd = p.segs[s];
            const int64_t seg_end = sd.vec_begin + sd.nvec;
            const int64_t lo = v0 - sd.vec_begin;
            const int64_t hi = (v1 < seg_end ? v1 : seg_end) - sd.vec_begin;
            const int ve = 16 >> sd.esz_log2;
            const bool head_partial = sd.lead > 0;
            const bool tail_partial = ((int64_t(sd.lead) + sd.numel) % ve) != 0;
            if (sd.coaligned) {
                if (head_partial && lo <= 0 && 0 < hi) ok = post({0, 1, kJobScalar, s, slot, 0}, sd);
                const int64_t kf0 = head_partial ? 1 : 0;
                const int64_t kf1 = tail_partial ? sd.nvec - 1 : sd.nvec;
                const int64_t a = lo > kf0 ? lo : kf0;
                const int64_t e = hi < kf1 ? hi : kf1;
                constexpr int64_t kCV = kMChunk / 16;
                for (int64_t x = a; ok && x < e; x += kCV)
                    ok = post({x, (x + kCV < e ? x + kCV : e), kJobChunk, s, slot, sd.esz_log2}, sd);
                const int64_t last = sd.nvec - 1;
                if (ok && tail_partial && last >= lo && last < hi && !(head_partial && last == 0))
                    ok = post({last, last + 1, kJobScalar, s, slot, 0}, sd);
            } else {
                ok = post({lo, hi, kJobScalar, s, slot, 0}, sd);
            }
            if (ok) ok = post({0, 0, kJobFlush, s, slot, 0}, sd);
            slot += kMeasureBulkSlotsPerRun;
            ++s;
            v0 = sd.vec_begin + hi;
        }
    }
    if (ok) ok = post({0, 0, kJobEnd, 0, 0, 0}, sd);
    if (!ok) {
        raise_fault(p.fault);
        // the loads of the last kMStages jobs may still be landing in shared memory
        const uint64_t first = k > uint64_t(kMStages) ? k - kMStages : 0;
        for (uint64_t c = first; c < k; ++c)
            mbar_wait_bounded(full_s + 8 * int(c % kMStages), uint32_t((c / kMStages) & 1), kDrainNs);
    }
}

// Consumers: warps 1.. (warps 2.. in accumulate mode, where warp 1 writes R).
template <bool WRITE_R>
__device__ void measure_consume(const MeasureParams& p, const uint8_t* ring, MRing& r) {
    constexpr int kFirstWarp = WRITE_R ? 2 : 1;
    constexpr int kThreads = 32 * (kMeasureThreads / 32 - kFirstWarp);
    const uint32_t full_s = smem_addr(r.full), empty_s = smem_addr(r.empty);
    const int tid = int(threadIdx.x) - 32 * kFirstWarp;
    const int warp = tid >> 5, lane = tid & 31;
    double dd = 0.0, da = 0.0;
    for (uint64_t k = 0;; ++k) {
        const int st = int(k % kMStages);
        const uint32_t parity = uint32_t((k / kMStages) & 1);
        int ok = 1;
        if (lane == 0) ok = mbar_wait_bounded(full_s + 8 * st, parity, kWaitNs) ? 1 : 0;
        ok = __shfl_sync(0xffffffffu, ok, 0);
        if (!ok) {
            if (lane == 0) raise_fault(p.fault);
            break;
        }
        mbar_try_wait(full_s + 8 * st, parity);   // completed: orders this lane's reads after the loads
        const MJob j = r.jobs[st];
        if (j.kind == kJobEnd) break;
        if (j.kind == kJobChunk) {
            const uint4* W = reinterpret_cast<const uint4*>(ring + size_t(st) * 2 * kMChunk);
            const uint4* R = W + kMChunk / 16;
            const int n = int(j.k1 - j.k0);
            float ad[8], aa[8];
#pragma unroll
            for (int q = 0; q < 8; ++q) { ad[q] = 0.f; aa[q] = 0.f; }
            if (j.esz_log2 == 1) {
#pragma unroll 4
                for (int v = tid; v < n; v += kThreads) accumulate<1>(W[v], R[v], ad, aa);
            } else {
#pragma unroll 4
                for (int v = tid; v < n; v += kThreads) accumulate<2>(W[v], R[v], ad, aa);
            }
            dd += double(tree8(ad));
            da += double(tree8(aa));
        } else if (j.kind == kJobScalar) {
            const SegDev sd = p.segs[j.seg];
            for (int64_t v = j.k0 + tid; v < j.k1; v += kThreads) scalar_vector<WRITE_R>(sd, v, dd, da);
        } else {   // flush: this warp's share of the run, in a fixed order
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) {
                dd += __shfl_down_sync(0xffffffffu, dd, off);
                da += __shfl_down_sync(0xffffffffu, da, off);
            }
            if (lane == 0)
                run_box_put<kMConsumerWarps - (WRITE_R ? 1 : 0)>(r.box, st, warp, dd, da, p.partials + j.slot);
            dd = 0.0;
            da = 0.0;
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(empty_s + 8 * st);
    }
}

// Accumulate mode (R <- W after the measure, Eq. 1 against W(t-1)): one
// thread stores every staged W chunk to R with a bulk store once the chunk
// (and with it the old R) has landed, and hands the buffer back when the
// store has read it.
__device__ void measure_store_r(const MeasureParams& p, const uint8_t* ring, MRing& r) {
    const uint32_t full_s = smem_addr(r.full), empty_s = smem_addr(r.empty);
    const uint32_t ring_s = smem_addr(ring);
    for (uint64_t k = 0;; ++k) {
        const int st = int(k % kMStages);
        if (!mbar_wait_bounded(full_s + 8 * st, uint32_t((k / kMStages) & 1), kWaitNs)) {
            raise_fault(p.fault);
            break;
        }
        const MJob j = r.jobs[st];
        if (j.kind == kJobEnd) break;
        if (j.kind == kJobChunk) {
            const SegDev sd = p.segs[j.seg];
            uint8_t* rb = sd.r - (int64_t(sd.lead) << sd.esz_log2) + 16 * j.k0;
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(rb),
                         "r"(ring_s + uint32_t(st) * 2 * kMChunk), "r"(uint32_t(j.k1 - j.k0) * 16u)
                         : "memory");
            asm volatile("cp.async.bulk.commit_group;" ::: "memory");
            asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
        }
        mbar_arrive(empty_s + 8 * st);
    }
    asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
}

template <bool WRITE_R>
__global__ void __launch_bounds__(kMeasureThreads, 1) measure_bulk_kernel(const MeasureParams p) {
    extern __shared__ __align__(128) uint8_t ring[];
    __shared__ __align__(8) MRing r;
    __shared__ unsigned int s_ticket;
    if (threadIdx.x == 0) {
        for (int st = 0; st < kMStages; ++st) {
            mbar_init(smem_addr(&r.full[st]), 1);
            mbar_init(smem_addr(&r.empty[st]), kMConsumerWarps);
            r.box.count[st] = 0u;
        }
        mbar_init_fence();
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        measure_produce(p, ring, r);
    } else if (WRITE_R && threadIdx.x < 64) {
        if (threadIdx.x == 32) measure_store_r(p, ring, r);
    } else if (threadIdx.x >= 32) {
        measure_consume<WRITE_R>(p, ring, r);
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        s_ticket = atomicAdd(p.ticket, 1u);
    }
    __syncthreads();
    if (s_ticket != gridDim.x - 1) return;
    __threadfence();
    // the ring's loads have all landed (or the CTA gave up): it stages the combine
    finalize(p, reinterpret_cast<double2*>(ring), int32_t(kMeasureBulkSmem / sizeof(double2)));
}

}  // namespace

cudaError_t launch_measure(const MeasureParams& p, int grid, bool write_ref, cudaStream_t s) {
    cudaGetLastError();  // a stale non-sticky status must not be blamed on this launch
    if (write_ref) measure_kernel<true><<<grid, kMeasureThreads, 0, s>>>(p);
    else measure_kernel<false><<<grid, kMeasureThreads, 0, s>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_measure_bulk(const MeasureParams& p, int grid, bool write_ref, cudaStream_t s) {
    cudaGetLastError();
    if (write_ref) measure_bulk_kernel<true><<<grid, kMeasureThreads, kMeasureBulkSmem, s>>>(p);
    else measure_bulk_kernel<false><<<grid, kMeasureThreads, kMeasureBulkSmem, s>>>(p);
    return cudaGetLastError();
}

cudaError_t measure_bulk_prepare(int* blocks_per_sm) {
    cudaError_t e = cudaFuncSetAttribute(measure_bulk_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         int(kMeasureBulkSmem));
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(measure_bulk_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 int(kMeasureBulkSmem));
    if (e != cudaSuccess) return e;
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks_per_sm, measure_bulk_kernel<false>,
                                                         kMeasureThreads, kMeasureBulkSmem);
}

cudaError_t measure_occupancy(int* blocks_per_sm) {
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks_per_sm, measure_kernel<false>,
                                                         kMeasureThreads, 0);
}

}  // namespace lc
