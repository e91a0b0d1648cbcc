// lc_internal.cuh -- device-side tables and kernel launchers shared by the
// translation units of liblayercheck.so (not part of the public ABI).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace lc {

constexpr int kMeasureThreads = 256;   // threads per measure CTA
constexpr int kCopyThreads = 256;      // threads per copy CTA
constexpr int kSelectThreads = 512;    // the select kernel is a single CTA

// Work-range boundaries of the CTAs are rounded to these granules so that
// every warp's 512-byte access starts on a 32-byte sector: a store that
// covers only part of a sector makes L2 fetch the rest from DRAM first.
#ifndef LC_MEASURE_ALIGN_VECS
#define LC_MEASURE_ALIGN_VECS 32       // 16-byte vectors (512 bytes)
#endif
#ifndef LC_COPY_ALIGN_BYTES
#define LC_COPY_ALIGN_BYTES 512
#endif

// One registered segment in measure order (layers ascending, registration
// order within a layer).  The segment is covered by "virtual vectors":
// 16-byte windows aligned to absolute 16-byte addresses of w; vector k
// covers elements [k*VE - lead, (k+1)*VE - lead) with VE = 16 / element
// size, so only the first and the last vector can be partial.
struct SegDev {
    const uint8_t* w;
    uint8_t* r;
    int64_t numel;
    int64_t vec_begin;   // first vector of the segment in the measure work space
    int64_t nvec;        // number of vectors covering the segment
    int32_t lead;        // elements of vector 0 in front of the segment start
    int32_t esz_log2;    // 1 = bf16, 2 = fp32
    int32_t coaligned;   // w and r have the same address modulo 16
    int32_t layer;
};

struct MeasureParams {
    const SegDev* segs;
    const int64_t* cta_vec_begin;    // [G+1] vector range of every CTA
    const int32_t* cta_seg0;         // [G]   first segment each CTA touches
    const int32_t* cta_slot0;        // [G]   first partial slot of each CTA
    const int32_t* seg_slot_begin;   // [nseg+1] slots of segment s: [begin[s], begin[s+1])
    const int32_t* layer_seg_begin;  // [nlayers+1] segments of layer l
    double2* partials;               // [nslots] (sum|W-R|, sum|R|) per (CTA, segment) run
    double* seg_sums;                // [2*nseg]  per-segment (D, A)
    double* sums;                    // [3*nlayers] per-layer (D, A, n)
    unsigned int* ticket;            // CTA completion counter (reset by the last CTA)
    int32_t nseg;
    int32_t nlayers;
    // bulk-load measure only: host-mapped fault word (a bounded wait ran
    // out) and the test of that bound (each CTA's first load announces 16
    // bytes more than it brings)
    uint32_t* fault;
    int32_t stall_first;
    // bulk kernels: after its own range b (of gridDim.x), a CTA takes the
    // ranges gridDim.x + u of a pool of `units` small ones, u from
    // atomicAdd(unit_next, 1), until the pool is empty; 0: no pool
    int32_t units;
    unsigned int* unit_next;         // reset by the last CTA
};

// One copy entry.  The entries of a launch tile a linear "work space"
// without gaps: entry i occupies [woff, woff + span), span a multiple of 16
// and >= nbytes.  Payload bytes [0, nbytes) move from src to dst (and to
// dst2 if set); in GATHER mode bytes [nbytes, span) of the destination
// stream are written as zero.
struct CopyDesc {
    uint64_t woff;
    uint64_t nbytes;
    uint64_t span;
    const uint8_t* src;   // GATHER / COPY: absolute source
    uint8_t* dst;         // SCATTER / COPY: absolute destination
    uint8_t* dst2;        // optional second destination of the payload
};

enum CopyMode : int32_t {
    kGather = 0,    // src absolute  -> dst = stream base + (woff - lo)
    kScatter = 1,   // src = stream base + (woff - lo) -> dst absolute
    kCopy = 2       // src absolute  -> dst absolute
};

struct CopyParams {
    const CopyDesc* desc;
    int32_t ndesc;
    int32_t mode;
    uint64_t lo, hi;     // work range of this launch; lo and hi multiples of 16
    uint8_t* base;       // stream buffer holding work offset lo (GATHER / SCATTER)
    // Device-driven launches (no host round trip): when set, the entry count
    // and the end of the range are read from device memory at kernel start.
    const int32_t* ndesc_dev;
    const uint64_t* hi_dev;
    // Host-mapped word a bulk-engine copy sets to 1 when a bounded wait
    // runs out (never cleared by the device).
    uint32_t* fault;
    // Its copy in device memory, set together with it: every CTA of a bulk
    // copy reads it before its first load and returns at once if it is set,
    // so the later waves of a launch whose first wave gave up end at once.
    uint32_t* fault_dev;
    // Test of that bound: each CTA's first bulk load announces 16 bytes more
    // than it brings, so its wait can only run out.
    int32_t stall_first;
};

// A section of a layer's packed block (one segment's W, exp_avg or exp_avg_sq).
struct SectionDev {
    uint64_t off_in_layer;
    uint64_t nbytes;
    uint64_t span;
    const uint8_t* src;
    uint8_t* ref;         // snapshot of a W section (for the fused commit), else null
    uint64_t commit_off;  // W section: its offset in the layer's commit work space
    int32_t layer;
    int32_t idx;          // position among the layer's sections
};

// Layout of the decision block written by the select kernel and mirrored
// to pinned host memory.
struct ResultHeader {
    int64_t step;
    int32_t n_selected;
    int32_t n_nonfinite;
    uint64_t bytes;            // packed stream bytes
    int32_t n_pack_desc;
    int32_t n_commit_desc;
    uint64_t commit_work;      // work-space bytes of the commit list
    int64_t max_staleness;
    double weighted_staleness;
    uint32_t magic;
    uint32_t status;           // kStatusOk, or kStatusCapacity: nothing persisted
    uint64_t pack_bytes;       // bytes the pack moves: `bytes`, or 0 after kStatusCapacity
};
constexpr uint32_t kResultMagic = 0x4C43534Cu;
constexpr uint32_t kStatusOk = 0;
constexpr uint32_t kStatusCapacity = 1;

struct ResultLayout {
    size_t mask_off, u_off, off_off, total;
};
__host__ __device__ inline ResultLayout result_layout(int nlayers) {
    ResultLayout L;
    size_t h = (sizeof(ResultHeader) + 15) & ~size_t(15);
    L.mask_off = h;
    L.u_off = L.mask_off + ((size_t(nlayers) + 15) & ~size_t(15));
    L.off_off = L.u_off + size_t(nlayers) * 8;
    L.total = L.off_off + size_t(nlayers) * 8;
    return L;
}

struct SelectParams {
    const double* sums;              // [3*nlayers]
    double* delta;                   // [nlayers] accumulators Delta_l
    int64_t* t_last;                 // [nlayers] last persistence steps t_l
    const double* tau_mult;          // [nlayers]
    const int64_t* layer_numel;      // [nlayers]
    const uint64_t* layer_bytes;     // [nlayers] packed block bytes
    const int32_t* layer_sec_begin;  // [nlayers+1] sections of layer l (packed order)
    const int32_t* layer_wsec_count; // [nlayers] W sections of layer l (first in its range)
    const uint64_t* layer_commit_work; // [nlayers] commit work bytes of layer l's W sections
    const SectionDev* secs;
    int64_t* layer_scratch;          // [3*nlayers] per-layer output indices
    uint8_t* result;                 // decision block (device)
    CopyDesc* pack_desc;             // [nsec]
    CopyDesc* commit_desc;           // [nseg]
    double* acc_save;                // [nlayers] the step's accumulated drift (for a rollback)
    int64_t* tl_save;                // [nlayers] t_l before the step
    int64_t* step_counter;           // last step decided on the device
    double tau;
    double eps_w;
    int64_t step;                    // the step, unless step_from_counter
    uint64_t capacity;               // bytes the destination holds (UINT64_MAX: unchecked)
    int32_t step_from_counter;       // 1: step = *step_counter + 1 (captured graphs)
    int32_t max_staleness;
    int32_t nlayers;
    int32_t mode;                    // lc_drift_mode
    int32_t fuse_commit;
};

// Optimizer inputs of one segment in measure order (fused AdamW step).
struct OptSegDev {
    const uint8_t* grad;   // bf16 or fp32 gradient
    uint8_t* model;        // bf16 model copy, or null
    float* m;              // exp_avg
    float* v;              // exp_avg_sq
    int32_t grad_bf16;
    int32_t fast;          // W, m, v, grad and model line up with W's 16-byte vectors
};

// fp32 constants of one AdamW step (formed in binary64, rounded once).
struct AdamConsts {
    float decay;           // 1 - lr*wd
    float b1, omb1;        // beta1, 1 - beta1
    float b2, omb2;        // beta2, 1 - beta2
    float step_size;       // lr / (1 - beta1^t)
    float rbc2;            // 1 / (1 - beta2^t)
    float eps;
};

// Launchers (return the launch error, if any).
cudaError_t launch_measure(const MeasureParams& p, int grid, bool write_ref, cudaStream_t s);
cudaError_t measure_occupancy(int* blocks_per_sm);
// Bulk-load measure: W and R stream through a shared-memory ring
// (cp.async.bulk); its partition gives every (CTA, segment) run
// kMeasureBulkSlotsPerRun partial slots (the CTA's consumer warps combine
// their shares into one).  W and R must be device memory.  write_ref:
// accumulate mode (R <- W as well).
constexpr int kMeasureBulkSlotsPerRun = 1;
cudaError_t launch_measure_bulk(const MeasureParams& p, int grid, bool write_ref, cudaStream_t s);
cudaError_t measure_bulk_prepare(int* blocks_per_sm);
cudaError_t launch_adamw_measure(const MeasureParams& p, const OptSegDev* opt, const AdamConsts& c,
                                 int grid, cudaStream_t s);
// The fused step with its loads on the bulk engine: the bulk-load measure's
// partition (kMeasureBulkSlotsPerRun slots per run); every array device memory.
cudaError_t launch_adamw_bulk(const MeasureParams& p, const OptSegDev* opt, const AdamConsts& c, int grid,
                              cudaStream_t s);
cudaError_t adamw_bulk_prepare(int* blocks_per_sm);
cudaError_t launch_select(const SelectParams& p, cudaStream_t s);
cudaError_t launch_copy(const CopyParams& p, int grid, cudaStream_t s);
cudaError_t copy_occupancy(int* blocks_per_sm);
// Bulk-engine copy (cp.async.bulk through shared memory); every address the
// launch touches must be device memory.  copy_bulk_prepare raises the
// kernel's shared-memory limit and reports its CTAs per SM.
cudaError_t launch_copy_bulk(const CopyParams& p, int grid, cudaStream_t s);
cudaError_t copy_bulk_prepare(int* blocks_per_sm);

// Sets the thread-local message returned by lc_last_error().
void set_last_error(const char* msg);

}  // namespace lc
