// lc_api.cu -- host side of liblayercheck.so: the C ABI of layercheck.h.
//
// Owns the per-context tables (measure work partition, packed-layout
// sections), the per-layer state (Delta_l, t_l), the pinned decision block,
// the device staging ring and the pinned-host version stores, and drives
// the kernels of lc_measure.cu, lc_select.cu and lc_copy.cu on the caller's
// stream.  No compute happens here: every step of the path runs on the GPU.
#include "layercheck.h"
#include "lc_host.h"
#include "lc_internal.cuh"

#include <nvtx3/nvToolsExt.h>

#include <algorithm>
#include <chrono>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <exception>
#include <iterator>
#include <map>
#include <mutex>
#include <set>
#include <string>
#include <thread>
#include <vector>

using namespace lc;

// CTAs of a bulk-engine launch, in waves of one CTA per resident slot.  With
// more than one wave each CTA takes a smaller share of the range, and SMs
// that finish early start the next CTAs, which shortens the launch's tail.
#ifndef LC_MEASURE_BULK_WAVES
#define LC_MEASURE_BULK_WAVES 1
#endif
#ifndef LC_COPY_BULK_WAVES
#define LC_COPY_BULK_WAVES 8
#endif
// The bulk measure (and the fused step on its partition): a CTA walks an
// equal share of the first (100 - LC_MEASURE_POOL_PCT)% of the work space,
// then takes small units of the rest, LC_MEASURE_POOL_UNITS per CTA in all,
// from a counter.  CTAs that stream faster take more units, so the launch
// ends when the pool runs dry rather than when its slowest share is done.
#ifndef LC_MEASURE_POOL_PCT
#define LC_MEASURE_POOL_PCT 10
#endif
#ifndef LC_MEASURE_POOL_UNITS
#define LC_MEASURE_POOL_UNITS 8
#endif

// ---------------------------------------------------------------------------
// errors
// ---------------------------------------------------------------------------
namespace {

thread_local std::string g_err;

lc_status fail(lc_status st, const char* fmt, ...) {
    char buf[1024];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    g_err = buf;
    return st;
}

#define LC_CUDA(call)                                                                   \
    do {                                                                                \
        cudaError_t e_ = (call);                                                        \
        if (e_ != cudaSuccess) {                                                        \
            cudaGetLastError();                                                         \
            return fail(e_ == cudaErrorMemoryAllocation ? LC_ERR_OOM : LC_ERR_CUDA,     \
                        "%s failed: %s (%s:%d)", #call, cudaGetErrorString(e_), __FILE__, \
                        __LINE__);                                                      \
        }                                                                               \
    } while (0)

#define LC_TRY(expr)                  \
    do {                              \
        lc_status st_ = (expr);       \
        if (st_ != LC_OK) return st_; \
    } while (0)

// Restores the caller's current device on scope exit.
struct DeviceGuard {
    int prev = -1;
    explicit DeviceGuard(int dev) {
        if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
        if (prev != dev) cudaSetDevice(dev);
    }
    ~DeviceGuard() {
        int cur = -1;
        if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
    }
};

uint64_t round_up(uint64_t x, uint64_t a) { return (x + a - 1) / a * a; }

// An NVTX range over one entry point, so a profiler's timeline shows the
// library's calls (a no-op unless a tool is attached).
struct Range {
    explicit Range(const char* name) { nvtxRangePushA(name); }
    ~Range() { nvtxRangePop(); }
    Range(const Range&) = delete;
    Range& operator=(const Range&) = delete;
};

// Polls an event until it completes or timeout_ms passes.
lc_status wait_event(cudaEvent_t ev, int timeout_ms, const char* what) {
    using clk = std::chrono::steady_clock;
    const auto t0 = clk::now();
    long spins = 0;
    for (;;) {
        const cudaError_t q = cudaEventQuery(ev);
        if (q == cudaSuccess) return LC_OK;
        if (q != cudaErrorNotReady) {
            cudaGetLastError();
            return fail(LC_ERR_CUDA, "%s: %s", what, cudaGetErrorString(q));
        }
        const auto ms = std::chrono::duration_cast<std::chrono::milliseconds>(clk::now() - t0).count();
        if (ms > timeout_ms) return fail(LC_ERR_TIMEOUT, "%s: not complete after %d ms", what, timeout_ms);
        if (++spins > 20000) std::this_thread::sleep_for(std::chrono::microseconds(50));
    }
}

lc_status check_device_ptr(const void* p, int device, const char* what, bool allow_host) {
    cudaPointerAttributes a;
    const cudaError_t e = cudaPointerGetAttributes(&a, p);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return fail(LC_ERR_INVALID_ARG, "%s: not a CUDA-visible pointer (%s)", what, cudaGetErrorString(e));
    }
    if (a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged) {
        if (a.type == cudaMemoryTypeDevice && a.device != device)
            return fail(LC_ERR_INVALID_ARG, "%s: memory of device %d, context is on device %d", what,
                        a.device, device);
        return LC_OK;
    }
    if (allow_host && a.type == cudaMemoryTypeHost) return LC_OK;
    return fail(LC_ERR_INVALID_ARG, "%s: not device memory", what);
}

std::mutex g_store_mu;
std::set<const lc_store*> g_live_stores;

}  // namespace

// ---------------------------------------------------------------------------
// objects
// ---------------------------------------------------------------------------
struct StoreVersion {
    int64_t id;
    int32_t layer;
    int32_t durable;
    int64_t step;
    uint64_t off;      // byte offset in the arena
    uint64_t bytes;
    int32_t slot;      // ring slot (ring mode) or -1
};

struct lc_store {
    int32_t nlayers = 0;
    int32_t per_layer = 0;                 // 0 = log, 1 = newest-only, V >= 2 = ring
    uint64_t capacity = 0;
    uint8_t* arena = nullptr;
    uint64_t top = 0;                      // log mode
    std::vector<uint64_t> layer_bytes;
    std::vector<uint64_t> layer_base;      // ring mode
    std::vector<int64_t> layer_writes;     // ring mode: versions ever written
    std::map<uint64_t, uint64_t> excluded; // ranges kept out of use (lc_store_exclude), disjoint
    // slow regions that lc_store_check_dma left in use to keep room for a
    // full step: a placement uses them only when it does not fit without them
    std::map<uint64_t, uint64_t> avoid;
    // newest-only mode: layers whose blocks have the same size share a class
    // of slots (its layers' slots plus spares); a free slot list per class
    std::vector<int32_t> layer_class;
    std::vector<uint64_t> class_bytes;     // slot size (block size rounded to 4096)
    std::vector<int32_t> class_layers;
    std::vector<int32_t> class_slots;      // slots laid out in the arena
    std::vector<std::vector<uint64_t>> class_free;
    std::vector<StoreVersion> versions;
    int64_t next_id = 0;
    std::vector<cudaEvent_t> inflight;     // copies still writing into the arena
};

namespace {

// Blocks of a newest-only store start on this boundary.
constexpr uint64_t kStoreGrain = 4096;

using RangeMap = std::map<uint64_t, uint64_t>;   // offset -> length, disjoint ranges

// The first offset >= `from` at which `len` bytes touch no range of `excl`.
// Only the last range beginning at or before `from` can contain it; the
// ranges after it are passed over while the block runs into them.
uint64_t place_around(const RangeMap& excl, uint64_t from, uint64_t len) {
    uint64_t at = from;
    auto it = excl.upper_bound(at);
    if (it != excl.begin()) {
        auto prev = std::prev(it);
        if (prev->first + prev->second > at) it = prev;
    }
    for (; it != excl.end(); ++it) {
        if (at + len <= it->first) break;
        at = it->first + it->second;
    }
    return at;
}

// The same for the union of two maps (each disjoint, possibly overlapping
// each other): alternate until neither moves the block.
uint64_t place_around(const RangeMap& a, const RangeMap& b, uint64_t from, uint64_t len) {
    uint64_t at = from;
    for (;;) {
        const uint64_t x = place_around(a, at, len);
        const uint64_t y = place_around(b, x, len);
        if (y == x) return x;
        at = y;
    }
}

// Log mode: the first offset >= `from` at which `len` bytes touch no
// excluded range.
uint64_t log_place(const lc_store* st, uint64_t from, uint64_t len) {
    return place_around(st->excluded, from, len);
}

// Adds [lo, hi) to `r`, merging it with the ranges it touches.
void add_range(RangeMap& r, uint64_t lo, uint64_t hi) {
    for (auto it = r.begin(); it != r.end();) {
        if (it->first <= hi && lo <= it->first + it->second) {
            lo = std::min(lo, it->first);
            hi = std::max(hi, it->first + it->second);
            it = r.erase(it);
        } else {
            ++it;
        }
    }
    r.emplace(lo, hi - lo);
}

// Newest-only mode: size classes in the order their slots are laid out
// (largest first; classes have distinct sizes).
std::vector<size_t> classes_largest_first(const lc_store* st) {
    const size_t nc = st->class_bytes.size();
    std::vector<size_t> order(nc);
    for (size_t c = 0; c < nc; ++c) order[c] = c;
    std::sort(order.begin(), order.end(),
              [&](size_t a, size_t b) { return st->class_bytes[a] > st->class_bytes[b]; });
    return order;
}

// The excluded ranges together with the ranges to avoid.
RangeMap excluded_and_avoided(const lc_store* st) {
    RangeMap m = st->excluded;
    for (const auto& x : st->avoid) add_range(m, x.first, x.first + x.second);
    return m;
}

// Whether the store, empty and with the ranges of `excl` (and of `more`)
// out of use, takes a step that persists every layer: in a log store every
// layer's block in layer order from offset 0; in a newest-only store each
// size class's slots for its layers plus its spare (the first pass of
// layout_slots).
bool full_step_fits(const lc_store* st, const RangeMap& excl, const RangeMap& more = RangeMap()) {
    uint64_t top = 0;
    auto put = [&](uint64_t z) {
        const uint64_t at = place_around(excl, more, top, z);
        if (at + z > st->capacity) return false;
        top = at + z;
        return true;
    };
    if (st->per_layer == 0) {
        for (uint64_t z : st->layer_bytes)
            if (!put(z)) return false;
        return true;
    }
    for (size_t c : classes_largest_first(st))
        for (int32_t k = 0; k <= st->class_layers[c]; ++k)
            if (!put(st->class_bytes[c])) return false;
    return true;
}

// Newest-only mode: lays the slots out in an empty store, skipping excluded
// ranges -- classes largest first, each its layers' slots plus one spare,
// then further spares class by class while they fit.  The slots keep off
// the ranges to avoid too, unless the layers' slots and spares then do not
// fit.
void layout_slots(lc_store* st) {
    const size_t nc = st->class_bytes.size();
    const std::vector<size_t> order = classes_largest_first(st);
    const RangeMap both = excluded_and_avoided(st);
    const RangeMap& keep_off = !st->avoid.empty() && full_step_fits(st, both) ? both : st->excluded;
    st->class_slots.assign(nc, 0);
    st->class_free.assign(nc, {});
    uint64_t top = 0;
    auto place = [&](size_t c) -> bool {
        const uint64_t z = st->class_bytes[c];
        const uint64_t at = place_around(keep_off, top, z);
        if (at + z > st->capacity) return false;
        st->class_free[c].push_back(at);
        st->class_slots[c] += 1;
        top = at + z;
        return true;
    };
    for (size_t c : order)
        for (int32_t k = 0; k <= st->class_layers[c]; ++k)
            if (!place(c)) return;
    for (bool grew = true; grew;) {
        grew = false;
        for (size_t c : order) grew = place(c) || grew;
    }
}

// Newest-only mode: once a layer has a durable version, its older durable
// versions are released (pending ones stay until they are durable).
void store_release_superseded(lc_store* st) {
    std::vector<int64_t> newest(size_t(st->nlayers), -1);
    for (size_t i = 0; i < st->versions.size(); ++i) {
        const StoreVersion& v = st->versions[i];
        if (!v.durable) continue;
        const int64_t cur = newest[size_t(v.layer)];
        if (cur < 0 || v.step > st->versions[size_t(cur)].step ||
            (v.step == st->versions[size_t(cur)].step && v.id > st->versions[size_t(cur)].id))
            newest[size_t(v.layer)] = int64_t(i);
    }
    std::vector<StoreVersion> keep;
    keep.reserve(st->versions.size());
    for (size_t i = 0; i < st->versions.size(); ++i) {
        const StoreVersion& v = st->versions[i];
        if (v.durable && newest[size_t(v.layer)] != int64_t(i))
            st->class_free[size_t(st->layer_class[size_t(v.layer)])].push_back(v.off);
        else
            keep.push_back(v);
    }
    st->versions.swap(keep);
}

}  // namespace

struct PendingPack {
    int64_t step;
    cudaEvent_t done;
    lc_store* store;
    std::vector<int64_t> ids;
};

enum State { kNew = 0, kReady, kMeasured, kSelected, kPacked };

struct lc_ctx {
    int device = 0;
    cudaStream_t stream = nullptr;
    cudaStream_t copy_stream = nullptr;
    lc_config cfg{};
    int sms = 0;
    State state = kNew;
    int64_t last_step = -1;

    int32_t nseg = 0, nlayers = 0;
    std::vector<lc_segment> segs;          // measure order
    std::vector<int32_t> layer_seg_begin;  // [nlayers+1]
    std::vector<int64_t> layer_numel;
    std::vector<uint64_t> layer_bytes;
    std::vector<SectionDev> secs;          // packed order, layer-major
    std::vector<int32_t> layer_sec_begin;  // [nlayers+1]
    std::vector<int32_t> sec_seg;          // segment (measure order) of each section
    std::vector<int32_t> sec_part;         // 0 = W, 1 = exp_avg, 2 = exp_avg_sq
    int measure_grid = 0, copy_grid = 0, nslots = 0;
    int bulk_grid = 0;                     // CTAs of a bulk-engine copy launch
    bool bulk_sources = false;             // every registered array is device memory
    uint32_t* h_fault = nullptr;           // pinned, mapped: a bulk copy gave up waiting
    uint32_t* d_fault = nullptr;           // its device address
    uint32_t* d_fault_dev = nullptr;       // its copy in device memory (read by every copy CTA)
    bool any_write_ref = false;
    std::vector<int32_t> order;            // measure position -> registration index
    bool snap_missing = false;             // some segment has no snapshot
    OptSegDev* d_opt = nullptr;            // optimizer table (lc_register_optimizer)

    // device memory
    void* d_tables = nullptr;
    MeasureParams mp{};
    MeasureParams mpb{};                   // bulk-load measure: its own partition and partials
    int measure_bulk_grid = 0;
    bool bulk_measure = false;             // lc_measure takes the bulk-load kernel
    bool bulk_adam = false;                // lc_adamw_step_measure takes the bulk-load kernel
    SelectParams sp{};
    CopyDesc* d_pack_desc = nullptr;
    CopyDesc* d_commit_desc = nullptr;
    CopyDesc* d_restore_desc = nullptr;
    uint8_t* d_result = nullptr;
    uint8_t* h_result = nullptr;           // pinned
    ResultLayout rl{};
    cudaEvent_t ev_result = nullptr;

    // staging ring
    uint8_t* d_staging = nullptr;
    uint64_t slot_bytes = 0;
    cudaEvent_t ev_slot_free[2] = {nullptr, nullptr};
    cudaEvent_t ev_slot_filled[2] = {nullptr, nullptr};
    bool slot_busy[2] = {false, false};

    // last decision
    bool have_select = false;
    ResultHeader hdr{};
    std::vector<uint8_t> mask;
    std::vector<uint64_t> offsets;
    std::vector<PendingPack> pending;
    lc_counters counters{};

    // device-driven steps: pinned decision blocks of steps still in flight
    struct AsyncSlot {
        uint8_t* host = nullptr;   // pinned copy of the decision block
        cudaEvent_t done = nullptr;
        int64_t step = -1;
        bool busy = false;
    };
    static constexpr int kAsyncSlots = 4;
    AsyncSlot slots[kAsyncSlots + 1];   // the last one belongs to the captured graph
    cudaStream_t capture_stream = nullptr;
    cudaGraphExec_t graph_exec = nullptr;
    lc_counters graph_delta{};             // what one replay of the graph launches

    // copy trace: two timing events per staged chunk (lc_copy_trace_*)
    struct Span {
        int32_t kind;
        int32_t chunk;
        int64_t step;
        uint64_t bytes;
        cudaEvent_t a, b;
    };
    bool trace_on = false;
    std::vector<Span> trace;
    std::vector<cudaEvent_t> trace_pool;   // events of cleared records, for reuse
    int64_t trace_dropped = 0;
};

namespace {

// True for memory of cudaMalloc (not managed, not host): the only kind the
// bulk-copy engine is given.
bool plain_device(const void* p) {
    cudaPointerAttributes a;
    if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return a.type == cudaMemoryTypeDevice;
}

// A bulk copy whose bounded wait ran out leaves the word set for good: the
// bytes of that copy (and so every later checkpoint) are not to be trusted.
lc_status check_copy_fault(const lc_ctx* ctx, const char* what) {
    if (ctx->h_fault && *reinterpret_cast<volatile const uint32_t*>(ctx->h_fault))
        return fail(LC_ERR_TIMEOUT, "%s: a bulk-engine copy gave up waiting for its loads", what);
    return LC_OK;
}

// Engine and grid of a copy launch whose stream-side buffer is `base`
// (nullptr when the launch has none).
bool use_bulk(const lc_ctx* ctx, const void* base) {
    return ctx->cfg.copy_engine == LC_COPY_BULK && ctx->bulk_sources && (!base || plain_device(base));
}

cudaError_t launch_copy_engine(lc_ctx* ctx, CopyParams p, bool bulk, uint64_t units, cudaStream_t s) {
    p.fault = ctx->d_fault;
    p.fault_dev = ctx->d_fault_dev;
    p.stall_first = (ctx->cfg.debug_flags & LC_DEBUG_BULK_STALL) ? 1 : 0;
    const uint64_t cap = uint64_t(bulk ? ctx->bulk_grid : ctx->copy_grid);
    const int grid = int(std::max<uint64_t>(1, std::min<uint64_t>(cap, units)));
    ctx->counters.kernel_launches += 1;
    ctx->counters.copy_launches += 1;
    if (bulk) ctx->counters.bulk_copy_launches += 1;
    return bulk ? launch_copy_bulk(p, grid, s) : launch_copy(p, grid, s);
}

// Copy trace.  A span's start event is recorded on its stream right before
// the span's work and its end event right after, so end - start is the work
// itself and a gap between spans of one stream is time that stream waited.
// Tracing never makes a call fail: a span that cannot be recorded is dropped.
constexpr size_t kMaxTraceSpans = size_t(1) << 16;

cudaEvent_t trace_event(lc_ctx* ctx) {
    if (!ctx->trace_pool.empty()) {
        cudaEvent_t e = ctx->trace_pool.back();
        ctx->trace_pool.pop_back();
        return e;
    }
    cudaEvent_t e = nullptr;
    if (cudaEventCreate(&e) != cudaSuccess) {
        cudaGetLastError();
        return nullptr;
    }
    return e;
}

int64_t trace_begin(lc_ctx* ctx, int32_t kind, int32_t chunk, int64_t step, uint64_t bytes, cudaStream_t s) {
    if (!ctx->trace_on) return -1;
    if (ctx->trace.size() >= kMaxTraceSpans) {
        ctx->trace_dropped += 1;
        return -1;
    }
    cudaEvent_t a = trace_event(ctx), b = a ? trace_event(ctx) : nullptr;
    if (!a || !b || cudaEventRecord(a, s) != cudaSuccess) {
        cudaGetLastError();
        if (a) ctx->trace_pool.push_back(a);
        if (b) ctx->trace_pool.push_back(b);
        ctx->trace_dropped += 1;
        return -1;
    }
    ctx->trace.push_back({kind, chunk, step, bytes, a, b});
    return int64_t(ctx->trace.size()) - 1;
}

void trace_end(lc_ctx* ctx, int64_t idx, cudaStream_t s) {
    if (idx < 0) return;
    // a failed record leaves the span untimed (lc_copy_trace_read reports NaN)
    if (cudaEventRecord(ctx->trace[size_t(idx)].b, s) != cudaSuccess) cudaGetLastError();
}

// The Eq. 1 scan on the context's engine.
lc_status launch_measure_engine(lc_ctx* ctx, cudaStream_t s) {
    if (ctx->bulk_measure) {
        LC_CUDA(launch_measure_bulk(ctx->mpb, ctx->measure_bulk_grid, ctx->cfg.mode == LC_DRIFT_ACCUMULATE, s));
        ctx->counters.bulk_measure_launches += 1;
    } else {
        LC_CUDA(launch_measure(ctx->mp, ctx->measure_grid, ctx->cfg.mode == LC_DRIFT_ACCUMULATE, s));
    }
    ctx->counters.kernel_launches += 1;
    ctx->counters.measure_launches += 1;
    return LC_OK;
}

}  // namespace

// ---------------------------------------------------------------------------
// config, errors, create, destroy
// ---------------------------------------------------------------------------
extern "C" void lc_config_default(lc_config* cfg) {
    if (!cfg) return;
    std::memset(cfg, 0, sizeof *cfg);
    cfg->eps_w = 1e-8;
    cfg->mode = LC_DRIFT_SNAPSHOT;
    cfg->pack_align = 256;
    cfg->fuse_commit = 1;
    cfg->timeout_ms = 60000;
    cfg->staging_bytes = 512ull << 20;
}

extern "C" const char* lc_last_error(void) { return g_err.c_str(); }

// Lets other translation units of the library report an error message.
void lc::set_last_error(const char* msg) { g_err = msg ? msg : ""; }

extern "C" lc_status lc_create(lc_ctx** out, int device, void* cuda_stream, const lc_config* cfg) {
    g_err.clear();
    if (!out) return fail(LC_ERR_INVALID_ARG, "lc_create: out is NULL");
    *out = nullptr;
    lc_config c;
    if (cfg) c = *cfg;
    else lc_config_default(&c);
    if (!(c.eps_w >= 0.0) || !std::isfinite(c.eps_w))
        return fail(LC_ERR_INVALID_ARG, "lc_create: eps_w must be finite and >= 0");
    if (c.mode != LC_DRIFT_SNAPSHOT && c.mode != LC_DRIFT_ACCUMULATE)
        return fail(LC_ERR_INVALID_ARG, "lc_create: unknown drift mode %d", c.mode);
    if (c.pack_align < 16 || (c.pack_align & (c.pack_align - 1)))
        return fail(LC_ERR_INVALID_ARG, "lc_create: pack_align must be a power of two >= 16");
    if (c.timeout_ms <= 0) return fail(LC_ERR_INVALID_ARG, "lc_create: timeout_ms must be > 0");
    if (c.staging_bytes < (2u << 20))
        return fail(LC_ERR_INVALID_ARG, "lc_create: staging_bytes must be >= 2 MiB");
    if (c.copy_engine != LC_COPY_THREADS && c.copy_engine != LC_COPY_BULK)
        return fail(LC_ERR_INVALID_ARG, "lc_create: unknown copy engine %d", c.copy_engine);
    if (c.debug_flags & ~(LC_DEBUG_BULK_STALL | LC_DEBUG_MEASURE_STALL))
        return fail(LC_ERR_INVALID_ARG, "lc_create: unknown debug flags 0x%x", unsigned(c.debug_flags));
    int ndev = 0;
    LC_CUDA(cudaGetDeviceCount(&ndev));
    if (device < 0 || device >= ndev)
        return fail(LC_ERR_INVALID_ARG, "lc_create: device %d out of range (%d devices)", device, ndev);
    cudaDeviceProp prop;
    LC_CUDA(cudaGetDeviceProperties(&prop, device));
    if (prop.major * 10 + prop.minor != 103)
        return fail(LC_ERR_INVALID_ARG,
                    "lc_create: liblayercheck is built for sm_103a only; device %d is sm_%d%d", device,
                    prop.major, prop.minor);
    DeviceGuard g(device);
    lc_ctx* ctx = new lc_ctx();
    ctx->device = device;
    ctx->stream = static_cast<cudaStream_t>(cuda_stream);
    ctx->cfg = c;
    ctx->sms = prop.multiProcessorCount;
    cudaError_t e = cudaStreamCreateWithFlags(&ctx->copy_stream, cudaStreamNonBlocking);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ctx->ev_result, cudaEventDisableTiming);
    for (int i = 0; i < 2 && e == cudaSuccess; ++i) {
        e = cudaEventCreateWithFlags(&ctx->ev_slot_free[i], cudaEventDisableTiming);
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ctx->ev_slot_filled[i], cudaEventDisableTiming);
    }
    if (e == cudaSuccess)
        e = cudaHostAlloc(reinterpret_cast<void**>(&ctx->h_fault), sizeof(uint32_t), cudaHostAllocMapped);
    if (e == cudaSuccess) {
        *ctx->h_fault = 0;
        e = cudaHostGetDevicePointer(reinterpret_cast<void**>(&ctx->d_fault), ctx->h_fault, 0);
    }
    if (e == cudaSuccess) e = cudaMalloc(reinterpret_cast<void**>(&ctx->d_fault_dev), 16);
    if (e == cudaSuccess) e = cudaMemset(ctx->d_fault_dev, 0, 16);
    int bocc = 0;
    if (e == cudaSuccess) e = copy_bulk_prepare(&bocc);
    if (e != cudaSuccess) {
        cudaGetLastError();
        lc_destroy(ctx);
        return fail(LC_ERR_CUDA, "lc_create: %s", cudaGetErrorString(e));
    }
    ctx->bulk_grid = ctx->sms * std::max(1, bocc) * LC_COPY_BULK_WAVES;
    *out = ctx;
    return LC_OK;
}

extern "C" void lc_destroy(lc_ctx* ctx) {
    if (!ctx) return;
    DeviceGuard g(ctx->device);
    if (ctx->stream || ctx->copy_stream) {
        cudaEvent_t ev;
        if (cudaEventCreateWithFlags(&ev, cudaEventDisableTiming) == cudaSuccess) {
            if (cudaEventRecord(ev, ctx->stream) == cudaSuccess) wait_event(ev, ctx->cfg.timeout_ms, "lc_destroy");
            if (ctx->copy_stream && cudaEventRecord(ev, ctx->copy_stream) == cudaSuccess)
                wait_event(ev, ctx->cfg.timeout_ms, "lc_destroy");
            cudaEventDestroy(ev);
        }
    }
    for (auto& pp : ctx->pending) cudaEventDestroy(pp.done);
    for (auto& sl : ctx->slots) {
        if (sl.host) cudaFreeHost(sl.host);
        if (sl.done) cudaEventDestroy(sl.done);
    }
    for (auto& sp : ctx->trace) {
        cudaEventDestroy(sp.a);
        cudaEventDestroy(sp.b);
    }
    for (cudaEvent_t e : ctx->trace_pool) cudaEventDestroy(e);
    if (ctx->graph_exec) cudaGraphExecDestroy(ctx->graph_exec);
    if (ctx->capture_stream) cudaStreamDestroy(ctx->capture_stream);
    cudaFree(ctx->d_tables);
    cudaFree(ctx->d_fault_dev);
    cudaFree(ctx->d_opt);
    cudaFree(ctx->d_staging);
    if (ctx->h_result) cudaFreeHost(ctx->h_result);
    if (ctx->h_fault) cudaFreeHost(ctx->h_fault);
    if (ctx->ev_result) cudaEventDestroy(ctx->ev_result);
    for (int i = 0; i < 2; ++i) {
        if (ctx->ev_slot_free[i]) cudaEventDestroy(ctx->ev_slot_free[i]);
        if (ctx->ev_slot_filled[i]) cudaEventDestroy(ctx->ev_slot_filled[i]);
    }
    if (ctx->copy_stream) cudaStreamDestroy(ctx->copy_stream);
    cudaGetLastError();
    delete ctx;
}

// ---------------------------------------------------------------------------
// layout registration
// ---------------------------------------------------------------------------
namespace {

// Bump allocator over one device allocation holding every table.
struct TablePlan {
    size_t size = 0;
    size_t take(size_t bytes) {
        size_t off = round_up(size, 256);
        size = off + bytes;
        return off;
    }
};

}  // namespace

static lc_status register_layout_impl(lc_ctx* ctx, const lc_segment* segs, int32_t nseg, int32_t nlayers,
                                      const double* tau_mult);

// The tables are host vectors sized by the layout: an allocation failure
// is reported as LC_ERR_OOM rather than thrown across the C ABI.
extern "C" lc_status lc_register_layout(lc_ctx* ctx, const lc_segment* segs, int32_t nseg,
                                        int32_t nlayers, const double* tau_mult) {
    try {
        return register_layout_impl(ctx, segs, nseg, nlayers, tau_mult);
    } catch (const std::exception& e) {
        return fail(LC_ERR_OOM, "lc_register_layout: %s", e.what());
    }
}

static lc_status register_layout_impl(lc_ctx* ctx, const lc_segment* segs, int32_t nseg, int32_t nlayers,
                                      const double* tau_mult) {
    g_err.clear();
    if (!ctx) return fail(LC_ERR_INVALID_ARG, "lc_register_layout: ctx is NULL");
    if (ctx->state != kNew) return fail(LC_ERR_STATE, "lc_register_layout: layout already registered");
    if (!segs || nseg <= 0) return fail(LC_ERR_INVALID_ARG, "lc_register_layout: no segments");
    if (nlayers <= 0) return fail(LC_ERR_INVALID_ARG, "lc_register_layout: nlayers must be > 0");
    DeviceGuard g(ctx->device);

    std::vector<int32_t> per_layer(nlayers, 0);
    for (int32_t i = 0; i < nseg; ++i) {
        const lc_segment& s = segs[i];
        if (s.layer < 0 || s.layer >= nlayers)
            return fail(LC_ERR_INVALID_ARG, "segment %d: layer %d outside [0, %d)", i, s.layer, nlayers);
        if (s.w_dtype != LC_BF16 && s.w_dtype != LC_F32)
            return fail(LC_ERR_INVALID_ARG, "segment %d: unknown dtype %d", i, s.w_dtype);
        if (s.numel <= 0) return fail(LC_ERR_INVALID_ARG, "segment %d: numel must be > 0", i);
        if (!s.w) return fail(LC_ERR_INVALID_ARG, "segment %d: w is required", i);
        if (!s.snap && ctx->cfg.mode != LC_DRIFT_ACCUMULATE)
            return fail(LC_ERR_INVALID_ARG, "segment %d: snap is required in snapshot mode", i);
        if ((s.exp_avg == nullptr) != (s.exp_avg_sq == nullptr))
            return fail(LC_ERR_INVALID_ARG, "segment %d: exp_avg and exp_avg_sq must both be set or both NULL", i);
        const uintptr_t esz = s.w_dtype == LC_BF16 ? 2 : 4;
        if ((uintptr_t(s.w) % esz) || (uintptr_t(s.snap) % esz))
            return fail(LC_ERR_INVALID_ARG, "segment %d: w/snap not aligned to the element size", i);
        if (s.snap && s.snap == s.w)
            return fail(LC_ERR_INVALID_ARG, "segment %d: snap must not alias w", i);
        if (s.exp_avg && ((uintptr_t(s.exp_avg) % 4) || (uintptr_t(s.exp_avg_sq) % 4)))
            return fail(LC_ERR_INVALID_ARG, "segment %d: Adam moments not 4-byte aligned", i);
        char what[64];
        snprintf(what, sizeof what, "segment %d w", i);
        LC_TRY(check_device_ptr(s.w, ctx->device, what, false));
        if (s.snap) {
            snprintf(what, sizeof what, "segment %d snap", i);
            LC_TRY(check_device_ptr(s.snap, ctx->device, what, false));
        }
        if (s.exp_avg) {
            snprintf(what, sizeof what, "segment %d exp_avg", i);
            LC_TRY(check_device_ptr(s.exp_avg, ctx->device, what, false));
            snprintf(what, sizeof what, "segment %d exp_avg_sq", i);
            LC_TRY(check_device_ptr(s.exp_avg_sq, ctx->device, what, false));
        }
        per_layer[s.layer] += 1;
    }
    for (int32_t l = 0; l < nlayers; ++l)
        if (per_layer[l] == 0) return fail(LC_ERR_INVALID_ARG, "layer %d has no segment", l);
    bool all_device = true;
    for (int32_t i = 0; i < nseg && all_device; ++i) {
        const lc_segment& s = segs[i];
        all_device = plain_device(s.w) && (!s.snap || plain_device(s.snap)) &&
                     (!s.exp_avg || (plain_device(s.exp_avg) && plain_device(s.exp_avg_sq)));
    }
    std::vector<double> mult(nlayers, 1.0);
    if (tau_mult) {
        for (int32_t l = 0; l < nlayers; ++l) {
            if (!std::isfinite(tau_mult[l]) || tau_mult[l] < 0.0)
                return fail(LC_ERR_INVALID_ARG, "tau_mult[%d] must be finite and >= 0", l);
            mult[l] = tau_mult[l];
        }
    }

    // measure order: layers ascending, registration order inside a layer
    std::vector<int32_t> order(nseg);
    for (int32_t i = 0; i < nseg; ++i) order[i] = i;
    std::stable_sort(order.begin(), order.end(),
                     [&](int32_t a, int32_t b) { return segs[a].layer < segs[b].layer; });
    ctx->nseg = nseg;
    ctx->bulk_sources = all_device;
    ctx->nlayers = nlayers;
    ctx->segs.resize(nseg);
    for (int32_t i = 0; i < nseg; ++i) ctx->segs[i] = segs[order[i]];
    ctx->order = order;
    ctx->snap_missing = false;
    for (int32_t i = 0; i < nseg; ++i) ctx->snap_missing |= segs[i].snap == nullptr;
    ctx->layer_seg_begin.assign(nlayers + 1, 0);
    for (int32_t i = 0; i < nseg; ++i) ctx->layer_seg_begin[ctx->segs[i].layer + 1] += 1;
    for (int32_t l = 0; l < nlayers; ++l) ctx->layer_seg_begin[l + 1] += ctx->layer_seg_begin[l];

    // measure work space: 16-byte virtual vectors
    std::vector<SegDev> sd(nseg);
    int64_t V = 0;
    for (int32_t i = 0; i < nseg; ++i) {
        const lc_segment& s = ctx->segs[i];
        const int esz_log2 = s.w_dtype == LC_BF16 ? 1 : 2;
        const int ve = 16 >> esz_log2;
        SegDev& d = sd[i];
        d.w = static_cast<const uint8_t*>(s.w);
        d.r = static_cast<uint8_t*>(s.snap);
        d.numel = s.numel;
        d.lead = int32_t((uintptr_t(s.w) & 15) >> esz_log2);
        d.esz_log2 = esz_log2;
        d.coaligned = s.snap && (uintptr_t(s.w) & 15) == (uintptr_t(s.snap) & 15);
        d.layer = s.layer;
        d.nvec = (int64_t(d.lead) + s.numel + ve - 1) / ve;
        d.vec_begin = V;
        V += d.nvec;
    }
    // CTA work ranges of the measure work space: G equal shares in granules
    // of LC_MEASURE_ALIGN_VECS, and `per_run` partial slots for every
    // (CTA, segment) run
    // (with a pool: G static ranges over the first granules, then `units`
    // ranges over the rest; range r's slots are fixed whichever CTA walks it)
    struct Partition {
        int64_t G = 0;
        int64_t units = 0;
        std::vector<int64_t> cta_vec;
        std::vector<int32_t> cta_seg0, cta_slot0, seg_slot_begin;
        int32_t nslots = 0;
    };
    auto partition = [&](int64_t grid, int32_t per_run, int64_t pool_pct = 0, int64_t units_per_cta = 0) {
        Partition pt;
        const int64_t gran = LC_MEASURE_ALIGN_VECS;
        const int64_t ngran = (V + gran - 1) / gran;
        pt.G = std::max<int64_t>(1, std::min<int64_t>(ngran, grid));
        const int64_t G = pt.G;
        // granules in the pool, in units of at least kMinUnit granules (512 KB
        // of W: a unit costs a counter fetch, a table lookup and a flush); a
        // pool too small to give every CTA a unit on average is not used
        constexpr int64_t kMinUnit = 1024;
        int64_t pool = pool_pct > 0 ? ngran * pool_pct / 100 : 0;
        pt.units = pool >= G * kMinUnit ? std::min<int64_t>(G * units_per_cta, pool / kMinUnit) : 0;
        if (pt.units == 0) pool = 0;
        const int64_t U = pt.units, R = G + U, ng_static = ngran - pool;
        pt.cta_vec.resize(R + 1);
        pt.cta_seg0.resize(R);
        pt.cta_slot0.resize(R);
        pt.seg_slot_begin.assign(nseg + 1, -1);
        for (int64_t b = 0; b <= G; ++b) pt.cta_vec[b] = std::min(V, ng_static * b / G * gran);
        for (int64_t u = 1; u <= U; ++u) pt.cta_vec[G + u] = std::min(V, (ng_static + pool * u / U) * gran);
        int32_t slot = 0, s = 0;
        for (int64_t b = 0; b < R; ++b) {
            const int64_t v0 = pt.cta_vec[b], v1 = pt.cta_vec[b + 1];
            while (s < nseg && sd[s].vec_begin + sd[s].nvec <= v0) ++s;
            pt.cta_seg0[b] = s;
            pt.cta_slot0[b] = slot;
            for (int32_t t = s; v0 < v1 && t < nseg && sd[t].vec_begin < v1; ++t) {
                if (pt.seg_slot_begin[t] < 0) pt.seg_slot_begin[t] = slot;
                slot += per_run;
            }
        }
        pt.seg_slot_begin[nseg] = slot;
        for (int32_t t = nseg - 1; t >= 0; --t)
            if (pt.seg_slot_begin[t] < 0) pt.seg_slot_begin[t] = pt.seg_slot_begin[t + 1];
        pt.nslots = slot;
        return pt;
    };
    int occ = 0;
    LC_CUDA(measure_occupancy(&occ));
    const Partition pa = partition(int64_t(ctx->sms) * std::max(1, occ), 1);
    int bocc = 0;
    LC_CUDA(measure_bulk_prepare(&bocc));
    const Partition pb = partition(int64_t(ctx->sms) * std::max(1, bocc) * LC_MEASURE_BULK_WAVES,
                                   kMeasureBulkSlotsPerRun, LC_MEASURE_POOL_PCT, LC_MEASURE_POOL_UNITS);
    const int64_t Rb = pb.G + pb.units;
    const int64_t G = pa.G, Gb = pb.G;
    ctx->measure_grid = int(G);
    ctx->measure_bulk_grid = int(Gb);
    ctx->nslots = pa.nslots;

    // packed layout: per layer all W sections, then exp_avg, then exp_avg_sq
    const uint64_t align = uint64_t(ctx->cfg.pack_align);
    ctx->layer_numel.assign(nlayers, 0);
    ctx->layer_bytes.assign(nlayers, 0);
    ctx->layer_sec_begin.assign(nlayers + 1, 0);
    std::vector<int32_t> wsec(nlayers, 0);
    std::vector<uint64_t> commit_work(nlayers, 0);
    ctx->secs.clear();
    ctx->sec_seg.clear();
    ctx->sec_part.clear();
    for (int32_t l = 0; l < nlayers; ++l) {
        ctx->layer_sec_begin[l] = int32_t(ctx->secs.size());
        uint64_t off = 0;
        for (int part = 0; part < 3; ++part) {
            for (int32_t i = ctx->layer_seg_begin[l]; i < ctx->layer_seg_begin[l + 1]; ++i) {
                const lc_segment& sg = ctx->segs[i];
                if (part == 0) ctx->layer_numel[l] += sg.numel;
                const uint64_t esz = sg.w_dtype == LC_BF16 ? 2 : 4;
                const uint64_t nbytes = part == 0 ? uint64_t(sg.numel) * esz
                                        : (sg.exp_avg ? uint64_t(sg.numel) * 4 : 0);
                if (nbytes == 0) continue;
                SectionDev sec;
                sec.off_in_layer = off;
                sec.nbytes = nbytes;
                sec.span = round_up(nbytes, align);
                sec.src = part == 0 ? static_cast<const uint8_t*>(sg.w)
                          : part == 1 ? reinterpret_cast<const uint8_t*>(sg.exp_avg)
                                      : reinterpret_cast<const uint8_t*>(sg.exp_avg_sq);
                sec.ref = part == 0 ? static_cast<uint8_t*>(sg.snap) : nullptr;
                sec.commit_off = part == 0 ? commit_work[l] : 0;
                sec.layer = l;
                sec.idx = int32_t(ctx->secs.size()) - ctx->layer_sec_begin[l];
                if (part == 0) commit_work[l] += round_up(nbytes, 16);
                ctx->secs.push_back(sec);
                ctx->sec_seg.push_back(i);
                ctx->sec_part.push_back(part);
                if (part == 0) wsec[l] += 1;
                off += sec.span;
            }
        }
        ctx->layer_bytes[l] = off;
    }
    ctx->layer_sec_begin[nlayers] = int32_t(ctx->secs.size());
    const int32_t nsec = int32_t(ctx->secs.size());

    int cocc = 0;
    LC_CUDA(copy_occupancy(&cocc));
    ctx->copy_grid = ctx->sms * std::max(1, cocc);

    // one device allocation for every table and small state array
    TablePlan tp;
    const size_t o_segs = tp.take(sizeof(SegDev) * nseg);
    const size_t o_ctav = tp.take(sizeof(int64_t) * (G + 1));
    const size_t o_ctas = tp.take(sizeof(int32_t) * G);
    const size_t o_ctal = tp.take(sizeof(int32_t) * G);
    const size_t o_segslot = tp.take(sizeof(int32_t) * (nseg + 1));
    const size_t o_lsb = tp.take(sizeof(int32_t) * (nlayers + 1));
    const size_t o_part = tp.take(sizeof(double2) * std::max(1, ctx->nslots));
    const size_t o_segsum = tp.take(sizeof(double) * 2 * nseg);
    const size_t o_sums = tp.take(sizeof(double) * 3 * nlayers);
    const size_t o_ticket = tp.take(sizeof(unsigned int));
    const size_t o_ctav_b = tp.take(sizeof(int64_t) * (Rb + 1));
    const size_t o_ctas_b = tp.take(sizeof(int32_t) * Rb);
    const size_t o_ctal_b = tp.take(sizeof(int32_t) * Rb);
    const size_t o_unit_b = tp.take(sizeof(unsigned int));
    const size_t o_segslot_b = tp.take(sizeof(int32_t) * (nseg + 1));
    const size_t o_part_b = tp.take(sizeof(double2) * std::max(1, pb.nslots));
    const size_t o_ticket_b = tp.take(sizeof(unsigned int));
    const size_t o_delta = tp.take(sizeof(double) * nlayers);
    const size_t o_tlast = tp.take(sizeof(int64_t) * nlayers);
    const size_t o_mult = tp.take(sizeof(double) * nlayers);
    const size_t o_lnumel = tp.take(sizeof(int64_t) * nlayers);
    const size_t o_lbytes = tp.take(sizeof(uint64_t) * nlayers);
    const size_t o_lsec = tp.take(sizeof(int32_t) * (nlayers + 1));
    const size_t o_lwsec = tp.take(sizeof(int32_t) * nlayers);
    const size_t o_lcw = tp.take(sizeof(uint64_t) * nlayers);
    const size_t o_secs = tp.take(sizeof(SectionDev) * std::max(1, nsec));
    const size_t o_scratch = tp.take(sizeof(int64_t) * 3 * nlayers);
    const size_t o_accsave = tp.take(sizeof(double) * nlayers);
    const size_t o_tlsave = tp.take(sizeof(int64_t) * nlayers);
    const size_t o_stepctr = tp.take(sizeof(int64_t));
    ctx->rl = result_layout(nlayers);
    const size_t o_result = tp.take(ctx->rl.total);
    const size_t o_pdesc = tp.take(sizeof(CopyDesc) * std::max(1, nsec));
    const size_t o_cdesc = tp.take(sizeof(CopyDesc) * nseg);
    const size_t o_rdesc = tp.take(sizeof(CopyDesc) * std::max(1, nsec));
    const size_t total = tp.size;

    std::vector<uint8_t> host(total, 0);
    {
        const int64_t before_first_step = -1;
        std::memcpy(host.data() + o_stepctr, &before_first_step, sizeof before_first_step);
    }
    auto put = [&](size_t off, const void* src, size_t n) { if (n) std::memcpy(host.data() + off, src, n); };
    put(o_segs, sd.data(), sizeof(SegDev) * nseg);
    put(o_ctav, pa.cta_vec.data(), sizeof(int64_t) * (G + 1));
    put(o_ctas, pa.cta_seg0.data(), sizeof(int32_t) * G);
    put(o_ctal, pa.cta_slot0.data(), sizeof(int32_t) * G);
    put(o_segslot, pa.seg_slot_begin.data(), sizeof(int32_t) * (nseg + 1));
    put(o_ctav_b, pb.cta_vec.data(), sizeof(int64_t) * (Rb + 1));
    put(o_ctas_b, pb.cta_seg0.data(), sizeof(int32_t) * Rb);
    put(o_ctal_b, pb.cta_slot0.data(), sizeof(int32_t) * Rb);
    put(o_segslot_b, pb.seg_slot_begin.data(), sizeof(int32_t) * (nseg + 1));
    put(o_lsb, ctx->layer_seg_begin.data(), sizeof(int32_t) * (nlayers + 1));
    put(o_mult, mult.data(), sizeof(double) * nlayers);
    put(o_lnumel, ctx->layer_numel.data(), sizeof(int64_t) * nlayers);
    put(o_lbytes, ctx->layer_bytes.data(), sizeof(uint64_t) * nlayers);
    put(o_lsec, ctx->layer_sec_begin.data(), sizeof(int32_t) * (nlayers + 1));
    put(o_lwsec, wsec.data(), sizeof(int32_t) * nlayers);
    put(o_lcw, commit_work.data(), sizeof(uint64_t) * nlayers);
    put(o_secs, ctx->secs.data(), sizeof(SectionDev) * nsec);
    // accumulators, t_l, ticket and partials start at zero (the host image is zeroed)

    void* dev = nullptr;
    LC_CUDA(cudaMalloc(&dev, total));
    ctx->d_tables = dev;
    LC_CUDA(cudaMemcpy(dev, host.data(), total, cudaMemcpyHostToDevice));
    uint8_t* base = static_cast<uint8_t*>(dev);

    MeasureParams& mp = ctx->mp;
    mp.segs = reinterpret_cast<const SegDev*>(base + o_segs);
    mp.cta_vec_begin = reinterpret_cast<const int64_t*>(base + o_ctav);
    mp.cta_seg0 = reinterpret_cast<const int32_t*>(base + o_ctas);
    mp.cta_slot0 = reinterpret_cast<const int32_t*>(base + o_ctal);
    mp.seg_slot_begin = reinterpret_cast<const int32_t*>(base + o_segslot);
    mp.layer_seg_begin = reinterpret_cast<const int32_t*>(base + o_lsb);
    mp.partials = reinterpret_cast<double2*>(base + o_part);
    mp.seg_sums = reinterpret_cast<double*>(base + o_segsum);
    mp.sums = reinterpret_cast<double*>(base + o_sums);
    mp.ticket = reinterpret_cast<unsigned int*>(base + o_ticket);
    mp.nseg = nseg;
    mp.nlayers = nlayers;
    mp.fault = ctx->d_fault;
    mp.stall_first = 0;
    MeasureParams& mpb = ctx->mpb;
    mpb = mp;
    mpb.cta_vec_begin = reinterpret_cast<const int64_t*>(base + o_ctav_b);
    mpb.cta_seg0 = reinterpret_cast<const int32_t*>(base + o_ctas_b);
    mpb.cta_slot0 = reinterpret_cast<const int32_t*>(base + o_ctal_b);
    mpb.seg_slot_begin = reinterpret_cast<const int32_t*>(base + o_segslot_b);
    mpb.partials = reinterpret_cast<double2*>(base + o_part_b);
    mpb.ticket = reinterpret_cast<unsigned int*>(base + o_ticket_b);
    mpb.units = int32_t(pb.units);
    ctx->counters.measure_pool_units = pb.units;
    mpb.unit_next = reinterpret_cast<unsigned int*>(base + o_unit_b);
    mpb.stall_first = (ctx->cfg.debug_flags & LC_DEBUG_MEASURE_STALL) ? 1 : 0;
    ctx->bulk_measure = ctx->cfg.copy_engine == LC_COPY_BULK && all_device && !ctx->snap_missing;

    SelectParams& sp = ctx->sp;
    sp.sums = mp.sums;
    sp.delta = reinterpret_cast<double*>(base + o_delta);
    sp.t_last = reinterpret_cast<int64_t*>(base + o_tlast);
    sp.tau_mult = reinterpret_cast<const double*>(base + o_mult);
    sp.layer_numel = reinterpret_cast<const int64_t*>(base + o_lnumel);
    sp.layer_bytes = reinterpret_cast<const uint64_t*>(base + o_lbytes);
    sp.layer_sec_begin = reinterpret_cast<const int32_t*>(base + o_lsec);
    sp.layer_wsec_count = reinterpret_cast<const int32_t*>(base + o_lwsec);
    sp.layer_commit_work = reinterpret_cast<const uint64_t*>(base + o_lcw);
    sp.secs = reinterpret_cast<const SectionDev*>(base + o_secs);
    sp.layer_scratch = reinterpret_cast<int64_t*>(base + o_scratch);
    sp.acc_save = reinterpret_cast<double*>(base + o_accsave);
    sp.tl_save = reinterpret_cast<int64_t*>(base + o_tlsave);
    sp.step_counter = reinterpret_cast<int64_t*>(base + o_stepctr);
    sp.capacity = UINT64_MAX;
    sp.step_from_counter = 0;
    sp.result = base + o_result;
    sp.pack_desc = reinterpret_cast<CopyDesc*>(base + o_pdesc);
    sp.commit_desc = reinterpret_cast<CopyDesc*>(base + o_cdesc);
    sp.nlayers = nlayers;
    sp.mode = ctx->cfg.mode;
    sp.fuse_commit = ctx->cfg.fuse_commit;
    sp.eps_w = ctx->cfg.eps_w;
    ctx->d_result = sp.result;
    ctx->d_pack_desc = sp.pack_desc;
    ctx->d_commit_desc = sp.commit_desc;
    ctx->d_restore_desc = reinterpret_cast<CopyDesc*>(base + o_rdesc);

    LC_CUDA(cudaHostAlloc(reinterpret_cast<void**>(&ctx->h_result), ctx->rl.total, cudaHostAllocDefault));
    ctx->mask.assign(nlayers, 0);
    ctx->offsets.assign(nlayers, 0);
    ctx->state = kReady;
    ctx->last_step = -1;
    return LC_OK;
}

// ---------------------------------------------------------------------------
// per-step path
// ---------------------------------------------------------------------------
namespace {

bool step_open(const lc_ctx* ctx) {
    if (ctx->state == kMeasured || ctx->state == kPacked) return true;
    if (ctx->state == kSelected) return ctx->hdr.n_selected > 0;
    return false;
}

}  // namespace

extern "C" lc_status lc_measure(lc_ctx* ctx, int64_t step) {
    Range range("lc_measure");
    g_err.clear();
    if (!ctx) return fail(LC_ERR_INVALID_ARG, "lc_measure: ctx is NULL");
    if (ctx->state == kNew) return fail(LC_ERR_STATE, "lc_measure: no layout registered");
    if (step_open(ctx)) return fail(LC_ERR_STATE, "lc_measure: the previous step is still open");
    if (step < 0 || step <= ctx->last_step)
        return fail(LC_ERR_INVALID_ARG, "lc_measure: step %lld must exceed the previous step %lld",
                    (long long)step, (long long)ctx->last_step);
    if (ctx->snap_missing)
        return fail(LC_ERR_STATE, "lc_measure: a segment has no snapshot (use lc_adamw_step_measure)");
    DeviceGuard g(ctx->device);
    LC_TRY(launch_measure_engine(ctx, ctx->stream));
    ctx->last_step = step;
    ctx->state = kMeasured;
    return LC_OK;
}

extern "C" lc_status lc_register_optimizer(lc_ctx* ctx, const lc_optim_segment* osegs, int32_t nseg) {
    g_err.clear();
    if (!ctx || !osegs) return fail(LC_ERR_INVALID_ARG, "lc_register_optimizer: NULL argument");
    if (ctx->state == kNew) return fail(LC_ERR_STATE, "lc_register_optimizer: no layout registered");
    if (ctx->cfg.mode != LC_DRIFT_ACCUMULATE)
        return fail(LC_ERR_STATE, "lc_register_optimizer: the fused step needs LC_DRIFT_ACCUMULATE mode");
    if (nseg != ctx->nseg)
        return fail(LC_ERR_INVALID_ARG, "lc_register_optimizer: %d segments, the layout has %d", nseg, ctx->nseg);
    DeviceGuard g(ctx->device);
    std::vector<OptSegDev> od(ctx->nseg);
    bool opt_device = true;
    for (int32_t pos = 0; pos < ctx->nseg; ++pos) {
        const int32_t i = ctx->order[pos];
        const lc_segment& s = ctx->segs[pos];
        const lc_optim_segment& o = osegs[i];
        if (s.w_dtype != LC_F32)
            return fail(LC_ERR_INVALID_ARG, "segment %d: the fused step updates fp32 weights", i);
        if (!s.exp_avg) return fail(LC_ERR_INVALID_ARG, "segment %d: the fused step needs Adam moments", i);
        if (!o.grad || (o.grad_dtype != LC_BF16 && o.grad_dtype != LC_F32))
            return fail(LC_ERR_INVALID_ARG, "segment %d: gradient pointer or dtype invalid", i);
        const uintptr_t gesz = o.grad_dtype == LC_BF16 ? 2 : 4;
        if (uintptr_t(o.grad) % gesz || uintptr_t(o.model_copy) % 2)
            return fail(LC_ERR_INVALID_ARG, "segment %d: gradient or model copy misaligned", i);
        char what[64];
        snprintf(what, sizeof what, "segment %d grad", i);
        LC_TRY(check_device_ptr(o.grad, ctx->device, what, false));
        if (o.model_copy) {
            snprintf(what, sizeof what, "segment %d model_copy", i);
            LC_TRY(check_device_ptr(o.model_copy, ctx->device, what, false));
        }
        OptSegDev& d = od[pos];
        d.grad = static_cast<const uint8_t*>(o.grad);
        d.model = static_cast<uint8_t*>(o.model_copy);
        d.m = s.exp_avg;
        d.v = s.exp_avg_sq;
        d.grad_bf16 = o.grad_dtype == LC_BF16;
        // vectors of w start at w - 4*lead (16-byte aligned); every other array
        // must line up with them for the vector path
        const uintptr_t w0 = uintptr_t(s.w) & ~uintptr_t(15);
        const uintptr_t lead = (uintptr_t(s.w) & 15) / 4;
        bool fast = (uintptr_t(s.exp_avg) - 4 * lead) % 16 == 0 && (uintptr_t(s.exp_avg_sq) - 4 * lead) % 16 == 0;
        fast = fast && (d.grad_bf16 ? (uintptr_t(o.grad) - 2 * lead) % 8 == 0
                                    : (uintptr_t(o.grad) - 4 * lead) % 16 == 0);
        if (o.model_copy) fast = fast && (uintptr_t(o.model_copy) - 2 * lead) % 8 == 0;
        (void)w0;
        d.fast = fast ? 1 : 0;
        opt_device = opt_device && plain_device(o.grad) && (!o.model_copy || plain_device(o.model_copy));
    }
    // the bulk-load step: weights, moments, gradients and model copies all device memory
    ctx->bulk_adam = ctx->cfg.copy_engine == LC_COPY_BULK && ctx->bulk_sources && opt_device;
    if (ctx->bulk_adam) {
        int occ = 0;
        LC_CUDA(adamw_bulk_prepare(&occ));
    }
    if (!ctx->d_opt) {
        void* p = nullptr;
        LC_CUDA(cudaMalloc(&p, sizeof(OptSegDev) * ctx->nseg));
        ctx->d_opt = static_cast<OptSegDev*>(p);
    }
    LC_CUDA(cudaMemcpy(ctx->d_opt, od.data(), sizeof(OptSegDev) * ctx->nseg, cudaMemcpyHostToDevice));
    return LC_OK;
}

extern "C" lc_status lc_adamw_step_measure(lc_ctx* ctx, int64_t step, const lc_adamw_hparams* hp) {
    Range range("lc_adamw_step_measure");
    g_err.clear();
    if (!ctx || !hp) return fail(LC_ERR_INVALID_ARG, "lc_adamw_step_measure: NULL argument");
    if (!ctx->d_opt) return fail(LC_ERR_STATE, "lc_adamw_step_measure: no optimizer registered");
    if (step_open(ctx)) return fail(LC_ERR_STATE, "lc_adamw_step_measure: the previous step is still open");
    if (step < 1 || step <= ctx->last_step)
        return fail(LC_ERR_INVALID_ARG, "lc_adamw_step_measure: step %lld must be >= 1 and exceed %lld",
                    (long long)step, (long long)ctx->last_step);
    const double vals[5] = {hp->lr, hp->beta1, hp->beta2, hp->eps, hp->weight_decay};
    for (double x : vals)
        if (!std::isfinite(x)) return fail(LC_ERR_INVALID_ARG, "lc_adamw_step_measure: non-finite hyperparameter");
    if (!(hp->beta1 >= 0.0 && hp->beta1 < 1.0 && hp->beta2 >= 0.0 && hp->beta2 < 1.0) || hp->lr < 0.0 ||
        hp->eps < 0.0)
        return fail(LC_ERR_INVALID_ARG, "lc_adamw_step_measure: hyperparameters out of range");
    AdamConsts c;
    c.decay = float(1.0 - hp->lr * hp->weight_decay);
    c.b1 = float(hp->beta1);
    c.omb1 = float(1.0 - hp->beta1);
    c.b2 = float(hp->beta2);
    c.omb2 = float(1.0 - hp->beta2);
    c.step_size = float(hp->lr / (1.0 - std::pow(hp->beta1, double(step))));
    c.rbc2 = float(1.0 / (1.0 - std::pow(hp->beta2, double(step))));
    c.eps = float(hp->eps);
    DeviceGuard g(ctx->device);
    if (ctx->bulk_adam) {
        LC_CUDA(launch_adamw_bulk(ctx->mpb, ctx->d_opt, c, ctx->measure_bulk_grid, ctx->stream));
        ctx->counters.bulk_measure_launches += 1;
    } else {
        LC_CUDA(launch_adamw_measure(ctx->mp, ctx->d_opt, c, ctx->measure_grid, ctx->stream));
    }
    ctx->counters.kernel_launches += 1;
    ctx->counters.measure_launches += 1;
    ctx->last_step = step;
    ctx->state = kMeasured;
    return LC_OK;
}

extern "C" lc_status lc_layer_sums_device(lc_ctx* ctx, double** sums_dev) {
    g_err.clear();
    if (!ctx || !sums_dev) return fail(LC_ERR_INVALID_ARG, "lc_layer_sums_device: NULL argument");
    if (ctx->state == kNew) return fail(LC_ERR_STATE, "lc_layer_sums_device: no layout registered");
    *sums_dev = ctx->mp.sums;
    return LC_OK;
}

extern "C" lc_status lc_set_layer_sums_buffer(lc_ctx* ctx, double* sums_dev) {
    g_err.clear();
    if (!ctx || !sums_dev) return fail(LC_ERR_INVALID_ARG, "lc_set_layer_sums_buffer: NULL argument");
    if (ctx->state == kNew) return fail(LC_ERR_STATE, "lc_set_layer_sums_buffer: no layout registered");
    if (step_open(ctx)) return fail(LC_ERR_STATE, "lc_set_layer_sums_buffer: a step is open");
    if (uintptr_t(sums_dev) & 7) return fail(LC_ERR_INVALID_ARG, "lc_set_layer_sums_buffer: buffer not 8-byte aligned");
    DeviceGuard g(ctx->device);
    LC_TRY(check_device_ptr(sums_dev, ctx->device, "lc_set_layer_sums_buffer", false));
    ctx->mp.sums = sums_dev;
    ctx->mpb.sums = sums_dev;
    ctx->sp.sums = sums_dev;
    return LC_OK;
}

extern "C" lc_status lc_select(lc_ctx* ctx, double tau, int32_t max_staleness, uint8_t* mask_out,
                               double* u_out, uint64_t* bytes_out) {
    Range range("lc_select");
    g_err.clear();
    if (!ctx) return fail(LC_ERR_INVALID_ARG, "lc_select: ctx is NULL");
    if (ctx->state != kMeasured) return fail(LC_ERR_STATE, "lc_select: call lc_measure first");
    if (!std::isfinite(tau)) return fail(LC_ERR_INVALID_ARG, "lc_select: tau must be finite");
    if (max_staleness < 0) return fail(LC_ERR_INVALID_ARG, "lc_select: max_staleness must be >= 0");
    DeviceGuard g(ctx->device);
    SelectParams p = ctx->sp;
    p.tau = tau;
    p.max_staleness = max_staleness;
    p.step = ctx->last_step;
    LC_CUDA(launch_select(p, ctx->stream));
    ctx->counters.kernel_launches += 1;
    ctx->counters.select_launches += 1;
    LC_CUDA(cudaMemcpyAsync(ctx->h_result, ctx->d_result, ctx->rl.total, cudaMemcpyDeviceToHost, ctx->stream));
    ctx->counters.d2h_bytes += ctx->rl.total;
    LC_CUDA(cudaEventRecord(ctx->ev_result, ctx->stream));
    LC_TRY(wait_event(ctx->ev_result, ctx->cfg.timeout_ms, "lc_select"));
    LC_TRY(check_copy_fault(ctx, "lc_select"));

    ResultHeader h;
    std::memcpy(&h, ctx->h_result, sizeof h);
    if (h.magic != kResultMagic || h.step != ctx->last_step || h.status != kStatusOk)
        return fail(LC_ERR_CUDA, "lc_select: decision block is corrupt");
    const uint8_t* m = ctx->h_result + ctx->rl.mask_off;
    const double* u = reinterpret_cast<const double*>(ctx->h_result + ctx->rl.u_off);
    const uint64_t* o = reinterpret_cast<const uint64_t*>(ctx->h_result + ctx->rl.off_off);
    uint64_t check = 0;
    for (int32_t l = 0; l < ctx->nlayers; ++l) {
        ctx->mask[l] = m[l];
        ctx->offsets[l] = o[l];
        if (m[l]) check += ctx->layer_bytes[l];
    }
    if (check != h.bytes) return fail(LC_ERR_CUDA, "lc_select: decision block byte count mismatch");
    if (mask_out) std::memcpy(mask_out, m, size_t(ctx->nlayers));
    if (u_out) std::memcpy(u_out, u, sizeof(double) * size_t(ctx->nlayers));
    if (bytes_out) *bytes_out = h.bytes;
    ctx->hdr = h;
    ctx->have_select = true;
    ctx->state = kSelected;
    return LC_OK;
}

extern "C" lc_status lc_last_select_info(const lc_ctx* ctx, lc_select_info* out) {
    g_err.clear();
    if (!ctx || !out) return fail(LC_ERR_INVALID_ARG, "lc_last_select_info: NULL argument");
    if (!ctx->have_select) return fail(LC_ERR_STATE, "lc_last_select_info: no lc_select yet");
    out->step = ctx->hdr.step;
    out->n_selected = ctx->hdr.n_selected;
    out->n_nonfinite = ctx->hdr.n_nonfinite;
    out->bytes = ctx->hdr.bytes;
    out->max_staleness = ctx->hdr.max_staleness;
    out->weighted_staleness = ctx->hdr.weighted_staleness;
    return LC_OK;
}

extern "C" lc_status lc_last_select_offsets(const lc_ctx* ctx, uint64_t* offsets_out) {
    g_err.clear();
    if (!ctx || !offsets_out) return fail(LC_ERR_INVALID_ARG, "lc_last_select_offsets: NULL argument");
    if (!ctx->have_select) return fail(LC_ERR_STATE, "lc_last_select_offsets: no lc_select yet");
    std::memcpy(offsets_out, ctx->offsets.data(), sizeof(uint64_t) * size_t(ctx->nlayers));
    return LC_OK;
}

namespace {

lc_status launch_copy_range(lc_ctx* ctx, const CopyDesc* desc, int ndesc, int mode, uint64_t lo,
                            uint64_t hi, uint8_t* base, cudaStream_t s) {
    if (hi <= lo || ndesc <= 0) return LC_OK;
    CopyParams p{};
    p.desc = desc;
    p.ndesc = ndesc;
    p.mode = mode;
    p.lo = lo;
    p.hi = hi;
    p.base = base;
    p.ndesc_dev = nullptr;
    p.hi_dev = nullptr;
    LC_CUDA(launch_copy_engine(ctx, p, use_bulk(ctx, base), (hi - lo) >> 4, s));
    return LC_OK;
}

lc_status ensure_staging(lc_ctx* ctx) {
    if (ctx->d_staging) return LC_OK;
    ctx->slot_bytes = (ctx->cfg.staging_bytes / 2) & ~uint64_t(4095);
    void* p = nullptr;
    LC_CUDA(cudaMalloc(&p, ctx->slot_bytes * 2));
    ctx->d_staging = static_cast<uint8_t*>(p);
    return LC_OK;
}

}  // namespace

extern "C" lc_status lc_pack_device(lc_ctx* ctx, void* dst, uint64_t dst_capacity) {
    Range range("lc_pack_device");
    g_err.clear();
    if (!ctx) return fail(LC_ERR_INVALID_ARG, "lc_pack_device: ctx is NULL");
    if (ctx->state != kSelected) return fail(LC_ERR_STATE, "lc_pack_device: call lc_select first");
    const uint64_t bytes = ctx->hdr.bytes;
    if (bytes > 0) {
        if (!dst) return fail(LC_ERR_INVALID_ARG, "lc_pack_device: dst is NULL");
        if (uintptr_t(dst) & 15) return fail(LC_ERR_INVALID_ARG, "lc_pack_device: dst must be 16-byte aligned");
        if (bytes > dst_capacity)
            return fail(LC_ERR_CAPACITY, "lc_pack_device: %llu bytes selected, capacity %llu",
                        (unsigned long long)bytes, (unsigned long long)dst_capacity);
        DeviceGuard g(ctx->device);
        LC_TRY(check_device_ptr(dst, ctx->device, "lc_pack_device dst", true));
        LC_TRY(launch_copy_range(ctx, ctx->d_pack_desc, ctx->hdr.n_pack_desc, kGather, 0, bytes,
                                 static_cast<uint8_t*>(dst), ctx->stream));
    }
    ctx->state = kPacked;
    return LC_OK;
}

extern "C" lc_status lc_pack_async(lc_ctx* ctx, lc_store* st) {
    Range range("lc_pack_async");
    g_err.clear();
    if (!ctx || !st) return fail(LC_ERR_INVALID_ARG, "lc_pack_async: NULL argument");
    if (ctx->state != kSelected) return fail(LC_ERR_STATE, "lc_pack_async: call lc_select first");
    if (st->nlayers != ctx->nlayers || st->layer_bytes != ctx->layer_bytes)
        return fail(LC_ERR_INVALID_ARG, "lc_pack_async: store was created for another layout");
    const uint64_t bytes = ctx->hdr.bytes;
    DeviceGuard g(ctx->device);
    if (bytes == 0) {
        // nothing persisted: the step is durable as soon as earlier copies are
        PendingPack pp;
        pp.step = ctx->hdr.step;
        pp.store = st;
        LC_CUDA(cudaEventCreateWithFlags(&pp.done, cudaEventDisableTiming));
        LC_CUDA(cudaEventRecord(pp.done, ctx->copy_stream));
        ctx->pending.push_back(std::move(pp));
        ctx->state = kPacked;
        return LC_OK;
    }
    // the staging ring first: a failure leaves the store untouched
    LC_TRY(ensure_staging(ctx));
    // reserve the destination of every selected layer block in the store
    struct Extent { uint64_t soff; uint8_t* host; uint64_t len; int32_t layer; };
    std::vector<Extent> ext;
    std::vector<StoreVersion> fresh;
    std::vector<std::vector<int32_t>> wait_before;   // newest-only: layers to see complete first
    if (st->per_layer == 0) {
        // each layer block goes to the next offset that touches no excluded
        // range, and no range to avoid unless the step does not fit that
        // way; blocks that land back to back share one extent
        std::vector<uint64_t> at_of(size_t(ctx->nlayers), 0);
        auto place_step = [&](const RangeMap& keep_off) -> bool {
            uint64_t c = st->top;
            for (int32_t l = 0; l < ctx->nlayers; ++l) {
                if (!ctx->mask[l]) continue;
                const uint64_t lb = ctx->layer_bytes[l];
                const uint64_t at = place_around(keep_off, c, lb);
                if (at + lb > st->capacity) return false;
                at_of[size_t(l)] = at;
                c = at + lb;
            }
            return true;
        };
        if (!(!st->avoid.empty() && place_step(excluded_and_avoided(st))) && !place_step(st->excluded))
            return fail(LC_ERR_CAPACITY, "lc_pack_async: store holds %llu of %llu bytes, %llu more needed",
                        (unsigned long long)st->top, (unsigned long long)st->capacity, (unsigned long long)bytes);
        uint64_t cur = st->top;
        for (int32_t l = 0; l < ctx->nlayers; ++l) {
            if (!ctx->mask[l]) continue;
            const uint64_t lb = ctx->layer_bytes[l];
            const uint64_t at = at_of[size_t(l)];
            uint8_t* host = st->arena + at;
            if (!ext.empty() && ext.back().soff + ext.back().len == ctx->offsets[l] &&
                ext.back().host + ext.back().len == host)
                ext.back().len += lb;
            else
                ext.push_back({ctx->offsets[l], host, lb, l});
            fresh.push_back({0, l, 0, ctx->hdr.step, at, lb, -1});
            cur = at + lb;
        }
        for (StoreVersion& v : fresh) v.id = st->next_id++;
        st->top = cur;
    } else if (st->per_layer == 1) {
        // Newest-only: the placement of the step's blocks is decided here,
        // before anything is enqueued.  Layers ascending take a free slot of
        // their size class.  When the class has none, the earliest layer of
        // the step in that class not yet counted complete is to be waited
        // for: once its copy has landed its previous version's slot is free.
        // With a spare slot per class every step fits; a CAPACITY error
        // (fewer slots, after exclusions) leaves everything untouched.
        for (const StoreVersion& v : st->versions)
            if (!v.durable)
                return fail(LC_ERR_STATE, "lc_pack_async: the newest-only store still holds a pending version "
                                          "of layer %d (call lc_wait_durable)", v.layer);
        std::vector<std::vector<uint64_t>> free = st->class_free;
        std::vector<int64_t> old(size_t(ctx->nlayers), -1);
        for (size_t i = 0; i < st->versions.size(); ++i) old[size_t(st->versions[i].layer)] = int64_t(i);
        const size_t nc = st->class_bytes.size();
        std::vector<std::vector<int32_t>> issued(nc);
        std::vector<size_t> next_done(nc, 0);
        wait_before.assign(size_t(ctx->nlayers), {});
        for (int32_t l = 0; l < ctx->nlayers; ++l) {
            if (!ctx->mask[l]) continue;
            const size_t c = size_t(st->layer_class[size_t(l)]);
            while (free[c].empty()) {
                if (next_done[c] == issued[c].size())
                    return fail(LC_ERR_CAPACITY,
                                "lc_pack_async: no slot for the %llu-byte block of layer %d in the newest-only "
                                "store (%d slots of that size for %d layers)",
                                (unsigned long long)ctx->layer_bytes[l], l, st->class_slots[c],
                                st->class_layers[c]);
                const int32_t x = issued[c][next_done[c]++];
                wait_before[size_t(l)].push_back(x);
                if (old[size_t(x)] >= 0) free[c].push_back(st->versions[size_t(old[size_t(x)])].off);
            }
            const uint64_t off = free[c].back();
            free[c].pop_back();
            issued[c].push_back(l);
            ext.push_back({ctx->offsets[l], st->arena + off, ctx->layer_bytes[l], l});
            fresh.push_back({st->next_id++, l, 0, ctx->hdr.step, off, ctx->layer_bytes[l], -1});
        }
        // the free slots once every waited-for layer's old version is gone;
        // the other old versions free theirs in lc_wait_durable
        st->class_free.swap(free);
    } else {
        for (int32_t l = 0; l < ctx->nlayers; ++l) {
            if (!ctx->mask[l]) continue;
            for (const StoreVersion& v : st->versions)
                if (v.layer == l && !v.durable)
                    return fail(LC_ERR_STATE,
                                "lc_pack_async: layer %d still has a pending version (call lc_wait_durable)", l);
        }
        for (int32_t l = 0; l < ctx->nlayers; ++l) {
            if (!ctx->mask[l]) continue;
            const int32_t slot = int32_t(st->layer_writes[l] % st->per_layer);
            const uint64_t off = st->layer_base[l] + uint64_t(slot) * st->layer_bytes[l];
            st->versions.erase(std::remove_if(st->versions.begin(), st->versions.end(),
                                              [&](const StoreVersion& v) { return v.layer == l && v.slot == slot; }),
                               st->versions.end());
            st->layer_writes[l] += 1;
            ext.push_back({ctx->offsets[l], st->arena + off, ctx->layer_bytes[l], l});
            fresh.push_back({st->next_id++, l, 0, ctx->hdr.step, off, ctx->layer_bytes[l], slot});
        }
    }
    // forget copies into this store that have completed
    st->inflight.erase(std::remove_if(st->inflight.begin(), st->inflight.end(),
                                      [](cudaEvent_t ev) {
                                          if (cudaEventQuery(ev) != cudaSuccess) return false;
                                          cudaEventDestroy(ev);
                                          return true;
                                      }),
                       st->inflight.end());
    // newest-only: an event after the copy that completes each layer's block,
    // waited for (and the layer's version then counted durable) before a
    // block that reuses the room of that layer's previous version is written
    const bool newest = st->per_layer == 1;
    std::vector<cudaEvent_t> layer_done(newest ? size_t(ctx->nlayers) : 0, nullptr);
    std::vector<size_t> fresh_of(newest ? size_t(ctx->nlayers) : 0, 0);
    for (size_t i = 0; i < fresh.size() && newest; ++i) fresh_of[size_t(fresh[i].layer)] = i;
    auto drop_layer_events = [&]() {
        for (cudaEvent_t e : layer_done)
            if (e) cudaEventDestroy(e);
    };
    // a layer's copy has landed: its new version is durable, the old one is
    // gone (its room was already counted free by the placement)
    auto complete_layer = [&](int32_t x) -> lc_status {
        lc_status rc = wait_event(layer_done[size_t(x)], ctx->cfg.timeout_ms, "lc_pack_async");
        if (rc != LC_OK) return rc;
        fresh[fresh_of[size_t(x)]].durable = 1;
        st->versions.erase(std::remove_if(st->versions.begin(), st->versions.end(),
                                          [&](const StoreVersion& v) { return v.layer == x; }),
                           st->versions.end());
        return LC_OK;
    };
    // If an error ends the loop below after copies into the arena were
    // enqueued, the store still learns when they are done, so that it is
    // not freed or cleared under them.
    struct InflightGuard {
        lc_store* st;
        cudaStream_t s;
        bool armed = false;
        ~InflightGuard() {
            if (!armed) return;
            cudaEvent_t ev = nullptr;
            if (cudaEventCreateWithFlags(&ev, cudaEventDisableTiming) == cudaSuccess) {
                if (cudaEventRecord(ev, s) == cudaSuccess) st->inflight.push_back(ev);
                else cudaEventDestroy(ev);
            }
            cudaGetLastError();
        }
    } guard{st, ctx->copy_stream};
    // ring: gather chunk c into slot c%2 on the stream, copy it out on the copy stream
    const uint64_t S = ctx->slot_bytes;
    for (uint64_t lo = 0, c = 0; lo < bytes; lo += S, ++c) {
        const int r = int(c & 1);
        const uint64_t hi = std::min(bytes, lo + S);
        uint8_t* slot = ctx->d_staging + uint64_t(r) * S;
        if (ctx->slot_busy[r]) LC_CUDA(cudaStreamWaitEvent(ctx->stream, ctx->ev_slot_free[r], 0));
        const int64_t tg = trace_begin(ctx, LC_SPAN_GATHER, int32_t(c), ctx->hdr.step, hi - lo, ctx->stream);
        LC_TRY(launch_copy_range(ctx, ctx->d_pack_desc, ctx->hdr.n_pack_desc, kGather, lo, hi, slot, ctx->stream));
        trace_end(ctx, tg, ctx->stream);
        LC_CUDA(cudaEventRecord(ctx->ev_slot_filled[r], ctx->stream));
        LC_CUDA(cudaStreamWaitEvent(ctx->copy_stream, ctx->ev_slot_filled[r], 0));
        const int64_t tc = trace_begin(ctx, LC_SPAN_D2H, int32_t(c), ctx->hdr.step, hi - lo, ctx->copy_stream);
        for (const Extent& e : ext) {
            const uint64_t a = std::max(lo, e.soff), b = std::min(hi, e.soff + e.len);
            if (a >= b) continue;
            if (newest && a == e.soff) {
                for (int32_t x : wait_before[size_t(e.layer)]) {
                    const lc_status rc = complete_layer(x);
                    if (rc != LC_OK) {
                        // keep the versions whose copies are known complete; the
                        // room of the others stays taken
                        for (const StoreVersion& v : fresh)
                            if (v.durable) st->versions.push_back(v);
                        drop_layer_events();
                        return rc;
                    }
                }
            }
            guard.armed = true;
            LC_CUDA(cudaMemcpyAsync(e.host + (a - e.soff), slot + (a - lo), b - a, cudaMemcpyDeviceToHost,
                                    ctx->copy_stream));
            ctx->counters.d2h_bytes += b - a;
            if (newest && b == e.soff + e.len) {
                cudaError_t ee = cudaEventCreateWithFlags(&layer_done[size_t(e.layer)], cudaEventDisableTiming);
                if (ee == cudaSuccess) ee = cudaEventRecord(layer_done[size_t(e.layer)], ctx->copy_stream);
                if (ee != cudaSuccess) {
                    cudaGetLastError();
                    drop_layer_events();
                    return fail(LC_ERR_CUDA, "lc_pack_async: %s", cudaGetErrorString(ee));
                }
            }
        }
        trace_end(ctx, tc, ctx->copy_stream);
        LC_CUDA(cudaEventRecord(ctx->ev_slot_free[r], ctx->copy_stream));
        ctx->slot_busy[r] = true;
    }
    drop_layer_events();
    PendingPack pp;
    pp.step = ctx->hdr.step;
    pp.store = st;
    cudaEvent_t inflight;
    LC_CUDA(cudaEventCreateWithFlags(&inflight, cudaEventDisableTiming));
    if (cudaEventRecord(inflight, ctx->copy_stream) != cudaSuccess) {
        cudaEventDestroy(inflight);
        LC_CUDA(cudaGetLastError());
    }
    st->inflight.push_back(inflight);
    guard.armed = false;   // the store tracks the copies from here on
    LC_CUDA(cudaEventCreateWithFlags(&pp.done, cudaEventDisableTiming));
    if (cudaEventRecord(pp.done, ctx->copy_stream) != cudaSuccess) {
        cudaEventDestroy(pp.done);
        LC_CUDA(cudaGetLastError());
    }
    for (const StoreVersion& v : fresh) {
        st->versions.push_back(v);
        pp.ids.push_back(v.id);
    }
    ctx->pending.push_back(std::move(pp));
    ctx->state = kPacked;
    return LC_OK;
}

extern "C" lc_status lc_commit_snapshot(lc_ctx* ctx) {
    Range range("lc_commit_snapshot");
    g_err.clear();
    if (!ctx) return fail(LC_ERR_INVALID_ARG, "lc_commit_snapshot: ctx is NULL");
    if (ctx->state == kSelected && ctx->hdr.n_selected == 0) {
        ctx->state = kReady;
        return LC_OK;
    }
    if (ctx->state != kPacked)
        return fail(LC_ERR_STATE, "lc_commit_snapshot: the persisted layers were not packed");
    if (ctx->cfg.mode == LC_DRIFT_SNAPSHOT && !ctx->cfg.fuse_commit && ctx->hdr.n_commit_desc > 0) {
        DeviceGuard g(ctx->device);
        LC_TRY(launch_copy_range(ctx, ctx->d_commit_desc, ctx->hdr.n_commit_desc, kCopy, 0,
                                 ctx->hdr.commit_work, nullptr, ctx->stream));
    }
    ctx->state = kReady;
    return LC_OK;
}

extern "C" lc_status lc_wait_durable(lc_ctx* ctx, int64_t step, int32_t timeout_ms) {
    Range range("lc_wait_durable");
    g_err.clear();
    if (!ctx) return fail(LC_ERR_INVALID_ARG, "lc_wait_durable: ctx is NULL");
    const int tmo = timeout_ms > 0 ? timeout_ms : ctx->cfg.timeout_ms;
    DeviceGuard g(ctx->device);
    bool found = false;
    for (size_t i = 0; i < ctx->pending.size();) {
        PendingPack& pp = ctx->pending[i];
        if (pp.step != step) { ++i; continue; }
        found = true;
        LC_TRY(wait_event(pp.done, tmo, "lc_wait_durable"));
        LC_TRY(check_copy_fault(ctx, "lc_wait_durable"));
        {
            std::lock_guard<std::mutex> lk(g_store_mu);
            if (g_live_stores.count(pp.store)) {
                for (StoreVersion& v : pp.store->versions)
                    if (std::find(pp.ids.begin(), pp.ids.end(), v.id) != pp.ids.end()) v.durable = 1;
                if (pp.store->per_layer == 1) store_release_superseded(pp.store);
            }
        }
        cudaEventDestroy(pp.done);
        ctx->pending.erase(ctx->pending.begin() + i);
    }
    if (!found) return fail(LC_ERR_NOT_FOUND, "lc_wait_durable: no pending pack of step %lld", (long long)step);
    return LC_OK;
}

// ---------------------------------------------------------------------------
// device-driven steps (no host round trip) and their captured graph
// ---------------------------------------------------------------------------
namespace {

lc_status ensure_slot_memory(lc_ctx* ctx, lc_ctx::AsyncSlot& sl) {
    if (!sl.host) LC_CUDA(cudaHostAlloc(reinterpret_cast<void**>(&sl.host), ctx->rl.total, cudaHostAllocDefault));
    if (!sl.done) LC_CUDA(cudaEventCreateWithFlags(&sl.done, cudaEventDisableTiming));
    return LC_OK;
}

lc_status check_step_dst(lc_ctx* ctx, void* dst, uint64_t capacity) {
    if (capacity > 0) {
        if (!dst) return fail(LC_ERR_INVALID_ARG, "step: dst is NULL");
        if (uintptr_t(dst) & 15) return fail(LC_ERR_INVALID_ARG, "step: dst must be 16-byte aligned");
        LC_TRY(check_device_ptr(dst, ctx->device, "step dst", true));
    }
    if (ctx->snap_missing) return fail(LC_ERR_STATE, "step: a segment has no snapshot to measure against");
    return LC_OK;
}

// Enqueues measure -> select -> pack -> commit -> decision readback on s.
lc_status enqueue_step(lc_ctx* ctx, cudaStream_t s, int64_t step, bool step_from_counter, double tau,
                       int32_t max_staleness, uint8_t* dst, uint64_t capacity, uint8_t* host_block) {
    LC_TRY(launch_measure_engine(ctx, s));
    SelectParams p = ctx->sp;
    p.tau = tau;
    p.max_staleness = max_staleness;
    p.step = step;
    p.step_from_counter = step_from_counter ? 1 : 0;
    p.capacity = capacity;
    LC_CUDA(launch_select(p, s));
    const ResultHeader* hdr_dev = reinterpret_cast<const ResultHeader*>(ctx->d_result);
    CopyParams c{};
    c.desc = ctx->d_pack_desc;
    c.ndesc = 0;
    c.mode = kGather;
    c.lo = 0;
    c.hi = 0;
    c.base = dst;
    c.ndesc_dev = &hdr_dev->n_pack_desc;
    c.hi_dev = &hdr_dev->pack_bytes;
    // sizes are decided on the device: full grids, idle CTAs return at once
    LC_CUDA(launch_copy_engine(ctx, c, use_bulk(ctx, dst), UINT64_MAX, s));
    if (ctx->cfg.mode == LC_DRIFT_SNAPSHOT && !ctx->cfg.fuse_commit) {
        CopyParams k = c;
        k.desc = ctx->d_commit_desc;
        k.mode = kCopy;
        k.base = nullptr;
        k.ndesc_dev = &hdr_dev->n_commit_desc;
        k.hi_dev = &hdr_dev->commit_work;
        LC_CUDA(launch_copy_engine(ctx, k, use_bulk(ctx, nullptr), UINT64_MAX, s));
    }
    LC_CUDA(cudaMemcpyAsync(host_block, ctx->d_result, ctx->rl.total, cudaMemcpyDeviceToHost, s));
    ctx->counters.kernel_launches += 1;
    ctx->counters.select_launches += 1;
    ctx->counters.d2h_bytes += ctx->rl.total;
    return LC_OK;
}

}  // namespace

extern "C" lc_status lc_step_async(lc_ctx* ctx, int64_t step, double tau, int32_t max_staleness,
                                   void* dst, uint64_t dst_capacity) {
    Range range("lc_step_async");
    g_err.clear();
    if (!ctx) return fail(LC_ERR_INVALID_ARG, "lc_step_async: ctx is NULL");
    if (ctx->state == kNew) return fail(LC_ERR_STATE, "lc_step_async: no layout registered");
    if (step_open(ctx)) return fail(LC_ERR_STATE, "lc_step_async: a step is open");
    if (step < 0 || step <= ctx->last_step)
        return fail(LC_ERR_INVALID_ARG, "lc_step_async: step %lld must exceed the previous step %lld",
                    (long long)step, (long long)ctx->last_step);
    if (!std::isfinite(tau) || max_staleness < 0)
        return fail(LC_ERR_INVALID_ARG, "lc_step_async: tau must be finite and max_staleness >= 0");
    DeviceGuard g(ctx->device);
    LC_TRY(check_step_dst(ctx, dst, dst_capacity));
    int free_slot = -1;
    for (int i = 0; i < lc_ctx::kAsyncSlots; ++i)
        if (!ctx->slots[i].busy) { free_slot = i; break; }
    if (free_slot < 0)
        return fail(LC_ERR_STATE, "lc_step_async: %d steps in flight; call lc_step_wait", lc_ctx::kAsyncSlots);
    lc_ctx::AsyncSlot& sl = ctx->slots[free_slot];
    LC_TRY(ensure_slot_memory(ctx, sl));
    LC_TRY(enqueue_step(ctx, ctx->stream, step, false, tau, max_staleness, static_cast<uint8_t*>(dst),
                        dst_capacity, sl.host));
    LC_CUDA(cudaEventRecord(sl.done, ctx->stream));
    sl.step = step;
    sl.busy = true;
    ctx->last_step = step;
    return LC_OK;
}

extern "C" lc_status lc_step_wait(lc_ctx* ctx, int64_t step, int32_t timeout_ms, uint8_t* mask_out,
                                  double* u_out, uint64_t* bytes_out) {
    Range range("lc_step_wait");
    g_err.clear();
    if (!ctx) return fail(LC_ERR_INVALID_ARG, "lc_step_wait: ctx is NULL");
    lc_ctx::AsyncSlot* sl = nullptr;
    for (auto& s : ctx->slots)
        if (s.busy && s.step == step) { sl = &s; break; }
    if (!sl) return fail(LC_ERR_NOT_FOUND, "lc_step_wait: no step %lld in flight", (long long)step);
    DeviceGuard g(ctx->device);
    LC_TRY(wait_event(sl->done, timeout_ms > 0 ? timeout_ms : ctx->cfg.timeout_ms, "lc_step_wait"));
    sl->busy = false;
    LC_TRY(check_copy_fault(ctx, "lc_step_wait"));
    ResultHeader h;
    std::memcpy(&h, sl->host, sizeof h);
    if (h.magic != kResultMagic || h.step != step)
        return fail(LC_ERR_CUDA, "lc_step_wait: decision block of step %lld is corrupt", (long long)step);
    const uint8_t* m = sl->host + ctx->rl.mask_off;
    const double* u = reinterpret_cast<const double*>(sl->host + ctx->rl.u_off);
    const uint64_t* o = reinterpret_cast<const uint64_t*>(sl->host + ctx->rl.off_off);
    for (int32_t l = 0; l < ctx->nlayers; ++l) {
        ctx->mask[l] = m[l];
        ctx->offsets[l] = o[l];
    }
    if (mask_out) std::memcpy(mask_out, m, size_t(ctx->nlayers));
    if (u_out) std::memcpy(u_out, u, sizeof(double) * size_t(ctx->nlayers));
    if (bytes_out) *bytes_out = h.bytes;
    ctx->hdr = h;
    ctx->have_select = true;
    if (h.status == kStatusCapacity)
        return fail(LC_ERR_CAPACITY,
                    "step %lld: the %llu-byte stream exceeded the destination; nothing was persisted",
                    (long long)step, (unsigned long long)h.bytes);
    return LC_OK;
}

extern "C" lc_status lc_step_graph_create(lc_ctx* ctx, double tau, int32_t max_staleness, void* dst,
                                          uint64_t dst_capacity) {
    Range range("lc_step_graph_create");
    g_err.clear();
    if (!ctx) return fail(LC_ERR_INVALID_ARG, "lc_step_graph_create: ctx is NULL");
    if (ctx->state == kNew) return fail(LC_ERR_STATE, "lc_step_graph_create: no layout registered");
    if (step_open(ctx)) return fail(LC_ERR_STATE, "lc_step_graph_create: a step is open");
    if (!std::isfinite(tau) || max_staleness < 0)
        return fail(LC_ERR_INVALID_ARG, "lc_step_graph_create: tau must be finite and max_staleness >= 0");
    DeviceGuard g(ctx->device);
    LC_TRY(check_step_dst(ctx, dst, dst_capacity));
    lc_ctx::AsyncSlot& sl = ctx->slots[lc_ctx::kAsyncSlots];
    if (sl.busy) return fail(LC_ERR_STATE, "lc_step_graph_create: the graph's last step was not waited for");
    LC_TRY(ensure_slot_memory(ctx, sl));
    if (!ctx->capture_stream) LC_CUDA(cudaStreamCreateWithFlags(&ctx->capture_stream, cudaStreamNonBlocking));
    if (ctx->graph_exec) {
        cudaGraphExecDestroy(ctx->graph_exec);
        ctx->graph_exec = nullptr;
    }
    const lc_counters before = ctx->counters;
    LC_CUDA(cudaStreamBeginCapture(ctx->capture_stream, cudaStreamCaptureModeThreadLocal));
    lc_status rc = enqueue_step(ctx, ctx->capture_stream, 0, true, tau, max_staleness,
                                static_cast<uint8_t*>(dst), dst_capacity, sl.host);
    cudaGraph_t graph = nullptr;
    const cudaError_t e = cudaStreamEndCapture(ctx->capture_stream, &graph);
    const lc_counters after = ctx->counters;
    ctx->counters = before;      // capture runs nothing; launches count when the graph is replayed
    ctx->graph_delta = lc_counters{};
    ctx->graph_delta.kernel_launches = after.kernel_launches - before.kernel_launches;
    ctx->graph_delta.measure_launches = after.measure_launches - before.measure_launches;
    ctx->graph_delta.select_launches = after.select_launches - before.select_launches;
    ctx->graph_delta.copy_launches = after.copy_launches - before.copy_launches;
    ctx->graph_delta.bulk_copy_launches = after.bulk_copy_launches - before.bulk_copy_launches;
    ctx->graph_delta.d2h_bytes = after.d2h_bytes - before.d2h_bytes;
    if (rc != LC_OK) {
        if (graph) cudaGraphDestroy(graph);
        return rc;
    }
    if (e != cudaSuccess) {
        cudaGetLastError();
        return fail(LC_ERR_CUDA, "lc_step_graph_create: capture failed: %s", cudaGetErrorString(e));
    }
    const cudaError_t ei = cudaGraphInstantiate(&ctx->graph_exec, graph, 0);
    cudaGraphDestroy(graph);
    if (ei != cudaSuccess) {
        cudaGetLastError();
        ctx->graph_exec = nullptr;
        return fail(LC_ERR_CUDA, "lc_step_graph_create: instantiate failed: %s", cudaGetErrorString(ei));
    }
    return LC_OK;
}

extern "C" lc_status lc_step_graph_launch(lc_ctx* ctx, int64_t* step_out) {
    Range range("lc_step_graph_launch");
    g_err.clear();
    if (!ctx) return fail(LC_ERR_INVALID_ARG, "lc_step_graph_launch: ctx is NULL");
    if (!ctx->graph_exec) return fail(LC_ERR_STATE, "lc_step_graph_launch: no graph (lc_step_graph_create)");
    if (step_open(ctx)) return fail(LC_ERR_STATE, "lc_step_graph_launch: a step is open");
    lc_ctx::AsyncSlot& sl = ctx->slots[lc_ctx::kAsyncSlots];
    if (sl.busy) return fail(LC_ERR_STATE, "lc_step_graph_launch: wait for step %lld first", (long long)sl.step);
    DeviceGuard g(ctx->device);
    LC_CUDA(cudaGraphLaunch(ctx->graph_exec, ctx->stream));
    LC_CUDA(cudaEventRecord(sl.done, ctx->stream));
    const lc_counters& d = ctx->graph_delta;
    ctx->counters.kernel_launches += d.kernel_launches;
    ctx->counters.measure_launches += d.measure_launches;
    ctx->counters.select_launches += d.select_launches;
    ctx->counters.copy_launches += d.copy_launches;
    ctx->counters.bulk_copy_launches += d.bulk_copy_launches;
    ctx->counters.d2h_bytes += d.d2h_bytes;
    ctx->last_step += 1;
    sl.step = ctx->last_step;
    sl.busy = true;
    if (step_out) *step_out = ctx->last_step;
    return LC_OK;
}

// ---------------------------------------------------------------------------
// restore (§3.5, Eq. 8)
// ---------------------------------------------------------------------------
extern "C" lc_status lc_restore(lc_ctx* ctx, lc_store* st, int64_t t_fail, int64_t* layer_steps_out) {
    Range range("lc_restore");
    g_err.clear();
    if (!ctx || !st) return fail(LC_ERR_INVALID_ARG, "lc_restore: NULL argument");
    if (ctx->state == kNew) return fail(LC_ERR_STATE, "lc_restore: no layout registered");
    if (step_open(ctx)) return fail(LC_ERR_STATE, "lc_restore: a step is open");
    if (st->nlayers != ctx->nlayers || st->layer_bytes != ctx->layer_bytes)
        return fail(LC_ERR_INVALID_ARG, "lc_restore: store was created for another layout");
    const int32_t N = ctx->nlayers;
    std::vector<int64_t> pick(N);
    LC_TRY(lc_store_plan(st, t_fail, pick.data()));
    DeviceGuard g(ctx->device);
    LC_TRY(ensure_staging(ctx));

    // restore stream: the picked blocks, layers ascending
    std::vector<uint64_t> soff(N);
    uint64_t total = 0;
    for (int32_t l = 0; l < N; ++l) {
        soff[l] = total;
        total += ctx->layer_bytes[l];
    }
    const int32_t nsec = int32_t(ctx->secs.size());
    std::vector<CopyDesc> desc(nsec);
    for (int32_t l = 0; l < N; ++l) {
        for (int32_t j = ctx->layer_sec_begin[l]; j < ctx->layer_sec_begin[l + 1]; ++j) {
            const SectionDev& sec = ctx->secs[j];
            const lc_segment& sg = ctx->segs[ctx->sec_seg[j]];
            CopyDesc& d = desc[j];
            d.woff = soff[l] + sec.off_in_layer;
            d.nbytes = sec.nbytes;
            d.span = sec.span;
            d.src = nullptr;
            const int part = ctx->sec_part[j];
            d.dst = part == 0 ? static_cast<uint8_t*>(sg.w)
                    : part == 1 ? reinterpret_cast<uint8_t*>(sg.exp_avg)
                                : reinterpret_cast<uint8_t*>(sg.exp_avg_sq);
            d.dst2 = part == 0 ? static_cast<uint8_t*>(sg.snap) : nullptr;
        }
    }
    LC_CUDA(cudaMemcpyAsync(ctx->d_restore_desc, desc.data(), sizeof(CopyDesc) * nsec,
                            cudaMemcpyHostToDevice, ctx->stream));
    // the descriptor upload must land before the first scatter; the copy
    // stream must not start overwriting staging before earlier users finish
    cudaEvent_t ev_desc;
    LC_CUDA(cudaEventCreateWithFlags(&ev_desc, cudaEventDisableTiming));
    const uint64_t S = ctx->slot_bytes;
    lc_status rc = LC_OK;
    for (uint64_t lo = 0, c = 0; lo < total && rc == LC_OK; lo += S, ++c) {
        const int r = int(c & 1);
        const uint64_t hi = std::min(total, lo + S);
        uint8_t* slot = ctx->d_staging + uint64_t(r) * S;
        cudaError_t e = cudaSuccess;
        if (ctx->slot_busy[r]) e = cudaStreamWaitEvent(ctx->copy_stream, ctx->ev_slot_free[r], 0);
        const int64_t th = trace_begin(ctx, LC_SPAN_H2D, int32_t(c), t_fail, hi - lo, ctx->copy_stream);
        for (int32_t l = 0; l < N && e == cudaSuccess; ++l) {
            const uint64_t a = std::max(lo, soff[l]), b = std::min(hi, soff[l] + ctx->layer_bytes[l]);
            if (a >= b) continue;
            const StoreVersion& v = st->versions[size_t(pick[l])];
            e = cudaMemcpyAsync(slot + (a - lo), st->arena + v.off + (a - soff[l]), b - a,
                                cudaMemcpyHostToDevice, ctx->copy_stream);
            ctx->counters.h2d_bytes += b - a;
        }
        trace_end(ctx, th, ctx->copy_stream);
        if (e == cudaSuccess) e = cudaEventRecord(ctx->ev_slot_filled[r], ctx->copy_stream);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(ctx->stream, ctx->ev_slot_filled[r], 0);
        if (e != cudaSuccess) {
            cudaGetLastError();
            rc = fail(LC_ERR_CUDA, "lc_restore: %s", cudaGetErrorString(e));
            break;
        }
        const int64_t ts = trace_begin(ctx, LC_SPAN_SCATTER, int32_t(c), t_fail, hi - lo, ctx->stream);
        rc = launch_copy_range(ctx, ctx->d_restore_desc, nsec, kScatter, lo, hi, slot, ctx->stream);
        trace_end(ctx, ts, ctx->stream);
        if (rc == LC_OK && cudaEventRecord(ctx->ev_slot_free[r], ctx->stream) != cudaSuccess) {
            cudaGetLastError();
            rc = fail(LC_ERR_CUDA, "lc_restore: event record failed");
        }
        ctx->slot_busy[r] = true;
    }
    // per-layer state of the restored composite: t_l = version step, Delta_l = 0
    std::vector<int64_t> steps(N);
    for (int32_t l = 0; l < N; ++l) steps[l] = st->versions[size_t(pick[l])].step;
    std::vector<double> zeros(N, 0.0);
    if (rc == LC_OK) {
        cudaError_t e = cudaMemcpyAsync(ctx->sp.t_last, steps.data(), sizeof(int64_t) * N,
                                        cudaMemcpyHostToDevice, ctx->stream);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(ctx->sp.delta, zeros.data(), sizeof(double) * N, cudaMemcpyHostToDevice, ctx->stream);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(ctx->sp.step_counter, &t_fail, sizeof t_fail, cudaMemcpyHostToDevice, ctx->stream);
        if (e == cudaSuccess) e = cudaEventRecord(ev_desc, ctx->stream);
        if (e != cudaSuccess) {
            cudaGetLastError();
            rc = fail(LC_ERR_CUDA, "lc_restore: %s", cudaGetErrorString(e));
        } else {
            rc = wait_event(ev_desc, ctx->cfg.timeout_ms, "lc_restore");
        }
    }
    cudaEventDestroy(ev_desc);
    if (rc == LC_OK) rc = check_copy_fault(ctx, "lc_restore");
    if (rc != LC_OK) return rc;
    if (layer_steps_out) std::memcpy(layer_steps_out, steps.data(), sizeof(int64_t) * N);
    ctx->last_step = t_fail;
    ctx->state = kReady;
    return LC_OK;
}

extern "C" lc_status lc_layer_block_bytes(const lc_ctx* ctx, int32_t layer, uint64_t* out) {
    g_err.clear();
    if (!ctx || !out) return fail(LC_ERR_INVALID_ARG, "lc_layer_block_bytes: NULL argument");
    if (ctx->state == kNew) return fail(LC_ERR_STATE, "lc_layer_block_bytes: no layout registered");
    if (layer < 0 || layer >= ctx->nlayers) return fail(LC_ERR_INVALID_ARG, "lc_layer_block_bytes: bad layer");
    *out = ctx->layer_bytes[layer];
    return LC_OK;
}

extern "C" lc_status lc_get_counters(const lc_ctx* ctx, lc_counters* out) {
    g_err.clear();
    if (!ctx || !out) return fail(LC_ERR_INVALID_ARG, "lc_get_counters: NULL argument");
    *out = ctx->counters;
    return LC_OK;
}

// ---------------------------------------------------------------------------
// copy trace
// ---------------------------------------------------------------------------
extern "C" lc_status lc_copy_trace_enable(lc_ctx* ctx, int32_t enable) {
    g_err.clear();
    if (!ctx) return fail(LC_ERR_INVALID_ARG, "lc_copy_trace_enable: ctx is NULL");
    for (auto& sp : ctx->trace) {
        ctx->trace_pool.push_back(sp.a);
        ctx->trace_pool.push_back(sp.b);
    }
    ctx->trace.clear();
    ctx->trace_dropped = 0;
    ctx->trace_on = enable != 0;
    return LC_OK;
}

extern "C" lc_status lc_copy_trace_read(lc_ctx* ctx, lc_copy_span* out, int64_t cap, int64_t* n_out,
                                        int64_t* dropped_out) {
    g_err.clear();
    if (!ctx) return fail(LC_ERR_INVALID_ARG, "lc_copy_trace_read: ctx is NULL");
    if (cap < 0 || (cap > 0 && !out)) return fail(LC_ERR_INVALID_ARG, "lc_copy_trace_read: bad output array");
    if (n_out) *n_out = int64_t(ctx->trace.size());
    if (dropped_out) *dropped_out = ctx->trace_dropped;
    const size_t n = std::min(ctx->trace.size(), size_t(cap));
    if (n == 0) return LC_OK;
    DeviceGuard g(ctx->device);
    for (size_t i = 0; i < n; ++i) {
        LC_TRY(wait_event(ctx->trace[i].a, ctx->cfg.timeout_ms, "lc_copy_trace_read"));
        LC_TRY(wait_event(ctx->trace[i].b, ctx->cfg.timeout_ms, "lc_copy_trace_read"));
    }
    const cudaEvent_t base = ctx->trace[0].a;
    for (size_t i = 0; i < n; ++i) {
        const lc_ctx::Span& sp = ctx->trace[i];
        float a = 0.f, b = 0.f;
        const bool ok = cudaEventElapsedTime(&a, base, sp.a) == cudaSuccess &&
                        cudaEventElapsedTime(&b, base, sp.b) == cudaSuccess;
        if (!ok) cudaGetLastError();
        out[i].kind = sp.kind;
        out[i].chunk = sp.chunk;
        out[i].step = sp.step;
        out[i].bytes = sp.bytes;
        out[i].start_ms = ok ? double(a) : std::nan("");
        out[i].end_ms = ok ? double(b) : std::nan("");
    }
    return LC_OK;
}

// ---------------------------------------------------------------------------
// stores
// ---------------------------------------------------------------------------
extern "C" lc_status lc_store_create(lc_store** out, const lc_ctx* ctx, uint64_t capacity_bytes,
                                     int32_t versions_per_layer) {
    g_err.clear();
    if (!out || !ctx) return fail(LC_ERR_INVALID_ARG, "lc_store_create: NULL argument");
    *out = nullptr;
    if (ctx->state == kNew) return fail(LC_ERR_STATE, "lc_store_create: no layout registered");
    if (versions_per_layer < 0)
        return fail(LC_ERR_INVALID_ARG, "lc_store_create: versions_per_layer must be >= 0");
    lc_store* st = new lc_store();
    st->nlayers = ctx->nlayers;
    st->per_layer = versions_per_layer;
    st->layer_bytes = ctx->layer_bytes;
    if (versions_per_layer == 0) {
        if (capacity_bytes == 0) {
            delete st;
            return fail(LC_ERR_INVALID_ARG, "lc_store_create: capacity_bytes must be > 0");
        }
        st->capacity = capacity_bytes;
    } else if (versions_per_layer == 1) {
        // size classes of the layer blocks; every layer's slot plus a spare per class
        st->layer_class.assign(size_t(ctx->nlayers), -1);
        uint64_t need = 0;
        for (int32_t l = 0; l < ctx->nlayers; ++l) {
            const uint64_t z = round_up(ctx->layer_bytes[size_t(l)], kStoreGrain);
            size_t c = 0;
            while (c < st->class_bytes.size() && st->class_bytes[c] != z) ++c;
            if (c == st->class_bytes.size()) {
                st->class_bytes.push_back(z);
                st->class_layers.push_back(0);
                need += z;
            }
            st->class_layers[c] += 1;
            st->layer_class[size_t(l)] = int32_t(c);
            need += z;
        }
        if (capacity_bytes < need) {
            delete st;
            return fail(LC_ERR_INVALID_ARG,
                        "lc_store_create: a newest-only store needs capacity_bytes >= %llu (every layer's "
                        "block plus one block of each distinct size), got %llu",
                        (unsigned long long)need, (unsigned long long)capacity_bytes);
        }
        st->capacity = capacity_bytes / kStoreGrain * kStoreGrain;
        layout_slots(st);
    } else {
        st->layer_base.resize(ctx->nlayers);
        st->layer_writes.assign(ctx->nlayers, 0);
        uint64_t off = 0;
        for (int32_t l = 0; l < ctx->nlayers; ++l) {
            st->layer_base[l] = off;
            off += uint64_t(versions_per_layer) * ctx->layer_bytes[l];
        }
        st->capacity = off;
    }
    DeviceGuard g(ctx->device);
    void* p = nullptr;
    const cudaError_t e = cudaHostAlloc(&p, st->capacity, cudaHostAllocDefault);
    if (e != cudaSuccess) {
        cudaGetLastError();
        delete st;
        return fail(LC_ERR_OOM, "lc_store_create: cannot pin %llu bytes: %s",
                    (unsigned long long)st->capacity, cudaGetErrorString(e));
    }
    st->arena = static_cast<uint8_t*>(p);
    {
        std::lock_guard<std::mutex> lk(g_store_mu);
        g_live_stores.insert(st);
    }
    *out = st;
    return LC_OK;
}

namespace {

// Waits (bounded) for copies still writing into a store's arena.
lc_status drain_inflight(lc_store* st, int timeout_ms) {
    lc_status rc = LC_OK;
    for (cudaEvent_t ev : st->inflight) {
        if (rc == LC_OK) rc = wait_event(ev, timeout_ms, "store copy");
        cudaEventDestroy(ev);
    }
    st->inflight.clear();
    return rc;
}

}  // namespace

extern "C" void lc_store_destroy(lc_store* st) {
    if (!st) return;
    {
        std::lock_guard<std::mutex> lk(g_store_mu);
        g_live_stores.erase(st);
    }
    if (drain_inflight(st, 60000) == LC_OK && st->arena) cudaFreeHost(st->arena);
    delete st;
}

extern "C" lc_status lc_store_clear(lc_store* st) {
    g_err.clear();
    if (!st) return fail(LC_ERR_INVALID_ARG, "lc_store_clear: store is NULL");
    for (const StoreVersion& v : st->versions)
        if (!v.durable) return fail(LC_ERR_STATE, "lc_store_clear: a version is still pending");
    LC_TRY(drain_inflight(st, 60000));
    st->versions.clear();
    st->top = 0;
    std::fill(st->layer_writes.begin(), st->layer_writes.end(), 0);
    if (st->per_layer == 1) layout_slots(st);
    return LC_OK;
}

extern "C" int64_t lc_store_num_versions(const lc_store* st) {
    return st ? int64_t(st->versions.size()) : 0;
}

extern "C" lc_status lc_store_get_info(const lc_store* st, lc_store_info* out) {
    g_err.clear();
    if (!st || !out) return fail(LC_ERR_INVALID_ARG, "lc_store_get_info: NULL argument");
    std::memset(out, 0, sizeof *out);
    out->arena = st->arena;
    out->capacity = st->capacity;
    for (const auto& x : st->excluded) out->excluded_bytes += x.second;
    for (const auto& x : st->avoid) out->avoided_bytes += x.second;
    for (const StoreVersion& v : st->versions) out->used_bytes += v.bytes;
    out->versions_per_layer = st->per_layer;
    return LC_OK;
}

extern "C" lc_status lc_store_get_version(const lc_store* st, int64_t index, lc_version* out) {
    g_err.clear();
    if (!st || !out) return fail(LC_ERR_INVALID_ARG, "lc_store_get_version: NULL argument");
    if (index < 0 || index >= int64_t(st->versions.size()))
        return fail(LC_ERR_INVALID_ARG, "lc_store_get_version: index %lld out of range", (long long)index);
    const StoreVersion& v = st->versions[size_t(index)];
    out->layer = v.layer;
    out->durable = v.durable;
    out->step = v.step;
    out->host_ptr = st->arena + v.off;
    out->bytes = v.bytes;
    return LC_OK;
}

extern "C" lc_status lc_store_plan(const lc_store* st, int64_t t_fail, int64_t* pick_out) {
    g_err.clear();
    if (!st || !pick_out) return fail(LC_ERR_INVALID_ARG, "lc_store_plan: NULL argument");
    for (int32_t l = 0; l < st->nlayers; ++l) pick_out[l] = -1;
    for (size_t i = 0; i < st->versions.size(); ++i) {
        const StoreVersion& v = st->versions[i];
        if (!v.durable || v.step > t_fail) continue;
        const int64_t cur = pick_out[v.layer];
        if (cur < 0 || v.step >= st->versions[size_t(cur)].step) pick_out[v.layer] = int64_t(i);
    }
    for (int32_t l = 0; l < st->nlayers; ++l)
        if (pick_out[l] < 0)
            return fail(LC_ERR_NOT_FOUND, "lc_store_plan: layer %d has no durable version at or before step %lld",
                        l, (long long)t_fail);
    return LC_OK;
}

extern "C" lc_status lc_store_exclude(lc_store* st, uint64_t offset, uint64_t bytes) {
    g_err.clear();
    if (!st) return fail(LC_ERR_INVALID_ARG, "lc_store_exclude: store is NULL");
    if (st->per_layer >= 2)
        return fail(LC_ERR_INVALID_ARG, "lc_store_exclude: a ring store's slots are fixed; use a log or "
                                        "newest-only store");
    if (bytes == 0 || offset >= st->capacity || bytes > st->capacity - offset)
        return fail(LC_ERR_INVALID_ARG, "lc_store_exclude: range [%llu, +%llu) outside the %llu-byte arena",
                    (unsigned long long)offset, (unsigned long long)bytes, (unsigned long long)st->capacity);
    // whole 4096-byte granules, so newest-only blocks stay aligned
    const uint64_t a = offset / kStoreGrain * kStoreGrain;
    const uint64_t b = std::min(st->capacity, round_up(offset + bytes, kStoreGrain));
    for (const StoreVersion& v : st->versions)
        if (v.off < b && a < v.off + v.bytes)
            return fail(LC_ERR_STATE, "lc_store_exclude: version of layer %d (step %lld) lies in the range",
                        v.layer, (long long)v.step);
    add_range(st->excluded, a, b);
    const uint64_t lo = a, hi = b;
    if (st->per_layer == 1) {
        if (st->versions.empty()) {
            layout_slots(st);          // an empty store lays its slots out anew
        } else {
            for (size_t c = 0; c < st->class_free.size(); ++c) {
                auto& fl = st->class_free[c];
                const uint64_t z = st->class_bytes[c];
                const size_t before = fl.size();
                fl.erase(std::remove_if(fl.begin(), fl.end(), [&](uint64_t o) { return o < hi && lo < o + z; }),
                         fl.end());
                st->class_slots[c] -= int32_t(before - fl.size());
            }
        }
    }
    return LC_OK;
}

extern "C" lc_status lc_store_check_dma(lc_store* st, lc_ctx* ctx, uint64_t region_bytes, int32_t passes,
                                        double min_fraction, double* rates_out, int64_t rates_cap,
                                        uint64_t* excluded_out) {
    Range range("lc_store_check_dma");
    g_err.clear();
    if (!st || !ctx) return fail(LC_ERR_INVALID_ARG, "lc_store_check_dma: NULL argument");
    if (st->per_layer >= 2) return fail(LC_ERR_INVALID_ARG, "lc_store_check_dma: ring stores are not supported");
    if (region_bytes == 0) region_bytes = 256ull << 20;
    if (region_bytes % kStoreGrain || region_bytes < (1ull << 20) || region_bytes > (1ull << 30))
        return fail(LC_ERR_INVALID_ARG, "lc_store_check_dma: region_bytes must be a multiple of 4096 in [1 MiB, 1 GiB]");
    if (!(min_fraction >= 0.0) || !std::isfinite(min_fraction))
        return fail(LC_ERR_INVALID_ARG, "lc_store_check_dma: min_fraction must be finite and >= 0");
    if (passes == 0) passes = 4;
    if (passes < 1 || passes > 64) return fail(LC_ERR_INVALID_ARG, "lc_store_check_dma: passes must be in [1, 64]");
    if (!st->versions.empty() || !st->inflight.empty())
        return fail(LC_ERR_STATE, "lc_store_check_dma: the store must be empty (it overwrites the arena)");
    const int64_t n = int64_t((st->capacity + region_bytes - 1) / region_bytes);
    if (rates_out && rates_cap < n)
        return fail(LC_ERR_INVALID_ARG, "lc_store_check_dma: rates_out needs %lld entries", (long long)n);
    DeviceGuard g(ctx->device);
    void* src = nullptr;
    cudaStream_t s = nullptr;
    std::vector<cudaEvent_t> ev(size_t(n) + 1, nullptr);
    std::vector<double> best(size_t(n), 0.0), worst(size_t(n), 0.0);
    lc_status rc = LC_OK;
    cudaError_t e = cudaMalloc(&src, region_bytes);
    if (e == cudaSuccess) e = cudaMemset(src, 0, region_bytes);
    if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&s, cudaStreamNonBlocking);
    for (size_t i = 0; i < ev.size() && e == cudaSuccess; ++i) e = cudaEventCreate(&ev[i]);
    // several passes: slow regions come and go (the same regions, slow in
    // about half of the passes on the hosts measured), so a region is judged
    // by its worst pass against the median of the regions' best passes
    for (int pass = 0; pass < passes && e == cudaSuccess && rc == LC_OK; ++pass) {
        e = cudaEventRecord(ev[0], s);
        for (int64_t i = 0; i < n && e == cudaSuccess; ++i) {
            const uint64_t off = uint64_t(i) * region_bytes;
            const uint64_t len = std::min(region_bytes, st->capacity - off);
            e = cudaMemcpyAsync(st->arena + off, src, len, cudaMemcpyDeviceToHost, s);
            if (e == cudaSuccess) e = cudaEventRecord(ev[size_t(i) + 1], s);
        }
        if (e != cudaSuccess) break;
        rc = wait_event(ev[size_t(n)], ctx->cfg.timeout_ms, "lc_store_check_dma");
        for (int64_t i = 0; i < n && rc == LC_OK && e == cudaSuccess; ++i) {
            float ms = 0.f;
            e = cudaEventElapsedTime(&ms, ev[size_t(i)], ev[size_t(i) + 1]);
            const uint64_t len = std::min(region_bytes, st->capacity - uint64_t(i) * region_bytes);
            if (e == cudaSuccess && ms > 0.f) {
                const double r = len / (1e6 * ms);
                best[size_t(i)] = std::max(best[size_t(i)], r);
                worst[size_t(i)] = pass == 0 ? r : std::min(worst[size_t(i)], r);
            }
        }
    }
    if (e != cudaSuccess && rc == LC_OK) {
        cudaGetLastError();
        rc = fail(LC_ERR_CUDA, "lc_store_check_dma: %s", cudaGetErrorString(e));
    }
    if (rc == LC_ERR_TIMEOUT) {
        // copies still in flight: leave the source buffer to them rather than
        // block in cudaFree (which waits for the whole device)
        cudaGetLastError();
        return rc;
    }
    if (s) cudaStreamSynchronize(s);
    for (cudaEvent_t x : ev)
        if (x) cudaEventDestroy(x);
    if (s) cudaStreamDestroy(s);
    if (src) cudaFree(src);
    cudaGetLastError();
    if (rc != LC_OK) return rc;
    std::vector<double> sorted = best;
    std::sort(sorted.begin(), sorted.end());
    const double median = sorted[sorted.size() / 2];
    // the slow regions, slowest first (lower index first on a tie), each
    // kept out of use unless that would leave no room for a step that
    // persists every layer; a store without that room to begin with loses
    // every slow region
    std::vector<int64_t> slow;
    for (int64_t i = 0; i < n; ++i) {
        if (rates_out) rates_out[i] = worst[size_t(i)];
        if (worst[size_t(i)] < min_fraction * median) slow.push_back(i);
    }
    std::stable_sort(slow.begin(), slow.end(),
                     [&](int64_t a, int64_t b) { return worst[size_t(a)] < worst[size_t(b)]; });
    const bool guard = full_step_fits(st, st->excluded);
    RangeMap taken;                      // regions of this call, disjoint from each other
    std::vector<char> take(size_t(n), 0);
    for (int64_t i : slow) {
        const uint64_t off = uint64_t(i) * region_bytes;
        taken.emplace(off, std::min(region_bytes, st->capacity - off));
        if (guard && !full_step_fits(st, st->excluded, taken)) {
            taken.erase(off);
            continue;
        }
        take[size_t(i)] = 1;
    }
    // the slow regions left in use are avoided while a step fits without them
    RangeMap avoid;
    for (int64_t i : slow) {
        if (take[size_t(i)]) continue;
        const uint64_t off = uint64_t(i) * region_bytes;
        add_range(avoid, off, off + std::min(region_bytes, st->capacity - off));
    }
    st->avoid.swap(avoid);
    uint64_t excluded = 0;
    for (int64_t i = 0; i < n; ++i) {
        if (!take[size_t(i)]) continue;
        const uint64_t off = uint64_t(i) * region_bytes;
        const uint64_t len = std::min(region_bytes, st->capacity - off);
        LC_TRY(lc_store_exclude(st, off, len));
        excluded += len;
    }
    if (st->per_layer == 1 && excluded == 0) layout_slots(st);   // with the new ranges to avoid
    if (excluded_out) *excluded_out = excluded;
    return LC_OK;
}

// ---------------------------------------------------------------------------
// host internals used by the file tier (lc_files.cu)
// ---------------------------------------------------------------------------
int32_t lc::ctx_nlayers(const lc_ctx* ctx) { return ctx->nlayers; }
int32_t lc::store_nlayers(const lc_store* st) { return st->nlayers; }
const uint64_t* lc::store_layer_bytes(const lc_store* st) { return st->layer_bytes.data(); }

uint8_t* lc::store_append(lc_store* st, int32_t layer, int64_t* index_out) {
    if (st->per_layer != 0 || layer < 0 || layer >= st->nlayers) return nullptr;
    const uint64_t bytes = st->layer_bytes[size_t(layer)];
    const uint64_t at = log_place(st, st->top, bytes);
    if (at + bytes > st->capacity) return nullptr;
    st->versions.push_back({st->next_id++, layer, 1, -1, at, bytes, -1});
    uint8_t* p = st->arena + at;
    st->top = at + bytes;
    if (index_out) *index_out = int64_t(st->versions.size()) - 1;
    return p;
}

void lc::store_set_step(lc_store* st, int64_t index, int64_t step) {
    if (index >= 0 && size_t(index) < st->versions.size()) st->versions[size_t(index)].step = step;
}

lc_status lc::fail_status(lc_status st, const char* fmt, ...) {
    char buf[1024];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    g_err = buf;
    return st;
}
