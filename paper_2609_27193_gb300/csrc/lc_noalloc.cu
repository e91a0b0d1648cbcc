// lc_noalloc.cu -- lc_measure_noalloc: the per-layer sums of lc_measure for
// callers that cannot allocate device memory.
//
// It launches the same measure kernel as lc_measure, but every table and
// scratch buffer that kernel needs (segment table, CTA partition, partial
// sums, completion counter) lives in one file-scope static device array of
// LC_NOALLOC_SCRATCH_BYTES.  Host code never uses the array's name as an
// address: at set-up, once per device and with that device current, the
// array's device address is looked up with cudaGetSymbolAddress and cached.
// The tables are built on the host and reach the array as the kernel
// parameters of small upload kernels launched on the caller's stream ahead
// of the measure, so the driver copies them when each upload is launched and
// nothing reads host memory once the call has returned.  The completion
// counter travels in the upload as zero.  No cudaMalloc, cudaFree or other
// allocating routine is called.
#include "layercheck.h"
#include "lc_internal.cuh"

#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>

using namespace lc;

namespace {

constexpr int kMaxSeg = LC_NOALLOC_MAX_SEGMENTS;
constexpr int kMaxLayers = LC_NOALLOC_MAX_LAYERS;
constexpr int kMaxCtas = 2048;
constexpr int kMaxDevices = 64;

constexpr size_t al256(size_t x) { return (x + 255) & ~size_t(255); }

constexpr size_t al16(size_t x) { return (x + 15) & ~size_t(15); }

// Where each table of one call sits in the array: the tables are packed
// back to back (16-byte aligned) for the call's sizes, so the upload moves
// only the bytes the measure will read.
struct TableLayout {
    size_t segs, cta_vec, cta_seg, cta_slot, seg_slot, layer_seg, ticket, bytes;
};

constexpr TableLayout table_layout(size_t nseg, size_t nlayers, size_t G) {
    TableLayout t{};
    t.segs = 0;
    t.cta_vec = al16(t.segs + sizeof(SegDev) * nseg);
    t.cta_seg = al16(t.cta_vec + sizeof(int64_t) * (G + 1));
    t.cta_slot = al16(t.cta_seg + sizeof(int32_t) * G);
    t.seg_slot = al16(t.cta_slot + sizeof(int32_t) * G);
    t.layer_seg = al16(t.seg_slot + sizeof(int32_t) * (nseg + 1));
    t.ticket = al16(t.layer_seg + sizeof(int32_t) * (nlayers + 1));
    t.bytes = al16(t.ticket + sizeof(unsigned int));
    return t;
}

// Scratch layout: the tables (at most kTableBytes), then the kernel scratch.
constexpr size_t kTableBytes = al256(table_layout(kMaxSeg, kMaxLayers, kMaxCtas).bytes);
constexpr size_t kOffPartials = kTableBytes;
constexpr size_t kOffSegSums = al256(kOffPartials + sizeof(double2) * (kMaxCtas + kMaxSeg));
constexpr size_t kScratchUsed = al256(kOffSegSums + sizeof(double) * 2 * kMaxSeg);
static_assert(kScratchUsed <= LC_NOALLOC_SCRATCH_BYTES, "scratch layout exceeds its array");

}  // namespace

// The scratch of every lc_measure_noalloc call on a device.
static __device__ __align__(256) unsigned char g_noalloc_scratch[LC_NOALLOC_SCRATCH_BYTES];

namespace {

// One upload: `nbytes` (a multiple of 16) of the table image, to be written
// at byte `dst_off` of the scratch array.  Passed by value, so the launch
// itself carries the bytes.
constexpr int kUploadVecs = 1024;   // 16 KB of payload per launch
struct UploadChunk {
    uint32_t dst_off;
    uint32_t nbytes;
    uint4 data[kUploadVecs];
};
static_assert(sizeof(UploadChunk) <= 32000, "kernel parameters are limited to 32764 bytes");

__global__ void __launch_bounds__(256) noalloc_upload_kernel(const __grid_constant__ UploadChunk c) {
    uint4* dst = reinterpret_cast<uint4*>(g_noalloc_scratch + c.dst_off);
    const uint32_t nv = c.nbytes / 16;
    for (uint32_t i = threadIdx.x; i < nv; i += blockDim.x) dst[i] = c.data[i];
}

}  // namespace

namespace {

struct DeviceScratch {
    bool ready = false;
    unsigned char* addr = nullptr;   // device address of g_noalloc_scratch
    int max_grid = 0;
};
DeviceScratch g_scratch[kMaxDevices];
std::mutex g_scratch_mu;

// Table image built on the host; one per host thread, no heap.  The upload
// launches copy it into their parameters, so it may be rebuilt as soon as
// the call returns.
thread_local unsigned char t_image[kTableBytes] __attribute__((aligned(16)));
thread_local UploadChunk t_chunk;

lc_status err(lc_status st, const char* fmt, ...) __attribute__((format(printf, 2, 3)));
lc_status err(lc_status st, const char* fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    set_last_error(buf);
    return st;
}

struct CurrentDevice {
    int prev = -1;
    bool ok = false;
    explicit CurrentDevice(int dev) {
        if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
        ok = (prev == dev) || cudaSetDevice(dev) == cudaSuccess;
    }
    ~CurrentDevice() {
        int cur = -1;
        if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
    }
};

// Once per device, with the device current: the array's device address.
lc_status setup_device(int device, DeviceScratch* out) {
    std::lock_guard<std::mutex> lk(g_scratch_mu);
    DeviceScratch& d = g_scratch[device];
    if (!d.ready) {
        void* addr = nullptr;
        cudaError_t e = cudaGetSymbolAddress(&addr, g_noalloc_scratch);
        if (e != cudaSuccess) {
            cudaGetLastError();
            return err(LC_ERR_CUDA, "lc_measure_noalloc: cudaGetSymbolAddress failed: %s",
                       cudaGetErrorString(e));
        }
        int sms = 0, occ = 0;
        e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, device);
        if (e == cudaSuccess) e = measure_occupancy(&occ);
        if (e != cudaSuccess) {
            cudaGetLastError();
            return err(LC_ERR_CUDA, "lc_measure_noalloc: device query failed: %s", cudaGetErrorString(e));
        }
        d.addr = static_cast<unsigned char*>(addr);
        d.max_grid = sms * (occ > 0 ? occ : 1);
        if (d.max_grid > kMaxCtas) d.max_grid = kMaxCtas;
        if (d.max_grid < 1) d.max_grid = 1;
        d.ready = true;
    }
    *out = d;
    return LC_OK;
}

bool is_device_memory(const void* p, int device) {
    cudaPointerAttributes a;
    if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    if (a.type == cudaMemoryTypeManaged) return true;
    return a.type == cudaMemoryTypeDevice && a.device == device;
}

}  // namespace

extern "C" lc_status lc_measure_noalloc(int device, void* cuda_stream, const lc_segment* segs,
                                        int32_t nseg, int32_t nlayers, double* sums_out) {
    set_last_error("");
    if (!segs || nseg <= 0) return err(LC_ERR_INVALID_ARG, "lc_measure_noalloc: no segments");
    if (nlayers <= 0) return err(LC_ERR_INVALID_ARG, "lc_measure_noalloc: nlayers must be > 0");
    if (nseg > kMaxSeg)
        return err(LC_ERR_CAPACITY, "lc_measure_noalloc: %d segments exceed LC_NOALLOC_MAX_SEGMENTS (%d)",
                   nseg, kMaxSeg);
    if (nlayers > kMaxLayers)
        return err(LC_ERR_CAPACITY, "lc_measure_noalloc: %d layers exceed LC_NOALLOC_MAX_LAYERS (%d)",
                   nlayers, kMaxLayers);
    if (!sums_out || (reinterpret_cast<uintptr_t>(sums_out) & 7))
        return err(LC_ERR_INVALID_ARG, "lc_measure_noalloc: sums_out must be 8-byte aligned device memory");
    int ndev = 0;
    if (cudaGetDeviceCount(&ndev) != cudaSuccess) {
        cudaGetLastError();
        return err(LC_ERR_CUDA, "lc_measure_noalloc: no CUDA device");
    }
    if (device < 0 || device >= ndev || device >= kMaxDevices)
        return err(LC_ERR_INVALID_ARG, "lc_measure_noalloc: device %d out of range", device);
    CurrentDevice cur(device);
    if (!cur.ok) return err(LC_ERR_CUDA, "lc_measure_noalloc: cannot make device %d current", device);
    if (!is_device_memory(sums_out, device))
        return err(LC_ERR_INVALID_ARG, "lc_measure_noalloc: sums_out is not device memory");

    // validate and order the segments: layers ascending, registration order within
    int32_t per_layer[kMaxLayers + 1];
    std::memset(per_layer, 0, sizeof per_layer);
    for (int32_t i = 0; i < nseg; ++i) {
        const lc_segment& s = segs[i];
        if (s.layer < 0 || s.layer >= nlayers)
            return err(LC_ERR_INVALID_ARG, "lc_measure_noalloc: segment %d layer %d outside [0, %d)", i,
                       s.layer, nlayers);
        if (s.w_dtype != LC_BF16 && s.w_dtype != LC_F32)
            return err(LC_ERR_INVALID_ARG, "lc_measure_noalloc: segment %d has unknown dtype", i);
        if (s.numel <= 0 || !s.w || !s.snap)
            return err(LC_ERR_INVALID_ARG, "lc_measure_noalloc: segment %d needs numel > 0, w and snap", i);
        if (s.snap == s.w)
            return err(LC_ERR_INVALID_ARG, "lc_measure_noalloc: segment %d: snap must not alias w", i);
        const uintptr_t esz = s.w_dtype == LC_BF16 ? 2 : 4;
        if ((reinterpret_cast<uintptr_t>(s.w) % esz) || (reinterpret_cast<uintptr_t>(s.snap) % esz))
            return err(LC_ERR_INVALID_ARG, "lc_measure_noalloc: segment %d not element-aligned", i);
        if (!is_device_memory(s.w, device) || !is_device_memory(s.snap, device))
            return err(LC_ERR_INVALID_ARG, "lc_measure_noalloc: segment %d is not device memory", i);
        per_layer[s.layer] += 1;
    }
    int32_t layer_begin[kMaxLayers + 1];
    layer_begin[0] = 0;
    for (int32_t l = 0; l < nlayers; ++l) {
        if (per_layer[l] == 0) return err(LC_ERR_INVALID_ARG, "lc_measure_noalloc: layer %d has no segment", l);
        layer_begin[l + 1] = layer_begin[l] + per_layer[l];
    }
    DeviceScratch ds;
    lc_status st = setup_device(device, &ds);
    if (st != LC_OK) return st;

    std::memset(t_image, 0, sizeof t_image);
    // the segment table sits at offset 0 whatever the grid; the rest of the
    // layout depends on the grid, known once the work space is measured
    SegDev* sd = reinterpret_cast<SegDev*>(t_image);
    int32_t fill[kMaxLayers];
    std::memcpy(fill, layer_begin, sizeof(int32_t) * nlayers);
    for (int32_t i = 0; i < nseg; ++i) {
        const lc_segment& s = segs[i];
        SegDev& d = sd[fill[s.layer]++];
        const int esz_log2 = s.w_dtype == LC_BF16 ? 1 : 2;
        const int ve = 16 >> esz_log2;
        d.w = static_cast<const uint8_t*>(s.w);
        d.r = static_cast<uint8_t*>(s.snap);
        d.numel = s.numel;
        d.lead = int32_t((reinterpret_cast<uintptr_t>(s.w) & 15) >> esz_log2);
        d.esz_log2 = esz_log2;
        d.coaligned = (reinterpret_cast<uintptr_t>(s.w) & 15) == (reinterpret_cast<uintptr_t>(s.snap) & 15);
        d.layer = s.layer;
        d.nvec = (int64_t(d.lead) + s.numel + ve - 1) / ve;
    }
    int64_t V = 0;
    for (int32_t i = 0; i < nseg; ++i) {
        sd[i].vec_begin = V;
        V += sd[i].nvec;
    }
    const int64_t ngran = (V + LC_MEASURE_ALIGN_VECS - 1) / LC_MEASURE_ALIGN_VECS;
    const int64_t G = ngran < ds.max_grid ? ngran : ds.max_grid;
    const TableLayout L = table_layout(size_t(nseg), size_t(nlayers), size_t(G));
    if (L.bytes > kTableBytes) return err(LC_ERR_CUDA, "lc_measure_noalloc: internal table overflow");
    int64_t* cta_vec = reinterpret_cast<int64_t*>(t_image + L.cta_vec);
    int32_t* cta_seg = reinterpret_cast<int32_t*>(t_image + L.cta_seg);
    int32_t* cta_slot = reinterpret_cast<int32_t*>(t_image + L.cta_slot);
    int32_t* seg_slot = reinterpret_cast<int32_t*>(t_image + L.seg_slot);
    int32_t* layer_seg = reinterpret_cast<int32_t*>(t_image + L.layer_seg);
    for (int32_t i = 0; i <= nseg; ++i) seg_slot[i] = -1;
    for (int64_t b = 0; b <= G; ++b) {
        const int64_t v = ngran * b / G * LC_MEASURE_ALIGN_VECS;
        cta_vec[b] = v < V ? v : V;
    }
    int32_t slot = 0, s = 0;
    for (int64_t b = 0; b < G; ++b) {
        const int64_t v0 = cta_vec[b], v1 = cta_vec[b + 1];
        while (s < nseg && sd[s].vec_begin + sd[s].nvec <= v0) ++s;
        cta_seg[b] = s;
        cta_slot[b] = slot;
        for (int32_t t = s; v0 < v1 && t < nseg && sd[t].vec_begin < v1; ++t) {
            if (seg_slot[t] < 0) seg_slot[t] = slot;
            ++slot;
        }
    }
    seg_slot[nseg] = slot;
    for (int32_t t = nseg - 1; t >= 0; --t)
        if (seg_slot[t] < 0) seg_slot[t] = seg_slot[t + 1];
    std::memcpy(layer_seg, layer_begin, sizeof(int32_t) * (nlayers + 1));
    if (slot > kMaxCtas + kMaxSeg) return err(LC_ERR_CUDA, "lc_measure_noalloc: internal slot overflow");

    cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
    // the tables and a zero completion counter into the scratch array,
    // stream-ordered before the measure; each launch carries its bytes
    cudaGetLastError();
    for (size_t off = 0; off < L.bytes; off += sizeof t_chunk.data) {
        const size_t n = L.bytes - off < sizeof t_chunk.data ? L.bytes - off : sizeof t_chunk.data;
        t_chunk.dst_off = uint32_t(off);
        t_chunk.nbytes = uint32_t(n);
        std::memcpy(t_chunk.data, t_image + off, n);
        noalloc_upload_kernel<<<1, 256, 0, stream>>>(t_chunk);
        const cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess)
            return err(LC_ERR_CUDA, "lc_measure_noalloc: table upload failed: %s", cudaGetErrorString(e));
    }
    MeasureParams p{};
    p.segs = reinterpret_cast<const SegDev*>(ds.addr + L.segs);
    p.cta_vec_begin = reinterpret_cast<const int64_t*>(ds.addr + L.cta_vec);
    p.cta_seg0 = reinterpret_cast<const int32_t*>(ds.addr + L.cta_seg);
    p.cta_slot0 = reinterpret_cast<const int32_t*>(ds.addr + L.cta_slot);
    p.seg_slot_begin = reinterpret_cast<const int32_t*>(ds.addr + L.seg_slot);
    p.layer_seg_begin = reinterpret_cast<const int32_t*>(ds.addr + L.layer_seg);
    p.partials = reinterpret_cast<double2*>(ds.addr + kOffPartials);
    p.seg_sums = reinterpret_cast<double*>(ds.addr + kOffSegSums);
    p.sums = sums_out;
    p.ticket = reinterpret_cast<unsigned int*>(ds.addr + L.ticket);
    p.nseg = nseg;
    p.nlayers = nlayers;
    const cudaError_t e = launch_measure(p, int(G), false, stream);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return err(LC_ERR_CUDA, "lc_measure_noalloc: launch failed: %s", cudaGetErrorString(e));
    }
    return LC_OK;
}
