// lc_select.cu -- §3.2 Eq. 2-4 and the §3.3 staleness guard on the device,
// plus the packed-stream layout of the persisted layers (one CTA).
//
// From the per-layer sums of Eq. 1 the kernel forms u_l, updates the
// accumulator Delta_l, persists a layer when Delta_l >= tau * tau_mult[l],
// when its staleness t - t_l has reached S_max, or when the drift is not
// finite; it resets Delta_l and sets t_l = t for persisted layers.  It then
// assigns each persisted layer its offset in the packed stream (layers
// ascending) and writes the copy lists of the pack and of the snapshot
// commit, so the host never builds them.  If the stream would not fit the
// destination, it persists nothing and restores every layer's state to the
// not-persisted update (the drift stays accumulated).  The step comes from
// the host, or from a device counter when the step runs as a CUDA graph.
#include "lc_internal.cuh"

namespace lc {
namespace {

__global__ void __launch_bounds__(kSelectThreads) select_kernel(const SelectParams p) {
    const ResultLayout L = result_layout(p.nlayers);
    ResultHeader* hdr = reinterpret_cast<ResultHeader*>(p.result);
    uint8_t* mask = p.result + L.mask_off;
    double* u_out = reinterpret_cast<double*>(p.result + L.u_off);
    uint64_t* off = reinterpret_cast<uint64_t*>(p.result + L.off_off);
    int64_t* scratch = p.layer_scratch;

    __shared__ int s_nonfinite;
    __shared__ int64_t s_step;
    __shared__ uint32_t s_status;
    if (threadIdx.x == 0) {
        s_nonfinite = 0;
        s_step = p.step_from_counter ? *p.step_counter + 1 : p.step;
        *p.step_counter = s_step;
    }
    __syncthreads();
    const int64_t step = s_step;

    for (int l = threadIdx.x; l < p.nlayers; l += blockDim.x) {
        const double d = p.sums[3 * l], a = p.sums[3 * l + 1], n = p.sums[3 * l + 2];
        const double u = (d / n) / (a / n + p.eps_w);                     // Eq. 1
        const double acc = p.mode == 1 ? p.delta[l] + u : u;              // Eq. 2
        const double threshold = p.tau * p.tau_mult[l];
        const int64_t staleness = step - p.t_last[l];
        const bool nonfinite = !isfinite(acc);
        const bool persist = nonfinite || acc >= threshold                // Eq. 3
                             || staleness >= int64_t(p.max_staleness);     // §3.3
        if (nonfinite) atomicAdd(&s_nonfinite, 1);
        p.acc_save[l] = acc;
        p.tl_save[l] = p.t_last[l];
        if (persist) {                                                     // Eq. 4
            p.delta[l] = 0.0;
            p.t_last[l] = step;
        } else {
            p.delta[l] = acc;
        }
        mask[l] = persist ? 1 : 0;
        u_out[l] = u;
    }
    __syncthreads();

    // Stream layout and staleness statistics, layers ascending, in one
    // thread so that the sums keep a fixed order; every per-layer input is
    // first staged in shared memory by the whole CTA, a tile at a time, so
    // the ordered loop reads no global memory.
    __shared__ int64_t t_st[kSelectThreads];
    __shared__ int64_t t_numel[kSelectThreads];
    __shared__ uint64_t t_bytes[kSelectThreads];
    __shared__ uint64_t t_cw[kSelectThreads];
    __shared__ int32_t t_nsec[kSelectThreads];
    __shared__ int32_t t_nwsec[kSelectThreads];
    __shared__ uint8_t t_sel[kSelectThreads];
    uint64_t run = 0, commit_work = 0;
    int nsel = 0, nsec = 0, ncommit = 0;
    int64_t mx = 0;
    double num = 0.0, den = 0.0;
    for (int base = 0; base < p.nlayers; base += kSelectThreads) {
        const int l = base + int(threadIdx.x);
        if (l < p.nlayers) {
            const bool sel = mask[l] != 0;
            t_st[threadIdx.x] = step - p.t_last[l];
            t_numel[threadIdx.x] = p.layer_numel[l];
            t_sel[threadIdx.x] = sel ? 1 : 0;
            uint64_t cw = 0;
            int ns = 0, nw = 0;
            if (sel) {
                ns = p.layer_sec_begin[l + 1] - p.layer_sec_begin[l];
                nw = p.layer_wsec_count[l];
                cw = p.layer_commit_work[l];
            }
            t_bytes[threadIdx.x] = sel ? p.layer_bytes[l] : 0;
            t_cw[threadIdx.x] = cw;
            t_nsec[threadIdx.x] = ns;
            t_nwsec[threadIdx.x] = nw;
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            const int n = p.nlayers - base < kSelectThreads ? p.nlayers - base : kSelectThreads;
            for (int i = 0; i < n; ++i) {
                const int64_t st = t_st[i];
                mx = st > mx ? st : mx;
                num = __dadd_rn(num, __dmul_rn(double(t_numel[i]), double(st)));
                den = __dadd_rn(den, double(t_numel[i]));
                if (t_sel[i]) {
                    off[base + i] = run;
                    run += t_bytes[i];
                    scratch[3 * (base + i)] = nsec;
                    scratch[3 * (base + i) + 1] = ncommit;
                    scratch[3 * (base + i) + 2] = int64_t(commit_work);
                    nsec += t_nsec[i];
                    ncommit += t_nwsec[i];
                    commit_work += t_cw[i];
                    ++nsel;
                } else {
                    off[base + i] = 0;
                }
            }
        }
        __syncthreads();
    }

    if (threadIdx.x == 0) {
        // a stream larger than the destination persists nothing this step
        const bool fits = run <= p.capacity;
        hdr->step = step;
        hdr->n_selected = nsel;
        hdr->n_nonfinite = s_nonfinite;
        hdr->bytes = run;
        hdr->n_pack_desc = fits ? nsec : 0;
        hdr->n_commit_desc = fits ? ncommit : 0;
        hdr->commit_work = fits ? commit_work : 0;
        hdr->max_staleness = mx;
        hdr->weighted_staleness = den > 0.0 ? num / den : 0.0;
        hdr->magic = kResultMagic;
        hdr->status = fits ? kStatusOk : kStatusCapacity;
        hdr->pack_bytes = fits ? run : 0;
        s_status = hdr->status;
    }
    __syncthreads();

    if (s_status != kStatusOk) {
        // roll back to "nothing persisted": the drift stays accumulated
        for (int l = threadIdx.x; l < p.nlayers; l += blockDim.x) {
            p.delta[l] = p.acc_save[l];
            p.t_last[l] = p.tl_save[l];
        }
        return;
    }
    // the copy lists, one section per thread: a persisted layer's sections
    // go to its pack entries (and its W sections to its commit entries) at
    // the indices and offsets laid out above
    const bool fused = p.fuse_commit != 0 && p.mode == 0;
    const int nsec_all = p.layer_sec_begin[p.nlayers];
    for (int j = threadIdx.x; j < nsec_all; j += blockDim.x) {
        const SectionDev sec = p.secs[j];
        const int l = sec.layer;
        if (!mask[l]) continue;
        CopyDesc d;
        d.woff = off[l] + sec.off_in_layer;
        d.nbytes = sec.nbytes;
        d.span = sec.span;
        d.src = sec.src;
        d.dst = nullptr;
        d.dst2 = (fused && sec.ref) ? sec.ref : nullptr;
        p.pack_desc[scratch[3 * l] + sec.idx] = d;
        if (sec.idx < p.layer_wsec_count[l]) {
            CopyDesc c;
            c.woff = uint64_t(scratch[3 * l + 2]) + sec.commit_off;
            c.nbytes = sec.nbytes;
            c.span = (sec.nbytes + 15) & ~uint64_t(15);
            c.src = sec.src;
            c.dst = sec.ref;
            c.dst2 = nullptr;
            p.commit_desc[scratch[3 * l + 1] + sec.idx] = c;
        }
    }
}

}  // namespace

cudaError_t launch_select(const SelectParams& p, cudaStream_t s) {
    cudaGetLastError();
    select_kernel<<<1, kSelectThreads, 0, s>>>(p);
    return cudaGetLastError();
}

}  // namespace lc
