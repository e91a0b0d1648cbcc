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

    if (threadIdx.x == 0) {
        uint64_t run = 0, commit_work = 0;
        int nsel = 0, nsec = 0, ncommit = 0;
        int64_t mx = 0;
        double num = 0.0, den = 0.0;
        for (int l = 0; l < p.nlayers; ++l) {
            const int64_t st = step - p.t_last[l];
            mx = st > mx ? st : mx;
            num = __dadd_rn(num, __dmul_rn(double(p.layer_numel[l]), double(st)));
            den = __dadd_rn(den, double(p.layer_numel[l]));
            if (mask[l]) {
                off[l] = run;
                run += p.layer_bytes[l];
                scratch[3 * l] = nsec;
                scratch[3 * l + 1] = ncommit;
                scratch[3 * l + 2] = int64_t(commit_work);
                const int s0 = p.layer_sec_begin[l];
                nsec += p.layer_sec_begin[l + 1] - s0;
                for (int j = s0; j < s0 + p.layer_wsec_count[l]; ++j) {
                    commit_work += (p.secs[j].nbytes + 15) & ~uint64_t(15);
                    ++ncommit;
                }
                ++nsel;
            } else {
                off[l] = 0;
            }
        }
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
    const bool fused = p.fuse_commit != 0 && p.mode == 0;
    for (int l = threadIdx.x; l < p.nlayers; l += blockDim.x) {
        if (!mask[l]) continue;
        const int s0 = p.layer_sec_begin[l], s1 = p.layer_sec_begin[l + 1];
        int64_t di = scratch[3 * l];
        for (int j = s0; j < s1; ++j, ++di) {
            const SectionDev sec = p.secs[j];
            CopyDesc d;
            d.woff = off[l] + sec.off_in_layer;
            d.nbytes = sec.nbytes;
            d.span = sec.span;
            d.src = sec.src;
            d.dst = nullptr;
            d.dst2 = (fused && sec.ref) ? sec.ref : nullptr;
            p.pack_desc[di] = d;
        }
        int64_t ci = scratch[3 * l + 1];
        uint64_t cw = uint64_t(scratch[3 * l + 2]);
        for (int j = s0; j < s0 + p.layer_wsec_count[l]; ++j, ++ci) {
            const SectionDev sec = p.secs[j];
            CopyDesc d;
            d.woff = cw;
            d.nbytes = sec.nbytes;
            d.span = (sec.nbytes + 15) & ~uint64_t(15);
            d.src = sec.src;
            d.dst = sec.ref;
            d.dst2 = nullptr;
            p.commit_desc[ci] = d;
            cw += d.span;
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
