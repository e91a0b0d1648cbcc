// lc_select.cu -- §3.2 Eq. 2-4 and the §3.3 staleness guard on the device,
// plus the packed-stream layout of the persisted layers (one CTA).
//
// From the per-layer sums of Eq. 1 the kernel forms u_l, updates the
// accumulator Delta_l, persists a layer when Delta_l >= tau * tau_mult[l],
// when its staleness t - t_l has reached S_max, or when the drift is not
// finite; it resets Delta_l and sets t_l = t for persisted layers.  It then
// assigns each persisted layer its offset in the packed stream (layers
// ascending) and writes the copy lists of the pack and of the snapshot
// commit, so the host never builds them.
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
    if (threadIdx.x == 0) s_nonfinite = 0;
    __syncthreads();

    for (int l = threadIdx.x; l < p.nlayers; l += blockDim.x) {
        const double d = p.sums[3 * l], a = p.sums[3 * l + 1], n = p.sums[3 * l + 2];
        const double u = (d / n) / (a / n + p.eps_w);                     // Eq. 1
        const double acc = p.mode == 1 ? p.delta[l] + u : u;              // Eq. 2
        const double threshold = p.tau * p.tau_mult[l];
        const int64_t staleness = p.step - p.t_last[l];
        const bool nonfinite = !isfinite(acc);
        const bool persist = nonfinite || acc >= threshold                // Eq. 3
                             || staleness >= int64_t(p.max_staleness);     // §3.3
        if (nonfinite) atomicAdd(&s_nonfinite, 1);
        if (persist) {                                                     // Eq. 4
            p.delta[l] = 0.0;
            p.t_last[l] = p.step;
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
            const int64_t st = p.step - p.t_last[l];
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
        hdr->step = p.step;
        hdr->n_selected = nsel;
        hdr->n_nonfinite = s_nonfinite;
        hdr->bytes = run;
        hdr->n_pack_desc = nsec;
        hdr->n_commit_desc = ncommit;
        hdr->commit_work = commit_work;
        hdr->max_staleness = mx;
        hdr->weighted_staleness = den > 0.0 ? num / den : 0.0;
        hdr->magic = kResultMagic;
        hdr->reserved = 0;
    }
    __syncthreads();

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
