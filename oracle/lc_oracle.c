/*
 * lc_oracle.c -- the LayerCheck reference oracle (plain C, single thread).
 *
 * TEST INFRASTRUCTURE ONLY: loaded by the tests, the smoke check and the
 * benchmark's CPU-baseline leg, never by the product library.  Every
 * function restates one passage of the paper in the most direct form; no
 * blocking, vectorisation or reordering.  Floating point is binary64 and
 * the file must be compiled with -ffp-contract=off.
 */
#include "lc_oracle.h"

#include <math.h>
#include <string.h>

double lco_bf16_value(uint16_t bits)
{
    /* bf16 keeps the sign, the 8 exponent bits and the top 7 mantissa bits
     * of a binary32 value, so the binary32 with these bits in its upper
     * half has exactly the bf16 value. */
    uint32_t word = ((uint32_t)bits) << 16;
    float f;
    memcpy(&f, &word, sizeof f);
    return (double)f;
}

/* Element i of a weight tensor, widened to binary64 (exact for both types). */
static double elem(const void* base, int32_t dtype, int64_t i)
{
    if (dtype == LCO_BF16) {
        uint16_t bits;
        memcpy(&bits, (const uint8_t*)base + 2 * i, sizeof bits);
        return lco_bf16_value(bits);
    } else {
        float f;
        memcpy(&f, (const uint8_t*)base + 4 * i, sizeof f);
        return (double)f;
    }
}

static uint64_t elem_size(int32_t dtype)
{
    return dtype == LCO_BF16 ? 2u : 4u;
}

/* Eq. 1 (§3.2).  The mean is taken element-wise over all of the layer's
 * parameters, so the layer is one list of elements: the tensors in the
 * order given, each in index order.  W - R is exact in binary64 for bf16
 * and fp32 inputs, so the only rounding is in the running sums. */
void lco_layer_sums(const lco_tensor* t, int32_t ntensors, double out[3])
{
    double d_sum = 0.0;  /* sum |W_l(t) - W_l(t-1)| */
    double a_sum = 0.0;  /* sum |W_l(t-1)|          */
    int64_t n = 0;
    for (int32_t k = 0; k < ntensors; ++k) {
        for (int64_t i = 0; i < t[k].numel; ++i) {
            double w = elem(t[k].w, t[k].dtype, i);
            double r = elem(t[k].r, t[k].dtype, i);
            d_sum += fabs(w - r);
            a_sum += fabs(r);
        }
        n += t[k].numel;
    }
    out[0] = d_sum;
    out[1] = a_sum;
    out[2] = (double)n;
}

/* Eq. 1 (§3.2): u_l = mean(|W_l(t) - W_l(t-1)|) / (mean(|W_l(t-1)|) + eps_w). */
double lco_update_measure(double d_sum, double a_sum, double n, double eps_w)
{
    double mean_abs_update = d_sum / n;
    double mean_abs_weight = a_sum / n;
    return mean_abs_update / (mean_abs_weight + eps_w);
}

/* One checkpoint opportunity; every training step is one (§4.3, the
 * checkpoint-per-iteration regime).
 *   Eq. 2: Delta_l <- Delta_l + u_l(t)   (LCO_ACCUMULATE: R = W(t-1));
 *          with R = the last persisted snapshot (LCO_SNAPSHOT), u_l already
 *          is the drift accumulated since the last persistence, so the
 *          accumulator takes u_l directly.
 *   Eq. 3: persist when Delta_l >= K(t) (here tau * tau_mult[l]; the
 *          caller passes tau already scaled by the learning rate, §3.2).
 *   §3.3 : persist when the layer's staleness t - t_l has reached
 *          S_max (max_staleness), even below the threshold.
 *   Non-finite accumulated drift also persists (conservative counting).
 *   Eq. 4: Delta_l <- 0 on persistence, and t_l <- t. */
int32_t lco_select_step(int32_t nlayers, const double* u, double* delta,
                        int64_t* t_last, const double* tau_mult, double tau,
                        int32_t max_staleness, int64_t t, int32_t mode,
                        uint8_t* mask_out, int32_t* nonfinite_out)
{
    if (nlayers < 0 || max_staleness < 0 || !isfinite(tau) ||
        (mode != LCO_SNAPSHOT && mode != LCO_ACCUMULATE))
        return -1;
    int32_t nsel = 0, nonfinite = 0;
    for (int32_t l = 0; l < nlayers; ++l) {
        double acc = (mode == LCO_ACCUMULATE) ? delta[l] + u[l] : u[l];
        double threshold = tau * (tau_mult ? tau_mult[l] : 1.0);
        int64_t staleness = t - t_last[l];
        int persist = 0;
        if (!isfinite(acc)) {
            persist = 1;
            nonfinite += 1;
        } else if (acc >= threshold) {
            persist = 1;
        }
        if (staleness >= (int64_t)max_staleness)
            persist = 1;
        if (persist) {
            delta[l] = 0.0;
            t_last[l] = t;
            nsel += 1;
        } else {
            delta[l] = acc;
        }
        mask_out[l] = (uint8_t)persist;
    }
    if (nonfinite_out)
        *nonfinite_out = nonfinite;
    return nsel;
}

/* §3.3: per-layer staleness t - t_l, its maximum, and the size-weighted
 * average in which larger layers count proportionally more. */
void lco_staleness(int32_t nlayers, const int64_t* t_last,
                   const int64_t* layer_numel, int64_t t,
                   int64_t* max_out, double* weighted_out)
{
    int64_t mx = 0;
    double num = 0.0, den = 0.0;
    for (int32_t l = 0; l < nlayers; ++l) {
        int64_t s = t - t_last[l];
        if (s > mx)
            mx = s;
        num += (double)layer_numel[l] * (double)s;
        den += (double)layer_numel[l];
    }
    *max_out = mx;
    *weighted_out = den > 0.0 ? num / den : 0.0;
}

static uint64_t round_up(uint64_t x, uint32_t align)
{
    return (x + align - 1) / align * align;
}

/* Byte sizes of the three sections of tensor k. */
static void section_sizes(const lco_tensor* t, uint64_t sz[3])
{
    uint64_t n = (uint64_t)t->numel;
    sz[0] = n * elem_size(t->dtype);
    sz[1] = t->m ? n * 4u : 0u;
    sz[2] = t->v ? n * 4u : 0u;
}

/* Size of a packed layer block: the full layer state of §3.1 (weights
 * plus their optimizer tensors), each section padded to `align`. */
uint64_t lco_layer_block_bytes(const lco_tensor* t, int32_t ntensors, uint32_t align)
{
    uint64_t total = 0;
    for (int32_t k = 0; k < ntensors; ++k) {
        uint64_t sz[3];
        section_sizes(&t[k], sz);
        total += round_up(sz[0], align) + round_up(sz[1], align) + round_up(sz[2], align);
    }
    return total;
}

uint64_t lco_pack_layer(const lco_tensor* t, int32_t ntensors, uint32_t align, uint8_t* dst)
{
    uint64_t off = 0;
    for (int part = 0; part < 3; ++part) {          /* W, then m, then v */
        for (int32_t k = 0; k < ntensors; ++k) {
            uint64_t sz[3];
            section_sizes(&t[k], sz);
            const void* src = part == 0 ? t[k].w : part == 1 ? (const void*)t[k].m
                                                             : (const void*)t[k].v;
            if (sz[part] > 0)
                memcpy(dst + off, src, sz[part]);
            uint64_t padded = round_up(sz[part], align);
            memset(dst + off + sz[part], 0, padded - sz[part]);
            off += padded;
        }
    }
    return off;
}

int32_t lco_unpack_layer(const uint8_t* src, uint64_t nbytes, lco_tensor* t,
                         int32_t ntensors, uint32_t align)
{
    if (nbytes != lco_layer_block_bytes(t, ntensors, align))
        return -1;
    uint64_t off = 0;
    for (int part = 0; part < 3; ++part) {
        for (int32_t k = 0; k < ntensors; ++k) {
            uint64_t sz[3];
            section_sizes(&t[k], sz);
            void* dst = part == 0 ? t[k].w : part == 1 ? (void*)t[k].m : (void*)t[k].v;
            if (sz[part] > 0)
                memcpy(dst, src + off, sz[part]);
            uint64_t padded = round_up(sz[part], align);
            for (uint64_t b = sz[part]; b < padded; ++b)
                if (src[off + b] != 0)
                    return -1;
            off += padded;
        }
    }
    return 0;
}

/* §3.5 (composite recovery) and Eq. 8: layer l is restored from its most
 * recent successfully persisted version t_l <= t_fail. */
void lco_composite_pick(int32_t nversions, const int32_t* v_layer,
                        const int64_t* v_step, const uint8_t* v_durable,
                        int32_t nlayers, int64_t t_fail, int64_t* pick_out)
{
    for (int32_t l = 0; l < nlayers; ++l)
        pick_out[l] = -1;
    for (int32_t i = 0; i < nversions; ++i) {
        int32_t l = v_layer[i];
        if (l < 0 || l >= nlayers || !v_durable[i] || v_step[i] > t_fail)
            continue;
        if (pick_out[l] < 0 || v_step[i] >= v_step[pick_out[l]])
            pick_out[l] = i;
    }
}

/* ------------------------------------------------------------------------
 * AdamW with the drift read off the update (§3.4.2).
 *
 * AdamW (Adam with decoupled weight decay) per element, with step count t:
 *   p  <- p * (1 - lr*wd)                       decoupled weight decay
 *   m  <- beta1*m + (1-beta1)*g                 first moment
 *   v  <- beta2*v + (1-beta2)*g*g               second moment
 *   p  <- p - lr * (m/(1-beta1^t)) / (sqrt(v/(1-beta2^t)) + eps)
 * in binary32, the precision of the optimizer state, with the two bias
 * corrections folded into constants: v_hat = v * (1/(1-beta2^t)) and
 * step = (m * (lr/(1-beta1^t))) / (sqrt(v_hat) + eps); one rounding per
 * operation in exactly this order.
 * ---------------------------------------------------------------------- */
void lco_adamw_constants(const lco_adamw* hp, int64_t t, float out[9])
{
    out[0] = (float)(1.0 - hp->lr * hp->weight_decay);
    out[1] = (float)hp->beta1;
    out[2] = (float)(1.0 - hp->beta1);
    out[3] = (float)hp->beta2;
    out[4] = (float)(1.0 - hp->beta2);
    out[5] = (float)(hp->lr / (1.0 - pow(hp->beta1, (double)t)));
    out[6] = (float)(1.0 / (1.0 - pow(hp->beta2, (double)t)));
    out[7] = (float)hp->eps;
    out[8] = 0.0f;
}

uint16_t lco_bf16_round(float f)
{
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    if ((u & 0x7f800000u) == 0x7f800000u && (u & 0x007fffffu))
        return (uint16_t)((u >> 16) | 0x0040u);          /* quiet NaN */
    /* nearest, ties to the even bf16: add half an ulp minus one, plus the
     * parity of the bit that stays */
    uint32_t keep_lsb = (u >> 16) & 1u;
    return (uint16_t)((u + 0x7fffu + keep_lsb) >> 16);
}

void lco_adamw_step(const lco_adamw* hp, int64_t t, int64_t n, float* p, float* m, float* v,
                    const void* grad, int32_t grad_bf16, uint16_t* model,
                    double* d_out, double* a_out)
{
    float c[9];
    lco_adamw_constants(hp, t, c);
    const float decay = c[0], b1 = c[1], omb1 = c[2], b2 = c[3], omb2 = c[4];
    const float step_size = c[5], rbc2 = c[6], eps = c[7];
    double d_sum = 0.0, a_sum = 0.0;
    for (int64_t i = 0; i < n; ++i) {
        float g;
        if (grad_bf16) {
            uint16_t bits;
            memcpy(&bits, (const uint8_t*)grad + 2 * i, sizeof bits);
            g = (float)lco_bf16_value(bits);
        } else {
            memcpy(&g, (const uint8_t*)grad + 4 * i, sizeof g);
        }
        const float p_old = p[i];
        const float p_decayed = p_old * decay;
        const float m1a = b1 * m[i];
        const float m1b = omb1 * g;
        const float m_new = m1a + m1b;
        const float gg = g * g;
        const float v1a = b2 * v[i];
        const float v1b = omb2 * gg;
        const float v_new = v1a + v1b;
        const float v_hat = v_new * rbc2;
        const float root = sqrtf(v_hat);
        const float denom = root + eps;
        const float m_scaled = m_new * step_size;
        const float step = m_scaled / denom;
        const float p_new = p_decayed - step;
        p[i] = p_new;
        m[i] = m_new;
        v[i] = v_new;
        if (model)
            model[i] = lco_bf16_round(p_new);
        /* Eq. 1 terms: W(t) - W(t-1) and W(t-1), exact in binary64 */
        d_sum += fabs((double)p_new - (double)p_old);
        a_sum += fabs((double)p_old);
    }
    *d_out = d_sum;
    *a_out = a_sum;
}
