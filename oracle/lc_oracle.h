/*
 * lc_oracle.h -- declarations of the LayerCheck reference oracle.
 *
 * TEST INFRASTRUCTURE ONLY.  This is a plain, slow, single-threaded CPU
 * restatement of the method of "LayerCheck: Adaptive Layer-wise
 * Checkpointing for Large Language Model Post-training" (§3.2-§3.6).  It
 * exists so that the CUDA path can be checked against something written
 * straight from the paper.  Only tests, the smoke check and the CPU
 * baseline of the benchmark may load it; the product library never does,
 * and the two share no source, header, table or helper.
 *
 * Floating-point arithmetic is IEEE binary64, summed in the plain order the
 * definitions state (tensor registration order, then element index order),
 * except the AdamW step, which runs in binary32, the precision of the
 * optimizer state it updates.  Build with -ffp-contract=off so no
 * multiply-add is fused.
 */
#ifndef LC_ORACLE_H
#define LC_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum { LCO_BF16 = 0, LCO_F32 = 1 };
enum { LCO_SNAPSHOT = 0, LCO_ACCUMULATE = 1 };

/* One parameter tensor of a layer.  w/r hold `numel` elements of `dtype`;
 * m/v hold `numel` fp32 Adam moments or are NULL (no optimizer state).
 * Pointers are const for every function except lco_unpack_layer, which
 * writes w, m and v. */
typedef struct {
    void*   w;       /* current weights W_l(t)                                */
    void*   r;       /* reference weights W_l(t-1) / last persisted snapshot  */
    float*  m;       /* exp_avg    (may be NULL)                              */
    float*  v;       /* exp_avg_sq (may be NULL)                              */
    int64_t numel;
    int32_t dtype;   /* LCO_BF16 or LCO_F32                                   */
    int32_t reserved;
} lco_tensor;

/* Exact value of a bf16 bit pattern (bf16 is the upper half of binary32). */
double lco_bf16_value(uint16_t bits);

/* Eq. 1 (§3.2), the two means: out[0] = sum_i |W_i - R_i|, out[1] =
 * sum_i |R_i|, out[2] = element count, over all tensors of one layer taken
 * as one concatenated element list. */
void lco_layer_sums(const lco_tensor* t, int32_t ntensors, double out[3]);

/* Eq. 1 (§3.2): u = mean|W - R| / (mean|R| + eps_w), from the sums above. */
double lco_update_measure(double d_sum, double a_sum, double n, double eps_w);

/* One checkpoint opportunity (§3.2 Eq. 2-4, §3.3 staleness guard).
 * Updates delta[] and t_last[] in place and writes mask_out[] (1 =
 * persist).  tau_mult may be NULL (all 1).  Returns the number of selected
 * layers, or -1 on a bad argument.  *nonfinite_out (nullable) receives the
 * number of layers whose accumulated drift was not finite. */
int32_t lco_select_step(int32_t nlayers, const double* u, double* delta,
                        int64_t* t_last, const double* tau_mult, double tau,
                        int32_t max_staleness, int64_t t, int32_t mode,
                        uint8_t* mask_out, int32_t* nonfinite_out);

/* §3.3 staleness after a step: max_l (t - t_l) and the parameter-size
 * weighted mean sum_l n_l (t - t_l) / sum_l n_l. */
void lco_staleness(int32_t nlayers, const int64_t* t_last,
                   const int64_t* layer_numel, int64_t t,
                   int64_t* max_out, double* weighted_out);

/* Packed layer block (the full layer state of §3.1: weights plus Adam
 * moments).  Layout: every tensor's W bytes, then every tensor's m bytes,
 * then every tensor's v bytes, in registration order; each section is
 * zero-padded up to a multiple of `align` bytes (a power of two). */
uint64_t lco_layer_block_bytes(const lco_tensor* t, int32_t ntensors, uint32_t align);
uint64_t lco_pack_layer(const lco_tensor* t, int32_t ntensors, uint32_t align, uint8_t* dst);

/* Inverse of lco_pack_layer: writes w, m, v of each tensor from a block.
 * Returns 0, or -1 if nbytes does not match the block size or a padding
 * byte is non-zero. */
int32_t lco_unpack_layer(const uint8_t* src, uint64_t nbytes, lco_tensor* t,
                         int32_t ntensors, uint32_t align);

/* §3.5 and Eq. 8: for each layer, the index of the durable version with
 * the largest step <= t_fail (the later-recorded one on a tie), or -1 when
 * the layer has none. */
void lco_composite_pick(int32_t nversions, const int32_t* v_layer,
                        const int64_t* v_step, const uint8_t* v_durable,
                        int32_t nlayers, int64_t t_fail, int64_t* pick_out);

/* AdamW hyperparameters of one optimizer step (binary64, as given by the
 * training script). */
typedef struct {
    double lr, beta1, beta2, eps, weight_decay;
} lco_adamw;

/* fp32 constants of one AdamW step at step count t >= 1: out[0] = 1 - lr*wd,
 * out[1] = beta1, out[2] = 1 - beta1, out[3] = beta2, out[4] = 1 - beta2,
 * out[5] = lr / (1 - beta1^t), out[6] = 1 / (1 - beta2^t), out[7] = eps,
 * out[8] = 0; each formed in binary64 and rounded once to binary32. */
void lco_adamw_constants(const lco_adamw* hp, int64_t t, float out[9]);

/* One AdamW step (decoupled weight decay) on n fp32 parameters in place,
 * with the drift sums of Eq. 1 taken on the same pass (§3.4.2: the drift is
 * read off the optimizer update): d_out = sum |p_new - p_old|, a_out =
 * sum |p_old| (binary64 sums of the binary32 values).  grad is bf16 bits
 * (grad_bf16 = 1) or fp32.  model (nullable) receives bf16(p_new) rounded
 * to nearest even.  Every fp32 operation rounds once, in the order written
 * in lc_oracle.c. */
void lco_adamw_step(const lco_adamw* hp, int64_t t, int64_t n, float* p, float* m, float* v,
                    const void* grad, int32_t grad_bf16, uint16_t* model,
                    double* d_out, double* a_out);

/* Round-to-nearest-even binary32 -> bf16 bits (NaN -> quiet NaN). */
uint16_t lco_bf16_round(float f);

#ifdef __cplusplus
}
#endif
#endif /* LC_ORACLE_H */
