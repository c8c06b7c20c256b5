/*
 * tq.h — C ABI of the grouped ternary (W1.58A16) linear layer on GB300 (sm_103a).
 *
 * The layer is the TernaryLinear of "Ternary Mamba: Grouped Quantization-Aware
 * Training of W1.58A16 State Space Models", §3.1: latent fp32 weights W [N, K]
 * (N = out_features, K = in_features) are split into groups of g consecutive
 * elements along K inside one row; each group gets the non-learned scale
 * s = mean |w| (recomputed at every call), codes round(clip(w / s, -1, 1)) in
 * {-1, 0, +1}, and the dequantised weight s * code. The forward product uses
 * 16-bit (bf16) activations; the backward is the straight-through estimator.
 *
 * Conventions for every entry point
 *   - Every pointer is DEVICE memory owned by the caller, contiguous row-major,
 *     16-byte aligned. The library keeps no pointer after a call returns.
 *   - Work is enqueued on `stream` (a cudaStream_t passed as void*; NULL is the
 *     legacy default stream). No entry point synchronises, except
 *     tq_device_status(). No entry point allocates device memory. The library
 *     holds fixed file-scope device arrays instead, present on every device
 *     that loads it until the process exits: 40 MB of dW stream-K workspace
 *     (tq_linear_bwd), 16 MB of transposed-code scratch (tq_linear_bwd_noalloc),
 *     and a few KB of work counters and status words.
 *   - Arguments are checked before anything is enqueued. A rejected call
 *     returns TQ_ERR_INVALID_ARG or TQ_ERR_UNSUPPORTED, writes nothing and
 *     leaves a message in tq_last_error().
 *   - A failed launch returns TQ_ERR_CUDA. Kernels bound every wait they
 *     make; a wait that runs out records TQ_ERR_TIMEOUT in a per-device status
 *     word that tq_device_status() returns (and clears). Outputs of such a
 *     call are undefined.
 *   - Sizes of zero are allowed and do nothing (except that dW is zeroed by
 *     tq_linear_bwd when M = 0 and accumulate_dw = 0).
 *   - Group sizes: g in {32, 64, 128, 256, 512}.
 *
 * Packed code layout (2 bits per weight; the paper asks only for "packed
 * 2-bit weight storage", §8 — this particular layout is this library's)
 *   codes is uint32 [N][K/16]; word w of row n holds k in [16w, 16w + 16).
 *   Code i = k % 16 sits at bit 2*(i/2) when i is even and at bit
 *   16 + 2*(i/2) when i is odd (even codes fill the low half-word, odd codes
 *   the high half-word, pair j = (2j, 2j+1) at bits 2j and 16+2j).
 *   Values: 0b00 -> 0, 0b01 -> +1, 0b11 -> -1; 0b10 is never written.
 *   With this layout a shift and a mask turn one pair into a bf16x2 holding
 *   (2*c_2j, 2*c_2j+1), because the 2-bit value v times 0x4000 is the bf16 bit
 *   pattern of 0, +2.0 or -2.0.
 *
 * Scales are fp32 [N][K/g]; zero counts are int32 [N][K/g].
 */
#ifndef TQ_H_
#define TQ_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#if defined(__GNUC__)
#define TQ_API __attribute__((visibility("default")))
#else
#define TQ_API
#endif

typedef enum {
  TQ_OK = 0,
  TQ_ERR_INVALID_ARG = 1, /* null/misaligned pointer, bad size or group size   */
  TQ_ERR_UNSUPPORTED = 2, /* valid request outside what the kernels handle      */
  TQ_ERR_CUDA = 3,        /* CUDA runtime or launch error                       */
  TQ_ERR_TIMEOUT = 4      /* a device-side wait ran out (tq_device_status only) */
} tq_status;

typedef enum {
  TQ_OUT_F32 = 0,  /* fp32 output (default: keeps the max-element error small) */
  TQ_OUT_BF16 = 1, /* bf16 output, round to nearest even                        */
  /* Flag OR-ed into an output type (y_dtype, dx_dtype, tq_fwd_desc.y_dtype): the
   * activations x and dy are fp16 instead of bf16 (the paper's A16 is FP16, §3.3).
   * The codes expand to the same +-1 values; the group scale is rounded to fp16
   * instead of bf16 where the kernels apply it to the expanded codes. */
  TQ_IN_F16 = 0x100
} tq_out_dtype;

/*
 * tq_quantize — §3.1 quantiser: per-group absmean scale, ternary codes, packing.
 *   w            fp32 [n][k], latent weights (read only).
 *   n, k         n >= 0; k >= 0, k % 16 == 0 and k % g == 0.
 *   g            group size along k.
 *   codes        out: uint32 [n][k/16], layout above.
 *   scales       out: fp32 [n][k/g], s = (1/g) * sum |w| over the group.
 *   zero_counts  out: int32 [n][k/g], number of zero codes in the group
 *                (the zero-ratio monitor of §4).
 * The code of w is +-1 when |w / s| > 0.5 with the division in fp32 (round
 * half to even sends 0.5 to 0), 0 otherwise; a group with s = 0 is all zeros.
 * Inputs must be finite.
 */
TQ_API tq_status tq_quantize(const float* w, int64_t n, int64_t k, int32_t g,
                      uint32_t* codes, float* scales, int32_t* zero_counts,
                      void* stream);

/*
 * tq_quantize_with_transpose — tq_quantize, and in the same launch the transposed
 * codes that tq_codes_transpose would make of its codes (the operand of the STE dX
 * product on codes_t, §3.1), bit for bit the same as the two calls in a row.
 *   w, n, k, g, codes, scales, zero_counts   as tq_quantize.
 *   codes_t      out: uint32 [k][4 * ceil(n / 64)], layout of tq_codes_transpose;
 *                must not overlap codes.
 * One cooperative launch: once every CTA has written its codes (a grid barrier
 * with the library's wait limit), the grid transposes them. A wait that runs out
 * is reported by tq_device_status (TQ_ERR_TIMEOUT; codes_t is then incomplete).
 * Returns TQ_ERR_CUDA if the device cannot hold the cooperative grid.
 */
TQ_API tq_status tq_quantize_with_transpose(const float* w, int64_t n, int64_t k, int32_t g,
                                            uint32_t* codes, float* scales, int32_t* zero_counts,
                                            uint32_t* codes_t, void* stream);

/* Largest entry count of the batched calls. */
#define TQ_MAX_BATCH 256

/* One matrix of a batched quantize call (tq_quantize_batched). */
typedef struct {
  const float* w;         /* fp32 [n][k] latent weights          */
  uint32_t* codes;        /* out: uint32 [n][k/16]               */
  float* scales;          /* out: fp32 [n][k/g]                  */
  int32_t* zero_counts;   /* out: int32 [n][k/g]                 */
  int64_t n;              /* rows                                */
  int64_t k;              /* columns, k % 16 == 0 and k % g == 0 */
} tq_quant_desc;

/*
 * tq_quantize_batched — tq_quantize of many matrices with the same group size
 * in one launch (e.g. the per-step requantize of every in_proj and out_proj of a
 * 48-block model, §3.1: the scale is recomputed at every forward). Each entry
 * gets exactly tq_quantize's result. descs is a HOST array (copied into the
 * launch; not kept); count <= TQ_MAX_BATCH; the outputs of different entries
 * must not overlap.
 */
TQ_API tq_status tq_quantize_batched(const tq_quant_desc* descs, int32_t count, int32_t g,
                                     void* stream);

/*
 * tq_quantize_decoupled — the decoupled quantizer of the paper's decoupled-
 * quantization ablation (appendix): the codes are decided against a threshold
 *   tau_g = row_factor[n] * s_g   (one fp32 product; s_g the absmean of §3.1)
 * instead of s_g itself, so that sparsity (tau) and output magnitude (a separate
 * learnable alpha_g the caller keeps and passes as the scales of tq_linear_fwd /
 * tq_linear_bwd) are decoupled; the asymmetric-gate variant uses 0.8 on the gate
 * rows 0..4095 of in_proj and 1 elsewhere.
 *   row_factor   fp32 [n] on the device, or NULL (every factor 1: tq_quantize).
 *   scales       out: the absmean s_g (not tau), e.g. to initialise alpha.
 *   Other arguments, layouts and errors as tq_quantize.
 */
TQ_API tq_status tq_quantize_decoupled(const float* w, int64_t n, int64_t k, int32_t g,
                                       const float* row_factor, uint32_t* codes, float* scales,
                                       int32_t* zero_counts, void* stream);

/*
 * tq_alpha_grad — gradient of the decoupled quantizer's magnitude: with
 * W^ = alpha_g * c, dalpha[n][j] = sum over group j of row n of dW^ * c, where dW^
 * is the dW of tq_linear_bwd (the STE hands the same matrix to the latent W).
 *   dw       fp32 [n][k] (device, 16-byte aligned).
 *   codes    uint32 [n][k/16], layout of tq_quantize (device, 16-byte aligned).
 *   dalpha   out: fp32 [n][k/g] (device).
 *   Summation: each 16-weight word in weight order, then the group's words as a
 *   binary tree; fp32. Requires k % g == 0 (and so k % 16 == 0); TQ_ERR_INVALID_ARG
 *   otherwise.
 */
TQ_API tq_status tq_alpha_grad(const float* dw, const uint32_t* codes, int64_t n, int64_t k,
                               int32_t g, float* dalpha, void* stream);

/*
 * tq_quantize_with_scales — the quantizer of the learnable-scale variant (§4,
 * "Zero-Ratio Collapse": s_g trained as a parameter instead of recomputed as the
 * absmean): the codes are decided against the caller's scales,
 *   c = round(clip(w / s_g, -1, 1))   (the fp32 quotient, rounding half to even),
 * for a scale of either sign (for s_g < 0 the codes flip with it, so s_g * c still
 * approximates w; s_g = 0 gives the sign of w, and 0 for w = 0).
 *   scales   fp32 [n][k/g]: the current s_g (device, 16-byte aligned); read only.
 *   codes, zero_counts   out: as tq_quantize.
 *   Other arguments, layouts and errors as tq_quantize; the forward and backward
 *   products take these scales as they take the absmean.
 */
TQ_API tq_status tq_quantize_with_scales(const float* w, int64_t n, int64_t k, int32_t g,
                                         const float* scales, uint32_t* codes,
                                         int32_t* zero_counts, void* stream);

/*
 * tq_scale_grad — gradient of the learnable scale. The paper does not give it;
 * this library takes the chain rule through W^ = s * round(clip(w / s)) with the
 * rounding passed straight through (the rule §3.1 applies to the latent weights):
 *   dW^/ds = c - q [|q| < 1],  q = w / s, so
 *   dscales[n][j] = sum_i dW^_i c_i - (1/s) sum_{i : |w_i| < |s|} dW^_i w_i
 * over group j of row n, where dW^ is the dW of tq_linear_bwd. The test |w| < |s|
 * compares the fp32 inputs exactly; for s = 0 the second sum is empty.
 *   w        fp32 [n][k], the latent weights the codes came from (device, 16-byte aligned).
 *   dw       fp32 [n][k] (device, 16-byte aligned).
 *   codes    uint32 [n][k/16] of tq_quantize_with_scales for (w, scales).
 *   scales   fp32 [n][k/g] (device, 4-byte aligned).
 *   dscales  out: fp32 [n][k/g] (device, 4-byte aligned).
 *   Summation: each 16-weight word in weight order, then the group's words as a
 *   binary tree, both sums in fp32, then one fp32 division. Requires k % g == 0;
 *   TQ_ERR_INVALID_ARG otherwise.
 */
TQ_API tq_status tq_scale_grad(const float* w, const float* dw, const uint32_t* codes,
                               const float* scales, int64_t n, int64_t k, int32_t g,
                               float* dscales, void* stream);

/* Hyperparameters of one AdamW step (tq_adamw_requantize). */
typedef struct tq_adamw_hparams {
  double lr;            /* learning rate of this step (after any schedule), >= 0       */
  double beta1, beta2;  /* in [0, 1); the paper uses (0.9, 0.95)                       */
  double eps;           /* > 0; the paper gives none, the usual default is 1e-8         */
  double weight_decay;  /* decoupled, >= 0; the paper uses 0.01                        */
  double grad_scale;    /* multiplies the gradient, >= 0 (global-norm clip factor; 1)  */
  int64_t step;         /* t >= 1: this update is the t-th of the moments              */
} tq_adamw_hparams;

/*
 * tq_adamw_requantize — the optimizer step of §3.3 (AdamW on the fp32 latent
 * weights, the training-hyperparameter table of the appendix) fused with the
 * requantization of §3.1 (per-group absmean scale, ternary codes), in one pass:
 *   g' = grad_scale * grad
 *   m  = beta1 m + (1 - beta1) g'          v = beta2 v + (1 - beta2) g'^2
 *   w  = w (1 - lr wd) - lr / (1 - beta1^t) * m / (sqrt(v) / sqrt(1 - beta2^t) + eps)
 *   then codes / scales / zero_counts of the new w exactly as tq_quantize.
 * Each operation is one fp32 operation in the order written (no fused
 * multiply-add); the step constants are computed in fp64 and rounded once to
 * fp32, so results are reproducible bit for bit.
 *   w, m, v      in/out: fp32 [n][k], updated in place (device, 16-byte aligned).
 *   grad         fp32 [n][k] (device).
 *   codes, scales, zero_counts   out: as tq_quantize, for the updated w.
 *   Requires the tq_quantize conditions on n, k, g; hp non-NULL with the ranges
 *   above; TQ_ERR_INVALID_ARG otherwise, before anything is launched.
 */
TQ_API tq_status tq_adamw_requantize(float* w, const float* grad, float* m, float* v, int64_t n,
                                     int64_t k, int32_t g, const tq_adamw_hparams* hp,
                                     uint32_t* codes, float* scales, int32_t* zero_counts,
                                     void* stream);

/*
 * tq_adamw_requantize_with_scales — tq_adamw_requantize for the learnable-scale
 * variant: the same AdamW update of w, m and v, then the codes and zero counts of
 * the new w against the caller's scales exactly as tq_quantize_with_scales (pass
 * the scales already updated for this step, e.g. by tq_adamw).
 *   scales   fp32 [n][k/g] (device, 16-byte aligned); read only.
 *   Other arguments, layouts and errors as tq_adamw_requantize.
 */
TQ_API tq_status tq_adamw_requantize_with_scales(float* w, const float* grad, float* m, float* v,
                                                 int64_t n, int64_t k, int32_t g,
                                                 const tq_adamw_hparams* hp, const float* scales,
                                                 uint32_t* codes, int32_t* zero_counts,
                                                 void* stream);

/*
 * tq_adamw — the AdamW update of tq_adamw_requantize (same operations, same
 * rounding) over a flat fp32 array without requantization, e.g. the scales of the
 * learnable-scale variant.
 *   p, m, v   in/out: fp32 [count] (device, 16-byte aligned).
 *   grad      fp32 [count] (device, 16-byte aligned).
 *   Requires count % 16 == 0 and hp as for tq_adamw_requantize;
 *   TQ_ERR_INVALID_ARG otherwise, before anything is launched.
 */
TQ_API tq_status tq_adamw(float* p, const float* grad, float* m, float* v, int64_t count,
                          const tq_adamw_hparams* hp, void* stream);

/*
 * tq_linear_fwd — W1.58A16 forward (§3.1, "W1.58A16" of the title):
 *   y[m][n] = sum_k x[m][k] * s[n][k/g] * code[n][k].
 *   x            bf16 [m][k] activations.
 *   codes/scales as produced by tq_quantize for W [n][k].
 *   y            out: [m][n], fp32 (TQ_OUT_F32) or bf16 (TQ_OUT_BF16); y_dtype may
 *                carry TQ_IN_F16 (x is fp16).
 *   Requires k % 64 == 0 and k % g == 0; n >= 1 when m >= 1.
 *   m <= 16 runs the decode kernel, larger m the tensor-core GEMM; both expand
 *   the codes on chip and accumulate in fp32 (the decode kernel folds the fp32
 *   scale into each group's sum for g >= 128, the others multiply the expanded
 *   codes by bf16(s)). The decode kernel takes k <= 2^30 and n < 2^31
 *   (TQ_ERR_UNSUPPORTED beyond). When a decode launch has fewer blocks of 256
 *   rows than the device has SMs, it cuts k into 2, 4 or 8 pieces, each block's
 *   pieces run by one thread-block cluster whose first CTA adds the others'
 *   partial sums to its own in piece order: the same result on every run (its
 *   rounding differs from that of an uncut launch by the order of the sums).
 *   Decode launches use programmatic dependent launch: one may start its CTAs
 *   while the previous kernel on the stream is still running, but before that
 *   kernel has completed it only prefetches codes and scales into L2 (coherent
 *   with any write still to come); every other read and every write waits.
 */
TQ_API tq_status tq_linear_fwd(const void* x, int64_t m, int64_t k,
                        const uint32_t* codes, const float* scales, int64_t n, int32_t g,
                        void* y, int32_t y_dtype, void* stream);

/*
 * tq_linear_bwd — straight-through-estimator backward (§3.1; STE = identity
 * through round and clip, no gradient to the non-learned scale):
 *   dx[m][k] = sum_n dy[m][n] * s[n][k/g] * code[n][k]      (through W^)
 *   dw[n][k] = sum_m dy[m][n] * x[m][k]                     (to latent W)
 *   dy           bf16 [m][n]; x bf16 [m][k] (the forward's input).
 *   dx           out: [m][k], fp32 or bf16 (dx_dtype); NULL skips dX.
 *   dw           out: fp32 [n][k]; NULL skips dW. accumulate_dw != 0 adds to
 *                dw instead of overwriting it.
 *   codes_t      optional: tq_codes_transpose's output for the same codes. With it
 *                dX expands the codes of W^T like the forward expands W's (faster);
 *                NULL makes dX read `codes` directly.
 *   Requires k % 64 == 0, k % g == 0, n % 8 == 0. x may be NULL when dw is.
 *   dW launches of one device share the library's 40 MB workspace (the partial
 *   sums of the tiles split across SMs): each dW launch waits for the device's
 *   previous dW launch, on whatever stream either was issued (an event the
 *   library records after every dW launch, waited on by the next one). A call
 *   made while `stream` is being captured into a CUDA graph takes no part in
 *   that: the graph's own dependencies order its dW nodes, so a graph must not
 *   leave two dW nodes unordered, nor be replayed beside a dW launch on another
 *   stream.
 */
TQ_API tq_status tq_linear_bwd(const void* dy, const void* x, int64_t m, int64_t n, int64_t k,
                        const uint32_t* codes, const uint32_t* codes_t, const float* scales,
                        int32_t g, void* dx, int32_t dx_dtype, float* dw,
                        int32_t accumulate_dw, void* stream);

/*
 * tq_linear_bwd_noalloc — tq_linear_bwd on the faster transposed-codes dX path
 * without a caller-provided codes_t: the codes are transposed (tq_codes_transpose)
 * into a 16 MB scratch array inside the library (a file-scope device array; no
 * allocation at any time), then the product runs as tq_linear_bwd with it. Same
 * arguments and results as tq_linear_bwd with codes_t = NULL.
 *   Returns TQ_ERR_UNSUPPORTED when the transposed codes (k * 4 * ceil(n/64)
 *   words) exceed the scratch; pass codes_t to tq_linear_bwd then.
 *   The scratch is one per device: calls on one device must not overlap in time
 *   (issue them on one stream).
 */
TQ_API tq_status tq_linear_bwd_noalloc(const void* dy, const void* x, int64_t m, int64_t n,
                                       int64_t k, const uint32_t* codes, const float* scales,
                                       int32_t g, void* dx, int32_t dx_dtype, float* dw,
                                       int32_t accumulate_dw, void* stream);

/*
 * tq_codes_transpose — the packed codes of W^T, a re-layout of tq_quantize's codes
 * (no arithmetic of the method) that the STE dX product streams along its
 * reduction (n):
 *   codes        uint32 [n][k/16], layout above.
 *   codes_t      out: uint32 [k][ldt] with ldt = 4 * ceil(n / 64) words per row;
 *                word w of row k holds the codes of (n', k) for n' in
 *                [16w, 16w + 16) at the bit of i = n' % 16 (same rule as codes);
 *                codes past n are 0.
 *   Requires k % 16 == 0.
 */
TQ_API tq_status tq_codes_transpose(const uint32_t* codes, int64_t n, int64_t k,
                                    uint32_t* codes_t, void* stream);

/* One matrix of a batched decode call (tq_linear_fwd_batched). */
typedef struct {
  const void* x;          /* bf16 [m][k]                         */
  const uint32_t* codes;  /* uint32 [n][k/16]                    */
  const float* scales;    /* fp32 [n][k/g]                       */
  void* y;                /* [m][n], dtype y_dtype               */
  int64_t n;              /* out_features                        */
  int64_t k;              /* in_features, k % 64 == 0            */
  int32_t g;              /* group size                          */
  int32_t y_dtype;        /* tq_out_dtype                        */
} tq_fwd_desc;

/*
 * tq_linear_fwd_batched — the decode forward of many matrices in one launch
 * (e.g. every in_proj and out_proj of a 48-block model for one token step):
 * for each i < count, y_i = x_i W^_i^T exactly as tq_linear_fwd, all with the
 * same token count m (1 <= m <= 16). descs is a HOST array (copied into the
 * launch; not kept); count <= TQ_MAX_BATCH.
 */
TQ_API tq_status tq_linear_fwd_batched(const tq_fwd_desc* descs, int32_t count, int64_t m,
                                void* stream);

/*
 * tq_device_status — synchronises `stream`, then returns and clears the status
 * word of the current device: TQ_OK, or TQ_ERR_TIMEOUT if a kernel's bounded
 * wait ran out since the last call; TQ_ERR_CUDA if the synchronise failed.
 * On TQ_ERR_TIMEOUT it first synchronises the whole device (every stream), then
 * clears the word and zeroes the dW kernel's stream-K tile counters, which a
 * launch that gave up may have left set; later calls then run normally.
 */
TQ_API tq_status tq_device_status(void* stream);

/*
 * tq_test_hooks — for testing the timeout path only; the paper has no counterpart.
 * Sets, for every later launch on the current device, the time limit of every
 * kernel wait (wait_limit_ns > 0; 0 restores the default of 2 s) and test flags
 * that make one kernel role withhold its first arrival on a barrier (0 in normal
 * use):
 *   1  tq_quantize / tq_quantize_batched: consumer warp 0 of CTA 0 does not
 *      release its first stage, so the producer's wait for that slot runs out;
 *   2  the dW product of tq_linear_bwd: the first epilogue warp of the first CTA
 *      pair's leader does not release its first accumulator, so the MMA issuer's
 *      wait for it runs out;
 *   4  a decode launch cut into pieces of k (tq_linear_fwd, m <= 16, fewer blocks
 *      of 256 rows than SMs): CTA 1 sends none of its partial sums, so the first
 *      CTA of its cluster waits for them in vain, and CTA 1 then for its release.
 * A launch made while a flag is set winds down at the limit (no copy or MMA left
 * in flight, every wait bounded) and reports TQ_ERR_TIMEOUT through
 * tq_device_status(); its outputs are undefined. Synchronises the device first.
 * Returns TQ_ERR_INVALID_ARG for a negative limit or an unknown flag.
 */
TQ_API tq_status tq_test_hooks(int64_t wait_limit_ns, uint32_t flags);

/* Message of the last failure on the calling thread ("" if none). */
TQ_API const char* tq_last_error(void);

/* Library version string. */
TQ_API const char* tq_version(void);

#ifdef __cplusplus
}
#endif

#endif /* TQ_H_ */
