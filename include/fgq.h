/*
 * fgq.h -- C ABI of libfgq, a GB300 (sm_103a) implementation of the data-parallel hot
 * path of Fine-Grained Quantization (FGQ), "Ternary Neural Networks with Fine-Grained
 * Quantization" (arXiv 1705.01462).
 *
 * The hot path: each output filter's weights are split into groups of G consecutive
 * weights along the reduction axis (Section 3.1, Eq. 2; Section 3.2 groups along the
 * input channels), each group is ternarized to codes t in {-1, 0, +1} with one fp32
 * scale alpha (Eq. 5; Eq. 4 reaches the same optimum), activations are quantized to
 * 8 or 4 bit dynamic fixed point (Section 4), and a convolution or fully connected layer
 * computes  y = s_x * sum_g alpha_g * (sum_{j in g} t_j * q_j)  with the inner sums held
 * in 32-bit integer accumulators (Section 4): one multiply per group instead of one per
 * weight (Section 4.1).
 *
 * Conventions for every call
 *   - All array pointers are DEVICE pointers owned by the caller (fgq_conv2d_host: host
 *     pointers).  Calls are asynchronous and ordered on the given CUDA stream.  The only
 *     allocations of the library are per-call temporaries (operands expanded or folded for
 *     the tensor cores) from a library-owned stream-ordered memory pool of the current
 *     device, allocated and freed on the call's stream; fgq_quantize_act_noalloc allocates
 *     nothing.
 *   - The return value reports errors found on the host (argument, alignment, unsupported
 *     shape, CUDA launch failure).  Errors found by a kernel (non-finite input, a bounded
 *     wait that ran out) are recorded in a device error word and returned by
 *     fgq_stream_status().
 *   - Shapes are int; products of shapes are computed in 64 bits.  Empty problems
 *     (M, P, n or B equal to 0) are valid and launch nothing.
 *
 * Data layouts
 *   Kred        reduction length.  Convolution: Kred = R*S*(C/groups), ordered (r, s, c)
 *               with c fastest (torch OIHW weights permuted to OHWI).
 *   Kp          ceil(Kred/G)*G, the row length padded with zero weights.
 *   ng          Kp/G groups per filter.
 *   codes       uint32 [M][ceil(Kp/16)].  Code of t: 0 -> 00, +1 -> 01, -1 -> 11 (10 is
 *               never written); element j of a row sits in word j/16, bits 2(j%16) and
 *               2(j%16)+1.  Unused bits are 0.  (This 2-bit encoding is the library's
 *               choice; the paper only states 2-bit weights, Section 4.)
 *   alpha       fp32 [M][ng].
 *   activations 8-bit types: one byte per element.  4-bit types: element 2i in the low
 *               nibble of byte i, 2i+1 in the high nibble (two's complement for S4).
 *               Convolution inputs are NHWC [B][H][W][C] (C even for 4-bit types); GEMM
 *               inputs are [P][Kred] (Kred even for 4-bit types).
 *   outputs     fp32 NHWC [B][Ho][Wo][M] (convolution), [P][M] (GEMM),
 *               Ho = (H + 2*pad - R)/stride + 1, Wo likewise.
 */
#ifndef FGQ_H_
#define FGQ_H_

#include <stddef.h>
#include <stdint.h>

#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  FGQ_OK = 0,
  FGQ_ERR_ARG = 1,          /* invalid argument: null pointer, negative size, bad G ... */
  FGQ_ERR_ALIGN = 2,        /* a pointer is not 16-byte aligned */
  FGQ_ERR_UNSUPPORTED = 3,  /* valid but unsupported combination (stated per call) */
  FGQ_ERR_NONFINITE = 4,    /* a kernel saw NaN or Inf in its fp32 input */
  FGQ_ERR_TIMEOUT = 5,      /* a kernel's bounded wait ran out; the kernel returned early */
  FGQ_ERR_CUDA = 6          /* a CUDA runtime call or a launch failed */
} fgq_status;

typedef enum { FGQ_U8 = 0, FGQ_S8 = 1, FGQ_U4 = 2, FGQ_S4 = 3 } fgq_act_type;

/* ABI version of this header (incremented on any signature change). */
int fgq_version(void);

/* Human-readable name of a status code (static string). */
const char* fgq_status_string(fgq_status s);

/* Number of uint32 code words per filter row: ceil(ceil(Kred/G)*G / 16); 0 on bad input. */
int64_t fgq_codes_words_per_row(int Kred, int G);

/* Number of groups per filter row, ceil(Kred/G); 0 on bad input. */
int64_t fgq_num_groups(int Kred, int G);

/*
 * FGQ ternarization (Section 3.1, Eq. 2 and Eq. 5, solved exactly per group -- the
 * paper's "brute-force" per-group solve, Section 4).
 *   w      fp32 [M][Kred] row-major, Kred in (r, s, c) order.
 *   G      group size, one of 1, 2, 4, 8, 16, 32, 64, 128.
 *   codes  out, uint32 [M][fgq_codes_words_per_row(Kred, G)], fully written.
 *   alpha  out, fp32 [M][fgq_num_groups(Kred, G)].
 * Per group: the kept set is {j : |w_j| >= tau} for the threshold tau maximising
 * (sum of kept |w|)^2 / (number kept), ties to the larger tau; alpha is the fp32 nearest
 * (ties to even) the exact mean of the kept |w|; t_j = sign(w_j) on the kept set.  An
 * all-zero group gives alpha = 0 and zero codes.  Decisions use exact integer arithmetic,
 * so results are bit-reproducible.  A group holding NaN/Inf gets zero codes and alpha,
 * and FGQ_ERR_NONFINITE is recorded.
 * Errors: FGQ_ERR_ARG (null pointer with M*Kred > 0, negative sizes, bad G),
 * FGQ_ERR_ALIGN (w, codes or alpha not 4-byte aligned), FGQ_ERR_CUDA.
 */
fgq_status fgq_ternarize(const float* w, int M, int Kred, int G, uint32_t* codes, float* alpha,
                         cudaStream_t stream);

/* Largest number of weight sets one fgq_ternarize_batch call takes. */
#define FGQ_TERNARIZE_BATCH_MAX 128

/*
 * fgq_ternarize for n weight sets of one group size G in one launch (the layers of a
 * network): set i is w[i] fp32 [M[i]][Kred[i]] -> codes[i], alpha[i], with the layouts,
 * results (bit for bit) and non-finite handling of fgq_ternarize.  w, M, Kred, codes,
 * alpha are HOST arrays of n entries holding device pointers and sizes (read during the
 * call, not kept); sets with M[i] * Kred[i] == 0 are skipped.  The sets must not overlap
 * one another's outputs.  One kernel launch for all sets (work items numbered across them),
 * so small layers do not each pay a launch and a partly idle grid.
 * Errors: FGQ_ERR_ARG (n < 0 or n > FGQ_TERNARIZE_BATCH_MAX, a null array with n > 0, or
 * any set that fgq_ternarize would reject for its arguments), FGQ_ERR_ALIGN (as
 * fgq_ternarize, per set), FGQ_ERR_CUDA.
 */
fgq_status fgq_ternarize_batch(int n, const float* const* w, const int* M, const int* Kred, int G,
                               uint32_t* const* codes, float* const* alpha, cudaStream_t stream);

/* Bytes of device workspace fgq_quantize_act needs for n elements (0 when n == 0). */
size_t fgq_quantize_act_workspace_bytes(size_t n);

/*
 * Dynamic-fixed-point activation quantization (Section 4: activations quantized to 8 or
 * 4 bits before each convolution, one shared exponent per tensor).
 *   x          fp32 [n].
 *   type       FGQ_U8 / FGQ_S8 / FGQ_U4 / FGQ_S4; qmax = 255 / 127 / 15 / 7, qmin = 0 /
 *              -128 / 0 / -8.
 *   scale_in   > 0: use this scale (must be a power of two, else FGQ_ERR_ARG); <= 0: derive
 *              it: E = smallest integer with max * 2^-E <= qmax (max = max|x|, or max(x, 0)
 *              for unsigned types), E = 0 when max = 0, E clamped to [-149, 127].
 *   q          out, n bytes (8-bit) or ceil(n/2) bytes (4-bit; an odd tail's high nibble
 *              is 0).
 *   scale_out  out, device fp32 [1]: 2^E.  May be NULL when scale_in > 0.
 *   workspace  device scratch of fgq_quantize_act_workspace_bytes(n) bytes (ignored when
 *              scale_in > 0); its contents on entry do not matter.
 * q_i = clamp(round_half_even(x_i * 2^-E), qmin, qmax), exact.  Two kernels when the scale
 * is derived (max reduction, then quantization); one when it is given.
 * Errors: FGQ_ERR_ARG, FGQ_ERR_ALIGN (x, q not 16-byte aligned; workspace not 4-byte
 * aligned or too small), FGQ_ERR_CUDA; NaN/Inf recorded as FGQ_ERR_NONFINITE.
 */
fgq_status fgq_quantize_act(const float* x, size_t n, fgq_act_type type, float scale_in, void* q,
                            float* scale_out, void* workspace, size_t workspace_bytes,
                            cudaStream_t stream);

/* Largest number of tensors one fgq_quantize_act_batch call takes. */
#define FGQ_QUANTIZE_BATCH_MAX 128

/* Bytes of device workspace fgq_quantize_act_batch needs for n tensors (0 on bad n). */
size_t fgq_quantize_act_batch_workspace_bytes(int n);

/*
 * fgq_quantize_act with a derived scale for n tensors (the inputs of a network's layers) in
 * few launches: tensor i is x[i] fp32 [nelem[i]] -> q[i] (type[i]) and scale_out[i] (device
 * fp32 [1]), with the results (bit for bit), layouts and non-finite handling of
 * fgq_quantize_act.  x, nelem, type, q, scale_out are HOST arrays of n entries holding device
 * pointers, sizes and types (read during the call, not kept); tensors with nelem[i] == 0 are
 * skipped.  The tensors are processed in order in chunks of up to 48 MB of input (a larger
 * tensor forms its own chunk); launch k reduces chunk k to its maxima and quantizes chunk
 * k - 1 (one launch more than there are chunks), so the second pass over a chunk follows the
 * first closely enough to find much of it in the L2.  workspace: device scratch of
 * fgq_quantize_act_batch_workspace_bytes(n) bytes, 4-byte aligned (its contents on entry
 * do not matter).  The outputs must not overlap the inputs or one another.
 * Errors: FGQ_ERR_ARG (n < 0 or n > FGQ_QUANTIZE_BATCH_MAX, a null array or pointer, a bad
 * type, a short workspace), FGQ_ERR_ALIGN (x[i], q[i] not 16-byte aligned; scale_out[i],
 * workspace not 4-byte aligned), FGQ_ERR_CUDA.
 */
fgq_status fgq_quantize_act_batch(int n, const float* const* x, const size_t* nelem, const fgq_act_type* type,
                                  void* const* q, float* const* scale_out, void* workspace, size_t workspace_bytes,
                                  cudaStream_t stream);

/*
 * Allocation-free variant of fgq_quantize_act (no counterpart in the paper).  For callers
 * that cannot allocate device memory themselves -- hosts whose device memory is owned by a
 * framework pool with a fixed budget, plugins that only receive pre-allocated buffers, or
 * latency-critical loops that cannot afford cudaMalloc/cudaFree (cudaFree synchronizes the
 * device) -- it keeps the derived-scale pass's per-block maxima in a static 16 KB device
 * array inside the library (4096 words), so no workspace argument is needed.  Arguments,
 * results and errors are those of fgq_quantize_act; the caller still passes x, q and
 * scale_out.  The call itself allocates nothing.  Its first call on each device looks up the
 * array's device address (cudaGetSymbolAddress) with that device current, so make that
 * first call before any stream capture.  Every GPU that loads the library holds the array
 * until exit; all calls share it, so calls that overlap on the GPU (other streams or host
 * threads) race and must be serialized.  Returns FGQ_ERR_UNSUPPORTED if the scale pass
 * would need more than 4096 blocks (devices with more than 512 SMs).
 */
fgq_status fgq_quantize_act_noalloc(const float* x, size_t n, fgq_act_type type, float scale_in,
                                    void* q, float* scale_out, cudaStream_t stream);

/* Threshold rules of fgq_ternarize_threshold. */
typedef enum { FGQ_RULE_EXP = 0, FGQ_RULE_GAUSS = 1 } fgq_threshold_rule;

/*
 * Ternarization at an analytical threshold instead of the exact search (Section 3:
 * t_j = sign(w_j) where |w_j| > Delta, else 0; Lemma 1 and its proof in the appendix).
 *   rule FGQ_RULE_EXP    Delta = mean |w| (Lemma 1: exponential magnitudes);
 *   rule FGQ_RULE_GAUSS  Delta = 0.6120031809624808 * rms(w) (Gaussian weights: rms is the
 *                        maximum-likelihood sigma the paper names; the constant is the z
 *                        maximising phi(z)^2 / (1 - Phi(z)), the Gaussian limit of the
 *                        threshold objective (sum of kept |w|)^2 / (number kept)).
 *   per_layer = 0        one Delta and one alpha per group of G;
 *   per_layer = 1        one Delta and one alpha for the whole M x Kred matrix (alpha
 *                        written to every entry): the one-scaling-factor-per-layer baseline.
 * alpha = fp32(mean of the kept |w|), 0 when nothing is kept.  The statistics cover the
 * real weights only (a row's zero padding is not counted).  Per group they are fp64 sums
 * in element order with explicitly rounded operations, so results are bit-reproducible;
 * per layer the sums run in a fixed tree order (deterministic, a few ulps from a
 * sequential sum).  codes and alpha layouts as fgq_ternarize (codes fully written).
 *   workspace  per_layer = 1: device scratch of fgq_ternarize_threshold_workspace_bytes()
 *              bytes, 16-byte aligned; ignored (may be NULL) when per_layer = 0.
 *   delta_out  per_layer = 1: device fp64 [1] receiving Delta (may be NULL); ignored
 *              otherwise.
 * A group (per_layer = 0) or layer (per_layer = 1) holding NaN/Inf gets zero codes and
 * alpha, and FGQ_ERR_NONFINITE is recorded.
 * Errors: as fgq_ternarize; FGQ_ERR_ARG for a bad rule or a missing or short workspace.
 */
size_t fgq_ternarize_threshold_workspace_bytes(void);
fgq_status fgq_ternarize_threshold(const float* w, int M, int Kred, int G, int rule, int per_layer,
                                   uint32_t* codes, float* alpha, void* workspace,
                                   size_t workspace_bytes, double* delta_out, cudaStream_t stream);

/*
 * Ternary error of each group (Section 3: the element-wise error ||W - alpha What||^2
 * restricted to the group):
 *   err[m][g] = sum_{j in g, j < Kred} (w[m][j] - alpha[m][g] * t[m][j])^2,
 * fp64, accumulated in element order with explicitly rounded operations.  codes and alpha
 * as from fgq_ternarize or fgq_ternarize_threshold for (M, Kred, G); err device fp64
 * [M][fgq_num_groups(Kred, G)].
 * Errors: FGQ_ERR_ARG, FGQ_ERR_ALIGN (w, codes, alpha not 4-byte aligned, err not 8-byte
 * aligned), FGQ_ERR_CUDA.
 */
fgq_status fgq_ternary_error(const float* w, int M, int Kred, int G, const uint32_t* codes,
                             const float* alpha, double* err, cudaStream_t stream);

/*
 * 8-bit weights for the first layer (Section 4: the first layer is kept at 8w-8a): each
 * filter row of w fp32 [M][Kred] is quantized as a signed 8-bit DFP vector, the same rule
 * as fgq_quantize_act with FGQ_S8 applied per row.  wq out int8 [M][Kred]; wscale out fp32
 * [M] (2^E per row).  Errors as fgq_ternarize.
 */
fgq_status fgq_quantize_weights_w8(const float* w, int M, int Kred, int8_t* wq, float* wscale,
                                   cudaStream_t stream);

/*
 * Grouped ternary GEMM (fully connected layer, Eq. 2 with 32-bit group accumulators,
 * Section 4):  y[p][m] = act_scale[0] * sum_g alpha[m][g] * s[m][g][p],
 *              s[m][g][p] = sum_{j in g} t[m][j] * q[p][j]   (exact int32).
 *   q          activations [P][Kred] of the given type.
 *   act_scale  device fp32 [1] (e.g. the scale_out of fgq_quantize_act).
 *   codes, alpha as produced by fgq_ternarize for (M, Kred, G).
 *   y          out, fp32 [P][M].
 * The fp32 result is within 1e-5 * act_scale * sum_g |alpha_g * s_g| of the exact value.
 * Memory: the tensor-core kernels take per-call temporaries from a library-owned
 * stream-ordered pool of the current device and return them on the same stream: the
 * activations as fp16 (2 bytes per element read), and the ternary operand -- at G >= 64
 * the codes as fp16 (2 * M * Kp bytes), at G = 4 its block-diagonal form (4 * 2 * M' * Kp
 * bytes per fp16 part, two parts for fp32 alphas, M' = M rounded up to 32 per conv group).
 * The pool keeps freed blocks, so only a call that needs more than the pool holds reaches
 * the device allocator.  The dp4a and few-row paths allocate nothing.
 * Errors: FGQ_ERR_ARG (null pointers, bad sizes, Kred odd for 4-bit types),
 * FGQ_ERR_ALIGN (any pointer not 16-byte aligned), FGQ_ERR_CUDA.
 */
fgq_status fgq_gemm(const void* q, fgq_act_type type, const float* act_scale, int P, int Kred,
                    const uint32_t* codes, const float* alpha, int M, int G, float* y,
                    cudaStream_t stream);

/*
 * Grouped ternary convolution as an implicit GEMM (Section 3.2 grouping along the input
 * channels, Eq. 2, Section 4):  out[b][ho][wo][m] = act_scale[0] * sum_g alpha[m][g] *
 * s[m][g][b,ho,wo], where the group sums run over the im2col column of (b, ho, wo):
 * element (r, s, c) is act[b][ho*stride-pad+r][wo*stride-pad+s][gi*C/groups + c], zero
 * outside the image, gi = the conv group of filter m (m / (M/groups)).
 *   act        NHWC [B][H][W][C] of the given type.
 *   codes, alpha  from fgq_ternarize with Kred = R*S*(C/groups).
 *   groups     convolution channel groups (C and M divisible by it); unrelated to G.
 *   out        fp32 NHWC [B][Ho][Wo][M].
 * Tolerance and errors as fgq_gemm (C odd for 4-bit types is FGQ_ERR_ARG).
 */
fgq_status fgq_conv2d(const void* act, fgq_act_type type, const float* act_scale, int B, int H,
                      int W, int C, int R, int S, int stride, int pad, int groups,
                      const uint32_t* codes, const float* alpha, int M, int G, float* out,
                      cudaStream_t stream);

/*
 * fgq_gemm and fgq_conv2d with the output requantized inside the kernel (Section 4: the
 * 32-bit outputs are converted to 8 bits and rounded before they are passed to the next
 * layer): instead of fp32 y the kernels write
 *   out_q[p][m] = clamp(round_half_even(y[p][m] * 2^-E), qmin, qmax)
 * of out_type FGQ_U8 (0..255: negative outputs become 0, a fused ReLU) or FGQ_S8
 * (-128..127), one byte each, for the given output scale out_scale[0] = 2^E (device fp32,
 * a power of two, e.g. a per-layer DFP scale found on a calibration batch).  y is the fp32
 * value the fp32-output call returns (same kernel, same rounding), so the codes equal
 * fgq_quantize_act applied to that output with scale_in = 2^E.  out_q: [P][M] bytes,
 * 4-byte aligned.  Errors as fgq_gemm / fgq_conv2d; FGQ_ERR_ARG for another out_type.
 */
fgq_status fgq_gemm_rq(const void* q, fgq_act_type type, const float* act_scale, int P, int Kred,
                       const uint32_t* codes, const float* alpha, int M, int G,
                       fgq_act_type out_type, const float* out_scale, void* out_q,
                       cudaStream_t stream);
fgq_status fgq_conv2d_rq(const void* act, fgq_act_type type, const float* act_scale, int B, int H,
                         int W, int C, int R, int S, int stride, int pad, int groups,
                         const uint32_t* codes, const float* alpha, int M, int G,
                         fgq_act_type out_type, const float* out_scale, void* out_q,
                         cudaStream_t stream);

/* fgq_conv2d_w8 (the 8-bit-weight first layer) with the output requantized in the kernel,
 * as fgq_conv2d_rq. */
fgq_status fgq_conv2d_w8_rq(const void* act, fgq_act_type type, const float* act_scale, int B, int H,
                            int W, int C, int R, int S, int stride, int pad, int groups,
                            const int8_t* wq, const float* wscale, int M, fgq_act_type out_type,
                            const float* out_scale, void* out_q, cudaStream_t stream);

/*
 * Max pooling of unsigned 8-bit codes (the pooling after the first layer of the ResNet
 * forward): out[b][ho][wo][c] = max over the R x R window at stride, padding pad (padded
 * positions do not take part) of in[b][h][w][c], NHWC, C a multiple of 4, pad < R.  Exact
 * in the code domain (one shared scale).  in, out 4-byte aligned.
 */
fgq_status fgq_maxpool_u8(const uint8_t* in, int B, int H, int W, int C, int R, int stride, int pad,
                          uint8_t* out, cudaStream_t stream);

/*
 * Residual addition of two 8-bit code tensors of n elements (the shortcut of a ResNet
 * block): v = a * a_scale[0] + b * b_scale[0] in fp32 (each product exact, the sum rounded
 * once).  out != NULL: fp32 v is stored there; otherwise v is requantized to out_q at
 * out_scale[0] = 2^E as fgq_conv2d_rq does (out_type FGQ_U8: negative sums become 0, the
 * ReLU after the addition; or FGQ_S8).  a_type, b_type: FGQ_U8 or FGQ_S8.
 */
fgq_status fgq_add_codes(const void* a, fgq_act_type a_type, const float* a_scale, const void* b,
                         fgq_act_type b_type, const float* b_scale, size_t n, float* out,
                         fgq_act_type out_type, const float* out_scale, void* out_q,
                         cudaStream_t stream);

/*
 * Fixed-point scaling factors (Section 4: the alphas are quantized to 8/4-bit fixed point).
 * The ng alphas of each filter row share one DFP exponent (this library's reading; the
 * paper does not say how the exponent is shared), chosen by fgq_quantize_act's rule for
 * the unsigned type of that width (alphas are >= 0):
 *   aq[m][g] = clamp(round_half_even(alpha[m][g] * 2^-E_m), 0, 2^bits - 1),
 *   ascale[m] = 2^E_m, E_m the smallest integer with max_g alpha[m][g] * 2^-E_m <= 2^bits - 1.
 *   alpha   fp32 [M][ng] (as from fgq_ternarize).
 *   bits    8 (aq: one byte per alpha, [M][ng]) or 4 (aq: two per byte along the row,
 *           element 2i in the low nibble, [M][ceil(ng/2)]).
 *   ascale  out, fp32 [M].
 * A row holding NaN/Inf gets zero codes and scale 0 and records FGQ_ERR_NONFINITE.
 * Errors: FGQ_ERR_ARG, FGQ_ERR_ALIGN (alpha, ascale not 4-byte aligned), FGQ_ERR_CUDA.
 */
fgq_status fgq_quantize_alpha(const float* alpha, int M, int ng, int bits, uint8_t* aq, float* ascale,
                              cudaStream_t stream);

/*
 * fgq_gemm and fgq_conv2d with fixed-point alphas (aq, abits, ascale as produced by
 * fgq_quantize_alpha): the same contraction with alpha'[m][g] = aq[m][g] * ascale[m] (exact
 * in fp32).  On the few-row path (P <= 8, see FGQ_PATH_GEMV in fgq_debug.h) the weights stream as 2-bit
 * codes plus 1 (or 1/2) byte per group instead of 4, and sum_g aq * s is accumulated
 * exactly in 64-bit integers: y = act_scale * ascale[m] * sum, rounded once.  Otherwise, with
 * 8-bit activations and Cg a multiple of 64, the automatic choice is the dense tensor-core
 * path (FGQ_PATH_DENSE): the integer weights aq * t are folded into an fp16 matrix in a pool
 * temporary (2 * M * Kp bytes) and one dense contraction sums the exact integer products in
 * an fp32 accumulator: y = act_scale * ascale[m] * sum is the exact value rounded once when
 * sum_k |aq t q| < 2^24 (which bounds every partial sum; e.g. always for Kred * 255 * 255 <
 * 2^24), and otherwise within (Kp / 16) * 2^-23 * act_scale * ascale[m] * sum_k |aq t q| of it
 * (the accumulator rounds at most once per 16 reduction elements).  On the group-sum
 * paths (forced, or shapes the dense path does not cover) the alphas are expanded to fp32
 * in a pool temporary (2-bit codes stay as they are) and the fgq_gemm tolerance holds with alpha';
 * errors as fgq_gemm / fgq_conv2d, FGQ_ERR_ARG for abits not 8 or 4.
 */
fgq_status fgq_gemm_qa(const void* q, fgq_act_type type, const float* act_scale, int P, int Kred,
                       const uint32_t* codes, const uint8_t* aq, int abits, const float* ascale, int M,
                       int G, float* y, cudaStream_t stream);
fgq_status fgq_conv2d_qa(const void* act, fgq_act_type type, const float* act_scale, int B, int H,
                         int W, int C, int R, int S, int stride, int pad, int groups,
                         const uint32_t* codes, const uint8_t* aq, int abits, const float* ascale,
                         int M, int G, float* out, cudaStream_t stream);

/*
 * Dense 8-bit-weight convolution for the first layer (8w-8a, Section 4):
 *   out = act_scale[0] * wscale[m] * sum_j wq[m][j] * col[j]   (exact int32 dot product).
 *   wq int8 [M][Kred], wscale fp32 [M] (as from fgq_quantize_weights_w8).  Other arguments
 *   as fgq_conv2d.  Errors as fgq_conv2d.  With 8-bit activations and groups == 1 (and unless
 *   FGQ_PATH_SIMT is forced) it runs on the dense tensor-core path (FGQ_PATH_DENSE): an
 *   explicit im2col of the activations into a stream-ordered pool temporary of P * Kc bytes
 *   (Kc = Kred rounded up to 64, at most 4096), then one dense contraction on integer fp16
 *   operands; the sums are exact while |sum_j wq col| < 2^24 (always for Kred <= 514).
 *   Otherwise the dp4a path.
 */
fgq_status fgq_conv2d_w8(const void* act, fgq_act_type type, const float* act_scale, int B,
                         int H, int W, int C, int R, int S, int stride, int pad, int groups,
                         const int8_t* wq, const float* wscale, int M, float* out,
                         cudaStream_t stream);

/*
 * One convolution layer end to end from HOST buffers (the inference pipeline of Section 4:
 * fp32 weights are ternarized per group of G (Eq. 5), the fp32 input is quantized to
 * dynamic fixed point, the grouped contraction runs, the fp32 output comes back):
 *   h_w    host fp32 weights [M][Kred] (Kred in (r, s, c) order).
 *   h_x    host fp32 activations NHWC [B][H][W][C].
 *   type   activation type of the quantized input (scale derived as fgq_quantize_act does).
 *   G      group size as fgq_ternarize; G = 0 selects the 8-bit-weight first layer instead
 *          (fgq_quantize_weights_w8 + fgq_conv2d_w8; 8-bit activation types only).
 *   h_out  host fp32 output NHWC [B][Ho][Wo][M].
 *   workspace  device buffer of fgq_conv2d_host_workspace_bytes(...) bytes, 256-byte
 *          aligned, owned by the caller (it holds the device copies, codes, alphas,
 *          quantized input and output).
 * Issues, in order on `stream`: one cudaMemcpyAsync per input buffer (weights, then
 * activations), the kernels of fgq_ternarize (or fgq_quantize_weights_w8), fgq_quantize_act
 * and fgq_conv2d (or fgq_conv2d_w8), and one cudaMemcpyAsync of the output back.  The call
 * is asynchronous: h_out is valid once the stream has completed; host buffers should be
 * page-locked (cudaHostAlloc) for the copies to overlap other work.  Calls on different
 * streams need workspaces of their own.  The contraction tolerance is fgq_conv2d's.
 * Errors: those of the calls it makes; FGQ_ERR_ARG (null pointer, workspace too small),
 * FGQ_ERR_ALIGN (workspace), FGQ_ERR_CUDA (a copy could not be issued).
 */
size_t fgq_conv2d_host_workspace_bytes(fgq_act_type type, int B, int H, int W, int C, int R, int S,
                                       int stride, int pad, int groups, int M, int G);
fgq_status fgq_conv2d_host(const float* h_w, const float* h_x, fgq_act_type type, int B, int H, int W,
                           int C, int R, int S, int stride, int pad, int groups, int M, int G,
                           float* h_out, void* workspace, size_t workspace_bytes, cudaStream_t stream);

/*
 * The 32-bit group accumulators themselves (Section 4), for verification:
 *   s[m][g][p] = sum_{j in g, j < Kred} t[m][j] * q[p][j],  int32 [M][ng][P].
 * q as in fgq_gemm.  Computed by the kernel family the fp32-output call of the same shape
 * uses (the automatic choice, or the family fgq_set_path forces, see fgq_debug.h): the
 * tensor-core kernels store each group's TMEM accumulator (an exact integer in fp32) as
 * int32, the CUDA-core kernel its dp4a sums.  The dense and few-row paths form no group
 * sums; where the automatic choice would take one of them the dp4a kernel runs, and
 * forcing either returns FGQ_ERR_UNSUPPORTED.  Errors as fgq_gemm.
 */
fgq_status fgq_group_sums(const void* q, fgq_act_type type, int P, int Kred,
                          const uint32_t* codes, int M, int G, int32_t* s, cudaStream_t stream);

/*
 * The group sums of a convolution (Section 3.2 grouping, Eq. 2, Section 4 accumulators):
 *   s[m][g][p] = sum_{j in g, j < Kred} t[m][j] * col_p[j],  int32 [M][ng][P],
 * col_p the im2col column of output position p = (b * Ho + ho) * Wo + wo for filter m's
 * conv group, as in fgq_conv2d.  Kernel family and errors as fgq_group_sums and
 * fgq_conv2d.
 */
fgq_status fgq_conv2d_group_sums(const void* act, fgq_act_type type, int B, int H, int W, int C, int R,
                                 int S, int stride, int pad, int groups, const uint32_t* codes, int M,
                                 int G, int32_t* s, cudaStream_t stream);

/*
 * Returns (and clears) the first error a kernel recorded on the current device since the
 * last call (FGQ_OK if none), or FGQ_ERR_CUDA if a CUDA call failed.  The error word is one
 * per device and shared by every stream: the call reads and clears it in one atomic step,
 * in order on `stream`, and synchronizes `stream` before it returns, so it covers every
 * kernel on `stream` and any kernel on another stream that recorded its error before the
 * read.  Synchronize the device first to cover the kernels of all streams.
 */
fgq_status fgq_stream_status(cudaStream_t stream);

/* Number of kernels this library has launched in this process (all calls, all threads). */
uint64_t fgq_launch_count(void);

/*
 * Failure-detection self test: launches one block that waits, with an iteration limit,
 * on an mbarrier that nothing arrives on, and records FGQ_ERR_TIMEOUT when the limit
 * runs out.  Read the result with fgq_stream_status().  Paper counterpart: none (library
 * health check).
 */
fgq_status fgq_selftest_wait_timeout(uint32_t max_iterations, cudaStream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* FGQ_H_ */
