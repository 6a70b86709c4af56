// Internal declarations shared by the libfgq translation units (not part of the ABI).
#pragma once

#include <cstddef>
#include <cstdint>

#include <cuda_runtime_api.h>

#include "../../include/fgq.h"
#include "../../include/fgq_debug.h"

namespace fgq {

// Geometry of one contraction call.  A GEMM is the convolution with B = P, H = W = 1,
// R = S = 1, C = Kred, stride 1, pad 0, groups 1.
struct Geom {
  int B, H, W, C, R, S, stride, pad, groups;
  int Ho, Wo, Cg, Kred, Kp, ng, M, Mg, G, wrow;
  int act_type;  // fgq_act_type
  int is_conv;
  int64_t P;     // B * Ho * Wo
  // fused output requantization (nullptr: fp32 output): codes [P][M] of 8-bit type
  // rq_signed ? FGQ_S8 : FGQ_U8 at the scale *rq_scale = 2^E
  uint8_t* rq_out;
  const float* rq_scale;
  int rq_signed;
};

// Device error word of the current device (first error wins; cleared by
// fgq_stream_status).  Returns nullptr if the symbol address cannot be obtained.
unsigned int* device_error_word();

// Counts one kernel launch (for fgq_launch_count) and converts a launch error.
fgq_status after_launch();
fgq_status after_launch(cudaError_t launch_result);  // the result of a cudaLaunchKernelEx

// Wait limit, in microseconds, that a test set on this host thread for the tensor-core
// kernels' mbarrier waits (fgq_debug_set_wait_limit_us), or -1 for the kernels' own limits.
int64_t debug_wait_limit_us();
// Whether the G = 4 output kernel runs on CTA pairs (this thread's setting, default off).
bool debug_cta_pairs();
int debug_max_ksplit();    // 1 .. 8
void note_ksplit(int k);   // group ranges of the G >= 64 tensor-core call just launched

// Kernel launchers (each returns FGQ_OK or FGQ_ERR_CUDA / FGQ_ERR_UNSUPPORTED).
fgq_status launch_ternarize(const float* w, int M, int Kred, int G, uint32_t* codes, float* alpha,
                            unsigned int* err, cudaStream_t s);
fgq_status launch_ternarize_batch(int n, const float* const* w, const int* M, const int* Kred, int G,
                                  uint32_t* const* codes, float* const* alpha, unsigned int* err, cudaStream_t s);
fgq_status launch_quantize_weights_w8(const float* w, int M, int Kred, int8_t* wq, float* wscale,
                                      unsigned int* err, cudaStream_t s);
size_t quantize_workspace_bytes(size_t n);
size_t threshold_workspace_bytes();
fgq_status launch_ternarize_threshold(const float* w, int M, int Kred, int G, int rule, int per_layer,
                                      uint32_t* codes, float* alpha, void* ws, double* delta_out, unsigned int* err,
                                      cudaStream_t s);
fgq_status launch_ternary_error(const float* w, int M, int Kred, int G, const uint32_t* codes, const float* alpha,
                                double* errv, cudaStream_t s);
fgq_status launch_quantize(const float* x, size_t n, int type, int E_given, bool derive, void* q,
                           float* scale_out, uint32_t* partials, unsigned int* err, cudaStream_t s);
// Batched derived-scale quantization of n tensors (tmax: n workspace words).
size_t quantize_batch_workspace_bytes(int n);
fgq_status launch_quantize_batch(int n, const float* const* x, const size_t* nelem, const int* type, void* const* q,
                                 float* const* scale_out, unsigned int* tmax, unsigned int* err, cudaStream_t s);

// CUDA-core contraction (dp4a).  codes/alpha for ternary weights, or wq/wscale for dense
// 8-bit weights (dense != 0).  sums != nullptr writes the int32 group sums [M][ng][P]
// instead of the fp32 output.
fgq_status launch_simt_contract(const void* act, const Geom& g, const void* weights,
                                const float* scales, int dense, const float* act_scale, float* out,
                                int32_t* sums, cudaStream_t s);
// Tensor-core contraction (tcgen05), G in {64, 128}; returns FGQ_ERR_UNSUPPORTED for shapes
// it does not cover.  sums != nullptr writes the int32 group sums [M][ng][P] (drained from
// TMEM) instead of the output.
bool tc_supports(const Geom& g);
fgq_status launch_tc_contract(const void* act, const Geom& g, const uint32_t* codes,
                              const float* alpha, const float* act_scale, float* out,
                              int32_t* sums, unsigned int* err, cudaStream_t s);


// Tensor-core contraction for G = 4 (block-diagonal activation operand).
bool tc4_supports(const Geom& g);
// sums != nullptr writes the int32 group sums [M][ng][P] instead of the output.
fgq_status launch_tc4_contract(const void* act, const Geom& g, const uint32_t* codes, const float* alpha,
                               const float* act_scale, float* out, int32_t* sums, unsigned int* err,
                               cudaStream_t s);

// Dense tensor-core contraction with the alphas folded into fp16 weights: fixed-point alphas
// (aq, abits 8 or 4, ascale) exactly, or fp32 alphas (aq == nullptr) split into two fp16
// parts.  8-bit activations, Cg % 64 == 0.
bool dense_supports(const Geom& g);
fgq_status launch_dense_contract(const void* act, const Geom& g, const uint32_t* codes, const float* alpha,
                                 const uint8_t* aq, int abits, const float* ascale, const float* act_scale, float* out,
                                 unsigned int* err, cudaStream_t s);
// fp32 alphas folded into the codes as two fp16 parts: a0[m][k] + a1[m][k] = alpha(m, k / G) *
// t[m][k] * 2^e_m to about 22 bits (a0 the fp16 nearest, a1 the fp16 nearest the remainder),
// with e_m putting row m's largest alpha in [2^14, 2^15), and rs[m] = 2^-e_m.  a0, a1 fp16
// [M][16 wrow]; codes 00 and padding give 0.
fgq_status launch_fold_alpha_split(const uint32_t* codes, int M, int wrow, int G, int ng, const float* alpha,
                                   void* a0, void* a1, float* rs, cudaStream_t s);
// The 8-bit-weight convolution (dense weights wq, per-filter scales) on the same kernel, through
// an explicit im2col of the activations in a pool temporary (any C, groups == 1); exact.
bool dense_w8_supports(const Geom& g);
fgq_status launch_dense_w8(const void* act, const Geom& g, const int8_t* wq, const float* wscale,
                           const float* act_scale, float* out, unsigned int* err, cudaStream_t s);

fgq_status launch_wait_timeout_selftest(uint32_t max_iter, unsigned int* err, cudaStream_t s);

// Chained-forward steps: max pooling of u8 codes, residual addition of two 8-bit code
// tensors (fp32 sum, or requantized when out_q is given).
fgq_status launch_maxpool_u8(const uint8_t* in, int B, int H, int W, int C, int R, int stride, int pad, uint8_t* out,
                             cudaStream_t s);
fgq_status launch_add_codes(const uint8_t* a, int a_signed, const float* a_scale, const uint8_t* b, int b_signed,
                            const float* b_scale, int64_t n, float* out, uint8_t* out_q, const float* out_scale,
                            int o_signed, cudaStream_t s);

// Stream-ordered memory pool of the current device for per-call temporaries (it keeps
// freed blocks: no release threshold).  nullptr if it cannot be created.
cudaMemPool_t scratch_pool();

// Fixed-point alphas (8- or 4-bit codes, one scale 2^E per filter row).
fgq_status launch_quantize_alpha(const float* alpha, int M, int ng, int bits, uint8_t* aq, float* ascale,
                                 unsigned int* err, cudaStream_t s);
fgq_status launch_dequantize_alpha(const uint8_t* aq, int bits, int M, int ng, const float* ascale, float* alpha,
                                   cudaStream_t s);

// Few-row contraction (P <= 8, 8-bit activations, Kred % 16 == 0, G >= 4); alphas fp32
// (abits = 0) or fixed point (abits 8 or 4 with aq, ascale).
bool gemv_supports(int P, int Kred, int G, int act_type);
fgq_status launch_gemv(const void* q, int act_type, int P, int Kred, int M, int G, const uint32_t* codes,
                       const float* alpha, const uint8_t* aq, int abits, const float* ascale, const float* act_scale,
                       float* y, uint8_t* rq_out, const float* rq_scale, int rq_signed, cudaStream_t s);

}  // namespace fgq
