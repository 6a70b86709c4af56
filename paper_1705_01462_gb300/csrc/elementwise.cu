// The non-contraction steps of a chained quantized ResNet forward (Section 4: activations
// stay 8-bit DFP codes between layers): max pooling of codes and the residual addition.
//
// Max pooling of unsigned codes is exact in the code domain (one shared scale, and the
// codes of post-ReLU activations are >= 0, so padding never wins).  The residual addition
// v = a * 2^Ea + b * 2^Eb is computed in fp32 (each product is exact; the sum is rounded
// once) and either stored as fp32 or requantized at a given scale 2^Eo with the rule of
// the activation quantizer (u8: negative sums become 0, the ReLU after the addition).
#include <cstdint>

#include "fgq_device.cuh"

namespace fgq {
namespace {

// One thread per 4 channels of one output pixel (C % 4 == 0), per-byte maxima with vmaxu4.
__global__ void __launch_bounds__(256) maxpool_u8_kernel(const uint8_t* __restrict__ in, int B, int H, int W, int C,
                                                         int R, int stride, int pad, int Ho, int Wo,
                                                         uint8_t* __restrict__ out) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int C4 = C / 4;
  if (i >= (int64_t)B * Ho * Wo * C4) return;
  const int c4 = (int)(i % C4);
  int64_t r = i / C4;
  const int wo = (int)(r % Wo);
  r /= Wo;
  const int ho = (int)(r % Ho);
  const int b = (int)(r / Ho);
  uint32_t m = 0;
  for (int dr = 0; dr < R; ++dr) {
    const int h = ho * stride - pad + dr;
    if (h < 0 || h >= H) continue;
    for (int ds = 0; ds < R; ++ds) {
      const int w = wo * stride - pad + ds;
      if (w < 0 || w >= W) continue;
      m = __vmaxu4(m, __ldg(reinterpret_cast<const uint32_t*>(in + (((int64_t)b * H + h) * W + w) * C) + c4));
    }
  }
  reinterpret_cast<uint32_t*>(out)[i] = m;
}

__device__ __forceinline__ float code_value(const uint8_t* p, int64_t i, int is_signed) {
  const uint8_t v = __ldg(p + i);
  return is_signed ? (float)(int8_t)v : (float)v;
}

__global__ void __launch_bounds__(256) add_codes_kernel(const uint8_t* __restrict__ a, int a_signed,
                                                        const float* __restrict__ a_scale,
                                                        const uint8_t* __restrict__ b, int b_signed,
                                                        const float* __restrict__ b_scale, int64_t n,
                                                        float* __restrict__ out, uint8_t* __restrict__ out_q,
                                                        const float* __restrict__ out_scale, int o_signed) {
  const float sa = __ldg(a_scale), sb = __ldg(b_scale);
  RqMul rq;
  if (out_q) rq = rq_mul(out_scale, o_signed);
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
    const float v = __fadd_rn(__fmul_rn(code_value(a, i, a_signed), sa), __fmul_rn(code_value(b, i, b_signed), sb));
    if (out_q)
      out_q[i] = rq_code(v, rq);
    else
      out[i] = v;
  }
}

}  // namespace

fgq_status launch_maxpool_u8(const uint8_t* in, int B, int H, int W, int C, int R, int stride, int pad, uint8_t* out,
                             cudaStream_t s) {
  const int Ho = (H + 2 * pad - R) / stride + 1, Wo = (W + 2 * pad - R) / stride + 1;
  const int64_t n = (int64_t)B * Ho * Wo * (C / 4);
  maxpool_u8_kernel<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(in, B, H, W, C, R, stride, pad, Ho, Wo, out);
  return after_launch();
}

fgq_status launch_add_codes(const uint8_t* a, int a_signed, const float* a_scale, const uint8_t* b, int b_signed,
                            const float* b_scale, int64_t n, float* out, uint8_t* out_q, const float* out_scale,
                            int o_signed, cudaStream_t s) {
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t want = (n + 255) / 256;
  const int blocks = (int)(want < 8 * sms ? (want > 0 ? want : 1) : 8 * sms);
  add_codes_kernel<<<blocks, 256, 0, s>>>(a, a_signed, a_scale, b, b_signed, b_scale, n, out, out_q, out_scale,
                                          o_signed);
  return after_launch();
}

}  // namespace fgq
