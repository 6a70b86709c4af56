// Dynamic-fixed-point activation quantization (Section 4: activations are quantized to 8
// or 4 bits before each convolution, with one shared exponent per tensor).
//
//   E   = smallest integer with max * 2^-E <= qmax (max = max|x|, or max(x, 0) for the
//         unsigned types), 0 when max = 0, clamped to [-149, 127];
//   q_i = clamp(round_half_even(x_i * 2^-E), qmin, qmax),   scale = 2^E.
//
// x * 2^-E is exact in fp32 whenever the result is at least 2^-126 (a power-of-two
// scaling), and a product below that rounds to the integer 0 whichever way it is rounded,
// so the codes are exact.  When 2^-E exceeds the fp32 range the scaling is applied as two
// exact factors.
//
// Pass 1 (derived scale only): per-block maxima of the magnitude bit patterns (non-negative
// floats order like their bits) into the caller's workspace.  Pass 2: every block reduces
// the block maxima, derives E, and quantizes a grid-stride share of 16-element chunks.
#include <climits>
#include <cstdint>
#include <cstring>
#include <mutex>

#include "fgq_device.cuh"

namespace fgq {
namespace {

constexpr int kThreads = 256;

__device__ __forceinline__ uint32_t mag_bits(float x, bool is_unsigned) {
  const uint32_t b = __float_as_uint(x);
  if (is_unsigned) return (b >> 31) ? 0u : b;  // negative (and -0) count as 0
  return b & 0x7fffffffu;
}

// float4 loads with an L2 eviction-priority hint: pass 1 marks the input evict-last so that
// as much of it as fits is still in L2 when pass 2 reads it (evict-first: not needed again).
__device__ __forceinline__ float4 ld_f4_policy(const float4* p, uint64_t pol) {
  float4 v;
  asm volatile("ld.global.nc.L2::cache_hint.v4.f32 {%0, %1, %2, %3}, [%4], %5;"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "l"(p), "l"(pol));
  return v;
}
__device__ __forceinline__ uint64_t policy_evict_last() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}
__device__ __forceinline__ uint64_t policy_evict_first() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}

__global__ void __launch_bounds__(kThreads) qa_max_kernel(const float* __restrict__ x, size_t n, int is_unsigned,
                                                          uint32_t* __restrict__ partials, unsigned int* err) {
  uint32_t mx = 0;
  bool bad = false;
  const size_t n4 = n / 4;
  const float4* x4 = reinterpret_cast<const float4*>(x);
  const size_t tid = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  const size_t nth = (size_t)gridDim.x * blockDim.x;
  const uint64_t keep = policy_evict_last();
  for (size_t i = tid; i < n4; i += nth) {
    const float4 f = ld_f4_policy(x4 + i, keep);
    const float e[4] = {f.x, f.y, f.z, f.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      bad |= (__float_as_uint(e[j]) & 0x7fffffffu) >= 0x7f800000u;
      mx = max(mx, mag_bits(e[j], is_unsigned));
    }
  }
  for (size_t i = n4 * 4 + tid; i < n; i += nth) {
    const float e = __ldg(x + i);
    bad |= (__float_as_uint(e) & 0x7fffffffu) >= 0x7f800000u;
    mx = max(mx, mag_bits(e, is_unsigned));
  }
  __shared__ uint32_t red[kThreads / 32];
  mx = __reduce_max_sync(FULL_MASK, mx);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = mx;
  if (__syncthreads_or(bad) && threadIdx.x == 0) record_error(err, FGQ_ERR_NONFINITE);
  if (threadIdx.x == 0) {
    uint32_t m = 0;
    for (int i = 0; i < kThreads / 32; ++i) m = max(m, red[i]);
    partials[blockIdx.x] = m;
  }
}

__device__ __forceinline__ int dfp_exponent(uint32_t mbits, int qmax) {
  if (mbits == 0 || mbits >= 0x7f800000u) return 0;
  const double md = (double)__uint_as_float(mbits);
  int E = (int)((__double_as_longlong(md) >> 52) & 0x7ff) - 1023 - 10;  // condition fails here
  while (md * pow2d(-E) > (double)qmax) ++E;
  return max(-149, min(127, E));
}

template <int TYPE>
struct QTraits;
template <> struct QTraits<FGQ_U8> { static constexpr int qmin = 0, qmax = 255, bits = 8; };
template <> struct QTraits<FGQ_S8> { static constexpr int qmin = -128, qmax = 127, bits = 8; };
template <> struct QTraits<FGQ_U4> { static constexpr int qmin = 0, qmax = 15, bits = 4; };
template <> struct QTraits<FGQ_S4> { static constexpr int qmin = -8, qmax = 7, bits = 4; };

template <int TYPE>
__device__ __forceinline__ uint32_t qcode(float x, float mul1, float mul2) {
  using T = QTraits<TYPE>;
  int r = __float2int_rn(x * mul1 * mul2);
  r = max(T::qmin, min(T::qmax, r));
  return (uint32_t)r & ((1u << T::bits) - 1u);
}

template <int TYPE>
__global__ void __launch_bounds__(kThreads) qa_quant_kernel(const float* __restrict__ x, size_t n,
                                                            const uint32_t* __restrict__ partials, int nparts,
                                                            int E_given, uint8_t* __restrict__ q,
                                                            float* __restrict__ scale_out) {
  using T = QTraits<TYPE>;
  __shared__ int sE;
  __shared__ uint32_t red[kThreads / 32];
  int E = E_given;
  if (partials != nullptr) {
    uint32_t mx = 0;
    for (int i = threadIdx.x; i < nparts; i += blockDim.x) mx = max(mx, partials[i]);
    mx = __reduce_max_sync(FULL_MASK, mx);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = mx;
    __syncthreads();
    if (threadIdx.x == 0) {
      uint32_t m = 0;
      for (int i = 0; i < kThreads / 32; ++i) m = max(m, red[i]);
      sE = dfp_exponent(m, T::qmax);
    }
    __syncthreads();
    E = sE;
  }
  if (blockIdx.x == 0 && threadIdx.x == 0 && scale_out != nullptr) *scale_out = pow2f(E);
  const float mul1 = (-E <= 127) ? pow2f(-E) : pow2f(64);
  const float mul2 = (-E <= 127) ? 1.0f : pow2f(-E - 64);

  const size_t n16 = n / 16;
  const size_t tid = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  const size_t nth = (size_t)gridDim.x * blockDim.x;
  const float4* x4 = reinterpret_cast<const float4*>(x);
  const uint64_t drop = policy_evict_first();
  // chunks in reverse of pass 1's order: the part of x pass 1 read last is the part most
  // likely still in L2
  for (size_t c0 = tid; c0 < n16; c0 += nth) {
    const size_t c = n16 - 1 - c0;
    float e[16];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float4 f = ld_f4_policy(x4 + 4 * c + j, drop);
      e[4 * j] = f.x; e[4 * j + 1] = f.y; e[4 * j + 2] = f.z; e[4 * j + 3] = f.w;
    }
    if (T::bits == 8) {
      uint4 o;
      uint32_t wv[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        wv[j] = qcode<TYPE>(e[4 * j], mul1, mul2) | (qcode<TYPE>(e[4 * j + 1], mul1, mul2) << 8) |
                (qcode<TYPE>(e[4 * j + 2], mul1, mul2) << 16) | (qcode<TYPE>(e[4 * j + 3], mul1, mul2) << 24);
      }
      o.x = wv[0]; o.y = wv[1]; o.z = wv[2]; o.w = wv[3];
      reinterpret_cast<uint4*>(q)[c] = o;
    } else {
      uint32_t wv[2] = {0u, 0u};
#pragma unroll
      for (int j = 0; j < 16; ++j) wv[j / 8] |= qcode<TYPE>(e[j], mul1, mul2) << (4 * (j % 8));
      reinterpret_cast<uint2*>(q)[c] = make_uint2(wv[0], wv[1]);
    }
  }
  if (tid == 0) {  // ragged tail of fewer than 16 elements
    for (size_t i = n16 * 16; i < n; ++i) {
      const uint32_t code = qcode<TYPE>(x[i], mul1, mul2);
      if (T::bits == 8) {
        q[i] = (uint8_t)code;
      } else if ((i & 1) == 0) {
        q[i / 2] = (uint8_t)code;  // the high nibble of an odd tail stays 0
      } else {
        q[i / 2] = (uint8_t)(q[i / 2] | (code << 4));
      }
    }
  }
}

int num_sms() {
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  return sms;
}

int max_blocks(size_t n) {
  const size_t need = (n / 16 + kThreads - 1) / kThreads;
  const size_t cap = (size_t)num_sms() * 8;
  return (int)(need < 1 ? 1 : (need < cap ? need : cap));
}

}  // namespace

namespace {

// Fixed-point alphas (Section 4): one warp per filter row; the row's DFP exponent from its
// maximum (the activation quantizer's rule, unsigned 8- or 4-bit), then the codes (4-bit:
// two per byte, element 2i in the low nibble) and the row scale 2^E.  A row holding
// NaN/Inf gets zero codes and scale 0 and records FGQ_ERR_NONFINITE.
template <int TYPE>
__global__ void __launch_bounds__(256) quantize_alpha_kernel(const float* __restrict__ alpha, int M, int ng,
                                                            uint8_t* __restrict__ aq, float* __restrict__ ascale,
                                                            unsigned int* err) {
  using T = QTraits<TYPE>;
  const int m = blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (m >= M) return;
  const float* row = alpha + (int64_t)m * ng;
  uint32_t mx = 0;
  bool bad = false;
  for (int g = lane; g < ng; g += 32) {
    const float v = __ldg(row + g);
    bad |= (__float_as_uint(v) & 0x7fffffffu) >= 0x7f800000u;
    mx = max(mx, mag_bits(v, true));
  }
  mx = __reduce_max_sync(FULL_MASK, mx);
  bad = __any_sync(FULL_MASK, bad);
  const int rb = T::bits == 8 ? ng : (ng + 1) / 2;  // code bytes per row
  uint8_t* out = aq + (int64_t)m * rb;
  if (bad) {
    if (lane == 0) {
      record_error(err, FGQ_ERR_NONFINITE);
      ascale[m] = 0.0f;
    }
    for (int i = lane; i < rb; i += 32) out[i] = 0;
    return;
  }
  const int E = dfp_exponent(mx, T::qmax);
  const float mul1 = (-E <= 127) ? pow2f(-E) : pow2f(64);
  const float mul2 = (-E <= 127) ? 1.0f : pow2f(-E - 64);
  if (lane == 0) ascale[m] = pow2f(E);
  for (int i = lane; i < rb; i += 32) {
    if (T::bits == 8) {
      out[i] = (uint8_t)qcode<TYPE>(__ldg(row + i), mul1, mul2);
    } else {
      const uint32_t lo = qcode<TYPE>(__ldg(row + 2 * i), mul1, mul2);
      const uint32_t hi = 2 * i + 1 < ng ? qcode<TYPE>(__ldg(row + 2 * i + 1), mul1, mul2) : 0u;
      out[i] = (uint8_t)(lo | (hi << 4));
    }
  }
}

// alpha' = a * scale per row (exact in fp32), for the paths that take fp32 alphas.
__global__ void __launch_bounds__(256) dequantize_alpha_kernel(const uint8_t* __restrict__ aq, int bits, int M, int ng,
                                                              const float* __restrict__ ascale,
                                                              float* __restrict__ alpha) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (int64_t)M * ng) return;
  const int m = (int)(i / ng), g = (int)(i - (int64_t)m * ng);
  uint32_t a;
  if (bits == 8) {
    a = __ldg(aq + i);
  } else {
    const uint8_t b = __ldg(aq + (int64_t)m * ((ng + 1) / 2) + g / 2);
    a = (g & 1) ? (b >> 4) : (b & 0xfu);
  }
  alpha[i] = (float)a * __ldg(ascale + m);
}

}  // namespace

fgq_status launch_quantize_alpha(const float* alpha, int M, int ng, int bits, uint8_t* aq, float* ascale,
                                 unsigned int* err, cudaStream_t s) {
  const unsigned blocks = (unsigned)((M + 7) / 8);
  if (bits == 8)
    quantize_alpha_kernel<FGQ_U8><<<blocks, 256, 0, s>>>(alpha, M, ng, aq, ascale, err);
  else
    quantize_alpha_kernel<FGQ_U4><<<blocks, 256, 0, s>>>(alpha, M, ng, aq, ascale, err);
  return after_launch();
}

fgq_status launch_dequantize_alpha(const uint8_t* aq, int bits, int M, int ng, const float* ascale, float* alpha,
                                   cudaStream_t s) {
  const int64_t n = (int64_t)M * ng;
  dequantize_alpha_kernel<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(aq, bits, M, ng, ascale, alpha);
  return after_launch();
}

size_t quantize_workspace_bytes(size_t n) {
  if (n == 0) return 0;
  return sizeof(uint32_t) * (size_t)max_blocks(n);
}

fgq_status launch_quantize(const float* x, size_t n, int type, int E_given, bool derive, void* q,
                           float* scale_out, uint32_t* partials, unsigned int* err, cudaStream_t s) {
  const int blocks = max_blocks(n);
  if (derive) {
    qa_max_kernel<<<blocks, kThreads, 0, s>>>(x, n, (type == FGQ_U8 || type == FGQ_U4) ? 1 : 0, partials, err);
    fgq_status st = after_launch();
    if (st != FGQ_OK) return st;
  } else {
    partials = nullptr;
  }
  uint8_t* qb = static_cast<uint8_t*>(q);
  switch (type) {
    case FGQ_U8: qa_quant_kernel<FGQ_U8><<<blocks, kThreads, 0, s>>>(x, n, partials, blocks, E_given, qb, scale_out); break;
    case FGQ_S8: qa_quant_kernel<FGQ_S8><<<blocks, kThreads, 0, s>>>(x, n, partials, blocks, E_given, qb, scale_out); break;
    case FGQ_U4: qa_quant_kernel<FGQ_U4><<<blocks, kThreads, 0, s>>>(x, n, partials, blocks, E_given, qb, scale_out); break;
    case FGQ_S4: qa_quant_kernel<FGQ_S4><<<blocks, kThreads, 0, s>>>(x, n, partials, blocks, E_given, qb, scale_out); break;
    default: return FGQ_ERR_ARG;
  }
  return after_launch();
}

}  // namespace fgq

// ----------------------------------------------------------------------------------------
// fgq_quantize_act_batch: the same quantization for many tensors (the inputs of a network's
// layers), with far fewer launches.  The tensors are taken in order in chunks of at most
// kBatchChunkBytes of fp32 input (a larger tensor forms a chunk of its own), so that what pass
// 1 reads is still in the L2 when pass 2 re-reads it.  The passes are pipelined: launch k
// quantizes chunk k - 1 (pass 2, from the L2) while it reduces chunk k (pass 1, from HBM),
// so C chunks take C + 1 launches and the two passes overlap.  Every block covers
// kBatchElems consecutive elements of one tensor.  Pass 1 folds its maximum into the
// tensor's word with atomicMax (magnitude bit patterns order like the floats); pass 2 takes
// the tensor's exponent from that word and quantizes its elements, blocks in reverse order
// (the data pass 1 read last first).
namespace fgq {
namespace {

constexpr int kBatchThreads = 256;
constexpr int64_t kBatchElems = 16384;             // elements per block (64 KB of fp32)
constexpr int kBatchChunk = 32;                    // tensors per launch
constexpr size_t kBatchChunkBytes = (size_t)48 << 20;  // two chunks (one per pass) share the L2

struct QTensor {
  const float* x;
  uint8_t* q;
  float* scale;
  unsigned int* tmax;  // the tensor's maximum word
  int64_t n;
  int type;
  int block0;   // first block of this tensor in the launch
};

struct QBatch {
  QTensor t[kBatchChunk];
  int n;
  int nblocks;
};

__device__ __forceinline__ int qbatch_tensor(const QBatch& b, int blk) {
  int lo = 0, hi = b.n - 1;
  while (lo < hi) {  // largest tensor whose first block is <= blk
    const int mid = (lo + hi + 1) >> 1;
    if (b.t[mid].block0 <= blk) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

__device__ __forceinline__ void qab_max_block(const QBatch& b, int blk, unsigned int* err) {
  const QTensor& T = b.t[qbatch_tensor(b, blk)];
  const int64_t e0 = (int64_t)(blk - T.block0) * kBatchElems;
  const int64_t e1 = e0 + kBatchElems < T.n ? e0 + kBatchElems : T.n;
  const bool is_unsigned = T.type == FGQ_U8 || T.type == FGQ_U4;
  uint32_t mx = 0;
  bool bad = false;
  const float4* x4 = reinterpret_cast<const float4*>(T.x + e0);  // e0 is a multiple of 4: aligned
  const int64_t n4 = (e1 - e0) / 4;
  const uint64_t keep = policy_evict_last();
  constexpr int U = 8;  // independent 16-byte loads in flight per thread
  int64_t i = threadIdx.x;
  for (; i + (U - 1) * kBatchThreads < n4; i += U * kBatchThreads) {
    float4 f[U];
#pragma unroll
    for (int u = 0; u < U; ++u) f[u] = ld_f4_policy(x4 + i + u * kBatchThreads, keep);
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const float e[4] = {f[u].x, f[u].y, f[u].z, f[u].w};
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        bad |= (__float_as_uint(e[j]) & 0x7fffffffu) >= 0x7f800000u;
        mx = max(mx, mag_bits(e[j], is_unsigned));
      }
    }
  }
  for (; i < n4; i += kBatchThreads) {
    const float4 f = ld_f4_policy(x4 + i, keep);
    const float e[4] = {f.x, f.y, f.z, f.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      bad |= (__float_as_uint(e[j]) & 0x7fffffffu) >= 0x7f800000u;
      mx = max(mx, mag_bits(e[j], is_unsigned));
    }
  }
  for (int64_t i = e0 + n4 * 4 + threadIdx.x; i < e1; i += kBatchThreads) {
    const float e = __ldg(T.x + i);
    bad |= (__float_as_uint(e) & 0x7fffffffu) >= 0x7f800000u;
    mx = max(mx, mag_bits(e, is_unsigned));
  }
  __shared__ uint32_t red[kBatchThreads / 32];
  mx = __reduce_max_sync(FULL_MASK, mx);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = mx;
  if (__syncthreads_or(bad) && threadIdx.x == 0) record_error(err, FGQ_ERR_NONFINITE);
  if (threadIdx.x == 0) {
    uint32_t m = 0;
    for (int i = 0; i < kBatchThreads / 32; ++i) m = max(m, red[i]);
    atomicMax(T.tmax, m);
  }
}

template <int TYPE>
__device__ __forceinline__ void qab_quant_range(const QTensor& T, int64_t e0, int64_t e1, bool write_scale) {
  using Tr = QTraits<TYPE>;
  const int E = dfp_exponent(*reinterpret_cast<const volatile unsigned int*>(T.tmax), Tr::qmax);
  if (write_scale && threadIdx.x == 0) *T.scale = pow2f(E);
  const float mul1 = (-E <= 127) ? pow2f(-E) : pow2f(64);
  const float mul2 = (-E <= 127) ? 1.0f : pow2f(-E - 64);
  const int64_t n16 = (e1 - e0) / 16;
  const float4* x4 = reinterpret_cast<const float4*>(T.x + e0);
  const uint64_t drop = policy_evict_first();
  constexpr int CU = 2;  // 16-element chunks in flight per thread (8 independent 16-byte loads)
  for (int64_t c0 = threadIdx.x; c0 < n16; c0 += CU * kBatchThreads) {
    float e[CU][16];
#pragma unroll
    for (int u = 0; u < CU; ++u) {
      const int64_t c = c0 + u * kBatchThreads;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const float4 f = c < n16 ? ld_f4_policy(x4 + 4 * c + j, drop) : make_float4(0.f, 0.f, 0.f, 0.f);
        e[u][4 * j] = f.x; e[u][4 * j + 1] = f.y; e[u][4 * j + 2] = f.z; e[u][4 * j + 3] = f.w;
      }
    }
#pragma unroll
    for (int u = 0; u < CU; ++u) {
      const int64_t c = c0 + u * kBatchThreads;
      if (c >= n16) break;
      if (Tr::bits == 8) {
        uint32_t wv[4];
#pragma unroll
        for (int j = 0; j < 4; ++j)
          wv[j] = qcode<TYPE>(e[u][4 * j], mul1, mul2) | (qcode<TYPE>(e[u][4 * j + 1], mul1, mul2) << 8) |
                  (qcode<TYPE>(e[u][4 * j + 2], mul1, mul2) << 16) | (qcode<TYPE>(e[u][4 * j + 3], mul1, mul2) << 24);
        reinterpret_cast<uint4*>(T.q + e0)[c] = make_uint4(wv[0], wv[1], wv[2], wv[3]);
      } else {
        uint32_t wv[2] = {0u, 0u};
#pragma unroll
        for (int j = 0; j < 16; ++j) wv[j / 8] |= qcode<TYPE>(e[u][j], mul1, mul2) << (4 * (j % 8));
        reinterpret_cast<uint2*>(T.q + e0 / 2)[c] = make_uint2(wv[0], wv[1]);
      }
    }
  }
  if (threadIdx.x == 0) {  // the tensor's ragged tail (last block only): fewer than 16 elements
    for (int64_t i = e0 + n16 * 16; i < e1; ++i) {
      const uint32_t code = qcode<TYPE>(T.x[i], mul1, mul2);
      if (Tr::bits == 8) {
        T.q[i] = (uint8_t)code;
      } else if ((i & 1) == 0) {
        T.q[i / 2] = (uint8_t)code;  // the high nibble of an odd tail stays 0
      } else {
        T.q[i / 2] = (uint8_t)(T.q[i / 2] | (code << 4));
      }
    }
  }
}

__device__ __forceinline__ void qab_quant_block(const QBatch& b, int blk) {
  const QTensor& T = b.t[qbatch_tensor(b, blk)];
  const int64_t e0 = (int64_t)(blk - T.block0) * kBatchElems;
  const int64_t e1 = e0 + kBatchElems < T.n ? e0 + kBatchElems : T.n;
  const bool first = blk == T.block0;
  switch (T.type) {
    case FGQ_U8: qab_quant_range<FGQ_U8>(T, e0, e1, first); break;
    case FGQ_S8: qab_quant_range<FGQ_S8>(T, e0, e1, first); break;
    case FGQ_U4: qab_quant_range<FGQ_U4>(T, e0, e1, first); break;
    default: qab_quant_range<FGQ_S4>(T, e0, e1, first); break;
  }
}

// One pipelined launch: blocks [0, q.nblocks) quantize chunk q (reverse block order), the
// rest reduce chunk m.
struct QPair {
  QBatch q, m;
};

__global__ void __launch_bounds__(kBatchThreads) qab_kernel(const __grid_constant__ QPair p, unsigned int* err) {
  pdl_wait();  // the previous launch's maxima (and the zeroed words) are complete
  pdl_trigger();
  const int bx = (int)blockIdx.x;
  if (bx < p.q.nblocks) qab_quant_block(p.q, p.q.nblocks - 1 - bx);
  else qab_max_block(p.m, bx - p.q.nblocks, err);
}

}  // namespace

size_t quantize_batch_workspace_bytes(int n) { return n > 0 ? sizeof(unsigned int) * (size_t)n : 0; }

fgq_status launch_quantize_batch(int n, const float* const* x, const size_t* nelem, const int* type, void* const* q,
                                 float* const* scale_out, unsigned int* tmax, unsigned int* err, cudaStream_t s) {
  if (cudaMemsetAsync(tmax, 0, sizeof(unsigned int) * (size_t)n, s) != cudaSuccess) return FGQ_ERR_CUDA;
  QPair p;
  memset(&p, 0, sizeof p);  // p.q: the chunk waiting for pass 2 (none yet)
  int i = 0;
  auto launch = [&]() -> fgq_status {
    const int64_t blocks = (int64_t)p.q.nblocks + p.m.nblocks;
    if (blocks == 0) return FGQ_OK;
    if (blocks > INT32_MAX) return FGQ_ERR_UNSUPPORTED;
    return after_launch(launch_pdl(qab_kernel, dim3((unsigned)blocks), dim3(kBatchThreads), 0, s, p, err));
  };
  while (i < n) {
    QBatch& b = p.m;
    memset(&b, 0, sizeof b);
    size_t bytes = 0;
    int blocks = 0;
    // a chunk: consecutive tensors up to kBatchChunkBytes of input (at least one tensor)
    while (i < n && b.n < kBatchChunk) {
      if (nelem[i] == 0) {
        ++i;
        continue;
      }
      const size_t tb = nelem[i] * sizeof(float);
      if (b.n > 0 && bytes + tb > kBatchChunkBytes) break;
      const int64_t nb = ((int64_t)nelem[i] + kBatchElems - 1) / kBatchElems;
      if ((int64_t)blocks + nb > INT32_MAX) {
        if (b.n == 0) return FGQ_ERR_UNSUPPORTED;  // one tensor beyond the grid's reach
        break;
      }
      QTensor& T = b.t[b.n++];
      T.x = x[i];
      T.q = static_cast<uint8_t*>(q[i]);
      T.scale = scale_out[i];
      T.tmax = tmax + i;
      T.n = (int64_t)nelem[i];
      T.type = type[i];
      T.block0 = blocks;
      blocks += (int)nb;
      bytes += tb;
      ++i;
    }
    if (b.n == 0) continue;
    b.nblocks = blocks;
    // pass 2 of the previous chunk and pass 1 of this one
    const fgq_status st = launch();
    if (st != FGQ_OK) return st;
    p.q = p.m;
  }
  memset(&p.m, 0, sizeof p.m);
  return launch();  // pass 2 of the last chunk
}

}  // namespace fgq

// ----------------------------------------------------------------------------------------
// fgq_quantize_act_noalloc: the derived-scale quantizer for callers that cannot allocate
// device memory.  Some hosts own every device allocation themselves (a framework's memory
// pool with a fixed budget, a plugin that only receives pre-allocated tensors) or cannot
// afford cudaMalloc/cudaFree on the inference path (cudaFree synchronizes the device, and a
// fresh allocation can stall or fail under memory pressure).  For them the per-block maxima
// of pass 1 live in this file-scope device array instead of a caller-provided workspace.
//
// The array is a host-side stand-in in host code, not a device address, so its address is
// obtained once per device with cudaGetSymbolAddress (with that device current) and passed
// to the kernels.  That set-up happens in the first call on each device, which should
// therefore come before any stream capture.  Every GPU that loads the library keeps the
// array (16 KB) until exit.  All calls share it: each call fully rewrites the slots it uses
// before reading them, so nothing needs clearing, but calls that overlap on the GPU (in
// different streams, or from different threads) race on it and must be serialized.
namespace fgq {
namespace {

constexpr int kNoallocScratchWords = 4096;  // maximum number of pass-1 blocks
static __device__ __align__(256) uint32_t g_noalloc_scratch[kNoallocScratchWords];

constexpr int kNoallocMaxDevices = 64;
uint32_t* g_noalloc_ptr[kNoallocMaxDevices];
std::mutex g_noalloc_mu;

// Device address of the scratch array on the current device (nullptr on failure).
uint32_t* noalloc_scratch() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kNoallocMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lk(g_noalloc_mu);
  if (!g_noalloc_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess) return nullptr;
    g_noalloc_ptr[dev] = static_cast<uint32_t*>(p);
  }
  return g_noalloc_ptr[dev];
}

}  // namespace
}  // namespace fgq

extern "C" fgq_status fgq_quantize_act_noalloc(const float* x, size_t n, fgq_act_type type, float scale_in,
                                               void* q, float* scale_out, cudaStream_t stream) {
  using namespace fgq;
  if (type != FGQ_U8 && type != FGQ_S8 && type != FGQ_U4 && type != FGQ_S4) return FGQ_ERR_ARG;
  int E = 0;
  const bool derive = !(scale_in > 0.0f);
  if (!derive) {  // a given scale must be a power of two 2^E (subnormal ones included)
    uint32_t b;
    memcpy(&b, &scale_in, sizeof b);
    const uint32_t ex = b >> 23, man = b & 0x7fffffu;
    if (ex == 255) return FGQ_ERR_ARG;
    if (ex > 0) {
      if (man != 0) return FGQ_ERR_ARG;
      E = (int)ex - 127;
    } else {
      if (man & (man - 1)) return FGQ_ERR_ARG;
      E = -149 + (31 - __builtin_clz(man));
    }
  }
  if (n == 0) return FGQ_OK;
  if (!x || !q || (derive && !scale_out)) return FGQ_ERR_ARG;
  if ((reinterpret_cast<uintptr_t>(x) & 15) || (reinterpret_cast<uintptr_t>(q) & 15) ||
      (scale_out && (reinterpret_cast<uintptr_t>(scale_out) & 3)))
    return FGQ_ERR_ALIGN;
  uint32_t* scratch = nullptr;
  if (derive) {
    if (quantize_workspace_bytes(n) > sizeof(uint32_t) * (size_t)kNoallocScratchWords) return FGQ_ERR_UNSUPPORTED;
    scratch = noalloc_scratch();
    if (!scratch) return FGQ_ERR_CUDA;
  }
  return launch_quantize(x, n, type, E, derive, q, scale_out, scratch, device_error_word(), stream);
}
