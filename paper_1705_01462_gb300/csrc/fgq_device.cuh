// Device-side helpers shared by the libfgq kernels.
#pragma once

#include <cstdint>
#include <utility>

#include "fgq_internal.h"

namespace fgq {

constexpr unsigned FULL_MASK = 0xffffffffu;

__device__ __forceinline__ void record_error(unsigned int* err, unsigned code) {
  if (err) atomicCAS(err, 0u, code);
}

// 2^k as fp32 bits for k in [-149, 127] (subnormal for k < -126).
__device__ __forceinline__ float pow2f(int k) {
  return k >= -126 ? __uint_as_float((uint32_t)(k + 127) << 23) : __uint_as_float(1u << (k + 149));
}

// 2^k as fp64 for k in [-1022, 1023].
__device__ __forceinline__ double pow2d(int k) {
  return __longlong_as_double((long long)(k + 1023) << 52);
}

// u8 x s8 dot product of four lanes plus c (PTX dp4a.u32.s32).
__device__ __forceinline__ int dp4a_us(uint32_t a, uint32_t b, int c) {
  int d;
  asm("dp4a.u32.s32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
  return d;
}

// s8 x s8 dot product of four lanes plus c.
__device__ __forceinline__ int dp4a_ss(uint32_t a, uint32_t b, int c) {
  int d;
  asm("dp4a.s32.s32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
  return d;
}

// Packed fp32x2 helpers (sm_100+ f32x2 arithmetic).
__device__ __forceinline__ unsigned long long pack_f2(float lo, float hi) {
  unsigned long long r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void unpack_f2(unsigned long long v, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ unsigned long long add_f2(unsigned long long a, unsigned long long b) {
  unsigned long long r;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ unsigned long long fma_f2(unsigned long long a, unsigned long long b,
                                                     unsigned long long c) {
  unsigned long long r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
  return r;
}

// Integer dot-product results are read back as fp32 without a conversion instruction:
// the accumulator starts at the bit pattern of 1.5 * 2^23, so for |s| < 2^22 the int32
// result's bits are the fp32 number 1.5 * 2^23 + s, and subtracting 1.5 * 2^23 (exact)
// gives s as fp32.
constexpr int kMagicI = 0x4B400000;
constexpr float kMagicF = 12582912.0f;

// Expansion of one code byte (four 2-bit codes, 00 -> 0, 01 -> +1, 11 -> -1) to four int8
// lanes, lane i from bits 2i, 2i+1.
__host__ __device__ constexpr uint32_t expand_code_byte(uint32_t b) {
  uint32_t r = 0;
  for (int i = 0; i < 4; ++i) {
    uint32_t c = (b >> (2 * i)) & 3u;
    uint32_t v = c == 1u ? 0x01u : (c == 3u ? 0xffu : 0x00u);
    r |= v << (8 * i);
  }
  return r;
}

// Fused output requantization (Section 4: the 32-bit outputs are converted to 8 bits and
// rounded before they are passed to the next layer): q = clamp(round_half_even(v * 2^-E),
// qmin, qmax) for the output scale 2^E, the rule of the activation quantizer; the two
// multipliers keep 2^-E representable for every E in [-149, 127].
struct RqMul {
  float m1, m2;
  int qmin, qmax;
};
__device__ __forceinline__ RqMul rq_mul(const float* scale, int is_signed) {
  const int E = ilogbf(__ldg(scale));
  RqMul r;
  r.m1 = (-E <= 127) ? pow2f(-E) : pow2f(64);
  r.m2 = (-E <= 127) ? 1.0f : pow2f(-E - 64);
  r.qmin = is_signed ? -128 : 0;
  r.qmax = is_signed ? 127 : 255;
  return r;
}
__device__ __forceinline__ uint8_t rq_code(float v, const RqMul& r) {
  int x = __float2int_rn(v * r.m1 * r.m2);
  x = max(r.qmin, min(r.qmax, x));
  return (uint8_t)(x & 0xff);
}

// Programmatic dependent launch: a kernel launched by launch_pdl may be scheduled while the
// kernel before it on the stream is still running (once every block of that kernel has
// called pdl_trigger or exited).  It must call pdl_wait -- which returns when the previous
// kernel has completed and its memory operations are visible -- before it reads or writes
// any global memory; what comes before (barrier initialisation, tensor-memory allocation,
// descriptor prefetch) overlaps the previous kernel's tail.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                       Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

}  // namespace fgq
