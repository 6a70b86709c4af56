// Operand preparation for the tensor-core kernels (device side): the activation codes and
// the ternary codes turned into the MMA operand types, 16 elements at a time.  sm_103a has no
// integer tcgen05 MMA; 8- and 4-bit codes are exact in fp16, 4-bit codes also in e4m3, and
// the ternary codes {0, +1, -1} in both.
#pragma once

#include <cstdint>

#include "tc_common.cuh"

namespace fgq {
namespace prep {

// 16 activation codes -> 16 fp16 integers (NHWC order kept).  8-bit: w holds 16 bytes;
// 4-bit: w[0], w[1] hold 16 nibbles, element 2i in the low nibble of byte i.  Signed codes are
// offset to unsigned and the offset subtracted in fp16 (1024 + v - bias, exact).
template <int ABITS, bool SIGNED>
__device__ __forceinline__ void f16x16(uint32_t (&w)[4], uint4& o0, uint4& o1) {
  if (ABITS == 8) {
    if (SIGNED) {
#pragma unroll
      for (int q = 0; q < 4; ++q) w[q] ^= 0x80808080u;
    }
  } else {
    const uint32_t x2[2] = {w[0], w[1]};
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      // 8 nibbles -> 8 bytes (element order preserved)
      const uint32_t x = x2[q];
      const uint32_t lo = (x & 0x000f000fu) | ((x & 0x00f000f0u) << 4);                // e0 e1 e4 e5
      const uint32_t hi = ((x >> 8) & 0x000f000fu) | (((x >> 8) & 0x00f000f0u) << 4);  // e2 e3 e6 e7
      w[2 * q] = (lo & 0xffffu) | ((hi & 0xffffu) << 16);                               // e0 e1 e2 e3
      w[2 * q + 1] = (lo >> 16) | (hi & 0xffff0000u);                                   // e4 e5 e6 e7
      if (SIGNED) {
        w[2 * q] ^= 0x08080808u;
        w[2 * q + 1] ^= 0x08080808u;
      }
    }
  }
  constexpr uint32_t bias2 =
      ABITS == 8 ? (SIGNED ? 0x64806480u : 0x64006400u) : (SIGNED ? 0x64086408u : 0x64006400u);
  o0.x = tc::u8pair_to_h2(w[0], 0x4140, bias2); o0.y = tc::u8pair_to_h2(w[0], 0x4342, bias2);
  o0.z = tc::u8pair_to_h2(w[1], 0x4140, bias2); o0.w = tc::u8pair_to_h2(w[1], 0x4342, bias2);
  o1.x = tc::u8pair_to_h2(w[2], 0x4140, bias2); o1.y = tc::u8pair_to_h2(w[2], 0x4342, bias2);
  o1.z = tc::u8pair_to_h2(w[3], 0x4140, bias2); o1.w = tc::u8pair_to_h2(w[3], 0x4342, bias2);
}

// 16 packed 4-bit activation codes (8 bytes, element 2i in the low nibble of byte i) -> 16
// e4m3 bytes in element order.  Every 4-bit value is exact in e4m3: 0 -> 0x00, 1 -> 0x38 (1.0),
// n = 2^e (1 + f/8) -> (e + 7) << 3 | f; negative s4 values carry the sign bit.  The 16-entry
// table is looked up with byte permutes (low and high half of the table, chosen per byte by
// the value's bit 3).
template <bool SIGNED>
__device__ __forceinline__ uint4 e4m3x16(uint32_t x0, uint32_t x1) {
  constexpr uint32_t T0 = 0x44403800u, T1 = 0x4E4C4A48u;       // 0 .. 7
  constexpr uint32_t T2 = SIGNED ? 0xCACCCED0u : 0x53525150u;  // 8 .. 11 (s4: -8 .. -5)
  constexpr uint32_t T3 = SIGNED ? 0xB8C0C4C8u : 0x57565554u;  // 12 .. 15 (s4: -4 .. -1)
  const uint32_t xs[2] = {x0, x1};
  uint32_t o[4];
#pragma unroll
  for (int q = 0; q < 2; ++q) {
    const uint32_t x = xs[q];
    const uint32_t lo = (x & 0x000f000fu) | ((x & 0x00f000f0u) << 4);                // e0 e1 e4 e5
    const uint32_t hi = ((x >> 8) & 0x000f000fu) | (((x >> 8) & 0x00f000f0u) << 4);  // e2 e3 e6 e7
    const uint32_t bw[2] = {(lo & 0xffffu) | ((hi & 0xffffu) << 16), (lo >> 16) | (hi & 0xffff0000u)};
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const uint32_t b = bw[h];  // four values 0 .. 15, one per byte
      const uint32_t sel = (b & 7u) | ((b >> 4) & 0x70u) | ((b >> 8) & 0x700u) | ((b >> 12) & 0x7000u);
      const uint32_t vlo = __byte_perm(T0, T1, sel), vhi = __byte_perm(T2, T3, sel);
      const uint32_t mask = ((b >> 3) & 0x01010101u) * 0xffu;
      o[2 * q + h] = (vhi & mask) | (vlo & ~mask);
    }
  }
  return make_uint4(o[0], o[1], o[2], o[3]);
}

// One layer's activations as the source of an expansion: the NHWC tensor, or -- for a 1x1
// unpadded convolution with stride > 1 -- only the pixels it reads, gathered into [P][C].
struct ActSrc {
  const uint8_t* act;
  int abits;    // 8 or 4
  int sgn;      // signed codes
  int strided;  // gather the strided pixels
  int H, W, C, Ho, Wo, stride;
  int64_t nchunks;  // 16-element chunks of the expanded tensor
};

inline ActSrc act_src(const void* act, const Geom& g) {
  ActSrc s;
  s.act = static_cast<const uint8_t*>(act);
  s.abits = (g.act_type == FGQ_U4 || g.act_type == FGQ_S4) ? 4 : 8;
  s.sgn = (g.act_type == FGQ_S8 || g.act_type == FGQ_S4) ? 1 : 0;
  s.strided = (g.R == 1 && g.S == 1 && g.pad == 0 && g.stride > 1) ? 1 : 0;
  s.H = g.H;
  s.W = g.W;
  s.C = g.C;
  s.Ho = g.Ho;
  s.Wo = g.Wo;
  s.stride = g.stride;
  s.nchunks = (s.strided ? g.P * g.C : (int64_t)g.B * g.H * g.W * g.C) / 16;
  return s;
}

// Source chunk of expanded chunk i (16 consecutive channels of one pixel).
__device__ __forceinline__ int64_t src_chunk(const ActSrc& s, int64_t i) {
  if (!s.strided) return i;
  const int cpp = s.C / 16;
  const int64_t p = i / cpp;
  const int c = (int)(i - p * cpp);
  const int wo = (int)(p % s.Wo);
  const int64_t q = p / s.Wo;
  const int ho = (int)(q % s.Ho);
  const int64_t b = q / s.Ho;
  return ((b * s.H + (int64_t)ho * s.stride) * s.W + (int64_t)wo * s.stride) * cpp + c;
}

// Expanded chunk i as fp16 (32 bytes at out + 2 i).
__device__ __forceinline__ void act_f16(const ActSrc& s, int64_t i, uint4* out) {
  const int64_t src = src_chunk(s, i);
  uint32_t w[4];
  uint4 o0, o1;
  if (s.abits == 8) {
    const uint4 v = __ldg(reinterpret_cast<const uint4*>(s.act) + src);
    w[0] = v.x; w[1] = v.y; w[2] = v.z; w[3] = v.w;
    if (s.sgn) f16x16<8, true>(w, o0, o1);
    else f16x16<8, false>(w, o0, o1);
  } else {
    const uint2 v = __ldg(reinterpret_cast<const uint2*>(s.act) + src);
    w[0] = v.x; w[1] = v.y; w[2] = 0u; w[3] = 0u;
    if (s.sgn) f16x16<4, true>(w, o0, o1);
    else f16x16<4, false>(w, o0, o1);
  }
  out[2 * i] = o0;
  out[2 * i + 1] = o1;
}

// Expanded chunk i of 4-bit codes as e4m3 (16 bytes at out + i).
__device__ __forceinline__ void act_e4m3(const ActSrc& s, int64_t i, uint4* out) {
  const uint2 v = __ldg(reinterpret_cast<const uint2*>(s.act) + src_chunk(s, i));
  out[i] = s.sgn ? e4m3x16<true>(v.x, v.y) : e4m3x16<false>(v.x, v.y);
}

// Expanded chunks first, first + step, ... of the activations (fp16, or e4m3 when F8):
// four chunks' source loads are issued before any is converted, so that each thread keeps
// four independent loads in flight (a single load per thread and iteration left these
// streaming loops bound by the load latency).
template <bool F8>
__device__ __forceinline__ void act_expand(const ActSrc& s, int64_t first, int64_t step, uint4* out) {
  constexpr int U = 4;
  int64_t i = first;
  for (; i + (U - 1) * step < s.nchunks; i += U * step) {
    uint4 v[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int64_t src = src_chunk(s, i + u * step);
      if (s.abits == 8) {
        v[u] = __ldg(reinterpret_cast<const uint4*>(s.act) + src);
      } else {
        const uint2 h = __ldg(reinterpret_cast<const uint2*>(s.act) + src);
        v[u] = make_uint4(h.x, h.y, 0u, 0u);
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int64_t c = i + u * step;
      if (F8) {
        out[c] = s.sgn ? e4m3x16<true>(v[u].x, v[u].y) : e4m3x16<false>(v[u].x, v[u].y);
      } else {
        uint32_t w[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
        uint4 o0, o1;
        if (s.abits == 8) {
          if (s.sgn) f16x16<8, true>(w, o0, o1);
          else f16x16<8, false>(w, o0, o1);
        } else {
          if (s.sgn) f16x16<4, true>(w, o0, o1);
          else f16x16<4, false>(w, o0, o1);
        }
        out[2 * c] = o0;
        out[2 * c + 1] = o1;
      }
    }
  }
  for (; i < s.nchunks; i += step) {
    if (F8) act_e4m3(s, i, out);
    else act_f16(s, i, out);
  }
}

// One code word (16 two-bit codes: 00 = 0, 01 = +1, 11 = -1) as 16 fp16 (32 bytes at
// out + 2 i) or 16 e4m3 (16 bytes at out + i: 0x00, 0x38, 0xB8).
__device__ __forceinline__ void codes_f16(const uint32_t* codes, int64_t i, uint4* out) {
  const uint32_t w = __ldg(codes + i);
  uint32_t h[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) {
    const uint32_t c0 = (w >> (4 * e)) & 3u, c1 = (w >> (4 * e + 2)) & 3u;
    const uint32_t lo = (c0 & 1u) ? ((c0 & 2u) ? 0xBC00u : 0x3C00u) : 0u;
    const uint32_t hi = (c1 & 1u) ? ((c1 & 2u) ? 0xBC00u : 0x3C00u) : 0u;
    h[e] = lo | (hi << 16);
  }
  out[2 * i] = make_uint4(h[0], h[1], h[2], h[3]);
  out[2 * i + 1] = make_uint4(h[4], h[5], h[6], h[7]);
}

__device__ __forceinline__ void codes_e4m3(const uint32_t* codes, int64_t i, uint4* out) {
  const uint32_t w = __ldg(codes + i);
  uint32_t o[4];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    uint32_t v = 0;
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const uint32_t c = (w >> (2 * (4 * q + e))) & 3u;
      v |= (((c & 1u) ? 0x38u : 0u) | ((c & 2u) << 6)) << (8 * e);
    }
    o[q] = v;
  }
  out[i] = make_uint4(o[0], o[1], o[2], o[3]);
}

// Blocks of 256 threads for n work items: up to a full device (8 blocks of 256 threads per
// SM), each thread looping.
inline int blocks_for(int64_t n) {
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t want = (n + 255) / 256;
  return (int)(want < 8LL * sms ? (want > 0 ? want : 1) : 8LL * sms);
}

}  // namespace prep
}  // namespace fgq
