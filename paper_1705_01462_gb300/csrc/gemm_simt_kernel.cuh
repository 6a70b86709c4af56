// CUDA-core grouped ternary contraction (Eq. 2 on a convolution or fully connected layer,
// 32-bit group accumulators of Section 4, one multiply per group as counted in Section 4.1).
//
// For each group of G weights (G a multiple of 4) the int32 group sum is a chain of G/4
// dp4a instructions over int8x4 activation words and int8x4 code words expanded from the
// 2-bit codes; the sum is then scaled by alpha into an fp32 accumulator.  The dp4a chain
// starts at the bit pattern of 1.5*2^23, so its int32 result reads directly as the fp32
// number 1.5*2^23 + s and one fp32 add recovers s exactly (no int->fp32 conversion
// instruction).  Per (filter, position, group): one dp4a per 4 weights (FMA-heavy pipe)
// plus one fp32 add and one fp32 FMA, which the heavy and lite FMA pipes share.
//
// Tiling: a 256-thread block computes 64 filters x 128 output positions; each thread owns
// 4 filters x 8 positions.  The reduction axis is staged through shared memory in chunks
// of max(16, G/4) words: activation words gathered from the implicit im2col (zero outside
// the image), code words expanded through a 256-entry byte table, and the chunk's alphas.
// The next chunk's global loads are issued into registers before the current chunk's
// math (double-buffered shared tiles, one barrier per chunk).
//
// The same kernel runs the dense 8-bit-weight first layer (int32 dot product over the
// whole row, scaled once at the end) and can write the raw int32 group sums.
//
// This header holds the tiled kernel and its launcher template; gemm_simt_g*.cu instantiate
// them per group size and gemm_simt.cu dispatches.
#pragma once

#include <cstdint>

#include "fgq_device.cuh"

namespace fgq {
namespace {

constexpr int BM = 64;    // filters per block
constexpr int BP = 128;   // positions per block
constexpr int NT = 256;   // threads per block

// Per-thread view of one output position for the im2col gather.
struct PosInfo {
  int valid;
  int b, hb, wb;  // image, and the input row/col of tap (0, 0): ho*stride - pad, wo*stride - pad
};

__device__ __forceinline__ PosInfo pos_info(const Geom& g, int64_t p) {
  PosInfo pi;
  pi.valid = p < g.P;
  if (!pi.valid) p = 0;
  const int wo = (int)(p % g.Wo);
  const int64_t t = p / g.Wo;
  const int ho = (int)(t % g.Ho);
  pi.b = (int)(t / g.Ho);
  pi.hb = ho * g.stride - g.pad;
  pi.wb = wo * g.stride - g.pad;
  return pi;
}

// Element offset of reduction index k (k < Kred) for position pi in conv group gi, or -1
// if it falls in the zero padding.
__device__ __forceinline__ int64_t act_elem(const Geom& g, const PosInfo& pi, int gi, int k) {
  const int tap = k / g.Cg;
  const int c = k - tap * g.Cg;
  const int r = tap / g.S;
  const int s = tap - r * g.S;
  const int hi = pi.hb + r, wi = pi.wb + s;
  if (hi < 0 || hi >= g.H || wi < 0 || wi >= g.W) return -1;
  return (((int64_t)pi.b * g.H + hi) * g.W + wi) * g.C + (int64_t)gi * g.Cg + c;
}

// One activation element as a byte lane (8-bit types: the byte; 4-bit types: the nibble,
// sign-extended for S4).
__device__ __forceinline__ uint32_t act_byte(const uint8_t* act, int type, int64_t e) {
  if (e < 0) return 0;
  if (type == FGQ_U8 || type == FGQ_S8) return act[e];
  uint32_t nib = (act[e >> 1] >> (4 * (e & 1))) & 0xfu;
  if (type == FGQ_S4) nib = (uint32_t)(((int)nib ^ 8) - 8) & 0xffu;
  return nib;
}

// Four consecutive reduction elements k..k+3 as an int8x4 word.
// mode 0: 8-bit, 4-byte aligned word within one tap; 1: 4-bit, 2-byte word within one tap;
// 2: byte-by-byte gather.  (Mode 3, whole 16-byte runs inside one tap, is handled by the
// tiled kernel's staging directly.)
__device__ __forceinline__ uint32_t act_word(const uint8_t* act, const Geom& g, const PosInfo& pi,
                                             int gi, int k, int mode) {
  if (!pi.valid || k >= g.Kred) return 0;
  if (mode == 0) {
    const int64_t e = act_elem(g, pi, gi, k);
    return e < 0 ? 0u : __ldg(reinterpret_cast<const uint32_t*>(act + e));
  }
  if (mode == 1) {
    const int64_t e = act_elem(g, pi, gi, k);
    if (e < 0) return 0u;
    const uint32_t h = __ldg(reinterpret_cast<const uint16_t*>(act + (e >> 1)));
    uint32_t v = (h & 0xfu) | ((h & 0xf0u) << 4) | ((h & 0xf00u) << 8) | ((h & 0xf000u) << 12);
    if (g.act_type == FGQ_S4) v = __vsub4(v ^ 0x08080808u, 0x08080808u);
    return v;
  }
  uint32_t v = 0;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    if (k + i < g.Kred) v |= act_byte(act, g.act_type, act_elem(g, pi, gi, k + i)) << (8 * i);
  }
  return v;
}

#ifndef FGQ_SIMT_MIN_BLOCKS
#define FGQ_SIMT_MIN_BLOCKS 2  // resident blocks per SM the register allocation targets
#endif
#ifndef FGQ_SIMT_PACKED_FP
#define FGQ_SIMT_PACKED_FP 0  // 1: packed fp32x2 add/FMA for the per-group scaling (measured 2-3% slower)
#endif

// Thread layout: tid -> filters 4*(tid % 16) .. +3 and positions {64j + 4*(tid / 16) + e :
// j = 0, 1; e = 0..3}.  Lanes run along the filters, so each 16-byte output store of a warp
// covers two whole 256-byte rows of y; the transposed activation tile As[word][position]
// gives a thread 4 positions per 16-byte shared load.
// Mode 4: the byte gather of mode 2 driven by a per-block table tbl[k] = r | s << 8 | c << 16
// of the reduction index's filter tap and channel (all ones past Kred), built once per block.
__device__ __forceinline__ uint32_t act_word_tbl(const uint8_t* act, const Geom& g, const PosInfo& pi, int gi,
                                                 int k, const uint32_t* tbl) {
  if (!pi.valid) return 0;
  uint32_t v = 0;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const uint32_t e = tbl[k + i];
    if (e == 0xffffffffu) continue;
    const int hi = pi.hb + (int)(e & 0xffu), wi = pi.wb + (int)((e >> 8) & 0xffu);
    if (hi < 0 || hi >= g.H || wi < 0 || wi >= g.W) continue;
    const int64_t el = (((int64_t)pi.b * g.H + hi) * g.W + wi) * g.C + (int64_t)gi * g.Cg + (int)(e >> 16);
    v |= act_byte(act, g.act_type, el) << (8 * i);
  }
  return v;
}

template <int G, bool SA, bool DW, bool SUMS>
__global__ void __launch_bounds__(NT, FGQ_SIMT_MIN_BLOCKS) simt_contract_kernel(const uint8_t* __restrict__ act, const Geom g,
                                                              const void* __restrict__ weights,
                                                              const float* __restrict__ scales,
                                                              const float* __restrict__ act_scale,
                                                              float* __restrict__ out, int32_t* __restrict__ sums,
                                                              int mode, int mtiles) {
  constexpr int KW = (G / 4 > 16) ? G / 4 : 16;  // words (4 elements) per chunk
  constexpr int GPC = DW ? 1 : (KW * 4) / G;     // groups per chunk
  constexpr int WPG = G / 4;                      // words per group
  constexpr int SW = (BP * KW) / NT;              // activation words staged per thread
  constexpr int CW = (BM * (KW / 4) + NT - 1) / NT;  // code words staged per thread
  constexpr int AW = (BM * GPC + NT - 1) / NT;    // alphas staged per thread

  extern __shared__ __align__(16) uint8_t smem_simt[];
  uint32_t (*As)[KW][BP] = reinterpret_cast<uint32_t (*)[KW][BP]>(smem_simt);
  uint32_t (*Ws)[KW][BM] = reinterpret_cast<uint32_t (*)[KW][BM]>(smem_simt + 2 * KW * BP * 4);
  float (*Al)[GPC][BM] = reinterpret_cast<float (*)[GPC][BM]>(smem_simt + 2 * KW * BP * 4 + 2 * KW * BM * 4);
  uint32_t* lut = reinterpret_cast<uint32_t*>(smem_simt + 2 * KW * BP * 4 + 2 * KW * BM * 4 + 2 * GPC * BM * 4);
  uint32_t* ktab = lut + 256;  // mode 4 only: one entry per reduction index of all chunks

  const int tid = threadIdx.x;
  const int ty = tid % 16, tx = tid / 16;
  const int gi = blockIdx.y / mtiles;
  const int mt = blockIdx.y - gi * mtiles;
  const int mlo = gi * g.Mg + mt * BM;
  const int mhi = min(gi * g.Mg + g.Mg, g.M);
  const int64_t p0 = (int64_t)blockIdx.x * BP;

  if (!DW) {
    for (int i = tid; i < 256; i += NT) lut[i] = expand_code_byte((uint32_t)i);
  }
  const int nchunks = (g.Kp + 4 * KW - 1) / (4 * KW);
  if (mode == 4) {
    for (int k = tid; k < nchunks * 4 * KW; k += NT) {
      uint32_t e = 0xffffffffu;
      if (k < g.Kred) {
        const int tap = k / g.Cg, c = k - (k / g.Cg) * g.Cg;
        const int r = tap / g.S, s2 = tap - (tap / g.S) * g.S;
        e = (uint32_t)r | ((uint32_t)s2 << 8) | ((uint32_t)c << 16);
      }
      ktab[k] = e;
    }
    __syncthreads();
  }

  // staging assignment: activations -- one position, SW consecutive words of the chunk
  const int spl = tid % BP;
  const int sw0 = (tid / BP) * SW;
  const PosInfo spi = pos_info(g, p0 + spl);
  const uint32_t* codes = static_cast<const uint32_t*>(weights);
  const int8_t* wq = static_cast<const int8_t*>(weights);

  uint32_t ra[SW];  // prefetched activation words
  uint32_t rc[DW ? (BM * KW + NT - 1) / NT : CW];  // prefetched code words / dense weight words
  float ral[AW];

  auto fetch = [&](int c) {
    const int k0 = c * 4 * KW;
    if (mode == 3) {
      // fast path: this thread's 4*SW elements lie inside one filter tap (C/groups is a
      // multiple of 4*SW) and start 16-byte aligned: one decomposition, 16-byte loads
      const int k = k0 + 4 * sw0;
      int64_t e = -1;
      if (spi.valid && k < g.Kred) e = act_elem(g, spi, gi, k);
#pragma unroll
      for (int i = 0; i < SW; i += 4) {
        uint4 v = make_uint4(0u, 0u, 0u, 0u);
        if (e >= 0) v = __ldg(reinterpret_cast<const uint4*>(act + e) + i / 4);
        ra[i] = v.x; ra[i + 1] = v.y; ra[i + 2] = v.z; ra[i + 3] = v.w;
      }
    } else if (mode == 4) {
#pragma unroll
      for (int i = 0; i < SW; ++i) ra[i] = act_word_tbl(act, g, spi, gi, k0 + 4 * (sw0 + i), ktab);
    } else {
#pragma unroll
      for (int i = 0; i < SW; ++i) ra[i] = act_word(act, g, spi, gi, k0 + 4 * (sw0 + i), mode);
    }
    if (!DW) {
#pragma unroll
      for (int r = 0; r < CW; ++r) {
        const int idx = tid + r * NT;
        const int ml = idx % BM, cw = idx / BM;
        const int m = mlo + ml, wi = k0 / 16 + cw;
        rc[r] = (idx < BM * (KW / 4) && m < mhi && wi < g.wrow) ? __ldg(codes + (int64_t)m * g.wrow + wi) : 0u;
      }
      if (!SUMS) {
#pragma unroll
        for (int r = 0; r < AW; ++r) {
          const int idx = tid + r * NT;
          const int ml = idx % BM, gl = idx / BM;
          const int m = mlo + ml, gg = c * GPC + gl;
          ral[r] = (idx < BM * GPC && m < mhi && gg < g.ng) ? __ldg(scales + (int64_t)m * g.ng + gg) : 0.0f;
        }
      }
    } else {
#pragma unroll
      for (int r = 0; r < (BM * KW + NT - 1) / NT; ++r) {
        const int idx = tid + r * NT;
        const int ml = idx % BM, kw = idx / BM;
        const int m = mlo + ml;
        uint32_t v = 0;
        if (idx < BM * KW && m < mhi) {
#pragma unroll
          for (int b = 0; b < 4; ++b) {
            const int k = k0 + 4 * kw + b;
            if (k < g.Kred) v |= ((uint32_t)(uint8_t)wq[(int64_t)m * g.Kred + k]) << (8 * b);
          }
        }
        rc[r] = v;
      }
    }
  };
  auto stash = [&](int buf) {
#pragma unroll
    for (int i = 0; i < SW; ++i) As[buf][sw0 + i][spl] = ra[i];
    if (!DW) {
#pragma unroll
      for (int r = 0; r < CW; ++r) {
        const int idx = tid + r * NT;
        if (idx < BM * (KW / 4)) {
          const int ml = idx % BM, cw = idx / BM;
#pragma unroll
          for (int b = 0; b < 4; ++b) Ws[buf][cw * 4 + b][ml] = lut[(rc[r] >> (8 * b)) & 0xffu];
        }
      }
      if (!SUMS) {
#pragma unroll
        for (int r = 0; r < AW; ++r) {
          const int idx = tid + r * NT;
          if (idx < BM * GPC) Al[buf][idx / BM][idx % BM] = ral[r];
        }
      }
    } else {
#pragma unroll
      for (int r = 0; r < (BM * KW + NT - 1) / NT; ++r) {
        const int idx = tid + r * NT;
        if (idx < BM * KW) Ws[buf][idx / BM][idx % BM] = rc[r];
      }
    }
  };

  float acc[4][8];
  int iacc[4][8];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      acc[i][j] = 0.0f;
      iacc[i][j] = 0;
    }

  fetch(0);
  __syncthreads();  // lut ready
  stash(0);
  __syncthreads();

  for (int c = 0; c < nchunks; ++c) {
    const int buf = c & 1;
    if (c + 1 < nchunks) fetch(c + 1);  // global loads in flight during this chunk's math

    if (DW) {
#pragma unroll 4
      for (int kw = 0; kw < KW; ++kw) {
        const uint4 bw = *reinterpret_cast<const uint4*>(&Ws[buf][kw][ty * 4]);
        const uint32_t bv[4] = {bw.x, bw.y, bw.z, bw.w};
        const uint4 a0 = *reinterpret_cast<const uint4*>(&As[buf][kw][4 * tx]);
        const uint4 a1 = *reinterpret_cast<const uint4*>(&As[buf][kw][64 + 4 * tx]);
        const uint32_t a[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
          for (int j = 0; j < 8; ++j) iacc[i][j] = SA ? dp4a_ss(a[j], bv[i], iacc[i][j]) : dp4a_us(a[j], bv[i], iacc[i][j]);
      }
    } else {
#pragma unroll 2
      for (int gl = 0; gl < GPC; ++gl) {
        int sm[4][8];
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
          for (int j = 0; j < 8; ++j) sm[i][j] = kMagicI;
#pragma unroll
        for (int wv = 0; wv < WPG; ++wv) {
          const int kw = gl * WPG + wv;
          const uint4 bw = *reinterpret_cast<const uint4*>(&Ws[buf][kw][ty * 4]);
          const uint32_t bv[4] = {bw.x, bw.y, bw.z, bw.w};
          const uint4 a0 = *reinterpret_cast<const uint4*>(&As[buf][kw][4 * tx]);
          const uint4 a1 = *reinterpret_cast<const uint4*>(&As[buf][kw][64 + 4 * tx]);
          const uint32_t a[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
#pragma unroll
          for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int j = 0; j < 8; ++j) sm[i][j] = SA ? dp4a_ss(a[j], bv[i], sm[i][j]) : dp4a_us(a[j], bv[i], sm[i][j]);
        }
        if (SUMS) {
          const int gg = c * GPC + gl;
          if (gg < g.ng) {
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              const int m = mlo + ty * 4 + i;
              if (m >= mhi) continue;
#pragma unroll
              for (int j = 0; j < 8; ++j) {
                const int64_t p = p0 + 64 * (j / 4) + 4 * tx + (j % 4);
                if (p < g.P) sums[((int64_t)m * g.ng + gg) * g.P + p] = sm[i][j] - kMagicI;
              }
            }
          }
        } else {
          const float4 al4 = *reinterpret_cast<const float4*>(&Al[buf][gl][ty * 4]);
          const float al[4] = {al4.x, al4.y, al4.z, al4.w};
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            if (FGQ_SIMT_PACKED_FP) {
              const unsigned long long negc = pack_f2(-kMagicF, -kMagicF);
              const unsigned long long a2 = pack_f2(al[i], al[i]);
#pragma unroll
              for (int j = 0; j < 8; j += 2) {
                const unsigned long long s2 =
                    add_f2(pack_f2(__int_as_float(sm[i][j]), __int_as_float(sm[i][j + 1])), negc);
                unsigned long long c2 = pack_f2(acc[i][j], acc[i][j + 1]);
                c2 = fma_f2(a2, s2, c2);
                unpack_f2(c2, acc[i][j], acc[i][j + 1]);
              }
            } else {
#pragma unroll
              for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(al[i], __int_as_float(sm[i][j]) - kMagicF, acc[i][j]);
            }
          }
        }
      }
    }

    if (c + 1 < nchunks) stash(buf ^ 1);
    __syncthreads();
  }

  if (SUMS) return;
  const float sx = __ldg(act_scale);
  const int m = mlo + ty * 4;
  const bool vec = (g.M % 4 == 0) && (m + 3 < mhi);
  if (g.rq_out) {  // fused requantization: 8-bit codes instead of fp32
    const RqMul r = rq_mul(g.rq_scale, g.rq_signed);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int64_t p = p0 + 64 * (j / 4) + 4 * tx + (j % 4);
      if (p >= g.P) continue;
      uint32_t b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i)
        b[i] = rq_code(DW ? sx * __ldg(scales + min(m + i, g.M - 1)) * (float)iacc[i][j] : sx * acc[i][j], r);
      uint8_t* orow = g.rq_out + p * g.M;
      if (vec) {
        *reinterpret_cast<uint32_t*>(orow + m) = b[0] | (b[1] << 8) | (b[2] << 16) | (b[3] << 24);
      } else {
#pragma unroll
        for (int i = 0; i < 4; ++i)
          if (m + i < mhi) orow[m + i] = (uint8_t)b[i];
      }
    }
    return;
  }
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const int64_t p = p0 + 64 * (j / 4) + 4 * tx + (j % 4);
    if (p >= g.P) continue;
    float v[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) v[i] = DW ? sx * __ldg(scales + min(m + i, g.M - 1)) * (float)iacc[i][j] : sx * acc[i][j];
    float* orow = out + p * g.M;
    if (vec) {
      *reinterpret_cast<float4*>(orow + m) = make_float4(v[0], v[1], v[2], v[3]);
    } else {
#pragma unroll
      for (int i = 0; i < 4; ++i)
        if (m + i < mhi) orow[m + i] = v[i];
    }
  }
}

template <int G, bool DW>
constexpr size_t simt_smem_bytes() {
  constexpr int KW = (G / 4 > 16) ? G / 4 : 16;
  constexpr int GPC = DW ? 1 : (KW * 4) / G;
  return (size_t)2 * KW * BP * 4 + 2 * KW * BM * 4 + 2 * GPC * BM * 4 + 256 * 4;
}

template <int G, bool SA, bool DW, bool SUMS>
void launch_one(const void* act, const Geom& g, const void* w, const float* sc, const float* as, float* out,
                int32_t* sums, int mode, cudaStream_t s) {
  constexpr int KW = (G / 4 > 16) ? G / 4 : 16;
  const size_t nk = (size_t)((g.Kp + 4 * KW - 1) / (4 * KW)) * 4 * KW;
  const size_t smem = simt_smem_bytes<G, DW>() + (mode == 4 ? 4 * nk : 0);
  static int attr_set = 0;
  if (attr_set < (int)smem) {
    cudaFuncSetAttribute(simt_contract_kernel<G, SA, DW, SUMS>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         (int)(smem > 48 * 1024 ? smem : 48 * 1024));
    attr_set = (int)(smem > 48 * 1024 ? smem : 48 * 1024);
  }
  const int mtiles = (g.Mg + BM - 1) / BM;
  dim3 grid((unsigned)((g.P + BP - 1) / BP), (unsigned)(mtiles * g.groups));
  simt_contract_kernel<G, SA, DW, SUMS><<<grid, NT, smem, s>>>(static_cast<const uint8_t*>(act), g, w, sc, as, out,
                                                               sums, mode, mtiles);
}

}  // namespace

// Launchers of the tiled kernel, one translation unit per set of group sizes (the kernel
// has 26 instantiations; spread over several files they compile in parallel).  Each
// returns false for a G it does not hold.
bool simt_launch_g4(bool sa, bool sums, const void* act, const Geom& g, const void* w, const float* sc,
                    const float* as, float* out, int32_t* sums_out, int mode, cudaStream_t s);
bool simt_launch_g8_16(bool sa, bool sums, const void* act, const Geom& g, const void* w, const float* sc,
                       const float* as, float* out, int32_t* sums_out, int mode, cudaStream_t s);
bool simt_launch_g32_64(bool sa, bool sums, const void* act, const Geom& g, const void* w, const float* sc,
                        const float* as, float* out, int32_t* sums_out, int mode, cudaStream_t s);
bool simt_launch_g128(bool sa, bool sums, const void* act, const Geom& g, const void* w, const float* sc,
                      const float* as, float* out, int32_t* sums_out, int mode, cudaStream_t s);
// The dense 8-bit-weight mode (G = 4 tiling, one scale per filter).
void simt_launch_dense(bool sa, const void* act, const Geom& g, const void* w, const float* sc, const float* as,
                       float* out, int mode, cudaStream_t s);

}  // namespace fgq
