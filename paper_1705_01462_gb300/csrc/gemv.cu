// Grouped ternary contraction for a few activation rows (P <= 8): fully connected layers
// at small batch, where every weight byte streams from HBM once and does little work.
// Math as the other contraction kernels (Eq. 2 with the 32-bit group accumulators of
// Section 4): s[m][g][p] = dp4a group sums, y[p][m] = s_x * sum_g alpha[m][g] s[m][g][p].
//
// One warp per filter row.  Lanes take consecutive code words (G < 16: each word holds
// 16 / G groups) or consecutive groups (G >= 16: G / 16 words each), so code, alpha and
// activation loads coalesce; each lane keeps its partial sums in registers and a fixed
// shuffle tree adds the lanes.  Alphas are fp32 [M][ng] (fp32 accumulation, like the
// tiled kernels) or fixed point (Section 4: 8-bit or 4-bit codes a[m][g] with one scale
// 2^E_m per row): then sum_g a_g * s_g is accumulated exactly in int64 and
// y = s_x * 2^E_m * sum, one rounding.  8-bit activations, Kred a multiple of 16.
#include <cstdint>

#include "fgq_device.cuh"

namespace fgq {
namespace {

constexpr int GV_WARPS = 8;
constexpr int GV_MAXP = 8;

__device__ __forceinline__ int dp4a_s(uint32_t a, uint32_t b, int c, bool sa) {
  int d;
  if (sa)
    asm("dp4a.s32.s32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
  else
    asm("dp4a.u32.s32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
  return d;
}

// alpha of group g of row m: fp32, or the fixed-point code (8-bit bytes; 4-bit nibbles,
// element 2i in the low nibble)
template <int QA>
__device__ __forceinline__ int alpha_code(const uint8_t* aq, int64_t rowbytes, int m, int g) {
  if (QA == 8) return __ldg(aq + (int64_t)m * rowbytes + g);
  const uint8_t b = __ldg(aq + (int64_t)m * rowbytes + g / 2);
  return (g & 1) ? (b >> 4) : (b & 0xf);
}

template <int G, bool SIGNED, int QA>
__global__ void __launch_bounds__(32 * GV_WARPS) gemv_kernel(const uint8_t* __restrict__ q, int P, int Kred, int M,
                                                             const uint32_t* __restrict__ codes,
                                                             const float* __restrict__ alpha,
                                                             const uint8_t* __restrict__ aq,
                                                             const float* __restrict__ ascale,
                                                             const float* __restrict__ act_scale,
                                                             float* __restrict__ y, uint8_t* __restrict__ rq_out,
                                                             const float* __restrict__ rq_scale, int rq_signed) {
  __shared__ uint32_t lut[256];  // byte of 4 codes -> 4 int8 weights
  for (int i = threadIdx.x; i < 256; i += blockDim.x) {
    uint32_t v = 0;
    for (int e = 0; e < 4; ++e) {
      const uint32_t c = (i >> (2 * e)) & 3u;
      v |= (c == 1u ? 0x01u : (c == 3u ? 0xffu : 0u)) << (8 * e);
    }
    lut[i] = v;
  }
  __syncthreads();
  const int m = blockIdx.x * GV_WARPS + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (m >= M) return;
  const int ng = (Kred + G - 1) / G;
  const int wrow = (ng * G + 15) / 16;
  const int kw = Kred / 16;  // code words that hold real elements
  const uint32_t* crow = codes + (int64_t)m * wrow;
  const int64_t arb = QA == 8 ? ng : (ng + 1) / 2;
  float acc[GV_MAXP];
  long long iacc[GV_MAXP];
#pragma unroll
  for (int p = 0; p < GV_MAXP; ++p) {
    acc[p] = 0.0f;
    iacc[p] = 0;
  }
  // the group sums of one 16-element word w for every position, folded into the
  // accumulators of group gofs + (element / G) (G < 16) or added to s (G >= 16)
  auto word = [&](int w, int (&s)[GV_MAXP]) {
    const uint32_t cw = __ldg(crow + w);
    const uint32_t wt[4] = {lut[cw & 0xffu], lut[(cw >> 8) & 0xffu], lut[(cw >> 16) & 0xffu], lut[cw >> 24]};
#pragma unroll
    for (int p = 0; p < GV_MAXP; ++p) {
      if (p >= P) break;
      const uint4 a = __ldg(reinterpret_cast<const uint4*>(q + (int64_t)p * Kred) + w);
      const uint32_t av[4] = {a.x, a.y, a.z, a.w};
      if (G >= 16) {
        int t = s[p];
#pragma unroll
        for (int b = 0; b < 4; ++b) t = dp4a_s(av[b], wt[b], t, SIGNED);
        s[p] = t;
      } else {
        constexpr int GPW = 16 / (G < 4 ? 4 : G);  // groups in the word (G = 4 or 8)
        constexpr int WPG = (G < 4 ? 4 : G) / 4;   // 4-element words per group
#pragma unroll
        for (int gg = 0; gg < GPW; ++gg) {
          int t = 0;
#pragma unroll
          for (int b = 0; b < WPG; ++b) t = dp4a_s(av[gg * WPG + b], wt[gg * WPG + b], t, SIGNED);
          const int g = w * GPW + gg;
          if (QA)
            iacc[p] += (long long)alpha_code<QA>(aq, arb, m, g) * t;
          else
            acc[p] = fmaf(__ldg(alpha + (int64_t)m * ng + g), (float)t, acc[p]);
        }
      }
    }
  };
  if (G < 16) {
    for (int w = lane; w < kw; w += 32) {
      int dummy[GV_MAXP];
      word(w, dummy);
    }
  } else {
    constexpr int WPG = G / 16;  // words per group
    for (int g = lane; g < ng; g += 32) {
      int s[GV_MAXP];
#pragma unroll
      for (int p = 0; p < GV_MAXP; ++p) s[p] = 0;
      for (int c = 0; c < WPG; ++c) {
        const int w = g * WPG + c;
        if (w < kw) word(w, s);  // padding words hold zero codes and no elements
      }
#pragma unroll
      for (int p = 0; p < GV_MAXP; ++p) {
        if (p >= P) break;
        if (QA)
          iacc[p] += (long long)alpha_code<QA>(aq, arb, m, g) * s[p];
        else
          acc[p] = fmaf(__ldg(alpha + (int64_t)m * ng + g), (float)s[p], acc[p]);
      }
    }
  }
  // fixed shuffle tree over the lanes
#pragma unroll
  for (int p = 0; p < GV_MAXP; ++p) {
    for (int o = 16; o > 0; o >>= 1) {
      if (QA)
        iacc[p] += __shfl_xor_sync(0xffffffffu, iacc[p], o);
      else
        acc[p] += __shfl_xor_sync(0xffffffffu, acc[p], o);
    }
  }
  const float sx = __ldg(act_scale);
#pragma unroll
  for (int p = 0; p < GV_MAXP; ++p) {
    if (p < P && lane == p) {
      const float v = QA ? (float)iacc[p] * (sx * __ldg(ascale + m)) : sx * acc[p];
      if (rq_out)  // fused requantization
        rq_out[(int64_t)p * M + m] = rq_code(v, rq_mul(rq_scale, rq_signed));
      else
        y[(int64_t)p * M + m] = v;
    }
  }
}

template <int G, bool SIGNED>
fgq_status launch_gemv_g(const void* q, int P, int Kred, int M, const uint32_t* codes, const float* alpha,
                         const uint8_t* aq, int abits, const float* ascale, const float* act_scale, float* y,
                         uint8_t* rq_out, const float* rq_scale, int rq_signed, cudaStream_t s) {
  const unsigned blocks = (unsigned)((M + GV_WARPS - 1) / GV_WARPS);
  const uint8_t* qb = static_cast<const uint8_t*>(q);
  if (abits == 8)
    gemv_kernel<G, SIGNED, 8><<<blocks, 32 * GV_WARPS, 0, s>>>(qb, P, Kred, M, codes, alpha, aq, ascale, act_scale, y,
                                                                 rq_out, rq_scale, rq_signed);
  else if (abits == 4)
    gemv_kernel<G, SIGNED, 4><<<blocks, 32 * GV_WARPS, 0, s>>>(qb, P, Kred, M, codes, alpha, aq, ascale, act_scale, y,
                                                                 rq_out, rq_scale, rq_signed);
  else
    gemv_kernel<G, SIGNED, 0><<<blocks, 32 * GV_WARPS, 0, s>>>(qb, P, Kred, M, codes, alpha, aq, ascale, act_scale, y,
                                                                 rq_out, rq_scale, rq_signed);
  return after_launch();
}

}  // namespace

bool gemv_supports(int P, int Kred, int G, int act_type) {
  return P >= 1 && P <= GV_MAXP && Kred % 16 == 0 && G >= 4 && (act_type == FGQ_U8 || act_type == FGQ_S8);
}

fgq_status launch_gemv(const void* q, int act_type, int P, int Kred, int M, int G, const uint32_t* codes,
                       const float* alpha, const uint8_t* aq, int abits, const float* ascale, const float* act_scale,
                       float* y, uint8_t* rq_out, const float* rq_scale, int rq_signed, cudaStream_t s) {
  if (!gemv_supports(P, Kred, G, act_type)) return FGQ_ERR_UNSUPPORTED;
  const bool sg = act_type == FGQ_S8;
#define FGQ_GEMV_CASE(GG)                                                                                   \
  case GG:                                                                                                  \
    return sg ? launch_gemv_g<GG, true>(q, P, Kred, M, codes, alpha, aq, abits, ascale, act_scale, y, rq_out, rq_scale, rq_signed, s)    \
              : launch_gemv_g<GG, false>(q, P, Kred, M, codes, alpha, aq, abits, ascale, act_scale, y, rq_out, rq_scale, rq_signed, s);
  switch (G) {
    FGQ_GEMV_CASE(4)
    FGQ_GEMV_CASE(8)
    FGQ_GEMV_CASE(16)
    FGQ_GEMV_CASE(32)
    FGQ_GEMV_CASE(64)
    FGQ_GEMV_CASE(128)
    default:
      return FGQ_ERR_UNSUPPORTED;
  }
#undef FGQ_GEMV_CASE
}

}  // namespace fgq
