// Analytical-threshold ternarization and the ternary error (Section 3; Lemma 1 and its
// proof in the appendix).  t_i = sign(w_i) where |w_i| > Delta, alpha = the mean of the
// kept magnitudes (the alpha of Eq. 4 for that support).  Delta comes from a model of the
// weight distribution instead of the exact search of Eq. 5:
//   FGQ_RULE_EXP   (exponential magnitudes, Lemma 1):  Delta = mean |w|;
//   FGQ_RULE_GAUSS (Gaussian weights):                 Delta = Z_GAUSS * rms(w), rms the
//     maximum-likelihood sigma the paper names and Z_GAUSS the maximiser of
//     phi(z)^2 / (1 - Phi(z)), the Gaussian limit of (sum_{|w|>Delta} |w|)^2 / |I_Delta|.
// Per group of G (one Delta and one alpha per group), or per layer (one Delta and one
// alpha for the whole M x Kred matrix: the one-scaling-factor baseline).
//
// Arithmetic: the statistics are fp64 sums in element order with explicitly rounded
// operations (no contraction into FMAs), the threshold comparison is in fp64 and
// alpha = fp32(S / k); a group's result is therefore the same on every run.  The
// per-layer rule sums in a fixed tree order (per-block partials, then a fixed reduction of
// the partials), so it is deterministic too, but its rounding differs from a sequential
// sum by a few ulps.
#include <algorithm>
#include <cmath>
#include <cstdint>

#include "fgq_device.cuh"

namespace fgq {
namespace {

constexpr double Z_GAUSS = 0.6120031809624808;
constexpr int THR_THREADS = 256;
constexpr int LAYER_BLOCKS = 1024;  // fixed partial count of the per-layer reductions

__device__ __forceinline__ double dabs(float v) { return fabs((double)v); }

__device__ __forceinline__ double threshold_of(double sa, double sq, int64_t n, int rule) {
  if (n == 0) return 0.0;
  if (rule == FGQ_RULE_EXP) return __ddiv_rn(sa, (double)n);
  return __dmul_rn(Z_GAUSS, __dsqrt_rn(__ddiv_rn(sq, (double)n)));
}

__device__ __forceinline__ uint32_t code_of(float v) { return v > 0.0f ? 1u : 3u; }

// Kept magnitudes of elements [j0, j1) of row wr against delta, in element order: bits
// of the code word(s) set in word (element j at bits 2 (j % 16)), sum and count added.
__device__ __forceinline__ void keep_range(const float* wr, int j0, int j1, double delta, uint32_t& word,
                                           double& kept, int& k) {
  for (int j = j0; j < j1; ++j) {
    const float v = __ldg(wr + j);
    if (dabs(v) > delta) {
      kept = __dadd_rn(kept, dabs(v));
      ++k;
      word |= code_of(v) << (2 * (j & 15));
    }
  }
}

// One thread per unit of U = max(G, 16) weights of a row: the 16 / G groups of one code
// word (G < 16), or one group and its G / 16 code words (G >= 16; valid G are powers of
// two, so G is then a multiple of 16).
__global__ void __launch_bounds__(THR_THREADS) thr_group_kernel(const float* __restrict__ w, int M, int Kred, int G,
                                                                int rule, int units_per_row, uint32_t* __restrict__ codes,
                                                                float* __restrict__ alpha, unsigned int* err) {
  const int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (u >= (int64_t)M * units_per_row) return;
  const int m = (int)(u / units_per_row);
  const int ui = (int)(u - (int64_t)m * units_per_row);
  const int ng = (Kred + G - 1) / G;
  const int wrow = (ng * G + 15) / 16;
  const int groups_per_unit = G < 16 ? 16 / G : 1;
  const float* wr = w + (int64_t)m * Kred;
  uint32_t* crow = codes + (int64_t)m * wrow;
  uint32_t word = 0;  // G < 16: the unit's code word
  for (int gg = 0; gg < groups_per_unit; ++gg) {
    const int g = ui * groups_per_unit + gg;
    if (g >= ng) break;
    const int j0 = g * G, j1 = min(j0 + G, Kred);
    double sa = 0.0, sq = 0.0;
    bool bad = false;
    for (int j = j0; j < j1; ++j) {
      const float v = __ldg(wr + j);
      bad |= !isfinite(v);
      sa = __dadd_rn(sa, dabs(v));
      sq = __dadd_rn(sq, __dmul_rn((double)v, (double)v));
    }
    double kept = 0.0;
    int k = 0;
    if (bad) {
      record_error(err, FGQ_ERR_NONFINITE);
      if (G >= 16)
        for (int c = j0 / 16; c < (j0 + G) / 16; ++c) crow[c] = 0u;
    } else {
      const double delta = threshold_of(sa, sq, j1 - j0, rule);
      if (G < 16) {
        keep_range(wr, j0, j1, delta, word, kept, k);
      } else {
        for (int c = j0 / 16; c < (j0 + G) / 16; ++c) {  // the group's words, padding included
          uint32_t wc = 0;
          keep_range(wr, min(16 * c, j1), min(16 * c + 16, j1), delta, wc, kept, k);
          crow[c] = wc;
        }
      }
    }
    alpha[(int64_t)m * ng + g] = k ? __double2float_rn(__ddiv_rn(kept, (double)k)) : 0.0f;
  }
  if (G < 16 && ui < wrow) crow[ui] = word;
}

// Per-layer rule, pass 1: per-block fp64 partial sums of |w| and w^2 over the row-major
// matrix (each block a contiguous range), and the non-finite flag.
__global__ void __launch_bounds__(THR_THREADS) thr_layer_stats_kernel(const float* __restrict__ w, int64_t n,
                                                                      double2* __restrict__ part, unsigned int* err) {
  const int64_t per = (n + gridDim.x - 1) / gridDim.x;
  const int64_t b0 = (int64_t)blockIdx.x * per, b1 = min(b0 + per, n);
  double sa = 0.0, sq = 0.0;
  bool bad = false;
  for (int64_t i = b0 + threadIdx.x; i < b1; i += blockDim.x) {
    const float v = __ldg(w + i);
    bad |= !isfinite(v);
    sa = __dadd_rn(sa, dabs(v));
    sq = __dadd_rn(sq, __dmul_rn((double)v, (double)v));
  }
  __shared__ double s_a[THR_THREADS], s_q[THR_THREADS];
  s_a[threadIdx.x] = sa;
  s_q[threadIdx.x] = sq;
  if (__syncthreads_or(bad) && threadIdx.x == 0) record_error(err, FGQ_ERR_NONFINITE);
  for (int h = THR_THREADS / 2; h > 0; h >>= 1) {
    if (threadIdx.x < h) {
      s_a[threadIdx.x] = __dadd_rn(s_a[threadIdx.x], s_a[threadIdx.x + h]);
      s_q[threadIdx.x] = __dadd_rn(s_q[threadIdx.x], s_q[threadIdx.x + h]);
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) part[blockIdx.x] = make_double2(s_a[0], s_q[0]);
}

// Sum of the block partials in a fixed order (thread t sums partials t, t + 256, ... in
// turn, then a fixed tree), so every block computes the same value.
__device__ double2 sum_parts(const double2* part, int nparts) {
  __shared__ double s_a[THR_THREADS], s_q[THR_THREADS];
  double a = 0.0, q = 0.0;
  for (int i = threadIdx.x; i < nparts; i += THR_THREADS) {
    const double2 v = part[i];
    a = __dadd_rn(a, v.x);
    q = __dadd_rn(q, v.y);
  }
  s_a[threadIdx.x] = a;
  s_q[threadIdx.x] = q;
  __syncthreads();
  for (int h = THR_THREADS / 2; h > 0; h >>= 1) {
    if (threadIdx.x < h) {
      s_a[threadIdx.x] = __dadd_rn(s_a[threadIdx.x], s_a[threadIdx.x + h]);
      s_q[threadIdx.x] = __dadd_rn(s_q[threadIdx.x], s_q[threadIdx.x + h]);
    }
    __syncthreads();
  }
  const double2 r = make_double2(s_a[0], s_q[0]);
  __syncthreads();  // the shared arrays are reused by the caller's own reduction
  return r;
}

// Per-layer rule, pass 2: the layer threshold, the code words (one thread per word), and
// per-block partials of the kept magnitudes and their count.
__global__ void __launch_bounds__(THR_THREADS) thr_layer_codes_kernel(const float* __restrict__ w, int M, int Kred,
                                                                      int G, int rule, const double2* __restrict__ part,
                                                                      int nparts, uint32_t* __restrict__ codes,
                                                                      double2* __restrict__ kept_part,
                                                                      double* delta_out) {
  const double2 st = sum_parts(part, nparts);
  const double delta = threshold_of(st.x, st.y, (int64_t)M * Kred, rule);
  if (blockIdx.x == 0 && threadIdx.x == 0 && delta_out) *delta_out = delta;
  const int ng = (Kred + G - 1) / G;
  const int wrow = (ng * G + 15) / 16;
  const int64_t nwords = (int64_t)M * wrow;
  double kept = 0.0;
  double cnt = 0.0;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < nwords; i += (int64_t)gridDim.x * blockDim.x) {
    const int m = (int)(i / wrow);
    const int c = (int)(i - (int64_t)m * wrow);
    uint32_t word = 0;
    for (int e = 0; e < 16; ++e) {
      const int j = 16 * c + e;
      if (j >= Kred) break;
      const float v = __ldg(w + (int64_t)m * Kred + j);
      if (dabs(v) > delta) {
        word |= code_of(v) << (2 * e);
        kept = __dadd_rn(kept, dabs(v));
        cnt += 1.0;
      }
    }
    codes[i] = word;
  }
  __shared__ double s_k[THR_THREADS], s_c[THR_THREADS];
  s_k[threadIdx.x] = kept;
  s_c[threadIdx.x] = cnt;
  __syncthreads();
  for (int h = THR_THREADS / 2; h > 0; h >>= 1) {
    if (threadIdx.x < h) {
      s_k[threadIdx.x] = __dadd_rn(s_k[threadIdx.x], s_k[threadIdx.x + h]);
      s_c[threadIdx.x] += s_c[threadIdx.x + h];  // integer counts, exact in fp64
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) kept_part[blockIdx.x] = make_double2(s_k[0], s_c[0]);
}

// Per-layer rule, pass 3: alpha = sum kept / count, written to every alpha[m][g].
__global__ void __launch_bounds__(THR_THREADS) thr_layer_alpha_kernel(const double2* __restrict__ kept_part,
                                                                      int nparts, int64_t nalpha,
                                                                      float* __restrict__ alpha) {
  const double2 st = sum_parts(kept_part, nparts);
  const float a = st.y > 0.0 ? __double2float_rn(__ddiv_rn(st.x, st.y)) : 0.0f;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < nalpha; i += (int64_t)gridDim.x * blockDim.x)
    alpha[i] = a;
}

// Ternary error of each group: err[m][g] = sum_j (w_j - alpha t_j)^2, fp64, element order.
__global__ void __launch_bounds__(THR_THREADS) ternary_error_kernel(const float* __restrict__ w, int M, int Kred,
                                                                    int G, const uint32_t* __restrict__ codes,
                                                                    const float* __restrict__ alpha,
                                                                    double* __restrict__ err) {
  const int ng = (Kred + G - 1) / G;
  const int64_t gi = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (gi >= (int64_t)M * ng) return;
  const int m = (int)(gi / ng), g = (int)(gi - (int64_t)m * ng);
  const int wrow = (ng * G + 15) / 16;
  const double a = (double)__ldg(alpha + gi);
  double e = 0.0;
  for (int j = g * G; j < min(g * G + G, Kred); ++j) {
    const uint32_t c = (__ldg(codes + (int64_t)m * wrow + j / 16) >> (2 * (j & 15))) & 3u;
    const double v = (double)__ldg(w + (int64_t)m * Kred + j);
    const double d = c == 1u ? __dsub_rn(v, a) : (c == 3u ? __dadd_rn(v, a) : v);
    e = __dadd_rn(e, __dmul_rn(d, d));
  }
  err[gi] = e;
}

}  // namespace

size_t threshold_workspace_bytes() { return (size_t)LAYER_BLOCKS * 2 * sizeof(double2) + 16; }

fgq_status launch_ternarize_threshold(const float* w, int M, int Kred, int G, int rule, int per_layer,
                                      uint32_t* codes, float* alpha, void* ws, double* delta_out, unsigned int* err,
                                      cudaStream_t s) {
  const int ng = (Kred + G - 1) / G;
  if (!per_layer) {
    const int U = G < 16 ? 16 : G;
    const int units_per_row = (ng * G + U - 1) / U;
    const int64_t units = (int64_t)M * units_per_row;
    thr_group_kernel<<<(unsigned)((units + THR_THREADS - 1) / THR_THREADS), THR_THREADS, 0, s>>>(
        w, M, Kred, G, rule, units_per_row, codes, alpha, err);
    return after_launch();
  }
  double2* part = static_cast<double2*>(ws);
  double2* kept_part = part + LAYER_BLOCKS;
  const int64_t n = (int64_t)M * Kred;
  thr_layer_stats_kernel<<<LAYER_BLOCKS, THR_THREADS, 0, s>>>(w, n, part, err);
  fgq_status st = after_launch();
  if (st != FGQ_OK) return st;
  thr_layer_codes_kernel<<<LAYER_BLOCKS, THR_THREADS, 0, s>>>(w, M, Kred, G, rule, part, LAYER_BLOCKS, codes,
                                                              kept_part, delta_out);
  st = after_launch();
  if (st != FGQ_OK) return st;
  const int64_t nalpha = (int64_t)M * ng;
  const int ab = (int)std::min<int64_t>((nalpha + THR_THREADS - 1) / THR_THREADS, 1024);
  thr_layer_alpha_kernel<<<ab > 0 ? ab : 1, THR_THREADS, 0, s>>>(kept_part, LAYER_BLOCKS, nalpha, alpha);
  return after_launch();
}

fgq_status launch_ternary_error(const float* w, int M, int Kred, int G, const uint32_t* codes, const float* alpha,
                                double* errv, cudaStream_t s) {
  const int64_t n = (int64_t)M * ((Kred + G - 1) / G);
  ternary_error_kernel<<<(unsigned)((n + THR_THREADS - 1) / THR_THREADS), THR_THREADS, 0, s>>>(w, M, Kred, G, codes,
                                                                                             alpha, errv);
  return after_launch();
}

}  // namespace fgq
