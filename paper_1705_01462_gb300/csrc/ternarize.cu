// FGQ ternarization kernels (Section 3.1: Eq. 2 splits each filter row into independent
// groups of G weights; each group is solved exactly for the threshold of Eq. 5, which is
// also the optimum of the asymmetric form Eq. 4) and the 8-bit first-layer weights
// (Section 4).
//
// Exact arithmetic.  Magnitudes are handled as their fp32 bit patterns, which order like
// the values.  With F = max(biased exponent of the group's largest magnitude, 1), every
// magnitude whose exponent is at least F - 8 is an integer multiple of 2^(F-158) below
// 2^32; sums of up to 128 of them are exact in uint64, and the objective comparison
// S_a^2 * k_b > S_b^2 * k_a is exact in 128 bits.  A threshold below that window never
// maximises Eq. 5's objective (dropping the smallest kept magnitude a does not raise the
// objective only if a > max|w| / (2k - 1) >= max|w| / 255), so only window values are
// candidates.  Equal magnitudes are kept or dropped together (a threshold rule), ties in
// the objective go to the smaller kept set, and alpha is the fp32 nearest the exact mean.
#include <cstdint>
#include <cstring>

#include "fgq_device.cuh"

namespace fgq {
namespace {

// S^2 * k as a 128-bit number (hi, lo); S < 2^40, k <= 128.
__device__ __forceinline__ void sq_times(uint64_t S, uint32_t k, uint64_t& hi, uint64_t& lo) {
  const uint64_t l = S * S, h = __umul64hi(S, S);
  lo = l * k;
  hi = h * k + __umul64hi(l, (uint64_t)k);
}

// Objective of (Sa, ka) strictly above that of (Sb, kb): Sa^2/ka > Sb^2/kb.
__device__ __forceinline__ bool j_greater(uint64_t Sa, uint32_t ka, uint64_t Sb, uint32_t kb) {
  uint64_t ah, al, bh, bl;
  sq_times(Sa, kb, ah, al);
  sq_times(Sb, ka, bh, bl);
  return ah > bh || (ah == bh && al > bl);
}

// fp32 nearest (ties to even) to S * 2^u / k, for 1 <= S < 2^40, 1 <= k <= 128, u >= -157.
// Only the top 32 bits of S enter a 32-bit division: with N = those bits (N >= 2^31) and
// the dropped low bits folded into a sticky flag, the exact quotient is
// q + (r + f) / k with q = N / k >= 2^24, r = N % k and 0 <= f < 1, so q is its floor and
// the quotient is exact iff r == 0 and nothing was dropped -- enough to round to 24 bits.
__device__ __forceinline__ float round_ratio_f32(uint64_t S, uint32_t k, int u) {
  if (S == 0 || k == 0) return 0.0f;
  const int nbS = 64 - __clzll((long long)S);
  int shift = nbS - 32;  // value = (N + dropped) * 2^(u + shift) / k
  uint32_t N;
  bool dropped;
  if (shift >= 0) {
    N = (uint32_t)(S >> shift);
    dropped = (S & ((1ull << shift) - 1)) != 0;
  } else {
    N = (uint32_t)(S << -shift);
    dropped = false;
  }
  const uint32_t q = N / k;
  const uint32_t r = N - q * k;
  const bool sticky = dropped || r != 0;
  const int nb = 32 - __clz((int)q);           // >= 25
  const int lead = nb - 1 + u + shift;         // binary exponent of the leading bit
  int lsb = lead >= -126 ? lead - 23 : -149;
  const int drop = lsb - (u + shift);          // bits of q below the fp32 lsb, >= 1
  uint64_t mant = 0, rem = 0, half = 1;
  if (drop < 64) {
    mant = (uint64_t)q >> drop;
    rem = (uint64_t)q & ((1ull << drop) - 1);
    half = 1ull << (drop - 1);
  }  // else: the value is below a quarter of the smallest subnormal step and rounds to 0
  if (rem > half || (rem == half && (sticky || (mant & 1)))) mant += 1;
  if (mant == (1ull << 24)) {
    mant >>= 1;
    lsb += 1;
  }
  if (mant >= (1ull << 23)) return __uint_as_float((uint32_t)(lsb + 23 + 127) << 23 | ((uint32_t)mant & 0x7fffffu));
  return __uint_as_float((uint32_t)mant);  // subnormal (lsb == -149)
}

// Fixed-point value of magnitude bits m in units of 2^(F-158); 0 outside the window.
__device__ __forceinline__ uint64_t fixed_of(uint32_t m, int F) {
  const int f = (int)(m >> 23);
  const int fe = f ? f : 1;
  if (m == 0 || fe < F - 8) return 0;
  const uint64_t sig = f ? ((m & 0x7fffffu) | 0x800000u) : (m & 0x7fffffu);
  return sig << (fe - F + 8);
}

__device__ __forceinline__ bool in_window(uint32_t m, int F) {
  const int f = (int)(m >> 23);
  return m != 0 && (f ? f : 1) >= F - 8;
}

// Magnitude bits sorted in descending order in registers by Batcher's odd-even merge
// network (N a power of two; 543 comparators for N = 64).
template <int N>
__device__ __forceinline__ void sort_desc(uint32_t (&s)[N]) {
  // stage (p, k) compares x with x + k where x - k % p lies in the first half of a block of
  // 2k and both lie in one block of 2p; the loops have constant trip counts so that the
  // network unrolls into register operations
#pragma unroll
  for (int p = 1; p < N; p <<= 1) {
#pragma unroll
    for (int k = p; k >= 1; k >>= 1) {
#pragma unroll
      for (int x = 0; x < N; ++x) {
        const int r = k % p;
        if (x >= r && x + k < N && (x - r) % (2 * k) < k && x / (2 * p) == (x + k) / (2 * p)) {
          const uint32_t a = s[x], b = s[x + k];
          s[x] = a > b ? a : b;
          s[x + k] = a > b ? b : a;
        }
      }
    }
  }
}

// The search of Eq. 5 over the sorted magnitudes, one element at a time in decreasing
// order: the best candidate so far (its exact sum bS in units of 2^(F-158), size bk and
// threshold tau) and fp32 estimates that decide all but near-tie comparisons.
//
// Fast form, for a group whose largest exponent F lies in [10, 253]: the window is every
// magnitude with bits >= wmin = (F - 8) << 23 (all normal), an element's fixed-point value
// is its significand shifted by its exponent's distance above F - 8, and the estimate fS is
// the running fp32 sum of the magnitudes scaled by c = 2^(127 - F) (exact scalings; after k
// adds its relative error is below k 2^-24 <= 2^-17 for k <= 128).  Candidate k's objective
// fS^2 / k is compared with the best's as fS^2 * bk against bQ * k, bQ = bfS^2 (1 +- 2^-14)
// kept from the best: each side is within 2^-16.5 of its exact value, so a comparison
// outside the 2^-14 band is decided correctly by the estimates, and one inside it by the
// exact 128-bit comparison (strict: a tie keeps the smaller k).  Elements past the window
// come after every candidate, so what they add to S and fS is never compared.
struct Eq5Scan {
  uint64_t S, bS;
  float fS, bQhi, bQlo, bkf;
  uint32_t bk, tau;
};

__device__ __forceinline__ void eq5_init(Eq5Scan& q) {
  q.S = 0;
  q.bS = 0;
  q.fS = 0.0f;
  q.bQhi = 0.0f;
  q.bQlo = 0.0f;
  q.bkf = 0.0f;
  q.bk = 0;
  q.tau = 0;
}

// Element k - 1 (k = 1 .. G) with magnitude bits m; `mn` the next element's bits (0 past
// the end).  Fast form only.
__device__ __forceinline__ void eq5_step(Eq5Scan& q, uint32_t m, uint32_t mn, uint32_t k, float kf, int F,
                                         uint32_t wmin, float c) {
  const uint32_t sig = (m & 0x7fffffu) | 0x800000u;
  q.S += (uint64_t)(sig << (((m >> 23) - (uint32_t)(F - 8)) & 31u));
  q.fS = fmaf(__uint_as_float(m), c, q.fS);
  if (mn < m && m >= wmin) {  // a threshold between distinct magnitudes, inside the window
    const float t = q.fS * q.fS;
    const float lhs = t * q.bkf;
    bool take;
    if (q.bk == 0 || lhs > q.bQhi * kf) take = true;
    else if (lhs < q.bQlo * kf) take = false;
    else take = j_greater(q.S, k, q.bS, q.bk);
    if (take) {
      q.bS = q.S;
      q.bk = k;
      q.bkf = kf;
      q.tau = m;
      q.bQhi = t * (1.0f + 0x1p-14f);
      q.bQlo = t * (1.0f - 0x1p-14f);
    }
  }
}

// General form (any F, subnormal magnitudes included): exact sums and comparisons only.
__device__ __forceinline__ void eq5_step_exact(Eq5Scan& q, uint32_t m, uint32_t mn, uint32_t k, int F) {
  q.S += fixed_of(m, F);
  if (mn < m && in_window(m, F) && (q.bk == 0 || j_greater(q.S, k, q.bS, q.bk))) {
    q.bS = q.S;
    q.bk = k;
    q.tau = m;
  }
}

__device__ __forceinline__ bool eq5_fast(int F) { return F >= 10 && F <= 253; }

__device__ __forceinline__ float eq5_scale(int F) { return __uint_as_float((uint32_t)(254 - F) << 23); }

// Solve one group held in registers (G <= 16).  Writes alpha and returns the 2G code bits.
template <int G>
__device__ __forceinline__ uint32_t solve_group_regs(const float (&v)[G], float& alpha, bool& bad) {
  uint32_t s[G];
#pragma unroll
  for (int i = 0; i < G; ++i) s[i] = __float_as_uint(v[i]) & 0x7fffffffu;
  sort_desc<G>(s);
  bad = s[0] >= 0x7f800000u;  // the largest magnitude: infinite or NaN if any is
  alpha = 0.0f;
  if (bad || s[0] == 0) return 0;
  const int F = max((int)(s[0] >> 23), 1);
  Eq5Scan q;
  eq5_init(q);
  if (eq5_fast(F)) {
    const uint32_t wmin = (uint32_t)(F - 8) << 23;
    const float c = eq5_scale(F);
#pragma unroll
    for (int i = 0; i < G; ++i) eq5_step(q, s[i], i + 1 < G ? s[i + 1] : 0u, i + 1, (float)(i + 1), F, wmin, c);
  } else {
#pragma unroll
    for (int i = 0; i < G; ++i) eq5_step_exact(q, s[i], i + 1 < G ? s[i + 1] : 0u, i + 1, F);
  }
  alpha = round_ratio_f32(q.bS, q.bk, F - 158);
  uint32_t bits = 0;
#pragma unroll
  for (int i = 0; i < G; ++i) {
    if ((__float_as_uint(v[i]) & 0x7fffffffu) >= q.tau) bits |= ((__float_as_uint(v[i]) >> 31) ? 3u : 1u) << (2 * i);
  }
  return bits;
}

// One unit of max(G, 4) consecutive weights of a row (one code byte for G <= 4): unit u of
// the layer, units_per_row units per filter row.
template <int G>
__device__ __forceinline__ void small_unit(const float* __restrict__ w, int Kred, int ng, int wrow,
                                           uint8_t* __restrict__ codes, float* __restrict__ alpha, unsigned int* err,
                                           int vec4, int64_t units_per_row, int64_t u) {
  constexpr int UNIT = G < 4 ? 4 : G;
  constexpr int NSUB = UNIT / G;
  const int m = (int)(u / units_per_row);
  const int ui = (int)(u - (int64_t)m * units_per_row);
  const int k0 = ui * UNIT;
  const float* row = w + (int64_t)m * Kred;
  float v[UNIT];
  if (vec4 && k0 + UNIT <= Kred) {
#pragma unroll
    for (int i = 0; i < UNIT; i += 4) {
      const float4 f = __ldg(reinterpret_cast<const float4*>(row + k0 + i));
      v[i] = f.x; v[i + 1] = f.y; v[i + 2] = f.z; v[i + 3] = f.w;
    }
  } else {
#pragma unroll
    for (int i = 0; i < UNIT; ++i) v[i] = (k0 + i < Kred) ? __ldg(row + k0 + i) : 0.0f;
  }
  uint32_t bits = 0;
#pragma unroll
  for (int sub = 0; sub < NSUB; ++sub) {
    const int g = ui * NSUB + sub;
    if (g < ng) {
      float gv[G];
#pragma unroll
      for (int i = 0; i < G; ++i) gv[i] = v[sub * G + i];
      float a;
      bool bad;
      const uint32_t b = solve_group_regs<G>(gv, a, bad);
      if (bad) record_error(err, FGQ_ERR_NONFINITE);
      alpha[(int64_t)m * ng + g] = a;
      bits |= b << (2 * sub * G);
    }
  }
  uint8_t* crow = codes + (int64_t)m * wrow * 4;
  const int byte0 = k0 / 4;
  if (UNIT == 4) {
    crow[byte0] = (uint8_t)bits;
  } else if (UNIT == 8) {
    *reinterpret_cast<uint16_t*>(crow + byte0) = (uint16_t)bits;
  } else {
    *reinterpret_cast<uint32_t*>(crow + byte0) = bits;
  }
  if (ui == units_per_row - 1) {  // zero the unused bytes of the row's last word
    for (int b = byte0 + UNIT / 4; b < wrow * 4; ++b) crow[b] = 0;
  }
}

// One thread per unit of max(G, 4) consecutive weights (one code byte for G <= 4).
template <int G>
__global__ void __launch_bounds__(256) ternarize_small_kernel(const float* __restrict__ w, int M, int Kred,
                                                              int ng, int wrow, uint8_t* __restrict__ codes,
                                                              float* __restrict__ alpha, unsigned int* err,
                                                              int vec4) {
  constexpr int UNIT = G < 4 ? 4 : G;
  const int Kp = ng * G;
  const int64_t units_per_row = (Kp + UNIT - 1) / UNIT;
  const int64_t total = (int64_t)M * units_per_row;
  for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < total; u += (int64_t)gridDim.x * blockDim.x)
    small_unit<G>(w, Kred, ng, wrow, codes, alpha, err, vec4, units_per_row, u);
}

// One group of G in {32, 64} weights (group grp = m ng + g of the layer) solved by one
// thread: the G magnitudes sorted in registers, then written to the thread's column of
// shared memory (`col`, stride TG_THREADS words: conflict-free) and scanned there by a
// rolled loop, which keeps the kernel's code small; the signs for the codes are read again
// (the group's bytes are still in L1).
constexpr int TG_THREADS = 128;

template <int G>
__device__ __forceinline__ void thread_group(const float* __restrict__ w, int Kred, int ng, int wrow,
                                             uint32_t* __restrict__ codes, float* __restrict__ alpha,
                                             unsigned int* err, int vec4, int64_t grp, uint32_t* col) {
  const int m = (int)(grp / ng);
  const int g = (int)(grp - (int64_t)m * ng);
  const float* src = w + (int64_t)m * Kred + (int64_t)g * G;
  const int nvalid = Kred - g * G < G ? Kred - g * G : G;
  uint32_t* crow = codes + (int64_t)m * wrow + g * (G / 16);
  uint32_t tau;
  {
    uint32_t s[G];
    if (vec4 && nvalid == G) {
#pragma unroll
      for (int i = 0; i < G; i += 4) {
        const float4 f = __ldg(reinterpret_cast<const float4*>(src + i));
        s[i] = __float_as_uint(f.x) & 0x7fffffffu;
        s[i + 1] = __float_as_uint(f.y) & 0x7fffffffu;
        s[i + 2] = __float_as_uint(f.z) & 0x7fffffffu;
        s[i + 3] = __float_as_uint(f.w) & 0x7fffffffu;
      }
    } else {
#pragma unroll
      for (int i = 0; i < G; ++i) s[i] = i < nvalid ? __float_as_uint(__ldg(src + i)) & 0x7fffffffu : 0u;
    }
    sort_desc<G>(s);
    if (s[0] >= 0x7f800000u) {  // the largest magnitude: infinite or NaN if any is
      record_error(err, FGQ_ERR_NONFINITE);
      alpha[grp] = 0.0f;
#pragma unroll
      for (int wd = 0; wd < G / 16; ++wd) crow[wd] = 0u;
      return;
    }
#pragma unroll
    for (int i = 0; i < G; ++i) col[i * TG_THREADS] = s[i];
  }
  const uint32_t top = col[0];
  Eq5Scan q;
  eq5_init(q);
  const int F = max((int)(top >> 23), 1);
  if (top != 0) {
    if (eq5_fast(F)) {
      const uint32_t wmin = (uint32_t)(F - 8) << 23;
      const float c = eq5_scale(F);
      uint32_t cur = top;
      float kf = 1.0f;
#pragma unroll 4
      for (int i = 0; i < G; ++i) {
        const uint32_t nxt = i + 1 < G ? col[(i + 1) * TG_THREADS] : 0u;
        eq5_step(q, cur, nxt, (uint32_t)(i + 1), kf, F, wmin, c);
        cur = nxt;
        kf += 1.0f;
      }
    } else {
      uint32_t cur = top;
      for (int i = 0; i < G; ++i) {
        const uint32_t nxt = i + 1 < G ? col[(i + 1) * TG_THREADS] : 0u;
        eq5_step_exact(q, cur, nxt, (uint32_t)(i + 1), F);
        cur = nxt;
      }
    }
  }
  alpha[grp] = q.bk ? round_ratio_f32(q.bS, q.bk, F - 158) : 0.0f;
  tau = q.bk ? q.tau : 0xffffffffu;  // codes: t = sign(w) where |w| >= tau
#pragma unroll 1
  for (int wd = 0; wd < G / 16; ++wd) {
    uint32_t b[16];
    if (vec4 && nvalid == G) {
#pragma unroll
      for (int e = 0; e < 16; e += 4) {
        const float4 f = __ldg(reinterpret_cast<const float4*>(src + 16 * wd + e));
        b[e] = __float_as_uint(f.x);
        b[e + 1] = __float_as_uint(f.y);
        b[e + 2] = __float_as_uint(f.z);
        b[e + 3] = __float_as_uint(f.w);
      }
    } else {
#pragma unroll
      for (int e = 0; e < 16; ++e) b[e] = 16 * wd + e < nvalid ? __float_as_uint(__ldg(src + 16 * wd + e)) : 0u;
    }
    uint32_t bits = 0;
#pragma unroll
    for (int e = 0; e < 16; ++e)
      if ((b[e] & 0x7fffffffu) >= tau) bits |= ((b[e] >> 31) ? 3u : 1u) << (2 * e);
    crow[wd] = bits;
  }
}

// One thread per group for G in {32, 64}.
template <int G>
__global__ void __launch_bounds__(TG_THREADS) ternarize_thread_kernel(const float* __restrict__ w, int M, int Kred,
                                                                      int ng, int wrow, uint32_t* __restrict__ codes,
                                                                      float* __restrict__ alpha, unsigned int* err,
                                                                      int vec4) {
  __shared__ uint32_t sorted[G * TG_THREADS];
  const int64_t total = (int64_t)M * ng;
  for (int64_t grp = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; grp < total;
       grp += (int64_t)gridDim.x * blockDim.x)
    thread_group<G>(w, Kred, ng, wrow, codes, alpha, err, vec4, grp, sorted + threadIdx.x);
}

// One group of G in {32, 64, 128} weights (group grp = m ng + g of the layer) solved by one
// warp: lane l holds elements l*E .. l*E+E-1.
template <int G>
__device__ __forceinline__ void warp_group(const float* __restrict__ w, int Kred, int ng, int wrow,
                                           uint32_t* __restrict__ codes, float* __restrict__ alpha, unsigned int* err,
                                           int64_t grp, int lane) {
  constexpr int E = G / 32;
  constexpr int L = 16 / E;  // lanes per code word
  const int m = (int)(grp / ng);
  const int g = (int)(grp - (int64_t)m * ng);
  const float* row = w + (int64_t)m * Kred;
  const int k0 = g * G + lane * E;
  float v[E];
  uint32_t mag[E], s[E];
  bool bad = false;
#pragma unroll
  for (int e = 0; e < E; ++e) {
    v[e] = (k0 + e < Kred) ? __ldg(row + k0 + e) : 0.0f;
    mag[e] = __float_as_uint(v[e]) & 0x7fffffffu;
    bad |= mag[e] >= 0x7f800000u;
    s[e] = mag[e];
  }
  if (__any_sync(FULL_MASK, bad)) {
    if (lane == 0) {
      record_error(err, FGQ_ERR_NONFINITE);
      alpha[grp] = 0.0f;
    }
    if (lane < G / 16) codes[(int64_t)m * wrow + g * (G / 16) + lane] = 0;
    return;
  }
  // bitonic sort of the G magnitudes across the warp, descending
#pragma unroll
  for (int size = 2; size <= G; size <<= 1) {
#pragma unroll
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      if (stride >= E) {
#pragma unroll
        for (int e = 0; e < E; ++e) {
          const int i = lane * E + e;
          const uint32_t p = __shfl_xor_sync(FULL_MASK, s[e], stride / E);
          const bool lower = (i & stride) == 0;
          const bool desc = (i & size) == 0;
          const uint32_t mx = s[e] > p ? s[e] : p, mn = s[e] > p ? p : s[e];
          s[e] = (lower == desc) ? mx : mn;
        }
      } else {
#pragma unroll
        for (int e = 0; e < E; ++e) {
          if ((e & stride) == 0) {
            const int i = lane * E + e;
            const bool desc = (i & size) == 0;
            const int e2 = (e + stride) < E ? e + stride : e;
            const uint32_t a = s[e], b = s[e2];
            const uint32_t mx = a > b ? a : b, mn = a > b ? b : a;
            s[e] = desc ? mx : mn;
            s[e2] = desc ? mn : mx;
          }
        }
      }
    }
  }
  const uint32_t mmax = __shfl_sync(FULL_MASK, s[0], 0);
  uint32_t bk = 0, tau = 0;
  uint64_t bS = 0;
  int F = 1;
  if (mmax != 0) {
    F = max((int)(mmax >> 23), 1);
    uint64_t pre[E];
    uint64_t run = 0;
#pragma unroll
    for (int e = 0; e < E; ++e) {
      run += fixed_of(s[e], F);
      pre[e] = run;
    }
    uint64_t incl = run;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint64_t n = __shfl_up_sync(FULL_MASK, incl, o);
      if (lane >= o) incl += n;
    }
    const uint64_t excl = incl - run;
    const uint32_t next_first = __shfl_down_sync(FULL_MASK, s[0], 1);
#pragma unroll
    for (int e = 0; e < E; ++e) {
      const int i = lane * E + e;
      const uint32_t nxt = (e + 1 < E) ? s[(e + 1) < E ? e + 1 : e] : next_first;
      const bool run_end = (i == G - 1) || (nxt < s[e]);
      if (run_end && in_window(s[e], F)) {
        const uint64_t S = excl + pre[e];
        if (bk == 0 || j_greater(S, (uint32_t)(i + 1), bS, bk)) {
          bS = S;
          bk = (uint32_t)(i + 1);
          tau = s[e];
        }
      }
    }
    // warp argmax of the objective; equal objectives keep the smaller kept count
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const uint64_t oS = __shfl_xor_sync(FULL_MASK, bS, o);
      const uint32_t ok = __shfl_xor_sync(FULL_MASK, bk, o);
      const uint32_t ot = __shfl_xor_sync(FULL_MASK, tau, o);
      bool take;
      if (ok == 0) take = false;
      else if (bk == 0) take = true;
      else if (j_greater(oS, ok, bS, bk)) take = true;
      else if (j_greater(bS, bk, oS, ok)) take = false;
      else take = ok < bk;
      if (take) {
        bS = oS;
        bk = ok;
        tau = ot;
      }
    }
  }
  const float a = bk ? round_ratio_f32(bS, bk, F - 158) : 0.0f;
  if (lane == 0) alpha[grp] = a;
  uint32_t bits = 0;
  if (bk) {
#pragma unroll
    for (int e = 0; e < E; ++e)
      if (mag[e] >= tau) bits |= ((__float_as_uint(v[e]) >> 31) ? 3u : 1u) << (2 * e);
  }
  bits <<= 2 * E * (lane % L);
#pragma unroll
  for (int o = 1; o < L; o <<= 1) bits |= __shfl_xor_sync(FULL_MASK, bits, o);
  if (lane % L == 0) codes[(int64_t)m * wrow + g * (G / 16) + lane / L] = bits;
}

// One warp per group for G in {32, 64, 128}.
template <int G>
__global__ void __launch_bounds__(256) ternarize_warp_kernel(const float* __restrict__ w, int M, int Kred,
                                                             int ng, int wrow, uint32_t* __restrict__ codes,
                                                             float* __restrict__ alpha, unsigned int* err) {
  const int lane = threadIdx.x & 31;
  const int64_t warp0 = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const int64_t total = (int64_t)M * ng;
  for (int64_t grp = warp0; grp < total; grp += nwarps) warp_group<G>(w, Kred, ng, wrow, codes, alpha, err, grp, lane);
}

// Many layers of one group size in one launch (fgq_ternarize_batch): work items (units of
// the thread-per-group kernel, groups of the warp-per-group kernel) are numbered across the
// layers; item i belongs to the last layer whose first item is <= i.
struct TernLayer {
  const float* w;
  uint32_t* codes;
  float* alpha;
  int64_t first;          // first work item of the layer
  int64_t units_per_row;  // thread-per-group kernel only
  int Kred, ng, wrow, vec4;
};
struct TernBatch {
  TernLayer l[FGQ_TERNARIZE_BATCH_MAX];
  int n;
  int64_t total;
};
// Passed by value as a __grid_constant__ kernel parameter: above the 4 KB limit of older
// toolkits, within the 32,764-byte parameter space of CUDA 12.1 and later (the toolkit this
// library is built with is 13.0).
static_assert(sizeof(TernBatch) <= 32764, "kernel parameter space");

// The layer of item i (the last layer whose first item is <= i), searched forward from
// layer l: each thread visits its items in increasing order.
__device__ __forceinline__ int batch_layer_from(const TernBatch& b, int l, int64_t i) {
  while (l + 1 < b.n && b.l[l + 1].first <= i) ++l;
  return l;
}

template <int G>
__global__ void __launch_bounds__(256) ternarize_small_batch_kernel(const __grid_constant__ TernBatch b,
                                                                    unsigned int* err) {
  int l = 0;
  for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < b.total; u += (int64_t)gridDim.x * blockDim.x) {
    l = batch_layer_from(b, l, u);
    const TernLayer& L = b.l[l];
    small_unit<G>(L.w, L.Kred, L.ng, L.wrow, reinterpret_cast<uint8_t*>(L.codes), L.alpha, err, L.vec4,
                  L.units_per_row, u - L.first);
  }
}

template <int G>
__global__ void __launch_bounds__(TG_THREADS) ternarize_thread_batch_kernel(const __grid_constant__ TernBatch b,
                                                                            unsigned int* err) {
  __shared__ uint32_t sorted[G * TG_THREADS];
  int l = 0;
  for (int64_t grp = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; grp < b.total;
       grp += (int64_t)gridDim.x * blockDim.x) {
    l = batch_layer_from(b, l, grp);
    const TernLayer& L = b.l[l];
    thread_group<G>(L.w, L.Kred, L.ng, L.wrow, L.codes, L.alpha, err, L.vec4, grp - L.first, sorted + threadIdx.x);
  }
}

template <int G>
__global__ void __launch_bounds__(256) ternarize_warp_batch_kernel(const __grid_constant__ TernBatch b,
                                                                   unsigned int* err) {
  const int lane = threadIdx.x & 31;
  const int64_t warp0 = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  int l = 0;
  for (int64_t grp = warp0; grp < b.total; grp += nwarps) {
    l = batch_layer_from(b, l, grp);
    const TernLayer& L = b.l[l];
    warp_group<G>(L.w, L.Kred, L.ng, L.wrow, L.codes, L.alpha, err, grp - L.first, lane);
  }
}

// Per-filter signed 8-bit dynamic fixed point (Section 4, first layer at 8w-8a): one block
// per row; E = smallest integer with max|w| * 2^-E <= 127, clamped to [-149, 127].
__global__ void __launch_bounds__(256) quantize_w8_kernel(const float* __restrict__ w, int Kred,
                                                          int8_t* __restrict__ wq, float* __restrict__ wscale,
                                                          unsigned int* err) {
  const int m = blockIdx.x;
  const float* row = w + (int64_t)m * Kred;
  uint32_t mx = 0;
  bool bad = false;
  for (int k = threadIdx.x; k < Kred; k += blockDim.x) {
    const uint32_t b = __float_as_uint(row[k]) & 0x7fffffffu;
    bad |= b >= 0x7f800000u;
    mx = max(mx, b);
  }
  __shared__ uint32_t red[8];
  __shared__ int sE;
  mx = __reduce_max_sync(FULL_MASK, mx);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = mx;
  if (__syncthreads_or(bad) && threadIdx.x == 0) record_error(err, FGQ_ERR_NONFINITE);
  if (threadIdx.x == 0) {
    uint32_t m2 = 0;
    for (int i = 0; i < (int)(blockDim.x >> 5); ++i) m2 = max(m2, red[i]);
    int E = 0;
    if (m2 != 0 && m2 < 0x7f800000u) {
      const double md = (double)__uint_as_float(m2);
      E = (int)((__double_as_longlong(md) >> 52) & 0x7ff) - 1023 - 10;
      while (md * pow2d(-E) > 127.0) ++E;
      E = max(-149, min(127, E));
    }
    sE = E;
    wscale[m] = pow2f(E);
  }
  __syncthreads();
  const int E = sE;
  const float mul1 = (-E <= 127) ? pow2f(-E) : pow2f(64);
  const float mul2 = (-E <= 127) ? 1.0f : pow2f(-E - 64);
  for (int k = threadIdx.x; k < Kred; k += blockDim.x) {
    const float x = row[k] * mul1 * mul2;
    int r = __float2int_rn(x);
    r = max(-128, min(127, r));
    wq[(int64_t)m * Kred + k] = (int8_t)r;
  }
}

int grid_for(int64_t work_items, int threads) {
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t need = (work_items + threads - 1) / threads;
  const int64_t cap = (int64_t)sms * 16;
  return (int)(need < 1 ? 1 : (need < cap ? need : cap));
}

}  // namespace

fgq_status launch_ternarize(const float* w, int M, int Kred, int G, uint32_t* codes, float* alpha,
                            unsigned int* err, cudaStream_t s) {
  const int ng = (Kred + G - 1) / G;
  const int wrow = (ng * G + 15) / 16;
  const int threads = 256;
  const int vec4 = (Kred % 4 == 0) && ((reinterpret_cast<uintptr_t>(w) & 15) == 0);
  uint8_t* cb = reinterpret_cast<uint8_t*>(codes);
  const int64_t unit = G < 4 ? 4 : G;
  const int64_t units = (int64_t)M * ((ng * (int64_t)G + unit - 1) / unit);
  switch (G) {
    case 1: ternarize_small_kernel<1><<<grid_for(units, threads), threads, 0, s>>>(w, M, Kred, ng, wrow, cb, alpha, err, vec4); break;
    case 2: ternarize_small_kernel<2><<<grid_for(units, threads), threads, 0, s>>>(w, M, Kred, ng, wrow, cb, alpha, err, vec4); break;
    case 4: ternarize_small_kernel<4><<<grid_for(units, threads), threads, 0, s>>>(w, M, Kred, ng, wrow, cb, alpha, err, vec4); break;
    case 8: ternarize_small_kernel<8><<<grid_for(units, threads), threads, 0, s>>>(w, M, Kred, ng, wrow, cb, alpha, err, vec4); break;
    case 16: ternarize_small_kernel<16><<<grid_for(units, threads), threads, 0, s>>>(w, M, Kred, ng, wrow, cb, alpha, err, vec4); break;
    case 32: ternarize_thread_kernel<32><<<grid_for((int64_t)M * ng, TG_THREADS), TG_THREADS, 0, s>>>(w, M, Kred, ng, wrow, codes, alpha, err, vec4); break;
    case 64: ternarize_thread_kernel<64><<<grid_for((int64_t)M * ng, TG_THREADS), TG_THREADS, 0, s>>>(w, M, Kred, ng, wrow, codes, alpha, err, vec4); break;
    case 128: ternarize_warp_kernel<128><<<grid_for((int64_t)M * ng * 32, threads), threads, 0, s>>>(w, M, Kred, ng, wrow, codes, alpha, err); break;
    default: return FGQ_ERR_ARG;
  }
  return after_launch();
}

fgq_status launch_ternarize_batch(int n, const float* const* w, const int* M, const int* Kred, int G,
                                  uint32_t* const* codes, float* const* alpha, unsigned int* err, cudaStream_t s) {
  if (n > FGQ_TERNARIZE_BATCH_MAX) return FGQ_ERR_ARG;
  TernBatch b;
  memset(&b, 0, sizeof b);
  const int64_t unit = G < 4 ? 4 : G;
  int64_t total = 0;
  for (int i = 0; i < n; ++i) {
    if ((int64_t)M[i] * Kred[i] == 0) continue;  // nothing to do for an empty layer
    TernLayer& L = b.l[b.n++];
    L.w = w[i];
    L.codes = codes[i];
    L.alpha = alpha[i];
    L.Kred = Kred[i];
    L.ng = (Kred[i] + G - 1) / G;
    L.wrow = (L.ng * G + 15) / 16;
    L.vec4 = (Kred[i] % 4 == 0) && ((reinterpret_cast<uintptr_t>(w[i]) & 15) == 0);
    L.units_per_row = (L.ng * (int64_t)G + unit - 1) / unit;
    L.first = total;
    total += G >= 32 ? (int64_t)M[i] * L.ng : (int64_t)M[i] * L.units_per_row;
  }
  b.total = total;
  if (total == 0) return FGQ_OK;
  const int threads = 256;
  switch (G) {
    case 1: ternarize_small_batch_kernel<1><<<grid_for(total, threads), threads, 0, s>>>(b, err); break;
    case 2: ternarize_small_batch_kernel<2><<<grid_for(total, threads), threads, 0, s>>>(b, err); break;
    case 4: ternarize_small_batch_kernel<4><<<grid_for(total, threads), threads, 0, s>>>(b, err); break;
    case 8: ternarize_small_batch_kernel<8><<<grid_for(total, threads), threads, 0, s>>>(b, err); break;
    case 16: ternarize_small_batch_kernel<16><<<grid_for(total, threads), threads, 0, s>>>(b, err); break;
    case 32: ternarize_thread_batch_kernel<32><<<grid_for(total, TG_THREADS), TG_THREADS, 0, s>>>(b, err); break;
    case 64: ternarize_thread_batch_kernel<64><<<grid_for(total, TG_THREADS), TG_THREADS, 0, s>>>(b, err); break;
    case 128: ternarize_warp_batch_kernel<128><<<grid_for(total * 32, threads), threads, 0, s>>>(b, err); break;
    default: return FGQ_ERR_ARG;
  }
  return after_launch();
}

fgq_status launch_quantize_weights_w8(const float* w, int M, int Kred, int8_t* wq, float* wscale,
                                      unsigned int* err, cudaStream_t s) {
  quantize_w8_kernel<<<M, 256, 0, s>>>(w, Kred, wq, wscale, err);
  return after_launch();
}

}  // namespace fgq
