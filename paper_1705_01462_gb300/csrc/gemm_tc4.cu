// Tensor-core (tcgen05) grouped ternary contraction for G = 4.
//
// Math (Eq. 2, 32-bit group accumulators of Section 4): y[p][m] = s_x * sum_g alpha[m][g]
// * s[m][g][p] with s an exact integer sum over a group of 4 reduction elements.  A dense
// MMA would sum across groups, so each K = 16 MMA step (4 groups) uses a block-diagonal
// ternary operand A' of 128 rows: row 4 m' + j holds filter m' of the tile (32 filters) only
// in the 4 columns of group slot j (zeros elsewhere), and D[4 m' + j][p] of one MMA
// (M = 128, N = 256, K = 16) receives the products of group 4 step + j alone.  A' depends
// only on the weights, so it is built once per call; the activations are the plain dense
// operand, expanded to fp16 once per call (one launch, prep4_kernel, prepares both) and
// loaded by TMA (2D rows or im2col boxes), and no thread builds operands inside the
// contraction.  Two variants:
//
//   output (FOLD): the group's scale multiplies inside the MMA (one multiply per group,
//     Section 4.1): A' carries the fp32 alpha folded into the codes as two fp16 parts,
//     alpha(m, g) t[m][k] 2^e_m = hi + lo to about 22 bits (hi the fp16 nearest, lo the fp16
//     nearest the remainder; e_m puts row m's largest alpha in [2^14, 2^15)).  Every product
//     hi t q and lo t q is exact in fp32 and so is each part's group sum hi s_g (11
//     significant bits times |s_g| <= 1020), so one step adds (hi + lo) s_g to the element its
//     slot owns.  The 8 MMAs of a K-tile (4 steps x 2 parts) accumulate in TMEM, and the
//     epilogue adds each K-tile's partials into fp32 registers with round-to-nearest adds:
//     every rounding is bounded by a K-tile's share of sum_g |alpha_g s_g|, far inside the
//     1e-5 sum_g |alpha_g s_g| tolerance.  At tile end the four slot rows of a filter are
//     summed across lanes (shuffles) and y = s_x 2^-e_m acc.
//   group sums (!FOLD): A' carries the codes in fp16 {0, +1, -1}; each step's D is exactly
//     s[m][g][p] (fp16 operands on exact integers), drained per step and stored as int32
//     (for verification of the integer accumulators).
//
// Tile: 32 filters x 256 positions; K-tile 64 (16 groups, 4 steps); TMEM: two 256-column
// accumulators.
// Warp roles (352 threads, one CTA per SM, persistent over tiles):
//   warps 0-7  epilogue: warp w reads TMEM lanes 32 (w % 4) .. (filter rows x slots) and the
//              128 positions of half w / 4 in 16-column loads, frees the buffer, and adds the
//              values into 128 fp32 registers (output) or stores them as int32 (group sums).
//              At tile end: the slot reduction, then the 32 x 256 output box through shared
//              memory by one TMA store when the output allows, else direct stores (or
//              requantized codes).
//   warps 8, 9 the MMA issuers (one thread each; warp 8 also allocates TMEM): alternate drain
//              units (K-tiles when folded, steps otherwise) into their own accumulator, so
//              one thread's barrier waits overlap the other's MMAs.
//   warp 10    the producer (one thread): per K-tile, the A' box(es) (64 reduction elements x
//              128 rows per part) and the activation box (64 channels x 256 positions) into
//              one ring stage.
// A stage is released by the epilogue when it sees the K-tile's last accumulator commit, so
// no commit is spent on the stages.  Every mbarrier wait is bounded in time; on expiry the
// kernel records FGQ_ERR_TIMEOUT, each role leaves its loop (uniformly within the epilogue,
// which uses named barriers), in-flight copies and MMAs are waited for, and TMEM is freed.
#include <cuda_fp16.h>

#include <cstdint>
#include <cstring>

#include "operand_prep.cuh"
#include "tc_common.cuh"

namespace fgq {
namespace {

using tc::encode_tiled;
using tc::make_map_2d;

constexpr int T4_FM = 32;       // filters per tile
constexpr int T4_ROWS = 128;    // MMA M: 4 slots x 32 filters, row 4 m' + j
constexpr int T4_BN = 256;      // positions per tile (MMA N)
constexpr int T4_KT = 64;       // reduction elements per K-tile: 16 groups, 4 MMA steps
constexpr int T4_NACC = 2;      // TMEM accumulators of 256 columns
constexpr int T4_EPI_WARPS = 8;
constexpr int T4_MMA_WARP = 8;  // warps 8 and 9
constexpr int T4_PROD_WARP = 10;
constexpr int T4_THREADS = 32 * (T4_PROD_WARP + 1);
constexpr int T4_TMEM_COLS = T4_NACC * T4_BN;
constexpr int T4_EPI_COLS = T4_BN / 2;             // positions per epilogue thread
constexpr uint64_t T4_TIMEOUT_NS = 1000000000ull;  // 1 s per wait
constexpr uint32_t T4_DRAIN_LIMIT = 1u << 20;      // polls of the final drains (never shortened)
constexpr uint32_t BAR_EPI4 = 2;

constexpr int A_TILE4 = T4_ROWS * T4_KT * 2;  // 16 KB fp16 block-diagonal operand, per part
constexpr int B_TILE4 = T4_BN * T4_KT * 2;    // 32 KB fp16 activations
constexpr int OUT_BOX4 = T4_BN * T4_FM * 4;   // 32 KB fp32 [256 positions][32 filters]

// Shared-memory plan of a variant: operand ring (A' parts + activations), output box, barriers.
template <bool FOLD>
struct T4Cfg {
  static constexpr int NPART = FOLD ? 2 : 1;
  static constexpr int STAGE = NPART * A_TILE4 + B_TILE4;
  static constexpr int NST = FOLD ? 3 : 4;
  static constexpr int OUT = FOLD ? OUT_BOX4 : 0;
  static constexpr int BAR = 8 * (2 * NST + 2 * T4_NACC + 1) + 16;
  static constexpr int SMEM = 1024 + NST * STAGE + OUT + BAR;
};
static_assert(T4Cfg<true>::SMEM <= 232448 && T4Cfg<false>::SMEM <= 232448, "shared memory budget");
static_assert(A_TILE4 % 1024 == 0 && B_TILE4 % 1024 == 0, "stage alignment");

struct T4Args {
  CUtensorMap a_map[2];   // fp16 A' [(groups * mtiles) * 128 rows][Kp] per part, box {64, 128}, 128B swizzle
  CUtensorMap act_map;    // fp16 activations: 2D [positions][C] or im2col, box 64 channels x 256 positions
  CUtensorMap out_map;    // fp32 [P][M], box {32 filters, 256 positions}; if out_tma
  const float* row_scale;  // FOLD: 2^-e_m [M]
  const float* act_scale;
  float* out;
  int32_t* sums;  // !FOLD: int32 group sums [M][ng][P]
  unsigned int* err;
  Geom g;
  int mtiles, ptiles, ntiles, ktiles;  // mtiles: 32-filter tiles per conv group
  int mtiles2;                         // CTA pairs: 64-filter tiles per conv group (ntiles counts pair tiles)
  int out_tma;
  uint64_t timeout_ns;
};

// Tiles are numbered with the filter tiles of one position tile consecutive, so that
// CTAs running at the same time share activation boxes in L2.
__device__ __forceinline__ void tile_coords4(const T4Args& a, int tile, int& gi, int& mt, int64_t& p0) {
  const int per_p = a.g.groups * a.mtiles;
  const int pt = tile / per_p;
  const int r = tile - pt * per_p;
  gi = r / a.mtiles;
  mt = r - gi * a.mtiles;
  p0 = (int64_t)pt * T4_BN;
}

// One launch prepares both operands of a call.  Blocks [0, fold_blocks) build the
// block-diagonal ternary operand A' straight from the 2-bit codes, one block per 32-filter
// tile and slice of the reduction axis: row 4 m' + j of tile (gi, mt) holds, for filter
// gi Mg + mt 32 + m', the elements of the groups whose index is j modulo 4 (slot j of every
// K = 16 step) and zeros elsewhere.  FOLD: the elements are alpha(m, g) 2^e_m t split into
// fp16 hi + lo (hi the fp16 nearest, lo the fp16 nearest the remainder), parts a0 and a1,
// where e_m puts the row's largest alpha in [2^14, 2^15) (clamped to [-100, 100]; an all-zero
// row keeps e = 0) so that the low part stays clear of fp16's subnormal range -- each block
// first finds e_m for its 32 filters (rs[m] = 2^-e_m written by the first slice); otherwise
// the codes as fp16 {0, +1, -1} in a0.  One thread per 16-byte chunk of A' (8 elements = 2
// groups, at most one of them in the row's slot).  The other blocks expand the activations
// to fp16.
constexpr int PREP4_CHUNKS = 8;  // 16-byte chunks of a row per fold block (64 elements)

template <bool FOLD>
__global__ void __launch_bounds__(256) prep4_kernel(const uint32_t* __restrict__ codes, int wrow,
                                                    const float* __restrict__ alpha, int ng, float* __restrict__ rs,
                                                    int Kp, int Mg, int mtiles, int ksplit, uint4* __restrict__ a0,
                                                    uint4* __restrict__ a1, int fold_blocks, const prep::ActSrc src,
                                                    uint4* __restrict__ x16) {
  pdl_wait();
  pdl_trigger();
  if ((int)blockIdx.x >= fold_blocks) {
    const int64_t nb = (int64_t)gridDim.x - fold_blocks;
    prep::act_expand<false>(src, ((int64_t)blockIdx.x - fold_blocks) * blockDim.x + threadIdx.x, nb * blockDim.x, x16);
    return;
  }
  const int tile = (int)blockIdx.x / ksplit, ks = (int)blockIdx.x - tile * ksplit;
  const int gi = tile / mtiles, mt = tile - gi * mtiles;
  __shared__ float mul[T4_FM];  // 2^e_m of the tile's filters
  if (FOLD) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
#pragma unroll
    for (int f = 0; f < T4_FM / 8; ++f) {
      const int mp = (T4_FM / 8) * warp + f;
      const int local = mt * T4_FM + mp;
      float mx = 0.0f;
      if (local < Mg) {
        const float* ar = alpha + ((int64_t)gi * Mg + local) * ng;
        for (int g = lane; g < ng; g += 32) mx = fmaxf(mx, __ldg(ar + g));
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      int e = mx > 0.0f ? 14 - ilogbf(mx) : 0;
      e = e < -100 ? -100 : (e > 100 ? 100 : e);
      if (lane == 0) {
        mul[mp] = ldexpf(1.0f, e);
        if (ks == 0 && local < Mg) rs[(int64_t)gi * Mg + local] = ldexpf(1.0f, -e);
      }
    }
    __syncthreads();
  }
  const int cpr = Kp / 8;  // chunks per row
  const int c0 = ks * PREP4_CHUNKS;
  const int nc = (cpr - c0) < PREP4_CHUNKS ? (cpr - c0) : PREP4_CHUNKS;
  for (int it = threadIdx.x; it < T4_ROWS * nc; it += blockDim.x) {
    const int rr = it / nc, c = c0 + (it - rr * nc);
    const int mp = rr >> 2, j = rr & 3;
    const int local = mt * T4_FM + mp;
    uint32_t h0[4] = {0u, 0u, 0u, 0u}, h1[4] = {0u, 0u, 0u, 0u};
    // group 2c occupies halves 0-3 of the chunk, group 2c + 1 halves 4-7; slot = group % 4
    const int grp = ((2 * c) & 3) == j ? 2 * c : (((2 * c + 1) & 3) == j ? 2 * c + 1 : -1);
    if (local < Mg && grp >= 0 && grp < ng) {
      const int64_t m = (int64_t)gi * Mg + local;
      const int k0 = 4 * grp;  // the group's 4 codes lie in one word, bits 2 (k0 % 16) ..
      const uint32_t cw = (__ldg(codes + m * wrow + k0 / 16) >> (2 * (k0 % 16))) & 0xffu;
      uint32_t hi = 0x3C00u, lo = 0u;  // fp16 +1 and 0: the codes themselves
      if (FOLD) {
        const float v = __ldg(alpha + m * ng + grp) * mul[mp];  // exact: a power-of-two scaling
        const __half hh = __float2half_rn(v);
        hi = __half_as_ushort(hh);
        lo = __half_as_ushort(__float2half_rn(v - __half2float(hh)));  // the remainder, exact in fp32
      }
      uint32_t e0[4], e1[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const uint32_t t = (cw >> (2 * e)) & 3u;  // 00 = 0, 01 = +1, 11 = -1
        const uint32_t sgn = t == 3u ? 0x8000u : 0u;
        const bool nz = t == 1u || t == 3u;
        e0[e] = nz ? (hi ^ sgn) : 0u;
        e1[e] = nz && lo ? (lo ^ sgn) : 0u;
      }
      // the group fills 32-bit words 0-1 of the chunk (group 2c) or 2-3 (group 2c + 1)
      const bool first = grp == 2 * c;
      const uint32_t p0 = e0[0] | (e0[1] << 16), p1 = e0[2] | (e0[3] << 16);
      const uint32_t q0 = e1[0] | (e1[1] << 16), q1 = e1[2] | (e1[3] << 16);
      h0[0] = first ? p0 : 0u;
      h0[1] = first ? p1 : 0u;
      h0[2] = first ? 0u : p0;
      h0[3] = first ? 0u : p1;
      h1[0] = first ? q0 : 0u;
      h1[1] = first ? q1 : 0u;
      h1[2] = first ? 0u : q0;
      h1[3] = first ? 0u : q1;
    }
    const int64_t i = ((int64_t)tile * T4_ROWS + rr) * cpr + c;
    a0[i] = make_uint4(h0[0], h0[1], h0[2], h0[3]);
    if (FOLD) a1[i] = make_uint4(h1[0], h1[1], h1[2], h1[3]);
  }
}

// Tile end of the output variant: the four slot rows 4 m' .. 4 m' + 3 of a filter are lanes
// 4 (lane / 4) .. + 3 of the warp; reduce them so that lane j ends with positions 4 i + j
// (i < 32) of its half, summed over the slots (two exchange rounds, each keeping half of the
// positions), scale by s_x 2^-e_m and store: one 32-filter x 256-position TMA box through
// shared memory (every epilogue thread of the CTA takes part), or direct / requantized stores.
__device__ __forceinline__ void store_tile4(const T4Args& a, float (&acc)[T4_EPI_COLS], float* otile, int gi, int mt,
                                            int64_t p0, int half, int mp, int j, bool mok, int m, float sx,
                                            bool leader) {
  const Geom& g = a.g;
  const bool b1 = (j >> 1) & 1, b0 = j & 1;
#pragma unroll
  for (int q = 0; q < T4_EPI_COLS / 4; ++q) {
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      // positions 4 q + e (slot bit 1 clear) and 4 q + 2 + e (set): keep the one whose bit 1
      // matches b1, send the other to lane ^ 2; the result goes to 4 q + e
      const float lo = acc[4 * q + e], hi = acc[4 * q + 2 + e];
      const float sent = __shfl_xor_sync(0xffffffffu, b1 ? lo : hi, 2);
      acc[4 * q + e] = (b1 ? hi : lo) + sent;
    }
    // positions 4 q + 2 b1 + 0 / + 1 (now at 4 q, 4 q + 1): keep bit 0 = b0
    const float e0 = acc[4 * q], e1 = acc[4 * q + 1];
    const float sent = __shfl_xor_sync(0xffffffffu, b0 ? e0 : e1, 1);
    acc[4 * q] = (b0 ? e1 : e0) + sent;  // position 4 q + j, all four slots
  }
  const float sc_m = mok ? sx * __ldg(a.row_scale + m) : 0.0f;
  const int64_t pbase = p0 + T4_EPI_COLS * half;
  if (a.out_tma) {
    if (leader) bulk_wait_read_all();  // the previous tile's box has been read out
    named_bar_sync(BAR_EPI4, 32 * T4_EPI_WARPS);
    float* ob = otile + (T4_EPI_COLS * half + j) * T4_FM + mp;
#pragma unroll
    for (int q = 0; q < T4_EPI_COLS / 4; ++q) ob[4 * q * T4_FM] = sc_m * acc[4 * q];
    fence_proxy_async_smem();
    named_bar_sync(BAR_EPI4, 32 * T4_EPI_WARPS);
    if (leader) {  // rows past P and filters past M are clipped by the tensor map
      tma_store_2d(&a.out_map, gi * g.Mg + mt * T4_FM, (int)p0, smem_u32(otile));
      bulk_commit();
    }
  } else if (mok) {
    if (g.rq_out) {  // fused requantization: 8-bit codes instead of fp32
      const RqMul r = rq_mul(g.rq_scale, g.rq_signed);
#pragma unroll
      for (int q = 0; q < T4_EPI_COLS / 4; ++q) {
        const int64_t p = pbase + 4 * q + j;
        if (p < g.P) g.rq_out[p * g.M + m] = rq_code(sc_m * acc[4 * q], r);
      }
    } else {
#pragma unroll
      for (int q = 0; q < T4_EPI_COLS / 4; ++q) {
        const int64_t p = pbase + 4 * q + j;
        if (p < g.P) a.out[p * g.M + m] = sc_m * acc[4 * q];
      }
    }
  }
}

template <bool TMAP, bool FOLD>
__global__ void __launch_bounds__(T4_THREADS, 1) tc4_contract_kernel(const __grid_constant__ T4Args a) {
  using Cfg = T4Cfg<FOLD>;
  constexpr int NST = Cfg::NST;
  extern __shared__ uint8_t smem_raw4[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw4) + 1023) & ~uintptr_t(1023));
  float* otile = reinterpret_cast<float*>(smem + NST * Cfg::STAGE);  // [256 positions][32 filters]
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + NST * Cfg::STAGE + Cfg::OUT);
  uint64_t* full = bars;
  uint64_t* empty = bars + NST;
  uint64_t* acc_full = empty + NST;
  uint64_t* acc_empty = acc_full + T4_NACC;
  uint64_t* drain_bar = acc_empty + T4_NACC;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_bar + 1);
  volatile uint32_t* abort_flag = tmem_slot + 1;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const Geom& g = a.g;
  const uint64_t tmo = a.timeout_ns;

  if (threadIdx.x == 0) {
    for (int i = 0; i < NST; ++i) {
      mbar_init(&full[i], 1);   // the producer's expect_tx, then the boxes' bytes
      mbar_init(&empty[i], 1);  // released by the epilogue (the K-tile's MMAs completed)
    }
    for (int i = 0; i < T4_NACC; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], T4_EPI_WARPS);
    }
    mbar_init(drain_bar, T4_NACC);  // one commit per MMA issuer
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == T4_MMA_WARP) {
    tmem_alloc(tmem_slot, T4_TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // the prologue above overlapped the previous kernel; global memory only from here on
  pdl_wait();
  pdl_trigger();
  const int my_tiles = (a.ntiles - (int)blockIdx.x + (int)gridDim.x - 1) / (int)gridDim.x;
  const int units_per_tile = FOLD ? a.ktiles : 4 * a.ktiles;  // drains per tile

  auto fail = [&]() {
    *abort_flag = 1;
    record_error(a.err, FGQ_ERR_TIMEOUT);
  };

  // ------------------------------------------------------------------ producer
  if (warp == T4_PROD_WARP && lane == 0) {
    const int total = my_tiles * a.ktiles;
    int gi = 0, mt = 0, tr = 0, ts = 0, tc0 = 0, kt = 0, tl = 0;
    int64_t p0 = 0;
    int n0 = 0, h0 = 0, w0 = 0;  // im2col: the tile's first window origin (input pixel coordinates)
    int issued = 0;
    bool ok = true;
    for (int j = 0; j < total; ++j) {
      if (kt == 0) {
        tile_coords4(a, (int)blockIdx.x + tl * (int)gridDim.x, gi, mt, p0);
        tr = ts = tc0 = 0;
        if (!TMAP) {
          const int pp = (int)p0;  // < P < 2^31
          const int wo = pp % g.Wo;
          const int q = pp / g.Wo;
          n0 = q / g.Ho;
          h0 = (q - n0 * g.Ho) * g.stride - g.pad;
          w0 = wo * g.stride - g.pad;
        }
      }
      const int s = j % NST;
      if (j >= NST && !mbar_wait_timed(&empty[s], ((j / NST) & 1) ^ 1, tmo, abort_flag, 64)) {
        ok = false;
        break;
      }
      uint8_t* sa = smem + s * Cfg::STAGE;
      const int arow = (gi * a.mtiles + mt) * T4_ROWS;
      const int ch = gi * g.Cg + tc0;  // a multiple of 64 (128-byte aligned in fp16)
      mbar_arrive_expect_tx(&full[s], Cfg::STAGE);
#pragma unroll
      for (int part = 0; part < Cfg::NPART; ++part)
        tma_load_2d(smem_u32(sa + part * A_TILE4), &a.a_map[part], kt * T4_KT, arow, &full[s]);
      uint8_t* sb = sa + Cfg::NPART * A_TILE4;
      if (TMAP)
        tma_load_2d(smem_u32(sb), &a.act_map, ch, (int)p0, &full[s]);
      else
        tma_load_im2col_4d(smem_u32(sb), &a.act_map, ch, w0, h0, n0, (uint16_t)ts, (uint16_t)tr, &full[s]);
      issued = j + 1;
      tc0 += T4_KT;
      if (tc0 == g.Cg) {
        tc0 = 0;
        if (++ts == g.S) {
          ts = 0;
          ++tr;
        }
      }
      if (++kt == a.ktiles) {
        kt = 0;
        ++tl;
      }
    }
    if (!ok && !*abort_flag) fail();
    // loads the MMA issuers may not have consumed: the last NST issued, one per stage, each
    // the latest phase of its stage's barrier; none may outlive the CTA
    for (int j = issued - NST < 0 ? 0 : issued - NST; j < issued; ++j)
      mbar_wait_bounded(&full[j % NST], (j / NST) & 1, T4_DRAIN_LIMIT);
  }

  // ------------------------------------------------------------------ MMA issuers
  if ((warp == T4_MMA_WARP || warp == T4_MMA_WARP + 1) && lane == 0) {
    const int b = warp - T4_MMA_WARP;  // this thread's accumulator: the units of its parity
    const uint32_t idesc = idesc_f16_f32(T4_ROWS, T4_BN);
    const int total = my_tiles * units_per_tile;
    const uint32_t d = tmem + (uint32_t)(b * T4_BN);
    bool ok = true;
    for (int u = b; u < total && ok; u += 2) {
      if (!mbar_wait_timed(&acc_empty[b], ((u >> 1) & 1) ^ 1, tmo, abort_flag, 0)) {
        ok = false;
        break;
      }
      const int kt = FOLD ? u : u >> 2;  // the CTA's K-tile sequence number
      const int s = kt % NST;
      if (!mbar_wait_timed(&full[s], (kt / NST) & 1, tmo, abort_flag, 0)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t abase = smem_u32(smem + s * Cfg::STAGE);
      const uint64_t bd = sdesc_k_sw128(abase + Cfg::NPART * A_TILE4);
      if (FOLD) {
        // the K-tile's 8 MMAs (4 steps x 2 parts) accumulate into this thread's buffer
#pragma unroll
        for (int st = 0; st < 4; ++st)
#pragma unroll
          for (int part = 0; part < 2; ++part)
            mma_f16(d, sdesc_k_sw128(abase + part * A_TILE4) + 2 * st, bd + 2 * st, idesc, (st | part) != 0 ? 1u : 0u);
      } else {
        const int st = u & 3;  // one step: the exact sums of its 4 groups
        mma_f16(d, sdesc_k_sw128(abase) + 2 * st, bd + 2 * st, idesc, 0u);
      }
      mma_commit(&acc_full[b]);
    }
    if (!ok && !*abort_flag) fail();
    // all MMAs issued by both threads are complete once the drain barrier flips
    mma_commit(drain_bar);
    mbar_wait_bounded(drain_bar, 0, T4_DRAIN_LIMIT);
  }

  // ------------------------------------------------------------------ epilogue
  if (warp < T4_EPI_WARPS) {
    const int quarter = warp & 3, half = warp >> 2;
    const int mp = 8 * quarter + (lane >> 2);  // filter of the tile
    const int j = lane & 3;                    // group slot of this TMEM lane
    const uint32_t tbase = tmem + ((uint32_t)(32 * quarter) << 16) + (uint32_t)(T4_EPI_COLS * half);
    const float sx = __ldg(a.act_scale);
    const bool leader = threadIdx.x == 0;
    int u = 0;  // drain units of this CTA so far
    bool ok = true;
    for (int tl = 0; tl < my_tiles; ++tl) {
      int gi, mt;
      int64_t p0;
      tile_coords4(a, (int)blockIdx.x + tl * (int)gridDim.x, gi, mt, p0);
      const int local = mt * T4_FM + mp;
      const int m = gi * g.Mg + local;
      const bool mok = local < g.Mg;
      const int64_t pbase = p0 + T4_EPI_COLS * half;
      float acc[T4_EPI_COLS];
#pragma unroll
      for (int i = 0; i < T4_EPI_COLS; ++i) acc[i] = 0.0f;
      for (int k = 0; k < units_per_tile; ++k, ++u) {
        if (!ok) continue;
        const int b = u & 1;
        if (!mbar_wait_timed(&acc_full[b], (u >> 1) & 1, tmo, abort_flag, 0)) {
          ok = false;
          continue;
        }
        if (leader && (FOLD || (u & 3) == 3)) {
          // the K-tile's MMAs have completed: its stage may be refilled
          const int kt = FOLD ? u : u >> 2;
          mbar_arrive(&empty[kt % NST]);
        }
        tc_fence_after();
        const uint32_t ta = tbase + (uint32_t)(b * T4_BN);
        if constexpr (FOLD) {
#pragma unroll
          for (int c = 0; c < T4_EPI_COLS / 16; ++c) {
            uint32_t r[16];
            tmem_ld16(ta + 16 * c, r);
            tmem_ld_wait_regs16(r);
            if (c == T4_EPI_COLS / 16 - 1) {
              tc_fence_before();
              __syncwarp();
              if (lane == 0) mbar_arrive(&acc_empty[b]);  // every column of the K-tile is in registers
            }
#pragma unroll
            for (int i = 0; i < 16; ++i) acc[16 * c + i] += __uint_as_float(r[i]);
          }
        } else {
          // exact sums of group 16 kt + 4 step + j, filter m, positions pbase + i
          const int grp = 16 * (k >> 2) + 4 * (k & 3) + j;
          int32_t* srow = a.sums + ((int64_t)(mok ? m : 0) * g.ng + (grp < g.ng ? grp : 0)) * g.P;
#pragma unroll
          for (int c = 0; c < T4_EPI_COLS / 16; ++c) {
            uint32_t r[16];
            tmem_ld16(ta + 16 * c, r);
            tmem_ld_wait_regs16(r);
            if (c == T4_EPI_COLS / 16 - 1) {
              tc_fence_before();
              __syncwarp();
              if (lane == 0) mbar_arrive(&acc_empty[b]);
            }
            if (mok && grp < g.ng) {
#pragma unroll
              for (int i = 0; i < 16; ++i) {
                const int64_t p = pbase + 16 * c + i;
                if (p < g.P) srow[p] = __float2int_rn(__uint_as_float(r[i]));
              }
            }
          }
        }
      }
      if (!ok && !*abort_flag) fail();
      if (named_bar_or(BAR_EPI4, 32 * T4_EPI_WARPS, !ok)) break;
      if constexpr (FOLD)
        store_tile4(a, acc, otile, gi, mt, p0, half, mp, j, mok, m, sx, leader);
    }
    if (leader) bulk_wait_all();
  }

  tc_fence_before();
  __syncthreads();
  if (warp == T4_MMA_WARP) {
    tc_fence_after();
    tmem_dealloc(tmem, T4_TMEM_COLS);
  }
}

// CTA-pair variant of the output kernel.  Two CTAs (a cluster) share a 64-filter x
// 256-position tile: CTA r holds the block-diagonal rows of filters 32 r .. of the pair's 64
// and positions 128 r .. of the 256, and one thread of CTA 0 issues M = 256, N = 256 MMAs
// (cta_group::2) that read both CTAs' operands and write each CTA's 128 TMEM lanes.  Per SM,
// a K-tile moves 48 KB into shared memory instead of 64 KB and each MMA reads 8 KB of it
// instead of 12 KB.  Synchronisation across the pair: CTA 1's loads complete on its own
// barriers and a forwarding thread passes each completion to CTA 0 (pfull); the MMA commit
// arrives on both CTAs' acc_full; CTA 1's epilogue warps free an accumulator with remote
// arrivals on CTA 0's acc_empty.  Each CTA frees its own stages (the epilogue relay).
constexpr int P4_NST = 4;
constexpr int P4_STAGE = 2 * A_TILE4 + B_TILE4 / 2;  // A' hi, lo + this CTA's 128 positions
constexpr int P4_BAR = 8 * (3 * P4_NST + 2 * T4_NACC + 1) + 16;
constexpr int P4_SMEM = 1024 + P4_NST * P4_STAGE + OUT_BOX4 + P4_BAR;
static_assert(P4_SMEM <= 232448, "shared memory budget");

__device__ __forceinline__ void pair_tile_coords(const T4Args& a, int tile, uint32_t rank, int& gi, int& mt,
                                                 int64_t& p0) {
  const int per_p = a.g.groups * a.mtiles2;
  const int pt = tile / per_p;
  const int r = tile - pt * per_p;
  gi = r / a.mtiles2;
  mt = 2 * (r - gi * a.mtiles2) + (int)rank;
  p0 = (int64_t)pt * T4_BN;
}

template <bool TMAP>
__global__ void __launch_bounds__(T4_THREADS, 1) tc4_pair_kernel(const __grid_constant__ T4Args a) {
  constexpr int NST = P4_NST;
  extern __shared__ uint8_t smem_raw4p[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw4p) + 1023) & ~uintptr_t(1023));
  float* otile = reinterpret_cast<float*>(smem + NST * P4_STAGE);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + NST * P4_STAGE + OUT_BOX4);
  uint64_t* full = bars;                // this CTA's stage loaded
  uint64_t* empty = bars + NST;         // this CTA's stage free
  uint64_t* pfull = bars + 2 * NST;     // CTA 0: CTA 1's stage loaded (forwarded)
  uint64_t* acc_full = bars + 3 * NST;
  uint64_t* acc_empty = acc_full + T4_NACC;  // CTA 0: both CTAs' epilogues drained
  uint64_t* drain_bar = acc_empty + T4_NACC;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_bar + 1);
  volatile uint32_t* abort_flag = tmem_slot + 1;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const Geom& g = a.g;
  const uint64_t tmo = a.timeout_ns;
  const uint32_t rank = cluster_ctarank();
  const int pair = (int)blockIdx.x >> 1, npairs = (int)gridDim.x >> 1;

  if (threadIdx.x == 0) {
    for (int i = 0; i < NST; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
      mbar_init(&pfull[i], 1);
    }
    for (int i = 0; i < T4_NACC; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], 2 * T4_EPI_WARPS);  // the epilogue warps of both CTAs
    }
    mbar_init(drain_bar, T4_NACC);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == T4_MMA_WARP) {
    tmem_alloc_pair(tmem_slot, T4_TMEM_COLS);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // both CTAs' barriers exist before any remote arrival
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const int my_tiles = (a.ntiles - pair + npairs - 1) / npairs;
  const int total = my_tiles * a.ktiles;

  auto fail = [&]() {
    *abort_flag = 1;
    record_error(a.err, FGQ_ERR_TIMEOUT);
  };

  // ------------------------------------------------------------------ producer (each CTA)
  if (warp == T4_PROD_WARP && lane == 0) {
    int gi = 0, mt = 0, tr = 0, ts = 0, tc0 = 0, kt = 0, tl = 0;
    int64_t p0 = 0;
    int n0 = 0, h0 = 0, w0 = 0;
    int issued = 0;
    bool ok = true;
    for (int j = 0; j < total; ++j) {
      if (kt == 0) {
        pair_tile_coords(a, pair + tl * npairs, rank, gi, mt, p0);
        tr = ts = tc0 = 0;
        if (!TMAP) {
          const int pp = (int)p0 + (T4_BN / 2) * (int)rank;  // this CTA's first position
          const int wo = pp % g.Wo;
          const int q = pp / g.Wo;
          n0 = q / g.Ho;
          h0 = (q - n0 * g.Ho) * g.stride - g.pad;
          w0 = wo * g.stride - g.pad;
        }
      }
      const int s = j % NST;
      if (j >= NST && !mbar_wait_timed(&empty[s], ((j / NST) & 1) ^ 1, tmo, abort_flag, 64)) {
        ok = false;
        break;
      }
      uint8_t* sa = smem + s * P4_STAGE;
      const int arow = (gi * a.mtiles + mt) * T4_ROWS;  // past the group's filters: masked at the end
      const int ch = gi * g.Cg + tc0;
      mbar_arrive_expect_tx(&full[s], P4_STAGE);
      tma_load_2d(smem_u32(sa), &a.a_map[0], kt * T4_KT, arow, &full[s]);
      tma_load_2d(smem_u32(sa + A_TILE4), &a.a_map[1], kt * T4_KT, arow, &full[s]);
      uint8_t* sb = sa + 2 * A_TILE4;
      if (TMAP)
        tma_load_2d(smem_u32(sb), &a.act_map, ch, (int)p0 + (T4_BN / 2) * (int)rank, &full[s]);
      else
        tma_load_im2col_4d(smem_u32(sb), &a.act_map, ch, w0, h0, n0, (uint16_t)ts, (uint16_t)tr, &full[s]);
      issued = j + 1;
      tc0 += T4_KT;
      if (tc0 == g.Cg) {
        tc0 = 0;
        if (++ts == g.S) {
          ts = 0;
          ++tr;
        }
      }
      if (++kt == a.ktiles) {
        kt = 0;
        ++tl;
      }
    }
    if (!ok && !*abort_flag) fail();
    for (int j = issued - NST < 0 ? 0 : issued - NST; j < issued; ++j)
      mbar_wait_bounded(&full[j % NST], (j / NST) & 1, T4_DRAIN_LIMIT);
  }

  // ------------------------------------------------------------------ CTA 1: forwarder
  if (rank == 1 && warp == T4_MMA_WARP && lane == 0) {
    const uint32_t lead_pfull = mapa_shared(pfull, 0);
    bool ok = true;
    for (int j = 0; j < total; ++j) {
      const int s = j % NST;
      if (!mbar_wait_timed(&full[s], (j / NST) & 1, tmo, abort_flag, 0)) {
        ok = false;
        break;
      }
      mbar_arrive_cluster(lead_pfull + 8u * (uint32_t)s);
    }
    if (!ok && !*abort_flag) fail();
  }

  // ------------------------------------------------------------------ CTA 0: MMA issuers
  if (rank == 0 && (warp == T4_MMA_WARP || warp == T4_MMA_WARP + 1) && lane == 0) {
    const int b = warp - T4_MMA_WARP;
    const uint32_t idesc = idesc_f16_f32(2 * T4_ROWS, T4_BN);
    const uint32_t d = tmem + (uint32_t)(b * T4_BN);
    bool ok = true;
    for (int u = b; u < total && ok; u += 2) {
      if (!mbar_wait_timed(&acc_empty[b], ((u >> 1) & 1) ^ 1, tmo, abort_flag, 0)) {
        ok = false;
        break;
      }
      const int s = u % NST;
      if (!mbar_wait_timed(&full[s], (u / NST) & 1, tmo, abort_flag, 0) ||
          !mbar_wait_timed(&pfull[s], (u / NST) & 1, tmo, abort_flag, 0)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t abase = smem_u32(smem + s * P4_STAGE);
      const uint64_t bd = sdesc_k_sw128(abase + 2 * A_TILE4);
#pragma unroll
      for (int st = 0; st < 4; ++st)
#pragma unroll
        for (int part = 0; part < 2; ++part)
          mma_f16_pair(d, sdesc_k_sw128(abase + part * A_TILE4) + 2 * st, bd + 2 * st, idesc, (st | part) != 0 ? 1u : 0u);
      mma_commit_pair(&acc_full[b], 3);
    }
    if (!ok && !*abort_flag) fail();
    mma_commit_pair(drain_bar, 1);
    mbar_wait_bounded(drain_bar, 0, T4_DRAIN_LIMIT);
  }

  // ------------------------------------------------------------------ epilogue (each CTA)
  if (warp < T4_EPI_WARPS) {
    const int quarter = warp & 3, half = warp >> 2;
    const int mp = 8 * quarter + (lane >> 2);
    const int j = lane & 3;
    const uint32_t tbase = tmem + ((uint32_t)(32 * quarter) << 16) + (uint32_t)(T4_EPI_COLS * half);
    const uint32_t lead_acc_empty = mapa_shared(acc_empty, 0);
    const float sx = __ldg(a.act_scale);
    const bool leader = threadIdx.x == 0;
    int u = 0;
    bool ok = true;
    for (int tl = 0; tl < my_tiles; ++tl) {
      int gi, mt;
      int64_t p0;
      pair_tile_coords(a, pair + tl * npairs, rank, gi, mt, p0);
      const int local = mt * T4_FM + mp;
      const int m = gi * g.Mg + local;
      const bool mok = local < g.Mg;
      float acc[T4_EPI_COLS];
#pragma unroll
      for (int i = 0; i < T4_EPI_COLS; ++i) acc[i] = 0.0f;
      for (int k = 0; k < a.ktiles; ++k, ++u) {
        if (!ok) continue;
        const int b = u & 1;
        if (!mbar_wait_timed(&acc_full[b], (u >> 1) & 1, tmo, abort_flag, 0)) {
          ok = false;
          continue;
        }
        if (leader) mbar_arrive(&empty[u % NST]);  // the K-tile's MMAs are complete: free this CTA's stage
        tc_fence_after();
        const uint32_t ta = tbase + (uint32_t)(b * T4_BN);
#pragma unroll
        for (int c = 0; c < T4_EPI_COLS / 16; ++c) {
          uint32_t r[16];
          tmem_ld16(ta + 16 * c, r);
          tmem_ld_wait_regs16(r);
          if (c == T4_EPI_COLS / 16 - 1) {
            tc_fence_before();
            __syncwarp();
            if (lane == 0) {  // the accumulator is free once both CTAs have it in registers
              if (rank == 0) mbar_arrive(&acc_empty[b]);
              else mbar_arrive_cluster(lead_acc_empty + 8u * (uint32_t)b);
            }
          }
#pragma unroll
          for (int i = 0; i < 16; ++i) acc[16 * c + i] += __uint_as_float(r[i]);
        }
      }
      if (!ok && !*abort_flag) fail();
      if (named_bar_or(BAR_EPI4, 32 * T4_EPI_WARPS, !ok)) break;
      store_tile4(a, acc, otile, gi, mt, p0, half, mp, j, mok, m, sx, leader);
    }
    if (leader) bulk_wait_all();
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // no CTA leaves while the pair's MMAs or arrivals may still reach it
  if (warp == T4_MMA_WARP) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, T4_TMEM_COLS);
  }
}

// CTA pairs the device runs at once: not every SM can pair with a neighbour of its cluster
// domain, so a persistent grid of SMs / 2 pairs would leave some pairs waiting for others to
// finish all their tiles.  Queried once per device and kernel.
template <bool TMAP>
int resident_pairs() {
  constexpr int kDev = 64;
  static std::once_flag once[kDev];
  static int n[kDev];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kDev) return 0;
  std::call_once(once[dev], [&] {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(2);
    cfg.blockDim = dim3(T4_THREADS);
    cfg.dynamicSmemBytes = P4_SMEM;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int c = 0;
    n[dev] = cudaOccupancyMaxActiveClusters(&c, tc4_pair_kernel<TMAP>, &cfg) == cudaSuccess ? c : 0;
  });
  return n[dev];
}

template <bool TMAP>
fgq_status launch_tc4_pair(const T4Args& args, int ntiles, cudaStream_t s) {
  if (!tc::smem_attr_once<tc4_pair_kernel<TMAP>>(P4_SMEM)) return FGQ_ERR_CUDA;
  const int resident = resident_pairs<TMAP>();
  if (resident <= 0) return FGQ_ERR_CUDA;
  const int npairs = ntiles < resident ? ntiles : resident;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(2 * npairs));
  cfg.blockDim = dim3(T4_THREADS);
  cfg.dynamicSmemBytes = P4_SMEM;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (cudaLaunchKernelEx(&cfg, tc4_pair_kernel<TMAP>, args) != cudaSuccess) return FGQ_ERR_CUDA;
  return after_launch();
}

template <bool TMAP, bool FOLD>
fgq_status launch_tc4(const T4Args& args, int grid, cudaStream_t s) {
  constexpr int smem = T4Cfg<FOLD>::SMEM;
  if (!tc::smem_attr_once<tc4_contract_kernel<TMAP, FOLD>>(smem)) return FGQ_ERR_CUDA;
  return after_launch(launch_pdl(tc4_contract_kernel<TMAP, FOLD>, dim3(grid), dim3(T4_THREADS), smem, s, args));
}

// Both operands of a call in one launch: A' (both parts when folded) with the row scales rs,
// and the activations in fp16.
fgq_status launch_prep4(const Geom& g, const uint32_t* codes, const float* alpha, float* rs, int mtiles, void* a0,
                        void* a1, const void* act, void* x16, cudaStream_t s) {
  const int ksplit = (g.Kp / 8 + PREP4_CHUNKS - 1) / PREP4_CHUNKS;
  const int fold_blocks = g.groups * mtiles * ksplit;
  const prep::ActSrc src = prep::act_src(act, g);
  const int xb = prep::blocks_for(src.nchunks);
  const dim3 grid(fold_blocks + xb), block(256);
  if (a1)
    return after_launch(launch_pdl(prep4_kernel<true>, grid, block, 0, s, codes, g.wrow, alpha, g.ng, rs, g.Kp,
                                       g.Mg, mtiles, ksplit, static_cast<uint4*>(a0), static_cast<uint4*>(a1),
                                       fold_blocks, src, static_cast<uint4*>(x16)));
  return after_launch(launch_pdl(prep4_kernel<false>, grid, block, 0, s, codes, g.wrow,
                                     static_cast<const float*>(nullptr), g.ng, static_cast<float*>(nullptr), g.Kp, g.Mg,
                                     mtiles, ksplit, static_cast<uint4*>(a0), static_cast<uint4*>(nullptr), fold_blocks,
                                     src, static_cast<uint4*>(x16)));
}

}  // namespace

bool tc4_supports(const Geom& g) {
  if (g.G != 4) return false;
  if (g.P >= (int64_t)1 << 31) return false;  // positions decoded in 32 bits
  // every K-tile inside one filter tap (conv) or row (GEMM); activation boxes by 2D or
  // im2col maps of the fp16 copy
  return tc::act16_supported(g);
}

fgq_status launch_tc4_contract(const void* act, const Geom& g, const uint32_t* codes, const float* alpha,
                               const float* act_scale, float* out, int32_t* sums, unsigned int* err,
                               cudaStream_t s) {
  if (!tc4_supports(g)) return FGQ_ERR_UNSUPPORTED;
  T4Args a;
  memset(&a, 0, sizeof a);
  a.act_scale = act_scale;
  a.out = out;
  a.sums = sums;
  a.err = err;
  a.g = g;
  a.mtiles = (g.Mg + T4_FM - 1) / T4_FM;
  a.ptiles = (int)((g.P + T4_BN - 1) / T4_BN);
  a.ktiles = g.Kp / T4_KT;
  const bool fold = sums == nullptr;
  // fp32 outputs run on CTA pairs (64 filters x 256 positions per pair) unless a test asked
  // for single CTAs; the group sums always on single CTAs
  const bool pairs = fold && debug_cta_pairs();
  a.mtiles2 = (a.mtiles + 1) / 2;
  a.ntiles = g.groups * (pairs ? a.mtiles2 : a.mtiles) * a.ptiles;
  // a test may shorten the waits (debug_wait_limit_us), never the final drains
  const int64_t lim_us = debug_wait_limit_us();
  a.timeout_ns = lim_us < 0 ? T4_TIMEOUT_NS : (uint64_t)lim_us * 1000u;

  // temporaries from the stream-ordered pool: the block-diagonal ternary operand A' per part
  // (folded hi, lo; or the codes), the row scales, and the activations in fp16
  cudaMemPool_t pool = scratch_pool();
  if (!pool) return FGQ_ERR_CUDA;
  const int nparts = fold ? 2 : 1;
  const int64_t arows = (int64_t)g.groups * a.mtiles * T4_ROWS;
  const size_t diag_bytes = (size_t)arows * g.Kp * 2;
  const size_t x16_bytes = (size_t)tc::act16_elems(g) * 2;
  const size_t rs_bytes = fold ? ((size_t)g.M * 4 + 255) / 256 * 256 : 0;
  const size_t total = nparts * diag_bytes + rs_bytes + x16_bytes;
  void* tmp = nullptr;
  if (cudaMallocFromPoolAsync(&tmp, total, pool, s) != cudaSuccess) return FGQ_ERR_CUDA;
  uint8_t* diag = static_cast<uint8_t*>(tmp);
  float* rs = reinterpret_cast<float*>(diag + nparts * diag_bytes);
  uint8_t* x16 = diag + nparts * diag_bytes + rs_bytes;
  if (fold) a.row_scale = rs;
  fgq_status st =
      launch_prep4(g, codes, alpha, rs, a.mtiles, diag, fold ? diag + diag_bytes : nullptr, act, x16, s);
  for (int part = 0; st == FGQ_OK && part < nparts; ++part)
    if (!make_map_2d(&a.a_map[part], CU_TENSOR_MAP_DATA_TYPE_FLOAT16, diag + part * diag_bytes, (uint64_t)g.Kp,
                     (uint64_t)arows, (uint64_t)g.Kp * 2, T4_KT, T4_ROWS, CU_TENSOR_MAP_SWIZZLE_128B))
      st = FGQ_ERR_CUDA;
  const bool tmap = tc::act_pointwise(g);
  if (st == FGQ_OK && !tc::act16_map(&a.act_map, x16, g, pairs ? T4_BN / 2 : T4_BN)) st = FGQ_ERR_CUDA;
  if (st == FGQ_OK && fold && g.groups == 1 && g.M % 4 == 0 && !g.rq_out)
    a.out_tma = make_map_2d(&a.out_map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, out, (uint64_t)g.M, (uint64_t)g.P,
                            (uint64_t)g.M * 4, T4_FM, T4_BN, CU_TENSOR_MAP_SWIZZLE_NONE)
                    ? 1
                    : 0;
  if (st == FGQ_OK) {
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int grid = a.ntiles < sms ? a.ntiles : sms;
    if (pairs)
      st = tmap ? launch_tc4_pair<true>(a, a.ntiles, s) : launch_tc4_pair<false>(a, a.ntiles, s);
    else if (fold)
      st = tmap ? launch_tc4<true, true>(a, grid, s) : launch_tc4<false, true>(a, grid, s);
    else
      st = tmap ? launch_tc4<true, false>(a, grid, s) : launch_tc4<false, false>(a, grid, s);
  }
  // the temporary returns to the pool once the work queued on s before this point is done
  if (cudaFreeAsync(tmp, s) != cudaSuccess && st == FGQ_OK) st = FGQ_ERR_CUDA;
  return st;
}

}  // namespace fgq
