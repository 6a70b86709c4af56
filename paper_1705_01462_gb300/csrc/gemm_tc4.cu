// Tensor-core (tcgen05) grouped ternary contraction for G = 4.
//
// Math (Eq. 2, 32-bit group accumulators of Section 4): y[p][m] = s_x * sum_g alpha[m][g]
// * s[m][g][p] with s an exact integer sum over a group of 4 reduction elements.  A dense
// MMA would sum across groups, so each K = 16 MMA step (4 groups) uses a block-diagonal
// ternary operand A' of 128 rows: row 4 m' + j holds filter m' of the tile (32 filters) only
// in the 4 columns of group slot j (zeros elsewhere), and D[4 m' + j][p] of one MMA
// (M = 128, N = 256, K = 16) receives the products of group 4 step + j alone.  A' depends
// only on the weights, so it is built once per call; the activations are the plain dense
// operand, expanded to fp16 once per call and loaded by TMA (2D rows or im2col boxes), and
// no thread builds operands inside the contraction.  Two variants:
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
#include <cstdint>
#include <cstring>

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

// Expands 2-bit codes (00 = 0, 01 = +1, 11 = -1; element k in word k / 16, bits 2 (k % 16))
// to fp16 {0, +1, -1}: one thread per code word, 16 halves (32 bytes) out.
__global__ void __launch_bounds__(256) expand_codes_kernel(const uint32_t* __restrict__ codes, int64_t nwords,
                                                           uint4* __restrict__ a16) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= nwords) return;
  const uint32_t w = __ldg(codes + i);
  uint32_t h[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) {
    const uint32_t c0 = (w >> (4 * e)) & 3u, c1 = (w >> (4 * e + 2)) & 3u;
    const uint32_t lo = (c0 & 1u) ? ((c0 & 2u) ? 0xBC00u : 0x3C00u) : 0u;
    const uint32_t hi = (c1 & 1u) ? ((c1 & 2u) ? 0xBC00u : 0x3C00u) : 0u;
    h[e] = lo | (hi << 16);
  }
  a16[2 * i] = make_uint4(h[0], h[1], h[2], h[3]);
  a16[2 * i + 1] = make_uint4(h[4], h[5], h[6], h[7]);
}

// Block-diagonal A' from a dense fp16 operand src [M][Kp]: row 4 m' + j of tile (gi, mt)
// keeps, of filter gi Mg + mt 32 + m', the elements of the groups whose index is j modulo 4
// (slot j of every K = 16 step) and zeros elsewhere.  One thread per 16-byte chunk (8
// elements = 2 groups) of A'.
__global__ void __launch_bounds__(256) diag_kernel(const uint2* __restrict__ src, int Kp, int Mg, int mtiles,
                                                   int64_t nchunks, uint4* __restrict__ dst) {
  const int cpr = Kp / 8;  // chunks per row
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < nchunks; i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = i / cpr;
    const int c = (int)(i - r * cpr);
    const int64_t tile = r / T4_ROWS;
    const int rr = (int)(r - tile * T4_ROWS);
    const int mp = rr >> 2, j = rr & 3;
    const int gi = (int)(tile / mtiles), mt = (int)(tile - (int64_t)gi * mtiles);
    const int local = mt * T4_FM + mp;
    uint4 v = make_uint4(0u, 0u, 0u, 0u);
    if (local < Mg) {
      const int64_t m = (int64_t)gi * Mg + local;
      const int g0 = 2 * c;  // first group of the chunk; slot = group % 4
      if ((g0 & 3) == j) {
        const uint2 h = __ldg(src + (m * Kp + 8 * c) / 4);
        v.x = h.x;
        v.y = h.y;
      } else if (((g0 + 1) & 3) == j) {
        const uint2 h = __ldg(src + (m * Kp + 8 * c + 4) / 4);
        v.z = h.x;
        v.w = h.y;
      }
    }
    dst[i] = v;
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
      if constexpr (FOLD) {
        // the four slot rows 4 m' .. 4 m' + 3 of a filter are lanes 4 (lane / 4) .. + 3 of the
        // warp: reduce them so that lane j ends with positions 4 i + j (i < 32) of its half,
        // summed over the slots; two exchange rounds, each keeping half of the positions
        const bool b1 = (j >> 1) & 1, b0 = j & 1;
#pragma unroll
        for (int q = 0; q < T4_EPI_COLS / 4; ++q) {
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            // positions 4 q + e (slot bit 1 clear) and 4 q + 2 + e (set): keep the one whose
            // bit 1 matches b1, send the other to lane ^ 2; the result goes to 4 q + e
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

template <bool TMAP, bool FOLD>
fgq_status launch_tc4(const T4Args& args, int grid, cudaStream_t s) {
  constexpr int smem = T4Cfg<FOLD>::SMEM;
  if (!tc::smem_attr_once<tc4_contract_kernel<TMAP, FOLD>>(smem)) return FGQ_ERR_CUDA;
  tc4_contract_kernel<TMAP, FOLD><<<grid, T4_THREADS, smem, s>>>(args);
  return after_launch();
}

fgq_status launch_diag(const void* src, int Kp, int Mg, int mtiles, int64_t rows, void* dst, cudaStream_t s) {
  const int64_t nchunks = rows * (Kp / 8);
  if (nchunks <= 0) return FGQ_OK;
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t want = (nchunks + 255) / 256;
  const int blocks = (int)(want < 8LL * sms ? want : 8LL * sms);
  diag_kernel<<<blocks, 256, 0, s>>>(static_cast<const uint2*>(src), Kp, Mg, mtiles, nchunks,
                                     static_cast<uint4*>(dst));
  return after_launch();
}

}  // namespace

fgq_status launch_expand_codes(const uint32_t* codes, int64_t nwords, void* a16, cudaStream_t s) {
  if (nwords <= 0) return FGQ_OK;
  expand_codes_kernel<<<(unsigned)((nwords + 255) / 256), 256, 0, s>>>(codes, nwords, static_cast<uint4*>(a16));
  return after_launch();
}

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
  a.ntiles = g.groups * a.mtiles * a.ptiles;
  a.ktiles = g.Kp / T4_KT;
  // a test may shorten the waits (debug_wait_limit_us), never the final drains
  const int64_t lim_us = debug_wait_limit_us();
  a.timeout_ns = lim_us < 0 ? T4_TIMEOUT_NS : (uint64_t)lim_us * 1000u;
  const bool fold = sums == nullptr;

  // temporaries from the stream-ordered pool: the dense ternary operand fp16 [M][Kp] per part
  // (folded hi, lo; or the codes) and the row scales, its block-diagonal form A' per part, and
  // the activations in fp16
  cudaMemPool_t pool = scratch_pool();
  if (!pool) return FGQ_ERR_CUDA;
  const int nparts = fold ? 2 : 1;
  const size_t dense_bytes = (size_t)g.M * g.Kp * 2;
  const int64_t arows = (int64_t)g.groups * a.mtiles * T4_ROWS;
  const size_t diag_bytes = (size_t)arows * g.Kp * 2;
  const size_t x16_bytes = (size_t)tc::act16_elems(g) * 2;
  const size_t rs_bytes = fold ? ((size_t)g.M * 4 + 255) / 256 * 256 : 0;
  const size_t total = nparts * (dense_bytes + diag_bytes) + rs_bytes + x16_bytes;
  void* tmp = nullptr;
  if (cudaMallocFromPoolAsync(&tmp, total, pool, s) != cudaSuccess) return FGQ_ERR_CUDA;
  uint8_t* dense = static_cast<uint8_t*>(tmp);
  uint8_t* diag = dense + nparts * dense_bytes;
  float* rs = reinterpret_cast<float*>(diag + nparts * diag_bytes);
  uint8_t* x16 = diag + nparts * diag_bytes + rs_bytes;
  fgq_status st;
  if (fold) {
    a.row_scale = rs;
    st = launch_fold_alpha_split(codes, g.M, g.wrow, g.G, g.ng, alpha, dense, dense + dense_bytes, rs, s);
  } else {
    st = launch_expand_codes(codes, (int64_t)g.M * g.wrow, dense, s);
  }
  for (int part = 0; st == FGQ_OK && part < nparts; ++part)
    st = launch_diag(dense + part * dense_bytes, g.Kp, g.Mg, a.mtiles, arows, diag + part * diag_bytes, s);
  if (st == FGQ_OK) st = tc::expand_act16(act, g, x16, s);
  for (int part = 0; st == FGQ_OK && part < nparts; ++part)
    if (!make_map_2d(&a.a_map[part], CU_TENSOR_MAP_DATA_TYPE_FLOAT16, diag + part * diag_bytes, (uint64_t)g.Kp,
                     (uint64_t)arows, (uint64_t)g.Kp * 2, T4_KT, T4_ROWS, CU_TENSOR_MAP_SWIZZLE_128B))
      st = FGQ_ERR_CUDA;
  const bool tmap = tc::act_pointwise(g);
  if (st == FGQ_OK && !tc::act16_map(&a.act_map, x16, g, T4_BN)) st = FGQ_ERR_CUDA;
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
    if (fold)
      st = tmap ? launch_tc4<true, true>(a, grid, s) : launch_tc4<false, true>(a, grid, s);
    else
      st = tmap ? launch_tc4<true, false>(a, grid, s) : launch_tc4<false, false>(a, grid, s);
  }
  // the temporary returns to the pool once the work queued on s before this point is done
  if (cudaFreeAsync(tmp, s) != cudaSuccess && st == FGQ_OK) st = FGQ_ERR_CUDA;
  return st;
}

}  // namespace fgq
