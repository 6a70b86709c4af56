// Dense tensor-core (tcgen05) contraction with the group scales folded into the weights.
//
// Eq. 2 sums alpha_g * (sum over group g of t * x); with A[m][k] = alpha(m, k / G) * t[m][k] the
// same value is one dense contraction y[p][m] = s_x * rs[m] * sum_k A[m][k] q[p][k], with no
// multiply per group.  A is built once per call in fp16, in one or two parts (A = A0 + A1):
//
//   * fixed-point alphas (Section 4: 8/4-bit codes a[m][g], one exponent E_m per filter row):
//     A = a * t, integers of magnitude <= 255 and exact in fp16; rs = 2^E_m.  Products and
//     every partial sum below 2^24 are exact in the fp32 accumulator, so y is the exact value
//     rounded once whenever |sum_k A q| < 2^24.
//   * fp32 alphas (an ablation): alpha * 2^e_m = hi + lo with hi = fp16(alpha 2^e_m) and lo =
//     fp16(the remainder); e_m puts the row's largest alpha in [2^14, 2^15), so the pair
//     carries about 22 bits of alpha; A0 = hi t, A1 = lo t, rs = 2^-e_m.  The accumulator
//     rounds once per K = 16 step.
//
// Tile: 128 filters x 256 positions, K-tile 64.  Each K-tile is 4 (or 8, two parts) MMAs
// M = 128, N = 256, K = 16 into the tile's TMEM accumulator (256 columns); the epilogue runs
// once per tile.  Two accumulators: the epilogue of tile i overlaps the MMAs of tile i + 1.
// Warp roles (448 threads, one CTA per SM, persistent over tiles):
//   warps 0-7  epilogue: warp w reads TMEM lanes 32 (w % 4) .. (filters), columns 128 (w / 4)
//              .. +127 (positions), scales by s_x rs[m] and stores fp32 (through shared memory
//              and TMA box stores where the output allows, single-part weights) or requantized
//              codes;
//   warps 8-11 loaders/converters: thread t brings the activation rows of tile positions t and
//              t + 128 (TMA boxes for 1x1 stride-1 layers and GEMMs, else cp.async gathers) and
//              converts them to the fp16 operand B (two stages);
//   warp 12    TMEM allocation and the MMA issuer;
//   warp 13    streams the folded-weight boxes (A) by TMA into their own ring of four stages
//              (two for split weights), released by the MMAs' commits, so the boxes arrive
//              ahead of the K-tiles that use them.
// Every mbarrier wait is bounded in time; on expiry the kernel records FGQ_ERR_TIMEOUT, each
// role leaves its loop, in-flight copies and MMAs are waited for, and TMEM is freed.
#include <cuda_fp16.h>

#include <cstdint>
#include <cstring>

#include "tc_common.cuh"

namespace fgq {
namespace {

using tc::encode_tiled;
using tc::make_map_2d;
using tc::st_off;
using tc::sw128;
using tc::u8pair_to_h2;

constexpr int TD_BM = 128;   // filters per tile (MMA M, TMEM lanes)
constexpr int TD_BN = 256;   // positions per tile (MMA N)
constexpr int TD_KT = 64;    // reduction elements per K-tile (4 MMA steps of K = 16)
constexpr int TD_NS = 4;     // staging ring depth
constexpr int TD_NACC = 2;   // TMEM accumulators of 256 columns (one tile each)
constexpr int TD_EPI_WARPS = 8;
constexpr int TD_LOAD_WARP0 = 8;
constexpr int TD_LOADERS = 128;
constexpr int TD_MMA_WARP = 12;
constexpr int TD_A_WARP = 13;  // lane 0 streams the folded-weight boxes
constexpr int TD_THREADS = 32 * (TD_A_WARP + 1);
constexpr int TD_TMEM_COLS = TD_NACC * 256;
constexpr uint64_t TD_TIMEOUT_NS = 1000000000ull;  // 1 s per wait
constexpr uint32_t BAR_EPID = 3;

constexpr int A_TILED = TD_BM * TD_KT * 2;  // 16 KB fp16 [128 filters][64 K] per part
constexpr int B_TILED = TD_BN * TD_KT * 2;  // 32 KB fp16 [256 positions][64 K]
constexpr int ST_STAGED = TD_BN * TD_KT;    // 16 KB: 256 raw activation rows of 64 bytes
constexpr int OUT_BOXD = 64 * TD_BM * 4;    // 32 KB: fp32 [64 positions][128 filters]

template <int NA>
struct DenseCfg {
  static constexpr int NAS = NA == 1 ? 4 : 2;  // folded-weight (A) ring depth
  static constexpr int NB = 2;                 // activation operand (B) ring depth
  static constexpr int A_STAGE = NA * A_TILED;
  static constexpr int SMEM_A = NAS * A_STAGE;
  static constexpr int SMEM_B = NB * B_TILED;
  static constexpr int SMEM_ST = TD_NS * ST_STAGED;
  // output staging for TMA box stores: one [64 positions][128 filters] fp32 box, single-part
  // weights only (two parts leave no room)
  static constexpr int SMEM_OUT = NA == 1 ? OUT_BOXD : 0;
  static constexpr int SMEM_BAR = 8 * (2 * NAS + 2 * NB + 2 * TD_NS + 2 * TD_NACC + 1) + 16;
  static constexpr int SMEM = 1024 + SMEM_A + SMEM_B + SMEM_ST + SMEM_OUT + SMEM_BAR;
};
static_assert(DenseCfg<1>::SMEM <= 232448 && DenseCfg<2>::SMEM <= 232448, "shared memory budget");
static_assert(A_TILED % 1024 == 0 && B_TILED % 1024 == 0 && ST_STAGED % 1024 == 0, "stage alignment");

struct TDArgs {
  CUtensorMap a_map[2];  // fp16 [M][Kp] folded weights (part 0, part 1), box {64, 128 rows}, 128-byte swizzle
  CUtensorMap act_map;   // uint8 [pixels][C], box {64 bytes, 256 rows}, 64-byte swizzle; TMA path
  CUtensorMap out_map;   // fp32 [P][M], box {128 filters, 64 positions}; if out_tma
  const uint8_t* act;
  const float* row_scale;  // rs [M]
  const float* act_scale;
  float* out;
  unsigned int* err;
  Geom g;
  int mtiles, ptiles, ntiles, ktiles;
  int out_tma;
  uint64_t timeout_ns;
};

// Filter tiles of one position tile are consecutive, so CTAs running at the same time share
// activation rows in L2.
__device__ __forceinline__ void tile_coords_d(const TDArgs& a, int tile, int& gi, int& m0, int64_t& p0) {
  const int per_p = a.g.groups * a.mtiles;
  const int pt = tile / per_p;
  const int r = tile - pt * per_p;
  gi = r / a.mtiles;
  m0 = gi * a.g.Mg + (r - gi * a.mtiles) * TD_BM;
  p0 = (int64_t)pt * TD_BN;
}

// Folded weights, one warp per filter row.  MODE 8 / 4: fixed-point alpha codes (8-bit, or
// 4-bit packed two per byte, element 2i in the low nibble) times t, and rs = ascale; MODE 0:
// fp32 alphas split into hi + lo after scaling the row by 2^e, rs = 2^-e.  Row m of part i
// is fp16 [Kp] at a_i + m Kp; codes 00 and padding give 0.
constexpr int FOLD_THREADS = 128;  // one block per filter row
template <int MODE>
__global__ void __launch_bounds__(FOLD_THREADS) fold_weights_kernel(const uint32_t* __restrict__ codes, int M,
                                                                    int wrow, int G, int ng,
                                                                    const float* __restrict__ alpha,
                                                                    const uint8_t* __restrict__ aq,
                                                                    const float* __restrict__ ascale,
                                                                    __half* __restrict__ a0, __half* __restrict__ a1,
                                                                    float* __restrict__ row_scale) {
  const int m = blockIdx.x;
  const int tid = threadIdx.x;
  float mul = 1.0f;
  if (MODE == 0) {
    float mx = 0.0f;
    for (int g = tid; g < ng; g += FOLD_THREADS) mx = fmaxf(mx, __ldg(alpha + (int64_t)m * ng + g));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    __shared__ float red[FOLD_THREADS / 32];
    if ((tid & 31) == 0) red[tid >> 5] = mx;
    __syncthreads();
#pragma unroll
    for (int i = 0; i < FOLD_THREADS / 32; ++i) mx = fmaxf(mx, red[i]);
    int e = mx > 0.0f ? 14 - ilogbf(mx) : 0;  // mx 2^e in [2^14, 2^15)
    e = e < -100 ? -100 : (e > 100 ? 100 : e);
    mul = ldexpf(1.0f, e);
    if (tid == 0) row_scale[m] = ldexpf(1.0f, -e);
  } else if (tid == 0) {
    row_scale[m] = __ldg(ascale + m);
  }
  const int64_t arow = MODE == 4 ? (ng + 1) / 2 : ng;
  for (int w = tid; w < wrow; w += FOLD_THREADS) {
    const uint32_t cw = __ldg(codes + (int64_t)m * wrow + w);
    uint32_t h0[8], h1[8];
#pragma unroll
    for (int e2 = 0; e2 < 8; ++e2) {
      uint32_t v0[2], v1[2];
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const int e = 2 * e2 + u;
        const uint32_t c = (cw >> (2 * e)) & 3u;
        const int g = (16 * w + e) / G;
        v0[u] = v1[u] = 0u;
        if ((c == 1u || c == 3u) && g < ng) {
          float v;
          if (MODE == 8) {
            v = (float)__ldg(aq + (int64_t)m * arow + g);
          } else if (MODE == 4) {
            const uint32_t b = __ldg(aq + (int64_t)m * arow + g / 2);
            v = (float)((g & 1) ? (b >> 4) : (b & 15u));
          } else {
            v = __ldg(alpha + (int64_t)m * ng + g) * mul;  // exact: a power-of-two scaling
          }
          const __half hi = __float2half_rn(v);
          const __half lo = __float2half_rn(v - __half2float(hi));  // the remainder, exact in fp32
          const uint32_t sgn = c == 3u ? 0x8000u : 0u;
          v0[u] = (uint32_t)__half_as_ushort(hi) ^ sgn;
          v1[u] = MODE == 0 ? ((uint32_t)__half_as_ushort(lo) ^ sgn) : 0u;
        }
      }
      h0[e2] = v0[0] | (v0[1] << 16);
      h1[e2] = v1[0] | (v1[1] << 16);
    }
    uint4* d0 = reinterpret_cast<uint4*>(a0 + ((int64_t)m * wrow + w) * 16);
    d0[0] = make_uint4(h0[0], h0[1], h0[2], h0[3]);
    d0[1] = make_uint4(h0[4], h0[5], h0[6], h0[7]);
    if (MODE == 0) {
      uint4* d1 = reinterpret_cast<uint4*>(a1 + ((int64_t)m * wrow + w) * 16);
      d1[0] = make_uint4(h1[0], h1[1], h1[2], h1[3]);
      d1[1] = make_uint4(h1[4], h1[5], h1[6], h1[7]);
    }
  }
}

template <int NA, bool SIGNED, bool TMAP>
__global__ void __launch_bounds__(TD_THREADS, 1) dense_contract_kernel(const __grid_constant__ TDArgs a) {
  using Cfg = DenseCfg<NA>;
  constexpr int NAS = Cfg::NAS;
  constexpr int NB = Cfg::NB;
  extern __shared__ uint8_t smem_rawd[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_rawd) + 1023) & ~uintptr_t(1023));
  uint8_t* abuf = smem;
  uint8_t* bbuf = smem + Cfg::SMEM_A;
  uint8_t* st = bbuf + Cfg::SMEM_B;
  float* otile = reinterpret_cast<float*>(st + Cfg::SMEM_ST);
  uint64_t* bars = reinterpret_cast<uint64_t*>(st + Cfg::SMEM_ST + Cfg::SMEM_OUT);
  uint64_t* a_full = bars;
  uint64_t* a_empty = bars + NAS;
  uint64_t* op_full = bars + 2 * NAS;
  uint64_t* op_empty = op_full + NB;
  uint64_t* st_full = op_empty + NB;
  uint64_t* st_empty = st_full + TD_NS;
  uint64_t* acc_full = st_empty + TD_NS;
  uint64_t* acc_empty = acc_full + TD_NACC;
  uint64_t* drain_bar = acc_empty + TD_NACC;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_bar + 1);
  volatile uint32_t* abort_flag = tmem_slot + 1;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const Geom& g = a.g;
  const uint64_t tmo = a.timeout_ns;

  if (threadIdx.x == 0) {
    for (int i = 0; i < NAS; ++i) {
      mbar_init(&a_full[i], 1);  // the A boxes' byte count
      mbar_init(&a_empty[i], 1);
    }
    for (int i = 0; i < NB; ++i) {
      mbar_init(&op_full[i], TD_LOADERS);  // B pieces
      mbar_init(&op_empty[i], 1);
    }
    for (int i = 0; i < TD_NS; ++i) {
      mbar_init(&st_full[i], TMAP ? 1 : TD_LOADERS);
      mbar_init(&st_empty[i], TD_LOADERS);
    }
    for (int i = 0; i < TD_NACC; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], TD_EPI_WARPS);
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == TD_MMA_WARP) {
    tmem_alloc(tmem_slot, TD_TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const int my_tiles = (a.ntiles - (int)blockIdx.x + (int)gridDim.x - 1) / (int)gridDim.x;

  auto fail = [&]() {
    *abort_flag = 1;
    record_error(a.err, FGQ_ERR_TIMEOUT);
  };

  // ------------------------------------------------------------------ loaders/converters
  if (warp >= TD_LOAD_WARP0 && warp < TD_MMA_WARP) {
    const int t = threadIdx.x - 32 * TD_LOAD_WARP0;  // tile positions t and t + 128
    const int total = my_tiles * a.ktiles;
    constexpr uint32_t TX_ACT = ST_STAGED;

    int cur_tile = -1, gi = 0, m0 = 0, tr = 0, ts = 0, tc0 = 0;
    int64_t p0 = 0;
    int pb[2] = {0, 0}, phb[2] = {0, 0}, pwb[2] = {0, 0};
    bool pvalid[2] = {false, false};
    int issued = 0;
    // activation rows of K-tile j (of this CTA's sequence) into staging slot j % NS
    auto issue = [&](int j) -> bool {
      const int tl = j / a.ktiles;
      if (tl != cur_tile) {
        cur_tile = tl;
        tile_coords_d(a, (int)blockIdx.x + tl * (int)gridDim.x, gi, m0, p0);
        tr = ts = tc0 = 0;
#pragma unroll
        for (int r = 0; r < 2; ++r) {
          const int64_t p = p0 + t + 128 * r;
          pvalid[r] = p < g.P;
          const int pp = pvalid[r] ? (int)p : 0;
          const int wo = pp % g.Wo;
          const int q = pp / g.Wo;
          const int ho = q % g.Ho;
          pb[r] = q / g.Ho;
          phb[r] = ho * g.stride - g.pad;
          pwb[r] = wo * g.stride - g.pad;
        }
      }
      const int slot = j % TD_NS;
      uint8_t* sa = st + slot * ST_STAGED;
      if (TMAP) {
        if (t == 0) {
          if (j >= TD_NS && !mbar_wait_timed(&st_empty[slot], ((j / TD_NS) & 1) ^ 1, tmo, abort_flag, 64))
            return false;
          mbar_arrive_expect_tx(&st_full[slot], TX_ACT);
          tma_load_2d(smem_u32(sa), &a.act_map, gi * g.Cg + tc0, (int)p0, &st_full[slot]);
          issued = j + 1;
        }
      } else {
        if (j >= TD_NS && !mbar_wait_timed(&st_empty[slot], ((j / TD_NS) & 1) ^ 1, tmo, abort_flag, 64))
          return false;
#pragma unroll
        for (int r = 0; r < 2; ++r) {
          const uint8_t* src = a.act;
          bool inside = false;
          if (pvalid[r]) {
            const int hi = phb[r] + tr, wi = pwb[r] + ts;
            if (hi >= 0 && hi < g.H && wi >= 0 && wi < g.W) {
              src = a.act + (((int64_t)pb[r] * g.H + hi) * g.W + wi) * g.C + (int64_t)gi * g.Cg + tc0;
              inside = true;
            }
          }
          const int row = t + 128 * r;
#pragma unroll
          for (int c = 0; c < 4; ++c)
            cp_async16(smem_u32(sa + st_off<8>(row, c)), inside ? (const void*)(src + 16 * c) : (const void*)a.act,
                       inside ? 16u : 0u);
        }
        cp_async_mbar_arrive_noinc(&st_full[slot]);
        issued = j + 1;
      }
      tc0 += TD_KT;
      if (tc0 == g.Cg) {
        tc0 = 0;
        if (++ts == g.S) {
          ts = 0;
          ++tr;
        }
      }
      return true;
    };

    bool ok = true;
    for (int j = 0; j < TD_NS - 1 && j < total && ok; ++j) ok = issue(j);
    int consumed = 0;
    for (int j = 0; j < total && ok; ++j) {
      if (j + TD_NS - 1 < total && !issue(j + TD_NS - 1)) {
        ok = false;
        break;
      }
      const int slot = j % TD_NS;
      const int os = j % NB;
      if (!mbar_wait_timed(&op_empty[os], ((j / NB) & 1) ^ 1, tmo, abort_flag, 64)) {
        ok = false;
        break;
      }
      uint8_t* Bt = bbuf + os * B_TILED;
      if (!mbar_wait_timed(&st_full[slot], (j / TD_NS) & 1, tmo, abort_flag, 32)) {
        ok = false;
        break;
      }
      consumed = j + 1;
      const uint8_t* sa = st + slot * ST_STAGED;
      constexpr uint32_t bias2 = SIGNED ? 0x64806480u : 0x64006400u;
      constexpr uint32_t flip = 0x80808080u;
#pragma unroll
      for (int r = 0; r < 2; ++r) {
        const int row = t + 128 * r;
#pragma unroll
        for (int c = 0; c < 4; ++c) {  // staging chunk c: activations 16 c .. 16 c + 15
          const uint4 v = *reinterpret_cast<const uint4*>(sa + st_off<8>(row, c));
          const uint32_t w[4] = {SIGNED ? v.x ^ flip : v.x, SIGNED ? v.y ^ flip : v.y, SIGNED ? v.z ^ flip : v.z,
                                 SIGNED ? v.w ^ flip : v.w};
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const uint4 o = make_uint4(u8pair_to_h2(w[2 * h], 0x4140, bias2), u8pair_to_h2(w[2 * h], 0x4342, bias2),
                                       u8pair_to_h2(w[2 * h + 1], 0x4140, bias2),
                                       u8pair_to_h2(w[2 * h + 1], 0x4342, bias2));
            *reinterpret_cast<uint4*>(Bt + sw128(row, 2 * c + h)) = o;
          }
        }
      }
      fence_proxy_async_smem();
      mbar_arrive(&op_full[os]);
      mbar_arrive(&st_empty[slot]);
    }
    if (!ok && !*abort_flag) fail();
    if (!TMAP) cp_async_wait_all();
    if (TMAP && t == 0) {
      for (int j = consumed; j < issued; ++j) mbar_wait_bounded(&st_full[j % TD_NS], (j / TD_NS) & 1, 1u << 16);
    }
  }

  // ------------------------------------------------------------------ folded-weight boxes
  if (warp == TD_A_WARP && lane == 0) {
    const int total = my_tiles * a.ktiles;
    int armed = 0;
    bool ok = true;
    for (int j = 0; j < total && ok; ++j) {
      const int as = j % NAS;
      if (!mbar_wait_timed(&a_empty[as], ((j / NAS) & 1) ^ 1, tmo, abort_flag, 64)) {
        ok = false;
        break;
      }
      const int tl = j / a.ktiles;
      int gj, mj;
      int64_t pj;
      tile_coords_d(a, (int)blockIdx.x + tl * (int)gridDim.x, gj, mj, pj);
      uint8_t* A = abuf + as * Cfg::A_STAGE;
      mbar_arrive_expect_tx(&a_full[as], Cfg::A_STAGE);
#pragma unroll
      for (int part = 0; part < NA; ++part)
        tma_load_2d(smem_u32(A + part * A_TILED), &a.a_map[part], (j - tl * a.ktiles) * TD_KT, mj, &a_full[as]);
      armed = j + 1;
    }
    if (!ok && !*abort_flag) fail();
    // boxes the MMA issuer did not consume may still be in flight
    for (int j = armed - NAS < 0 ? 0 : armed - NAS; j < armed; ++j)
      mbar_wait_bounded(&a_full[j % NAS], (j / NAS) & 1, 1u << 16);
  }

  // ------------------------------------------------------------------ MMA issuer
  if (warp == TD_MMA_WARP && lane == 0) {
    const uint32_t idesc = idesc_f16_f32(TD_BM, TD_BN);
    const int total = my_tiles * a.ktiles;
    bool ok = true;
    for (int j = 0; j < total && ok; ++j) {
      const int tl = j / a.ktiles;
      const int kt = j - tl * a.ktiles;
      const int b = tl & 1;
      if (kt == 0 && !mbar_wait_timed(&acc_empty[b], ((tl >> 1) & 1) ^ 1, tmo, abort_flag, 0)) {
        ok = false;
        break;
      }
      const int os = j % NB;
      const int as = j % NAS;
      if (!mbar_wait_timed(&op_full[os], (j / NB) & 1, tmo, abort_flag, 0) ||
          !mbar_wait_timed(&a_full[as], (j / NAS) & 1, tmo, abort_flag, 0)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t abase = smem_u32(abuf + as * Cfg::A_STAGE);
      const uint64_t bd = sdesc_k_sw128(smem_u32(bbuf + os * B_TILED));
#pragma unroll
      for (int part = 0; part < NA; ++part) {
        const uint64_t ad = sdesc_k_sw128(abase + part * A_TILED);
#pragma unroll
        for (int s = 0; s < 4; ++s)
          mma_f16(tmem + (uint32_t)(b * 256), ad + 2 * s, bd + 2 * s, idesc, (kt | part | s) != 0 ? 1u : 0u);
      }
      mma_commit(&op_empty[os]);
      mma_commit(&a_empty[as]);
      if (kt == a.ktiles - 1) mma_commit(&acc_full[b]);
    }
    if (!ok && !*abort_flag) fail();
    mma_commit(drain_bar);
    mbar_wait_bounded(drain_bar, 0, 1u << 20);
  }

  // ------------------------------------------------------------------ epilogue
  if (warp < TD_EPI_WARPS) {
    const int quarter = warp & 3, half = warp >> 2;
    const int t = 32 * quarter + lane;  // TMEM lane = filter row of the tile
    const uint32_t tbase = tmem + ((uint32_t)(32 * quarter) << 16) + (uint32_t)(128 * half);
    const float sx = __ldg(a.act_scale);
    const bool leader = threadIdx.x == 0;
    const bool out_tma = NA == 1 && a.out_tma;
    for (int tl = 0; tl < my_tiles; ++tl) {
      int gi, m0;
      int64_t p0;
      tile_coords_d(a, (int)blockIdx.x + tl * (int)gridDim.x, gi, m0, p0);
      const int m = m0 + t;
      const bool mok = m < gi * g.Mg + g.Mg && m < g.M;
      const float sc = mok ? sx * __ldg(a.row_scale + m) : 0.0f;
      const int b = tl & 1;
      const bool ok = mbar_wait_timed(&acc_full[b], (tl >> 1) & 1, tmo, abort_flag, 0);
      if (!ok && !*abort_flag) fail();
      if (named_bar_or(BAR_EPID, 32 * TD_EPI_WARPS, !ok)) break;
      tc_fence_after();
      const uint32_t ta = tbase + (uint32_t)(b * 256);
      const int64_t pw = p0 + 128 * half;  // this warp's first position
#pragma unroll 1
      for (int hh = 0; hh < 2; ++hh) {  // positions pw + 64 hh .. + 63
        uint32_t r0[32], r1[32];
        tmem_ld32(ta + 64 * hh, r0);
        tmem_ld32(ta + 64 * hh + 32, r1);
        tmem_ld_wait_regs(r0);
        reg_fence(r1);
        if (hh == 1) {  // every column of this accumulator is in registers: free it
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&acc_empty[b]);
        }
        if (out_tma) {
          // one staging box: positions p0 + 128 hb + 64 hh .. + 63 are written by the warps of
          // half hb, then stored by one thread
#pragma unroll 1
          for (int hb = 0; hb < 2; ++hb) {
            if (leader) bulk_wait_read_all();  // the previous box has been read out
            named_bar_sync(BAR_EPID, 32 * TD_EPI_WARPS);
            if (half == hb) {
#pragma unroll
              for (int i = 0; i < 32; ++i) {
                otile[i * TD_BM + t] = sc * __uint_as_float(r0[i]);
                otile[(32 + i) * TD_BM + t] = sc * __uint_as_float(r1[i]);
              }
            }
            fence_proxy_async_smem();
            named_bar_sync(BAR_EPID, 32 * TD_EPI_WARPS);
            if (leader) {  // a box that starts inside the output (its tail past P is not written)
              if (p0 + 128 * hb + 64 * hh < g.P) tma_store_2d(&a.out_map, m0, (int)(p0 + 128 * hb + 64 * hh), smem_u32(otile));
              bulk_commit();
            }
          }
        } else if (mok) {
          if (g.rq_out) {  // fused requantization: 8-bit codes instead of fp32
            const RqMul rq = rq_mul(g.rq_scale, g.rq_signed);
#pragma unroll
            for (int i = 0; i < 64; ++i) {
              const int64_t p = pw + 64 * hh + i;
              const uint32_t rv = i < 32 ? r0[i] : r1[i - 32];
              if (p < g.P) g.rq_out[p * g.M + m] = rq_code(sc * __uint_as_float(rv), rq);
            }
          } else {
#pragma unroll
            for (int i = 0; i < 64; ++i) {
              const int64_t p = pw + 64 * hh + i;
              const uint32_t rv = i < 32 ? r0[i] : r1[i - 32];
              if (p < g.P) a.out[p * g.M + m] = sc * __uint_as_float(rv);
            }
          }
        }
      }
    }
    if (leader) bulk_wait_all();
  }

  tc_fence_before();
  __syncthreads();
  if (warp == TD_MMA_WARP) {
    tc_fence_after();
    tmem_dealloc(tmem, TD_TMEM_COLS);
  }
}

template <int NA, bool SIGNED, bool TMAP>
fgq_status launch_dense(const TDArgs& args, int grid, cudaStream_t s) {
  if (!tc::smem_attr_once<dense_contract_kernel<NA, SIGNED, TMAP>>(DenseCfg<NA>::SMEM)) return FGQ_ERR_CUDA;
  dense_contract_kernel<NA, SIGNED, TMAP><<<grid, TD_THREADS, DenseCfg<NA>::SMEM, s>>>(args);
  return after_launch();
}

template <int NA>
fgq_status launch_dense_na(const TDArgs& args, bool sgn, bool tmap, int grid, cudaStream_t s) {
  if (sgn) return tmap ? launch_dense<NA, true, true>(args, grid, s) : launch_dense<NA, true, false>(args, grid, s);
  return tmap ? launch_dense<NA, false, true>(args, grid, s) : launch_dense<NA, false, false>(args, grid, s);
}

}  // namespace

bool dense_supports(const Geom& g) {
  if (g.act_type != FGQ_U8 && g.act_type != FGQ_S8) return false;
  if (g.Cg % TD_KT != 0) return false;        // every K-tile inside one filter tap (conv) or row (GEMM)
  if (g.C % 16 != 0) return false;            // 16-byte aligned activation rows
  if (g.Kp % 16 != 0) return false;           // fp16 rows of the folded weights: 32-byte multiples
  if (g.P >= (int64_t)1 << 31) return false;  // positions decoded in 32 bits
  if (encode_tiled() == nullptr) return false;
  return true;
}

namespace {

// Explicit im2col of 8-bit activations for the dense path (any channel count): row p (an
// output position, NHWC order) of col [P][Kc] holds act[b][ho stride - pad + r][wo stride - pad
// + s][c] at k = (r S + s) C + c, 0 outside the image and for Kred <= k < Kc.  One thread per
// position walks its row with running (r, s, c) counters and writes it in 16-byte pieces
// (measured faster than one thread per piece, and than staging rows in shared memory for
// contiguous warp stores).
constexpr int IM2COL_MAX_KC = 4096;
__global__ void __launch_bounds__(128) im2col_u8_kernel(const uint8_t* __restrict__ act, int B, int H, int W, int C,
                                                        int R, int S, int stride, int pad, int Ho, int Wo, int Kred,
                                                        int Kc, uint8_t* __restrict__ col) {
  const int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (p >= (int64_t)B * Ho * Wo) return;
  const int wo = (int)(p % Wo);
  const int64_t q = p / Wo;
  const int ho = (int)(q % Ho);
  const int b = (int)(q / Ho);
  const int h0 = ho * stride - pad, w0 = wo * stride - pad;
  uint4* dst = reinterpret_cast<uint4*>(col + p * Kc);
  int r = 0, sx = 0, c = 0;
  for (int k0 = 0; k0 < Kc; k0 += 16) {
    uint32_t wv[4] = {0u, 0u, 0u, 0u};
#pragma unroll
    for (int e = 0; e < 16; ++e) {
      uint32_t byte = 0u;
      if (k0 + e < Kred) {
        const int h = h0 + r, w = w0 + sx;
        if (h >= 0 && h < H && w >= 0 && w < W) byte = __ldg(act + (((int64_t)b * H + h) * W + w) * C + c);
        if (++c == C) {
          c = 0;
          if (++sx == S) {
            sx = 0;
            ++r;
          }
        }
      }
      wv[e >> 2] |= byte << (8 * (e & 3));
    }
    dst[k0 / 16] = make_uint4(wv[0], wv[1], wv[2], wv[3]);
  }
}

// The same im2col rows, one block per output row (b, ho): the R input rows that output
// row reads (zeros outside the image) are staged in shared memory with coalesced loads, and
// the Wo consecutive col rows -- one contiguous range of Wo * Kc bytes -- are written in
// 16-byte pieces by consecutive threads (coalesced stores), each piece gathered from the
// staged rows through a per-element table (row offset r * W * C + c, tap column s).
constexpr int IM2COL_ROWS_SMEM = 40 * 1024;
__global__ void __launch_bounds__(256) im2col_rows_kernel(const uint8_t* __restrict__ act, int H, int W, int C,
                                                         int R, int S, int stride, int pad, int Ho, int Wo, int Kred,
                                                         int Kc, uint8_t* __restrict__ col) {
  extern __shared__ uint8_t sm_i2c[];
  const int rowb = W * C;
  uint8_t* buf = sm_i2c;                                                       // [R][W * C]
  uint16_t* tab_off = reinterpret_cast<uint16_t*>(sm_i2c + ((R * rowb + 15) & ~15));  // [Kc]
  uint8_t* tab_s = reinterpret_cast<uint8_t*>(tab_off + Kc);                        // [Kc]
  const int ho = blockIdx.x % Ho;
  const int b = blockIdx.x / Ho;
  const int h0 = ho * stride - pad;
  for (int i = threadIdx.x; i < R * rowb; i += blockDim.x) {
    const int r = i / rowb, e = i - r * rowb;
    const int h = h0 + r;
    buf[i] = (h >= 0 && h < H) ? __ldg(act + ((int64_t)b * H + h) * rowb + e) : (uint8_t)0;
  }
  for (int j = threadIdx.x; j < Kc; j += blockDim.x) {
    if (j < Kred) {
      const int r = j / (S * C), rem = j - r * S * C;
      const int sx = rem / C, c = rem - sx * C;
      tab_off[j] = (uint16_t)(r * rowb + c);
      tab_s[j] = (uint8_t)sx;
    } else {
      tab_s[j] = 0xff;  // padding: zero
    }
  }
  __syncthreads();
  // thread t always writes piece jp = t % cpr of a row (its 16 table entries in registers),
  // for rows wo = t / cpr, t / cpr + rows_per_pass, ...; consecutive threads write
  // consecutive pieces
  const int cpr = Kc / 16;  // 16-byte pieces per col row (<= 256)
  const int rows_per_pass = blockDim.x / cpr;
  const int jp = threadIdx.x % cpr;
  const int wo0 = threadIdx.x / cpr;
  if (wo0 >= rows_per_pass) return;
  int off[16], sxs[16];
#pragma unroll
  for (int e = 0; e < 16; ++e) {
    const int j = jp * 16 + e;
    sxs[e] = tab_s[j];
    off[e] = sxs[e] != 0xff ? tab_off[j] : 0;
  }
  uint4* dst = reinterpret_cast<uint4*>(col + ((int64_t)b * Ho + ho) * Wo * Kc);
  for (int wo = wo0; wo < Wo; wo += rows_per_pass) {
    const int wbase = wo * stride - pad;
    uint32_t wv[4] = {0u, 0u, 0u, 0u};
#pragma unroll
    for (int e = 0; e < 16; ++e) {
      uint32_t byte = 0u;
      const int w = wbase + sxs[e];
      if (sxs[e] != 0xff && w >= 0 && w < W) byte = buf[off[e] + w * C];
      wv[e >> 2] |= byte << (8 * (e & 3));
    }
    dst[wo * cpr + jp] = make_uint4(wv[0], wv[1], wv[2], wv[3]);
  }
}

size_t im2col_rows_smem(const Geom& g, int Kc) { return (size_t)((g.R * g.W * g.C + 15) & ~15) + 3 * (size_t)Kc; }

// The same im2col rows for S C >= 16, where the 16 consecutive k of a 16-byte piece span at
// most two filter rows r, each a contiguous run of S C bytes of one input row.  One block per
// output row (b, ho): the R input rows are staged in shared memory (16-byte loads when the
// rows allow) at byte padB of a row of RS bytes whose margins stay zero (the padding
// columns), out-of-image rows all zero.  Piece q of col row wo is the 16-byte window of
// staged row r0 = 16 q / (S C) from its first element, completed from the window of row
// r0 + 1; each window is five 32-bit shared loads funnel-shifted to its byte offset, and
// k >= Kred reads zero.  Guards of IM2COL_SEG_GUARD bytes before and after the rows absorb
// the windows' reach past a row (those bytes are masked out).
constexpr int IM2COL_SEG_GUARD = 32;

__host__ __device__ inline int im2col_seg_padb(int pad, int C) { return (pad * C + 15) / 16 * 16; }
__host__ __device__ inline int im2col_seg_rs(int W, int C, int pad) {
  return (im2col_seg_padb(pad, C) + (W + pad) * C + 20 + 15) / 16 * 16;
}
size_t im2col_seg_smem(const Geom& g) { return 2 * (size_t)IM2COL_SEG_GUARD + (size_t)g.R * im2col_seg_rs(g.W, g.C, g.pad); }

__device__ __forceinline__ void window16(const uint8_t* p, uint32_t (&o)[4]) {
  const uint32_t* a = reinterpret_cast<const uint32_t*>(reinterpret_cast<uintptr_t>(p) & ~uintptr_t(3));
  const uint32_t sh = 8u * (uint32_t)(reinterpret_cast<uintptr_t>(p) & 3);
  uint32_t w[5];
#pragma unroll
  for (int i = 0; i < 5; ++i) w[i] = a[i];
#pragma unroll
  for (int i = 0; i < 4; ++i) o[i] = __funnelshift_r(w[i], w[i + 1], sh);
}

__device__ __forceinline__ uint32_t low_bytes_mask(int t) {  // the low t bytes (t clamped to 0 .. 4)
  return t >= 4 ? 0xffffffffu : (t <= 0 ? 0u : (1u << (8 * t)) - 1u);
}

// __byte_perm selector taking bytes [0, t) of a and the rest of b (t clamped to 0 .. 4).
__device__ __forceinline__ uint32_t merge_sel(int t) {
  t = t < 0 ? 0 : (t > 4 ? 4 : t);
  return 0x7654u - (0x4444u & ((1u << (4 * t)) - 1u));
}

constexpr int IM2COL_SEG_MAX_CPR = IM2COL_MAX_KC / 16;

__global__ void __launch_bounds__(256) im2col_seg_kernel(const uint8_t* __restrict__ act, int H, int W, int C, int R,
                                                        int S, int stride, int pad, int Ho, int Wo, int Kred,
                                                        int Kc, uint8_t* __restrict__ col) {
  extern __shared__ __align__(16) uint8_t sm_seg[];
  // per piece q of a col row (the same for every row): the offsets of its two windows from the
  // row's tap-0 byte, and n0 | nz << 8 (bytes from filter row r0; bytes below Kred)
  __shared__ int tab_a[IM2COL_SEG_MAX_CPR], tab_b[IM2COL_SEG_MAX_CPR], tab_n[IM2COL_SEG_MAX_CPR];
  const int padB = im2col_seg_padb(pad, C), RS = im2col_seg_rs(W, C, pad);
  uint8_t* rows = sm_seg + IM2COL_SEG_GUARD;  // [R][RS]
  const int ho = blockIdx.x % Ho;
  const int b = blockIdx.x / Ho;
  const int h0 = ho * stride - pad;
  const int rowb = W * C;
  const int SC = S * C;
  const int cpr = Kc / 16;  // 16-byte pieces per col row
  for (int q = threadIdx.x; q < cpr; q += blockDim.x) {
    const int k0 = 16 * q;
    const int r0 = k0 / SC, j0 = k0 - r0 * SC;
    const int n0 = SC - j0 < 16 ? SC - j0 : 16;
    const int nz = k0 >= Kred ? 0 : (Kred - k0 < 16 ? Kred - k0 : 16);
    tab_a[q] = r0 * RS + j0;
    tab_b[q] = (n0 < 16 && r0 + 1 < R) ? (r0 + 1) * RS - n0 : -1;
    tab_n[q] = n0 | (nz << 8);
  }
  const int nz16 = (2 * IM2COL_SEG_GUARD + R * RS) / 16;
  for (int i = threadIdx.x; i < nz16; i += blockDim.x) reinterpret_cast<uint4*>(sm_seg)[i] = make_uint4(0u, 0u, 0u, 0u);
  __syncthreads();
  if (rowb % 16 == 0 && (reinterpret_cast<uintptr_t>(act) & 15) == 0) {
    const int n16 = rowb / 16;
    for (int i = threadIdx.x; i < R * n16; i += blockDim.x) {
      const int r = i / n16, e = i - r * n16;
      const int h = h0 + r;
      if (h >= 0 && h < H)
        *reinterpret_cast<uint4*>(rows + r * RS + padB + 16 * e) =
            __ldg(reinterpret_cast<const uint4*>(act + ((int64_t)b * H + h) * rowb) + e);
    }
  } else {
    for (int i = threadIdx.x; i < R * rowb; i += blockDim.x) {
      const int r = i / rowb, e = i - r * rowb;
      const int h = h0 + r;
      if (h >= 0 && h < H) rows[r * RS + padB + e] = __ldg(act + ((int64_t)b * H + h) * rowb + e);
    }
  }
  __syncthreads();
  uint4* dst = reinterpret_cast<uint4*>(col + ((int64_t)b * Ho + ho) * Wo * Kc);
  // piece i = wo cpr + q, advanced by blockDim pieces without a division per piece
  const int dwo = (int)blockDim.x / cpr, dq = (int)blockDim.x - dwo * cpr;
  int wo = (int)threadIdx.x / cpr, q = (int)threadIdx.x - wo * cpr;
  for (int i = threadIdx.x; i < Wo * cpr; i += blockDim.x) {
    const int tn = tab_n[q];
    const int n0 = tn & 0xff, nz = tn >> 8;
    uint32_t o[4] = {0u, 0u, 0u, 0u};
    if (nz > 0) {
      const uint8_t* tap0 = rows + padB + (wo * stride - pad) * C;  // byte of filter tap s = 0 in staged row 0
      uint32_t A[4], Bw[4] = {0u, 0u, 0u, 0u};
      window16(tap0 + tab_a[q], A);
      const int ob = tab_b[q];
      if (ob >= 0) window16(tap0 + ob, Bw);
#pragma unroll
      for (int w = 0; w < 4; ++w) o[w] = __byte_perm(A[w], Bw[w], merge_sel(n0 - 4 * w));
      if (nz < 16) {  // the row's last piece below Kred: zero its bytes from nz on
#pragma unroll
        for (int w = 0; w < 4; ++w) o[w] &= low_bytes_mask(nz - 4 * w);
      }
    }
    dst[i] = make_uint4(o[0], o[1], o[2], o[3]);
    wo += dwo;
    q += dq;
    if (q >= cpr) {
      q -= cpr;
      ++wo;
    }
  }
}

// 8-bit weights wq [M][Kred] as fp16 [M][Kc] (zero-padded), rs = wscale: exact.
__global__ void __launch_bounds__(256) fold_w8_kernel(const int8_t* __restrict__ wq, const float* __restrict__ wscale,
                                                      int M, int Kred, int Kc, __half* __restrict__ a0,
                                                      float* __restrict__ row_scale) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (int64_t)M * Kc) return;
  const int m = (int)(i / Kc), k = (int)(i % Kc);
  a0[i] = __float2half_rn(k < Kred ? (float)__ldg(wq + (int64_t)m * Kred + k) : 0.0f);
  if (k == 0) row_scale[m] = __ldg(wscale + m);
}

// Tensor maps and launch of the dense kernel for folded weights a0 (+ a1) and row scales rs.
fgq_status run_dense(const void* act, const Geom& g, int NA, const __half* a0, const __half* a1, const float* rs,
                     const float* act_scale, float* out, unsigned int* err, cudaStream_t s) {
  TDArgs a;
  memset(&a, 0, sizeof a);
  a.act = static_cast<const uint8_t*>(act);
  a.row_scale = rs;
  a.act_scale = act_scale;
  a.out = out;
  a.err = err;
  a.g = g;
  a.mtiles = (g.Mg + TD_BM - 1) / TD_BM;
  a.ptiles = (int)((g.P + TD_BN - 1) / TD_BN);
  a.ntiles = g.groups * a.mtiles * a.ptiles;
  a.ktiles = g.Kred / TD_KT;
  // a test may shorten the waits (debug_wait_limit_us), never the final drains
  const int64_t lim_us = debug_wait_limit_us();
  a.timeout_ns = lim_us < 0 ? TD_TIMEOUT_NS : (uint64_t)lim_us * 1000u;
  for (int part = 0; part < NA; ++part)
    if (!make_map_2d(&a.a_map[part], CU_TENSOR_MAP_DATA_TYPE_FLOAT16, part ? (const void*)a1 : (const void*)a0,
                     (uint64_t)g.Kp, (uint64_t)g.M, (uint64_t)g.Kp * 2, TD_KT, TD_BM, CU_TENSOR_MAP_SWIZZLE_128B))
      return FGQ_ERR_CUDA;
  bool tmap = false;
  if (g.R == 1 && g.S == 1 && g.stride == 1 && g.pad == 0)
    tmap = make_map_2d(&a.act_map, CU_TENSOR_MAP_DATA_TYPE_UINT8, act, (uint64_t)g.C, (uint64_t)g.B * g.H * g.W,
                       (uint64_t)g.C, TD_KT, TD_BN, CU_TENSOR_MAP_SWIZZLE_64B);
  if (NA == 1 && g.groups == 1 && g.M % 4 == 0 && !g.rq_out)
    a.out_tma = make_map_2d(&a.out_map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, out, (uint64_t)g.M, (uint64_t)g.P,
                            (uint64_t)g.M * 4, TD_BM, 64, CU_TENSOR_MAP_SWIZZLE_NONE)
                    ? 1
                    : 0;
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int grid = a.ntiles < sms ? a.ntiles : sms;
  const bool sgn = g.act_type == FGQ_S8;
  return NA == 1 ? launch_dense_na<1>(a, sgn, tmap, grid, s) : launch_dense_na<2>(a, sgn, tmap, grid, s);
}

constexpr int64_t DENSE_W8_MAX_COL_BYTES = (int64_t)8 << 30;  // the im2col temporary

}  // namespace

fgq_status launch_dense_contract(const void* act, const Geom& g, const uint32_t* codes, const float* alpha,
                                 const uint8_t* aq, int abits, const float* ascale, const float* act_scale, float* out,
                                 unsigned int* err, cudaStream_t s) {
  if (!dense_supports(g)) return FGQ_ERR_UNSUPPORTED;
  if (aq ? (abits != 8 && abits != 4) || !ascale : !alpha) return FGQ_ERR_ARG;
  const int NA = aq ? 1 : 2;
  // folded weights fp16 [NA][M][Kp] and row scales [M], in one temporary from the pool
  cudaMemPool_t pool = scratch_pool();
  if (!pool) return FGQ_ERR_CUDA;
  const size_t part_bytes = (size_t)g.M * g.Kp * 2;
  void* tmp = nullptr;
  if (cudaMallocFromPoolAsync(&tmp, NA * part_bytes + (size_t)g.M * 4, pool, s) != cudaSuccess) return FGQ_ERR_CUDA;
  __half* a0 = static_cast<__half*>(tmp);
  __half* a1 = NA == 2 ? a0 + (size_t)g.M * g.Kp : nullptr;
  float* rs = reinterpret_cast<float*>(static_cast<uint8_t*>(tmp) + NA * part_bytes);
  const unsigned fblocks = (unsigned)g.M;
  if (!aq)
    fold_weights_kernel<0><<<fblocks, FOLD_THREADS, 0, s>>>(codes, g.M, g.wrow, g.G, g.ng, alpha, nullptr, nullptr, a0,
                                                            a1, rs);
  else if (abits == 8)
    fold_weights_kernel<8><<<fblocks, FOLD_THREADS, 0, s>>>(codes, g.M, g.wrow, g.G, g.ng, nullptr, aq, ascale, a0, a1,
                                                            rs);
  else
    fold_weights_kernel<4><<<fblocks, FOLD_THREADS, 0, s>>>(codes, g.M, g.wrow, g.G, g.ng, nullptr, aq, ascale, a0, a1,
                                                            rs);
  fgq_status st = after_launch();
  if (st == FGQ_OK) st = run_dense(act, g, NA, a0, a1, rs, act_scale, out, err, s);
  // the temporary returns to the pool once the work queued on s before this point is done
  if (cudaFreeAsync(tmp, s) != cudaSuccess && st == FGQ_OK) st = FGQ_ERR_CUDA;
  return st;
}

fgq_status launch_fold_alpha_split(const uint32_t* codes, int M, int wrow, int G, int ng, const float* alpha,
                                   void* a0, void* a1, float* rs, cudaStream_t s) {
  fold_weights_kernel<0><<<(unsigned)M, FOLD_THREADS, 0, s>>>(codes, M, wrow, G, ng, alpha, nullptr, nullptr,
                                                                static_cast<__half*>(a0), static_cast<__half*>(a1), rs);
  return after_launch();
}

bool dense_w8_supports(const Geom& g) {
  if (g.act_type != FGQ_U8 && g.act_type != FGQ_S8) return false;
  if (g.groups != 1 || g.P >= (int64_t)1 << 31) return false;
  const int64_t Kc = (g.Kred + TD_KT - 1) / TD_KT * TD_KT;
  if (Kc > IM2COL_MAX_KC || g.P * Kc > DENSE_W8_MAX_COL_BYTES) return false;
  return encode_tiled() != nullptr;
}

fgq_status launch_dense_w8(const void* act, const Geom& g, const int8_t* wq, const float* wscale,
                           const float* act_scale, float* out, unsigned int* err, cudaStream_t s) {
  if (!dense_w8_supports(g)) return FGQ_ERR_UNSUPPORTED;
  const int Kc = (g.Kred + TD_KT - 1) / TD_KT * TD_KT;
  cudaMemPool_t pool = scratch_pool();
  if (!pool) return FGQ_ERR_CUDA;
  const size_t col_bytes = (size_t)g.P * Kc, a_bytes = (size_t)g.M * Kc * 2;
  void* tmp = nullptr;
  if (cudaMallocFromPoolAsync(&tmp, col_bytes + a_bytes + (size_t)g.M * 4, pool, s) != cudaSuccess)
    return FGQ_ERR_CUDA;
  uint8_t* col = static_cast<uint8_t*>(tmp);
  __half* a0 = reinterpret_cast<__half*>(col + col_bytes);
  float* rs = reinterpret_cast<float*>(col + col_bytes + a_bytes);
  const size_t rows_smem = im2col_rows_smem(g, Kc), seg_smem = im2col_seg_smem(g);
  if (g.S * g.C >= 16 && seg_smem <= (size_t)IM2COL_ROWS_SMEM && (int64_t)g.B * g.Ho < INT32_MAX)
    im2col_seg_kernel<<<(unsigned)((int64_t)g.B * g.Ho), 256, seg_smem, s>>>(
        static_cast<const uint8_t*>(act), g.H, g.W, g.C, g.R, g.S, g.stride, g.pad, g.Ho, g.Wo, g.Kred, Kc, col);
  else if (rows_smem <= (size_t)IM2COL_ROWS_SMEM && g.S <= 254 && g.R * g.W * g.C < 65536 &&
      (int64_t)g.B * g.Ho < INT32_MAX)
    im2col_rows_kernel<<<(unsigned)((int64_t)g.B * g.Ho), 256, rows_smem, s>>>(
        static_cast<const uint8_t*>(act), g.H, g.W, g.C, g.R, g.S, g.stride, g.pad, g.Ho, g.Wo, g.Kred, Kc, col);
  else
    im2col_u8_kernel<<<(unsigned)((g.P + 127) / 128), 128, 0, s>>>(
        static_cast<const uint8_t*>(act), g.B, g.H, g.W, g.C, g.R, g.S, g.stride, g.pad, g.Ho, g.Wo, g.Kred, Kc, col);
  fgq_status st = after_launch();
  if (st == FGQ_OK) {
    fold_w8_kernel<<<(unsigned)(((int64_t)g.M * Kc + 255) / 256), 256, 0, s>>>(wq, wscale, g.M, g.Kred, Kc, a0, rs);
    st = after_launch();
  }
  if (st == FGQ_OK) {
    // the convolution as a GEMM over the im2col rows: P x Kc activations, M x Kc weights
    Geom gg = g;
    gg.B = (int)g.P;
    gg.H = gg.W = gg.Ho = gg.Wo = 1;
    gg.R = gg.S = gg.stride = 1;
    gg.pad = 0;
    gg.C = gg.Cg = gg.Kred = gg.Kp = Kc;
    gg.G = TD_KT;
    gg.ng = Kc / TD_KT;
    gg.wrow = Kc / 16;
    gg.Mg = g.M;
    gg.is_conv = 0;
    st = run_dense(col, gg, 1, a0, nullptr, rs, act_scale, out, err, s);
  }
  if (cudaFreeAsync(tmp, s) != cudaSuccess && st == FGQ_OK) st = FGQ_ERR_CUDA;
  return st;
}

}  // namespace fgq
