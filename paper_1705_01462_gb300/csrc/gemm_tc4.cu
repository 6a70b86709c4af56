// Tensor-core (tcgen05) grouped ternary contraction for G = 4.
//
// Math (Eq. 2, 32-bit group accumulators of Section 4): y[p][m] = s_x * sum_g alpha[m][g]
// * s[m][g][p] with s an exact integer sum over a group of 4 reduction elements.  A dense
// MMA would sum across groups, so each K = 16 MMA step (4 groups) uses a block-diagonal
// activation operand B' of 256 rows: row 64 j + P holds the activations of tile position P
// only in the 4 columns of group slot j (zeros elsewhere), and D[m][64 j + P] of one MMA
// (M = 128, N = 256, K = 16) receives the products of group 4 step + j alone.  The zeros of
// B' never change, so they are written once per CTA; each K-tile writes only the diagonal
// 8-byte pieces.  Two variants share the loaders:
//
//   output (FOLD): the group's scale multiplies inside the MMA (one multiply per group,
//     Section 4.1): the ternary operand is the fp32 alpha folded into the codes as two fp16
//     parts, alpha(m, g) t[m][k] 2^e_m = hi + lo to about 22 bits (hi the fp16 nearest, lo the
//     fp16 nearest the remainder; e_m puts row m's largest alpha in [2^14, 2^15)).  Every
//     product hi t q and lo t q is exact in fp32 and so is each part's group sum hi s_g (11
//     significant bits times |s_g| <= 1020), so one step adds (hi + lo) s_g to the element
//     its slot owns.  The 8 MMAs of a K-tile (4 steps x 2 parts) accumulate in TMEM, and the
//     epilogue adds the K-tile's four slot partials into fp32 registers with round-to-nearest
//     adds: every rounding is bounded by a K-tile's share of sum_g |alpha_g s_g|, far inside
//     the 1e-5 sum_g |alpha_g s_g| tolerance, and the accumulator is drained (and committed)
//     once per K-tile instead of once per step.  y = s_x 2^-e_m acc.
//   group sums (!FOLD): the ternary operand is the codes in fp16 {0, +1, -1}; each step's
//     D is exactly s[m][g][p] (fp16 operands on exact integers), stored as int32 (for
//     verification of the integer accumulators).
//
// The ternary operand reaches shared memory by TMA box loads in the MMA's swizzled layout,
// from a per-call stream-ordered temporary (folded: launch_fold_alpha_split; codes:
// expand_codes_kernel).
//
// Tile: 128 filters x 64 positions; K-tile 64 (16 groups, 4 steps).  TMEM: two 256-column
// buffers.  Output: one buffer per K-tile, so the MMAs of K-tile j + 1 run while the
// epilogue drains K-tile j.  Group sums: one buffer per step.
// Warp roles (416 threads, one CTA per SM, persistent over tiles):
//   warps 0-7  epilogue: warp w owns TMEM lanes 32 (w % 4) .. (filters) and the 32
//              positions of half w / 4; it loads its 32-column slices of the four slots
//              (two at a time), frees the buffer once they are in registers, and adds them
//              into 32 position accumulators (output), or stores them as int32 (group
//              sums).  At tile end the output is scaled by s_x 2^-e_m and written through
//              shared memory with TMA box stores (two 32-position boxes) when the output
//              allows, else directly (or requantized).
//   warps 8-11 loaders/converters: thread t builds, for position t % 64, MMA steps
//              2 (t / 64), 2 (t / 64) + 1 of B'; activations come by TMA boxes (1x1
//              stride-1 layers and GEMMs) or by per-thread cp.async gathers whose completion
//              is tracked on the stage's mbarrier; thread 0 also issues the A box loads.
//   warp 12    TMEM allocation and the MMA issuer.
// Every mbarrier wait is bounded in time; on expiry the kernel records FGQ_ERR_TIMEOUT,
// each role leaves its loop (uniformly within the epilogue, which uses named barriers),
// in-flight copies and MMAs are waited for, and TMEM is freed.
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

constexpr int T4_BM = 128;      // filters per tile (MMA M, TMEM lanes)
constexpr int T4_BP = 64;       // positions per tile
constexpr int T4_KT = 64;       // reduction elements per K-tile: 16 groups, 4 MMA steps
constexpr int T4_NB = 2;        // B' (activation operand) ring depth
constexpr int T4_NAS = 4;       // A (ternary operand) ring depth
constexpr int T4_NACC = 2;      // TMEM buffers of 256 columns
constexpr int T4_EPI_WARPS = 8;
constexpr int T4_LOAD_WARP0 = 8;  // loaders: warps 8-11
constexpr int T4_LOADERS = 128;
constexpr int T4_MMA_WARP = 12;
constexpr int T4_A_WARP = 13;     // lane 0 streams the A boxes
constexpr int T4_THREADS = 32 * (T4_A_WARP + 1);
constexpr int T4_TMEM_COLS = T4_NACC * 256;
constexpr uint64_t T4_TIMEOUT_NS = 1000000000ull;  // 1 s per wait
constexpr uint32_t T4_DRAIN_LIMIT = 1u << 20;      // polls of the final drains (never shortened)
constexpr uint32_t BAR_EPI4 = 2;

constexpr int A_TILE4 = 128 * T4_KT * 2;      // 16 KB fp16 ternary operand [128 filters][64 K], per part
constexpr int B_TILE4 = 256 * T4_KT * 2;      // 32 KB fp16 block-diagonal activations
constexpr int ST_STAGE4 = T4_BP * T4_KT;      // 4 KB: 64 raw activation rows (8-bit: 64 B each)
constexpr int OUT_BOX4 = 32 * T4_BM * 4;      // 16 KB fp32 [32 positions][128 filters]

// Shared-memory plan of a variant: A ring (the ternary operand's parts), B' ring, staging
// ring, output box, barriers.
template <bool FOLD>
struct T4Cfg {
  static constexpr int NPART = FOLD ? 2 : 1;
  static constexpr int A_STAGE = NPART * A_TILE4;
  static constexpr int NS = FOLD ? 4 : 6;  // staging ring depth
  static constexpr int OUT = FOLD ? OUT_BOX4 : 0;
  static constexpr int SMEM_A = T4_NAS * A_STAGE;
  static constexpr int SMEM_B = T4_NB * B_TILE4;
  static constexpr int BAR = 8 * (2 * T4_NAS + 2 * T4_NB + 2 * NS + 2 * T4_NACC + 1) + 16;
  static constexpr int SMEM = 1024 + SMEM_A + SMEM_B + NS * ST_STAGE4 + OUT + BAR;
};
static_assert(T4Cfg<true>::SMEM <= 232448 && T4Cfg<false>::SMEM <= 232448, "shared memory budget");
static_assert(ST_STAGE4 % 1024 == 0 && A_TILE4 % 1024 == 0 && B_TILE4 % 1024 == 0, "stage alignment");

struct T4Args {
  CUtensorMap a_map[2];   // fp16 [M][Kp] ternary operand parts (folded hi, lo; or codes), box {64, 128 rows},
                          // 128-byte swizzle
  CUtensorMap act_map;    // uint8 [pixels][row bytes], box {64 (or 32) bytes, 64 rows}; TMA path
  CUtensorMap out_map;    // fp32 [P][M], box {128 filters, 32 positions}; if out_tma
  const uint8_t* act;
  const float* row_scale;  // FOLD: 2^-e_m [M]
  const float* act_scale;
  float* out;
  int32_t* sums;  // !FOLD: int32 group sums [M][ng][P]
  unsigned int* err;
  Geom g;
  int mtiles, ptiles, ntiles, ktiles;
  int act_tma, out_tma;
  uint64_t timeout_ns;
};

// Tiles are numbered with the filter tiles of one position tile consecutive, so that
// CTAs running at the same time share activation rows in L2.
__device__ __forceinline__ void tile_coords4(const T4Args& a, int tile, int& gi, int& m0, int64_t& p0) {
  const int per_p = a.g.groups * a.mtiles;
  const int pt = tile / per_p;
  const int r = tile - pt * per_p;
  gi = r / a.mtiles;
  m0 = gi * a.g.Mg + (r - gi * a.mtiles) * T4_BM;
  p0 = (int64_t)pt * T4_BP;
}

__device__ __forceinline__ void add32(float (&acc)[32], const uint32_t (&r)[32]) {
#pragma unroll
  for (int i = 0; i < 32; ++i) acc[i] += __uint_as_float(r[i]);
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

template <int ABITS, bool SIGNED, bool TMAP, bool FOLD>
__global__ void __launch_bounds__(T4_THREADS, 1) tc4_contract_kernel(const __grid_constant__ T4Args a) {
  using Cfg = T4Cfg<FOLD>;
  constexpr int NS = Cfg::NS;
  extern __shared__ uint8_t smem_raw4[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw4) + 1023) & ~uintptr_t(1023));
  uint8_t* abuf = smem;
  uint8_t* bbuf = smem + Cfg::SMEM_A;
  uint8_t* st = bbuf + Cfg::SMEM_B;
  float* otile = reinterpret_cast<float*>(st + NS * ST_STAGE4);
  uint64_t* bars = reinterpret_cast<uint64_t*>(st + NS * ST_STAGE4 + Cfg::OUT);
  uint64_t* a_full = bars;
  uint64_t* a_empty = bars + T4_NAS;
  uint64_t* op_full = bars + 2 * T4_NAS;
  uint64_t* op_empty = op_full + T4_NB;
  uint64_t* st_full = op_empty + T4_NB;
  uint64_t* st_empty = st_full + NS;
  uint64_t* acc_full = st_empty + NS;
  uint64_t* acc_empty = acc_full + T4_NACC;
  uint64_t* drain_bar = acc_empty + T4_NACC;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_bar + 1);
  volatile uint32_t* abort_flag = tmem_slot + 1;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const Geom& g = a.g;
  const uint64_t tmo = a.timeout_ns;

  if (threadIdx.x == 0) {
    for (int i = 0; i < T4_NAS; ++i) {
      mbar_init(&a_full[i], 1);   // the A boxes' byte count
      mbar_init(&a_empty[i], 1);  // released by the epilogue once the K-tile's MMAs completed
    }
    for (int i = 0; i < T4_NB; ++i) {
      mbar_init(&op_full[i], T4_LOADERS);  // B' pieces
      mbar_init(&op_empty[i], 1);          // released like a_empty
    }
    for (int i = 0; i < NS; ++i) {
      mbar_init(&st_full[i], TMAP ? 1 : T4_LOADERS);
      mbar_init(&st_empty[i], T4_LOADERS);
    }
    for (int i = 0; i < T4_NACC; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], T4_EPI_WARPS);
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  // the off-diagonal zeros of every B' tile, written once
  for (int s = 0; s < T4_NB; ++s) {
    uint4* bt = reinterpret_cast<uint4*>(bbuf + s * B_TILE4);
    for (int i = threadIdx.x; i < B_TILE4 / 16; i += blockDim.x) bt[i] = make_uint4(0u, 0u, 0u, 0u);
  }
  fence_proxy_async_smem();
  if (warp == T4_MMA_WARP) {
    tmem_alloc(tmem_slot, T4_TMEM_COLS);
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
  if (warp >= T4_LOAD_WARP0 && warp < T4_MMA_WARP) {
    const int t = threadIdx.x - 32 * T4_LOAD_WARP0;
    const int P = t & (T4_BP - 1);  // tile position whose activations this thread copies/converts
    const int cpair = t >> 6;       // MMA steps 2 cpair, 2 cpair + 1 of the K-tile
    const int total = my_tiles * a.ktiles;
    constexpr int ROW_BYTES = T4_KT * ABITS / 8;
    constexpr int CPT = ROW_BYTES / 32;  // 16-byte chunks per thread and K-tile (2 or 1)
    constexpr uint32_t TX_ACT = T4_BP * ROW_BYTES;

    // walk of the K-tiles this thread issues copies for
    int cur_tile = -1, gi = 0, m0 = 0, tr = 0, ts = 0, tc0 = 0;
    int64_t p0 = 0;
    int pb = 0, phb = 0, pwb = 0;
    bool pvalid = false;
    int issued = 0;
    // activation copies of K-tile j (of this CTA's sequence) into staging slot j % NS
    auto issue = [&](int j) -> bool {
      const int tl = j / a.ktiles;
      if (tl != cur_tile) {
        cur_tile = tl;
        tile_coords4(a, (int)blockIdx.x + tl * (int)gridDim.x, gi, m0, p0);
        tr = ts = tc0 = 0;
        const int64_t p = p0 + P;
        pvalid = p < g.P;
        const int pp = pvalid ? (int)p : 0;
        const int wo = pp % g.Wo;
        const int q = pp / g.Wo;
        const int ho = q % g.Ho;
        pb = q / g.Ho;
        phb = ho * g.stride - g.pad;
        pwb = wo * g.stride - g.pad;
      }
      const int slot = j % NS;
      uint8_t* sa = st + slot * ST_STAGE4;
      if (TMAP) {
        if (t == 0) {
          if (j >= NS && !mbar_wait_timed(&st_empty[slot], ((j / NS) & 1) ^ 1, tmo, abort_flag, 64))
            return false;
          mbar_arrive_expect_tx(&st_full[slot], TX_ACT);
          tma_load_2d(smem_u32(sa), &a.act_map, (gi * g.Cg + tc0) * ABITS / 8, (int)p0, &st_full[slot]);
          issued = j + 1;
        }
      } else {
        if (j >= NS && !mbar_wait_timed(&st_empty[slot], ((j / NS) & 1) ^ 1, tmo, abort_flag, 64))
          return false;
        const uint8_t* src = a.act;
        bool inside = false;
        if (pvalid) {
          const int hi = phb + tr, wi = pwb + ts;
          if (hi >= 0 && hi < g.H && wi >= 0 && wi < g.W) {
            const int64_t e = (((int64_t)pb * g.H + hi) * g.W + wi) * g.C + (int64_t)gi * g.Cg + tc0;
            src = a.act + e * ABITS / 8;
            inside = true;
          }
        }
#pragma unroll
        for (int i = 0; i < CPT; ++i) {
          const int c = cpair * CPT + i;
          cp_async16(smem_u32(sa + st_off<ABITS>(P, c)), inside ? (const void*)(src + 16 * c) : (const void*)a.act,
                     inside ? 16u : 0u);
        }
        cp_async_mbar_arrive_noinc(&st_full[slot]);
        issued = j + 1;
      }
      tc0 += T4_KT;
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
    for (int j = 0; j < NS - 1 && j < total && ok; ++j) ok = issue(j);
    int consumed = 0;
    for (int j = 0; j < total && ok; ++j) {
      if (j + NS - 1 < total && !issue(j + NS - 1)) {
        ok = false;
        break;
      }
      const int slot = j % NS;
      const int os = j % T4_NB;
      if (!mbar_wait_timed(&op_empty[os], ((j / T4_NB) & 1) ^ 1, tmo, abort_flag, 64)) {
        ok = false;
        break;
      }
      uint8_t* Bt = bbuf + os * B_TILE4;
      if (!mbar_wait_timed(&st_full[slot], (j / NS) & 1, tmo, abort_flag, 32)) {
        ok = false;
        break;
      }
      consumed = j + 1;
      const uint8_t* sa = st + slot * ST_STAGE4;
      // B' rows 64 jj + P for slots jj = 0..3, MMA steps s of this thread: the 4 activations
      // of group slot jj at K offsets 16 s + 4 jj .. +3
      uint32_t wv[2][4];
      if (ABITS == 8) {
#pragma unroll
        for (int ss = 0; ss < 2; ++ss) {
          const uint4 v = *reinterpret_cast<const uint4*>(sa + st_off<8>(P, 2 * cpair + ss));
          wv[ss][0] = v.x;
          wv[ss][1] = v.y;
          wv[ss][2] = v.z;
          wv[ss][3] = v.w;
        }
      } else {
        // one 16-byte chunk = steps 2 cpair (bytes 0-7) and 2 cpair + 1 (bytes 8-15); the 4
        // nibbles of slot jj are 16-bit half jj of the step's 8 bytes
        const uint4 v = *reinterpret_cast<const uint4*>(sa + st_off<4>(P, cpair));
        const uint32_t half[2][2] = {{v.x, v.y}, {v.z, v.w}};
#pragma unroll
        for (int ss = 0; ss < 2; ++ss)
#pragma unroll
          for (int jj = 0; jj < 4; ++jj) {
            const uint32_t hw = (half[ss][jj >> 1] >> (16 * (jj & 1))) & 0xffffu;
            wv[ss][jj] = (hw & 0xfu) | ((hw & 0xf0u) << 4) | ((hw & 0xf00u) << 8) | ((hw & 0xf000u) << 12);
          }
      }
      constexpr uint32_t bias2 =
          ABITS == 8 ? (SIGNED ? 0x64806480u : 0x64006400u) : (SIGNED ? 0x64086408u : 0x64006400u);
      constexpr uint32_t flip = ABITS == 8 ? 0x80808080u : 0x08080808u;
#pragma unroll
      for (int ss = 0; ss < 2; ++ss) {
        const int s = 2 * cpair + ss;
#pragma unroll
        for (int jj = 0; jj < 4; ++jj) {
          const uint32_t w = SIGNED ? (wv[ss][jj] ^ flip) : wv[ss][jj];
          const uint2 hv = make_uint2(u8pair_to_h2(w, 0x4140, bias2), u8pair_to_h2(w, 0x4342, bias2));
          *reinterpret_cast<uint2*>(Bt + sw128(64 * jj + P, 2 * s + (jj >> 1)) + 8 * (jj & 1)) = hv;
        }
      }
      fence_proxy_async_smem();
      mbar_arrive(&op_full[os]);
      mbar_arrive(&st_empty[slot]);
    }
    if (!ok && !*abort_flag) fail();
    if (!TMAP) cp_async_wait_all();
    if (TMAP && t == 0) {
      for (int j = consumed; j < issued; ++j) mbar_wait_bounded(&st_full[j % NS], (j / NS) & 1, T4_DRAIN_LIMIT);
    }
  }

  // ------------------------------------------------------------------ A boxes
  if (warp == T4_A_WARP && lane == 0) {
    const int total = my_tiles * a.ktiles;
    int armed = 0;
    bool ok = true;
    for (int j = 0; j < total; ++j) {
      const int as = j % T4_NAS;
      if (!mbar_wait_timed(&a_empty[as], ((j / T4_NAS) & 1) ^ 1, tmo, abort_flag, 64)) {
        ok = false;
        break;
      }
      const int tl = j / a.ktiles;
      int gj, mj;
      int64_t pj;
      tile_coords4(a, (int)blockIdx.x + tl * (int)gridDim.x, gj, mj, pj);
      uint8_t* A = abuf + as * Cfg::A_STAGE;
      mbar_arrive_expect_tx(&a_full[as], Cfg::A_STAGE);
#pragma unroll
      for (int part = 0; part < Cfg::NPART; ++part)
        tma_load_2d(smem_u32(A + part * A_TILE4), &a.a_map[part], (j - tl * a.ktiles) * T4_KT, mj, &a_full[as]);
      armed = j + 1;
    }
    if (!ok && !*abort_flag) fail();
    // boxes the MMA issuer may not have consumed: the last T4_NAS armed ones, one per stage,
    // each the latest phase of its stage's barrier
    for (int j = armed - T4_NAS < 0 ? 0 : armed - T4_NAS; j < armed; ++j)
      mbar_wait_bounded(&a_full[j % T4_NAS], (j / T4_NAS) & 1, T4_DRAIN_LIMIT);
  }

  // ------------------------------------------------------------------ MMA issuer
  if (warp == T4_MMA_WARP && lane == 0) {
    const uint32_t idesc = idesc_f16_f32(128, 256);
    const int total = my_tiles * a.ktiles;
    int sc = 0;  // group sums: steps issued
    bool ok = true;
    for (int j = 0; j < total && ok; ++j) {
      const int os = j % T4_NB, as = j % T4_NAS;
      if (!mbar_wait_timed(&op_full[os], (j / T4_NB) & 1, tmo, abort_flag, 0) ||
          !mbar_wait_timed(&a_full[as], (j / T4_NAS) & 1, tmo, abort_flag, 0)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t abase = smem_u32(abuf + as * Cfg::A_STAGE);
      const uint64_t bd = sdesc_k_sw128(smem_u32(bbuf + os * B_TILE4));
      if (FOLD) {
        // the K-tile's 8 MMAs (4 steps x 2 parts) accumulate into buffer j % 2
        const int b = j & 1;
        if (!mbar_wait_timed(&acc_empty[b], ((j >> 1) & 1) ^ 1, tmo, abort_flag, 0)) {
          ok = false;
          break;
        }
        tc_fence_after();
#pragma unroll
        for (int s = 0; s < 4; ++s)
#pragma unroll
          for (int part = 0; part < Cfg::NPART; ++part)
            mma_f16(tmem + (uint32_t)(b * 256), sdesc_k_sw128(abase + part * A_TILE4) + 2 * s, bd + 2 * s, idesc,
                    (s | part) != 0 ? 1u : 0u);
        mma_commit(&acc_full[b]);
      } else {
        const uint64_t ad = sdesc_k_sw128(abase);
        for (int s = 0; s < 4; ++s, ++sc) {
          const int b = sc & 1;
          if (!mbar_wait_timed(&acc_empty[b], ((sc >> 1) & 1) ^ 1, tmo, abort_flag, 0)) {
            ok = false;
            break;
          }
          tc_fence_after();
          mma_f16(tmem + (uint32_t)(b * 256), ad + 2 * s, bd + 2 * s, idesc, 0u);
          mma_commit(&acc_full[b]);
        }
      }
      // the operand stages are released by the epilogue, which sees the K-tile's last
      // accumulator commit (one commit per buffer use, none spent on the stages)
    }
    if (!ok && !*abort_flag) fail();
    mma_commit(drain_bar);
    mbar_wait_bounded(drain_bar, 0, T4_DRAIN_LIMIT);
  }

  // ------------------------------------------------------------------ epilogue
  if (warp < T4_EPI_WARPS) {
    const int quarter = warp & 3, hsub = warp >> 2;
    const int t = 32 * quarter + lane;  // TMEM lane = filter row of the tile
    const uint32_t tbase = tmem + ((uint32_t)(32 * quarter) << 16) + (uint32_t)(32 * hsub);
    const float sx = __ldg(a.act_scale);
    const bool leader = threadIdx.x == 0;
    int sc = 0;  // buffer uses drained so far (K-tiles when folded, steps otherwise)
    bool ok = true;
    for (int tl = 0; tl < my_tiles; ++tl) {
      int gi, m0;
      int64_t p0;
      tile_coords4(a, (int)blockIdx.x + tl * (int)gridDim.x, gi, m0, p0);
      const int m = m0 + t;
      const bool mok = m < gi * g.Mg + g.Mg && m < g.M;
      const int64_t pw = p0 + 32 * hsub;  // this warp's first position
      float acc[32];
#pragma unroll
      for (int i = 0; i < 32; ++i) acc[i] = 0.0f;
      const int ndrain = FOLD ? a.ktiles : a.ktiles * 4;
      for (int u = 0; u < ndrain; ++u, ++sc) {
        if (!ok) continue;
        const int b = sc & 1;
        if (!mbar_wait_timed(&acc_full[b], (sc >> 1) & 1, tmo, abort_flag, 0)) {
          ok = false;
          continue;
        }
        if (leader && (FOLD || (u & 3) == 3)) {
          // the K-tile's MMAs have completed: its A and B' stages may be refilled
          const int kt = FOLD ? sc : sc >> 2;
          mbar_arrive(&a_empty[kt % T4_NAS]);
          mbar_arrive(&op_empty[kt % T4_NB]);
        }
        tc_fence_after();
        // slot j at columns 64 j .. 64 j + 63; this warp's 32 positions at + 32 hsub
        const uint32_t ta = tbase + (uint32_t)(b * 256);
        uint32_t r0[32], r1[32];
        if (FOLD) {
          tmem_ld32(ta, r0);
          tmem_ld32(ta + 64, r1);
          tmem_ld_wait_regs(r0);
          reg_fence(r1);
          add32(acc, r0);
          tmem_ld32(ta + 128, r0);
          add32(acc, r1);
          tmem_ld32(ta + 192, r1);
          tmem_ld_wait_regs(r0);
          reg_fence(r1);
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&acc_empty[b]);  // every column of the K-tile is in registers
          add32(acc, r0);
          add32(acc, r1);
        } else {
          // exact sums of groups 4 u + j, filter m, positions pw + i
          int32_t* s0 = a.sums + ((int64_t)(mok ? m : 0) * g.ng + 4 * u) * g.P;
#pragma unroll
          for (int hh = 0; hh < 2; ++hh) {
            tmem_ld32(ta + 128 * hh, r0);
            tmem_ld32(ta + 128 * hh + 64, r1);
            tmem_ld_wait_regs(r0);
            reg_fence(r1);
            if (hh == 1) {
              tc_fence_before();
              __syncwarp();
              if (lane == 0) mbar_arrive(&acc_empty[b]);
            }
            if (mok) {
#pragma unroll
              for (int i = 0; i < 32; ++i) {
                const int64_t p = pw + i;
                if (p < g.P) {
                  s0[(2 * hh) * g.P + p] = __float2int_rn(__uint_as_float(r0[i]));
                  s0[(2 * hh + 1) * g.P + p] = __float2int_rn(__uint_as_float(r1[i]));
                }
              }
            }
          }
        }
      }
      if (!ok && !*abort_flag) fail();
      if (named_bar_or(BAR_EPI4, 32 * T4_EPI_WARPS, !ok)) break;
      if (!FOLD) continue;  // the group sums are stored already
      const float sc_m = mok ? sx * __ldg(a.row_scale + m) : 0.0f;
      if (a.out_tma) {
        // two boxes of 32 positions, each written by the warps of its half, stored by one thread
#pragma unroll 1
        for (int hb = 0; hb < 2; ++hb) {
          if (leader) bulk_wait_read_all();  // the previous box has been read out
          named_bar_sync(BAR_EPI4, 32 * T4_EPI_WARPS);
          if (hsub == hb) {
#pragma unroll
            for (int i = 0; i < 32; ++i) otile[i * T4_BM + t] = sc_m * acc[i];
          }
          fence_proxy_async_smem();
          named_bar_sync(BAR_EPI4, 32 * T4_EPI_WARPS);
          if (leader) {  // a box that starts inside the output (its tail past P is not written)
            if (p0 + 32 * hb < g.P) tma_store_2d(&a.out_map, m0, (int)(p0 + 32 * hb), smem_u32(otile));
            bulk_commit();
          }
        }
      } else if (mok) {
        if (g.rq_out) {  // fused requantization: 8-bit codes instead of fp32
          const RqMul r = rq_mul(g.rq_scale, g.rq_signed);
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const int64_t p = pw + i;
            if (p < g.P) g.rq_out[p * g.M + m] = rq_code(sc_m * acc[i], r);
          }
        } else {
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const int64_t p = pw + i;
            if (p < g.P) a.out[p * g.M + m] = sc_m * acc[i];
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

template <int ABITS, bool SIGNED, bool TMAP, bool FOLD>
fgq_status launch_tc4(const T4Args& args, int grid, cudaStream_t s) {
  constexpr int smem = T4Cfg<FOLD>::SMEM;
  if (!tc::smem_attr_once<tc4_contract_kernel<ABITS, SIGNED, TMAP, FOLD>>(smem)) return FGQ_ERR_CUDA;
  tc4_contract_kernel<ABITS, SIGNED, TMAP, FOLD><<<grid, T4_THREADS, smem, s>>>(args);
  return after_launch();
}

template <int ABITS, bool SIGNED>
fgq_status launch_tc4_path(const T4Args& args, int grid, cudaStream_t s) {
  if (args.sums)
    return args.act_tma ? launch_tc4<ABITS, SIGNED, true, false>(args, grid, s)
                        : launch_tc4<ABITS, SIGNED, false, false>(args, grid, s);
  return args.act_tma ? launch_tc4<ABITS, SIGNED, true, true>(args, grid, s)
                      : launch_tc4<ABITS, SIGNED, false, true>(args, grid, s);
}

}  // namespace

fgq_status launch_expand_codes(const uint32_t* codes, int64_t nwords, void* a16, cudaStream_t s) {
  if (nwords <= 0) return FGQ_OK;
  expand_codes_kernel<<<(unsigned)((nwords + 255) / 256), 256, 0, s>>>(codes, nwords, static_cast<uint4*>(a16));
  return after_launch();
}

bool tc4_supports(const Geom& g) {
  if (g.G != 4) return false;
  if (g.Cg % T4_KT != 0) return false;        // every K-tile inside one filter tap (conv) or row (GEMM)
  if (g.C % 16 != 0) return false;            // 16-byte aligned activation rows
  if (g.P >= (int64_t)1 << 31) return false;  // positions decoded in 32 bits
  if (encode_tiled() == nullptr) return false;
  return true;
}

fgq_status launch_tc4_contract(const void* act, const Geom& g, const uint32_t* codes, const float* alpha,
                               const float* act_scale, float* out, int32_t* sums, unsigned int* err,
                               cudaStream_t s) {
  if (!tc4_supports(g)) return FGQ_ERR_UNSUPPORTED;
  T4Args a;
  memset(&a, 0, sizeof a);
  a.act = static_cast<const uint8_t*>(act);
  a.act_scale = act_scale;
  a.out = out;
  a.sums = sums;
  a.err = err;
  a.g = g;
  a.mtiles = (g.Mg + T4_BM - 1) / T4_BM;
  a.ptiles = (int)((g.P + T4_BP - 1) / T4_BP);
  a.ntiles = g.groups * a.mtiles * a.ptiles;
  a.ktiles = g.Kp / T4_KT;
  // a test may shorten the waits (debug_wait_limit_us), never the final drains
  const int64_t lim_us = debug_wait_limit_us();
  a.timeout_ns = lim_us < 0 ? T4_TIMEOUT_NS : (uint64_t)lim_us * 1000u;
  const int abits = (g.act_type == FGQ_U4 || g.act_type == FGQ_S4) ? 4 : 8;
  const bool fold = sums == nullptr;

  // the ternary operand, fp16 [M][Kp] (Kp = 16 wrow) per part, and (folded) the row scales,
  // in one temporary from the stream-ordered pool
  cudaMemPool_t pool = scratch_pool();
  if (!pool) return FGQ_ERR_CUDA;
  const size_t part_bytes = (size_t)g.M * g.wrow * 32;
  const int nparts = fold ? 2 : 1;
  void* tmp = nullptr;
  if (cudaMallocFromPoolAsync(&tmp, nparts * part_bytes + (fold ? (size_t)g.M * 4 : 0), pool, s) != cudaSuccess)
    return FGQ_ERR_CUDA;
  uint8_t* parts = static_cast<uint8_t*>(tmp);
  fgq_status st;
  if (fold) {
    float* rs = reinterpret_cast<float*>(parts + 2 * part_bytes);
    a.row_scale = rs;
    st = launch_fold_alpha_split(codes, g.M, g.wrow, g.G, g.ng, alpha, parts, parts + part_bytes, rs, s);
  } else {
    st = launch_expand_codes(codes, (int64_t)g.M * g.wrow, parts, s);
  }
  for (int part = 0; st == FGQ_OK && part < nparts; ++part)
    if (!make_map_2d(&a.a_map[part], CU_TENSOR_MAP_DATA_TYPE_FLOAT16, parts + part * part_bytes,
                     (uint64_t)g.wrow * 16, (uint64_t)g.M, (uint64_t)g.wrow * 32, T4_KT, T4_BM,
                     CU_TENSOR_MAP_SWIZZLE_128B))
      st = FGQ_ERR_CUDA;
  if (st == FGQ_OK && g.R == 1 && g.S == 1 && g.stride == 1 && g.pad == 0) {
    const uint64_t row_bytes = (uint64_t)g.C * abits / 8;
    a.act_tma = make_map_2d(&a.act_map, CU_TENSOR_MAP_DATA_TYPE_UINT8, act, row_bytes, (uint64_t)g.B * g.H * g.W,
                            row_bytes, (uint32_t)(T4_KT * abits / 8), T4_BP,
                            abits == 8 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_32B)
                    ? 1
                    : 0;
  }
  if (st == FGQ_OK && fold && g.groups == 1 && g.M % 4 == 0 && !g.rq_out) {
    a.out_tma = make_map_2d(&a.out_map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, out, (uint64_t)g.M, (uint64_t)g.P,
                            (uint64_t)g.M * 4, T4_BM, 32, CU_TENSOR_MAP_SWIZZLE_NONE)
                    ? 1
                    : 0;
  }
  if (st == FGQ_OK) {
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int grid = a.ntiles < sms ? a.ntiles : sms;
    const bool sgn = g.act_type == FGQ_S8 || g.act_type == FGQ_S4;
    if (abits == 4)
      st = sgn ? launch_tc4_path<4, true>(a, grid, s) : launch_tc4_path<4, false>(a, grid, s);
    else
      st = sgn ? launch_tc4_path<8, true>(a, grid, s) : launch_tc4_path<8, false>(a, grid, s);
  }
  // the temporary returns to the pool once the work queued on s before this point is done
  if (cudaFreeAsync(tmp, s) != cudaSuccess && st == FGQ_OK) st = FGQ_ERR_CUDA;
  return st;
}

}  // namespace fgq
