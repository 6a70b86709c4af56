// Tensor-core (tcgen05) grouped ternary contraction for G = 4.
//
// Math (Eq. 2, 32-bit group accumulators of Section 4): y[p][m] = s_x * sum_g alpha[m][g]
// * s[m][g][p] with s an exact integer sum over a group of 4 reduction elements.  A dense
// MMA would sum across groups, so each K = 16 MMA step (4 groups) uses a block-diagonal
// activation operand B': its 128 rows are (group slot j = 0..3, position p = 0..31), and
// row (j, p) holds the activations of position p only in the 4 columns of group slot j
// (zeros elsewhere).  Then D[m][32 j + p] = s[m][group 4 step + j][p] exactly (fp16
// operands on exact integers, |s| <= 4 * 255), each step into its own TMEM buffer, and the
// epilogue applies alpha once per group-output on the CUDA cores (Section 4.1).  The zeros
// of B' never change, so they are written once per CTA; each K-tile only writes the
// diagonal 8-byte pieces.
//
// Tile: 128 filters x 32 positions; K-tile 64 (16 groups, 4 MMA steps).
// Warp roles (416 threads, one CTA per SM, persistent over tiles):
//   warps 0-7  epilogue: warp w reads TMEM lanes 32*(w%4).. (filters) and the 64 columns
//              of group slots 2*(w/4), 2*(w/4)+1 of each step's buffer; 64 FMAs per step
//              with two alphas into 32 position accumulators; the two halves are summed
//              through shared memory at tile end and stored (TMA box store when possible).
//   warps 8-11 loaders/converters: thread t fills code row t of A (TMA box or cp.async)
//              and B' row t = (slot t/32, position t%32): 4 pieces of 4 activations.
//   warp 12    TMEM allocation and the MMA issuer: 4 tcgen05.mma (M = N = 128, K = 16)
//              per K-tile, one per TMEM buffer.
// Every mbarrier wait is bounded; on expiry the kernel records FGQ_ERR_TIMEOUT, each role
// leaves its loop (uniformly within the epilogue, which uses named barriers), in-flight
// copies and MMAs are waited for, and TMEM is freed.
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

constexpr int T4_BM = 128;       // filters per tile (MMA M, TMEM lanes)
constexpr int T4_BP = 32;        // positions per tile
constexpr int T4_KT = 64;        // reduction elements per K-tile: 16 groups, 4 MMA steps
constexpr int T4_NO = 3;         // operand ring depth
constexpr int T4_NS_TMA = 6;     // staging ring depth, TMA path
constexpr int T4_NS_GATHER = 10; // staging ring depth, gather path
constexpr int T4_NACC = 4;       // TMEM accumulator buffers, one per MMA step
constexpr int T4_EPI_WARPS = 8;
constexpr int T4_LOAD_WARP0 = 8;  // loaders: warps 8-11
constexpr int T4_MMA_WARP = 12;
constexpr int T4_THREADS = 32 * (T4_MMA_WARP + 1);
constexpr int T4_TMEM_COLS = T4_NACC * 128;
constexpr uint32_t T4_WAIT_LIMIT = 50000;  // polls of up to 20 us: about 1 s per wait
constexpr uint32_t BAR_EPI4 = 2;

constexpr int OP_TILE4 = 128 * T4_KT * 2;     // 16 KB fp16 operand tile (A or B')
constexpr int OP_STAGE4 = 2 * OP_TILE4;
constexpr int ST_ACT4 = 128 * T4_KT;          // 8 KB: one 64-byte raw row per loader thread
constexpr int ST_CODE4 = 128 * 16;            // 2 KB raw code words
constexpr int ST_STAGE4 = ST_ACT4 + ST_CODE4;
constexpr int OUT_TILE4 = T4_BP * T4_BM * 4;  // 16 KB fp32 [32 positions][128 filters]
constexpr int SMEM_OP4 = T4_NO * OP_STAGE4;
constexpr int SMEM_ST4 = T4_NS_GATHER * ST_STAGE4;
constexpr int SMEM_LUT4 = 16 * 32 * 4;
constexpr int SMEM_BAR4 = 8 * (2 * T4_NO + 2 * T4_NS_GATHER + 2 * T4_NACC + 1) + 16;
constexpr int T4_SMEM = 1024 + SMEM_OP4 + SMEM_ST4 + OUT_TILE4 + SMEM_LUT4 + SMEM_BAR4;

struct T4Args {
  CUtensorMap codes_map;  // uint32 [M][wrow], box {4 words, 128 rows}
  CUtensorMap act_map;    // uint8 [pixels][row bytes], box {64 (or 32) bytes, 32 rows}; TMA path
  CUtensorMap out_map;    // fp32 [P][M], box {128 filters, 32 positions}; if out_tma
  const uint8_t* act;
  const uint32_t* codes;
  const float* alpha;
  const float* act_scale;
  float* out;
  unsigned int* err;
  Geom g;
  int mtiles, ptiles, ntiles, ktiles;
  int act_tma, out_tma;
  uint32_t wait_limit;
};

__device__ __forceinline__ void tile_coords4(const T4Args& a, int tile, int& gi, int& m0, int64_t& p0) {
  const int per_p = a.g.groups * a.mtiles;
  const int pt = tile / per_p;
  const int r = tile - pt * per_p;
  gi = r / a.mtiles;
  m0 = gi * a.g.Mg + (r - gi * a.mtiles) * T4_BM;
  p0 = (int64_t)pt * T4_BP;
}

template <int ABITS, bool SIGNED, bool TMAP>
__global__ void __launch_bounds__(T4_THREADS, 1) tc4_contract_kernel(const __grid_constant__ T4Args a) {
  constexpr int NS = TMAP ? T4_NS_TMA : T4_NS_GATHER;
  extern __shared__ uint8_t smem_raw4[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw4) + 1023) & ~uintptr_t(1023));
  uint8_t* op = smem;
  uint8_t* st = smem + SMEM_OP4;
  float* otile = reinterpret_cast<float*>(smem + SMEM_OP4 + SMEM_ST4);
  uint32_t* lut = reinterpret_cast<uint32_t*>(smem + SMEM_OP4 + SMEM_ST4 + OUT_TILE4);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + SMEM_OP4 + SMEM_ST4 + OUT_TILE4 + SMEM_LUT4);
  uint64_t* op_full = bars;
  uint64_t* op_empty = bars + T4_NO;
  uint64_t* st_full = bars + 2 * T4_NO;
  uint64_t* st_empty = st_full + NS;
  uint64_t* acc_full = st_empty + NS;
  uint64_t* acc_empty = acc_full + T4_NACC;
  uint64_t* drain_bar = acc_empty + T4_NACC;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_bar + 1);
  volatile uint32_t* abort_flag = tmem_slot + 1;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const Geom& g = a.g;

  if (threadIdx.x == 0) {
    for (int i = 0; i < T4_NO; ++i) {
      mbar_init(&op_full[i], 128);
      mbar_init(&op_empty[i], 1);
    }
    for (int i = 0; i < NS; ++i) {
      mbar_init(&st_full[i], 1);
      mbar_init(&st_empty[i], 128);
    }
    for (int i = 0; i < T4_NACC; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], 32 * T4_EPI_WARPS);
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  tc::fill_code_lut(lut);
  // the off-diagonal zeros of every B' tile, written once
  for (int s = 0; s < T4_NO; ++s) {
    uint4* bt = reinterpret_cast<uint4*>(op + s * OP_STAGE4 + OP_TILE4);
    for (int i = threadIdx.x; i < OP_TILE4 / 16; i += blockDim.x) bt[i] = make_uint4(0u, 0u, 0u, 0u);
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
    const int slotj = t >> 5;   // group slot of B' row t
    const int pl = t & 31;      // position of B' row t within the tile
    const int total = my_tiles * a.ktiles;
    constexpr int ROW_BYTES = T4_KT * ABITS / 8;
    constexpr int CPR = ROW_BYTES / 16;
    constexpr uint32_t TX_CODES = 128 * 16;
    constexpr uint32_t TX_ACT = T4_BP * ROW_BYTES;

    int cur_tile = -1, gi = 0, m0 = 0, tr = 0, ts = 0, tc0 = 0;
    int64_t p0 = 0;
    int pb = 0, phb = 0, pwb = 0;
    bool pvalid = false;
    int issued = 0;
    auto issue = [&](int j) {
      const int tl = j / a.ktiles;
      if (tl != cur_tile) {
        cur_tile = tl;
        tile_coords4(a, (int)blockIdx.x + tl * (int)gridDim.x, gi, m0, p0);
        tr = ts = tc0 = 0;
        const int64_t p = p0 + pl;
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
      const int kk = j - tl * a.ktiles;
      if (TMAP) {
        if (t == 0) {
          bool free_ok = true;
          if (j >= NS) free_ok = mbar_wait_or_abort(&st_empty[slot], ((j / NS) & 1) ^ 1, a.wait_limit, abort_flag);
          if (free_ok) {
            mbar_arrive_expect_tx(&st_full[slot], TX_CODES + TX_ACT);
            tma_load_2d(smem_u32(sa + ST_ACT4), &a.codes_map, kk * (T4_KT / 16), m0, &st_full[slot]);
            tma_load_2d(smem_u32(sa), &a.act_map, (gi * g.Cg + tc0) * ABITS / 8, (int)p0, &st_full[slot]);
            issued = j + 1;
          } else if (!*abort_flag) {
            fail();
          }
        }
      } else {
        // own copies: the full activation row of position pl into staging row t, code row t
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
        for (int c = 0; c < CPR; ++c)
          cp_async16(smem_u32(sa + st_off<ABITS>(t, c)), inside ? (const void*)(src + 16 * c) : (const void*)a.act,
                     inside ? 16u : 0u);
        const int m = m0 + t;
        const bool mok = m < gi * g.Mg + g.Mg && m < g.M;
        const uint32_t* csrc = mok ? a.codes + (int64_t)m * g.wrow + kk * (T4_KT / 16) : a.codes;
        cp_async16(smem_u32(sa + ST_ACT4 + t * 16), csrc, mok ? 16u : 0u);
      }
      tc0 += T4_KT;
      if (tc0 == g.Cg) {
        tc0 = 0;
        if (++ts == g.S) {
          ts = 0;
          ++tr;
        }
      }
    };

    for (int j = 0; j < NS - 1; ++j) {
      if (j < total) issue(j);
      cp_async_commit();
    }
    int consumed = 0;
    const int srow = TMAP ? pl : t;  // staging row holding this thread's position
    for (int j = 0; j < total; ++j) {
      if (*abort_flag) break;
      if (j + NS - 1 < total) issue(j + NS - 1);
      cp_async_commit();
      if (!TMAP) cp_async_wait<NS - 1>();
      const int slot = j % NS;
      const int os = j % T4_NO;
      if ((TMAP && !mbar_wait_or_abort(&st_full[slot], (j / NS) & 1, a.wait_limit, abort_flag)) ||
          !mbar_wait_or_abort(&op_empty[os], ((j / T4_NO) & 1) ^ 1, a.wait_limit, abort_flag)) {
        if (!*abort_flag) fail();
        break;
      }
      consumed = j + 1;
      const uint8_t* sa = st + slot * ST_STAGE4;
      uint8_t* A = op + os * OP_STAGE4;
      uint8_t* Bt = A + OP_TILE4;
      tc::codes_row_to_fp16(sa + ST_ACT4 + t * 16, A, t, lut + lane);
      // B' row t: for each MMA step s the 4 activations of group slot slotj (K offsets
      // 16 s + 4 slotj .. +3) as 4 fp16 at the same K offsets of the row
#pragma unroll
      for (int s = 0; s < 4; ++s) {
        uint32_t w;
        if (ABITS == 8) {
          w = *reinterpret_cast<const uint32_t*>(sa + st_off<8>(srow, s) + 4 * slotj);
          if (SIGNED) w ^= 0x80808080u;
        } else {
          // 4 nibbles at byte offset 8 s + 2 slotj of the 32-byte row
          const uint32_t hword = *reinterpret_cast<const uint16_t*>(sa + st_off<4>(srow, s >> 1) + 8 * (s & 1) + 2 * slotj);
          w = (hword & 0xfu) | ((hword & 0xf0u) << 4) | ((hword & 0xf00u) << 8) | ((hword & 0xf000u) << 12);
          if (SIGNED) w ^= 0x08080808u;
        }
        const uint32_t bias2 = ABITS == 8 ? (SIGNED ? 0x64806480u : 0x64006400u) : (SIGNED ? 0x64086408u : 0x64006400u);
        const uint2 hv = make_uint2(u8pair_to_h2(w, 0x4140, bias2), u8pair_to_h2(w, 0x4342, bias2));
        *reinterpret_cast<uint2*>(Bt + sw128(t, 2 * s + (slotj >> 1)) + 8 * (slotj & 1)) = hv;
      }
      fence_proxy_async_smem();
      mbar_arrive(&op_full[os]);
      if (TMAP) mbar_arrive(&st_empty[slot]);
    }
    cp_async_wait_all();
    if (t == 0) {
      for (int j = consumed; j < issued; ++j) mbar_wait_bounded(&st_full[j % NS], (j / NS) & 1, 1u << 16);
    }
  }

  // ------------------------------------------------------------------ MMA issuer
  if (warp == T4_MMA_WARP && lane == 0) {
    const uint32_t idesc = idesc_f16_f32(128, 128);
    const uint32_t op_base = smem_u32(op);
    const int total = my_tiles * a.ktiles;
    int sc = 0;
    bool ok = true;
    for (int j = 0; j < total && ok; ++j) {
      const int os = j % T4_NO;
      if (!mbar_wait_or_abort(&op_full[os], (j / T4_NO) & 1, a.wait_limit, abort_flag)) {
        if (!*abort_flag) fail();
        break;
      }
      tc_fence_after();
      const uint32_t abase = op_base + os * OP_STAGE4;
      const uint64_t ad = sdesc_k_sw128(abase);
      const uint64_t bd = sdesc_k_sw128(abase + OP_TILE4);
      for (int s = 0; s < 4; ++s, ++sc) {
        const int b = sc % T4_NACC;
        if (!mbar_wait_or_abort(&acc_empty[b], ((sc / T4_NACC) & 1) ^ 1, a.wait_limit, abort_flag)) {
          if (!*abort_flag) fail();
          ok = false;
          break;
        }
        tc_fence_after();
        mma_f16(tmem + (uint32_t)(b * 128), ad + 2 * s, bd + 2 * s, idesc, 0u);
        mma_commit(&acc_full[b]);
      }
      mma_commit(&op_empty[os]);
    }
    mma_commit(drain_bar);
    mbar_wait_bounded(drain_bar, 0, a.wait_limit);
  }

  // ------------------------------------------------------------------ epilogue
  if (warp < T4_EPI_WARPS) {
    const int quarter = warp & 3, half = warp >> 2;
    const int t = 32 * quarter + lane;  // TMEM lane = filter row of the tile
    const uint32_t tbase = tmem + ((uint32_t)(32 * quarter) << 16) + (uint32_t)(64 * half);
    const float sx = __ldg(a.act_scale);
    const bool leader = threadIdx.x == 0;
    int sc = 0;
    bool ok = true;
    for (int tl = 0; tl < my_tiles; ++tl) {
      int gi, m0;
      int64_t p0;
      tile_coords4(a, (int)blockIdx.x + tl * (int)gridDim.x, gi, m0, p0);
      const int m = m0 + t;
      const bool mok = m < gi * g.Mg + g.Mg && m < g.M;
      const float* arow = a.alpha + (int64_t)(mok ? m : 0) * g.ng;
      float acc[32];
#pragma unroll
      for (int j = 0; j < 32; ++j) acc[j] = 0.0f;
      // alphas of step s of K-tile kk: groups 16 kk + 4 s + 2 half + {0, 1}
      float2 al_next = mok ? make_float2(__ldg(arow + 2 * half), __ldg(arow + 2 * half + 1)) : make_float2(0.f, 0.f);
      const int nsteps = a.ktiles * 4;
      for (int st4 = 0; st4 < nsteps; ++st4, ++sc) {
        if (!ok) continue;
        const int b = sc % T4_NACC;
        const float2 al = al_next;
        const int gn = 4 * (st4 + 1) + 2 * half;
        if (mok && st4 + 1 < nsteps) al_next = make_float2(__ldg(arow + gn), __ldg(arow + gn + 1));
        if (!mbar_wait_or_abort(&acc_full[b], (sc / T4_NACC) & 1, a.wait_limit, abort_flag)) {
          if (!*abort_flag) fail();
          ok = false;
          continue;
        }
        tc_fence_after();
        uint32_t r0[32], r1[32];
        tmem_ld32(tbase + (uint32_t)(b * 128), r0);
        tmem_ld32(tbase + (uint32_t)(b * 128 + 32), r1);
        tmem_ld_wait();
        tc_fence_before();
        mbar_arrive(&acc_empty[b]);
#pragma unroll
        for (int j = 0; j < 32; ++j)
          acc[j] = fmaf(al.y, __uint_as_float(r1[j]), fmaf(al.x, __uint_as_float(r0[j]), acc[j]));
      }
      if (named_bar_or(BAR_EPI4, 32 * T4_EPI_WARPS, !ok)) break;
      // sum the two halves' partials through the tile buffer
      if (leader && a.out_tma) bulk_wait_read_all();  // previous tile's store has read the buffer
      named_bar_sync(BAR_EPI4, 32 * T4_EPI_WARPS);
      if (half == 1) {
#pragma unroll
        for (int j = 0; j < 32; ++j) otile[j * T4_BM + t] = acc[j];
      }
      named_bar_sync(BAR_EPI4, 32 * T4_EPI_WARPS);
      if (half == 0) {
        if (a.out_tma) {
#pragma unroll
          for (int j = 0; j < 32; ++j) otile[j * T4_BM + t] = sx * (acc[j] + otile[j * T4_BM + t]);
          fence_proxy_async_smem();
        } else if (mok) {
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            const int64_t p = p0 + j;
            if (p < g.P) a.out[p * g.M + m] = sx * (acc[j] + otile[j * T4_BM + t]);
          }
        }
      }
      named_bar_sync(BAR_EPI4, 32 * T4_EPI_WARPS);
      if (leader && a.out_tma) {
        tma_store_2d(&a.out_map, m0, (int)p0, smem_u32(otile));
        bulk_commit();
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

template <int ABITS, bool SIGNED, bool TMAP>
fgq_status launch_tc4(const T4Args& args, int grid, cudaStream_t s) {
  static bool attr_set = false;
  if (!attr_set) {
    if (cudaFuncSetAttribute(tc4_contract_kernel<ABITS, SIGNED, TMAP>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             T4_SMEM) != cudaSuccess)
      return FGQ_ERR_CUDA;
    attr_set = true;
  }
  tc4_contract_kernel<ABITS, SIGNED, TMAP><<<grid, T4_THREADS, T4_SMEM, s>>>(args);
  return after_launch();
}

template <int ABITS, bool SIGNED>
fgq_status launch_tc4_path(const T4Args& args, int grid, cudaStream_t s) {
  return args.act_tma ? launch_tc4<ABITS, SIGNED, true>(args, grid, s) : launch_tc4<ABITS, SIGNED, false>(args, grid, s);
}

}  // namespace

bool tc4_supports(const Geom& g) {
  if (g.G != 4) return false;
  if (g.Cg % T4_KT != 0) return false;        // every K-tile inside one filter tap (conv) or row (GEMM)
  if (g.C % 16 != 0) return false;            // 16-byte aligned activation rows
  if (g.P >= (int64_t)1 << 31) return false;  // positions decoded in 32 bits
  if (encode_tiled() == nullptr) return false;
  return true;
}

fgq_status launch_tc4_contract(const void* act, const Geom& g, const uint32_t* codes, const float* alpha,
                               const float* act_scale, float* out, unsigned int* err, cudaStream_t s) {
  if (!tc4_supports(g)) return FGQ_ERR_UNSUPPORTED;
  T4Args a;
  memset(&a, 0, sizeof a);
  a.act = static_cast<const uint8_t*>(act);
  a.codes = codes;
  a.alpha = alpha;
  a.act_scale = act_scale;
  a.out = out;
  a.err = err;
  a.g = g;
  a.mtiles = (g.Mg + T4_BM - 1) / T4_BM;
  a.ptiles = (int)((g.P + T4_BP - 1) / T4_BP);
  a.ntiles = g.groups * a.mtiles * a.ptiles;
  a.ktiles = g.Kp / T4_KT;
  a.wait_limit = T4_WAIT_LIMIT;
  const int abits = (g.act_type == FGQ_U4 || g.act_type == FGQ_S4) ? 4 : 8;
  if (!make_map_2d(&a.codes_map, CU_TENSOR_MAP_DATA_TYPE_UINT32, codes, (uint64_t)g.wrow, (uint64_t)g.M,
                   (uint64_t)g.wrow * 4, T4_KT / 16, T4_BM, CU_TENSOR_MAP_SWIZZLE_NONE))
    return FGQ_ERR_CUDA;
  if (g.R == 1 && g.S == 1 && g.stride == 1 && g.pad == 0) {
    const uint64_t row_bytes = (uint64_t)g.C * abits / 8;
    a.act_tma = make_map_2d(&a.act_map, CU_TENSOR_MAP_DATA_TYPE_UINT8, act, row_bytes, (uint64_t)g.B * g.H * g.W,
                            row_bytes, (uint32_t)(T4_KT * abits / 8), T4_BP,
                            abits == 8 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_32B)
                    ? 1
                    : 0;
  }
  if (g.groups == 1 && g.M % 4 == 0) {
    a.out_tma = make_map_2d(&a.out_map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, out, (uint64_t)g.M, (uint64_t)g.P,
                            (uint64_t)g.M * 4, T4_BM, T4_BP, CU_TENSOR_MAP_SWIZZLE_NONE)
                    ? 1
                    : 0;
  }
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int grid = a.ntiles < sms ? a.ntiles : sms;
  const bool sgn = g.act_type == FGQ_S8 || g.act_type == FGQ_S4;
  if (abits == 4) return sgn ? launch_tc4_path<4, true>(a, grid, s) : launch_tc4_path<4, false>(a, grid, s);
  return sgn ? launch_tc4_path<8, true>(a, grid, s) : launch_tc4_path<8, false>(a, grid, s);
}

}  // namespace fgq
