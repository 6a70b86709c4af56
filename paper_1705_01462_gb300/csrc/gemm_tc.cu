// Tensor-core (tcgen05) grouped ternary contraction for G in {64, 128}, and the
// bounded-wait self test.
//
// Math (Eq. 2 with the 32-bit group accumulators of Section 4): per output filter m,
// position p and group g of G consecutive reduction elements, s[m][g][p] is an exact
// integer; y[p][m] = s_x * sum_g alpha[m][g] * s[m][g][p].  sm_103a has no integer
// tcgen05 MMA, so the group sums run as fp16 MMAs on exact integers: codes {-1, 0, +1}
// and 8-bit (or 4-bit) activations are exact in fp16, products are exact, and a group's
// fp32 accumulation stays an exact integer (|s| <= 128 * 255 < 2^24).  The K-tile of the
// MMA chain is 64 and aligned to the group, so after a group's MMAs the TMEM accumulator
// holds exactly s[m][g][p] for a 128-filter x 128-position tile; the epilogue multiplies
// it by alpha[m][g] and adds it into an fp32 register accumulator (one multiply per group,
// Section 4.1).  Four TMEM buffers let the MMAs of later groups run while a group drains.
// The group-sums variant (SUMS) stores each drained accumulator as the int32 s[m][g][p]
// instead (the exact integers themselves, for verification).
//
// Warp roles (480 threads, one CTA per SM, persistent over tiles):
//   warps 0-7  epilogue: warp w reads TMEM lanes 32*(w%4).. (filter rows) and columns
//              64*(w/4).. (positions) of the drained buffer: two 32-column tcgen05.ld per
//              group, release of the buffer, FMAs with alpha into fp32 registers.  At tile end
//              the fp32 tile goes to shared memory and one thread writes it to HBM with a TMA
//              box store (direct stores when the output has several conv groups, M % 4 != 0,
//              or the output is requantized).
//   warps 8-11 converters: thread t converts tile row t (one output position, 64 reduction
//              elements) of a staged K-tile to fp16 in the 128-byte-swizzled K-major layout
//              the MMA reads.
//   warp 12    TMEM allocation and the MMA issuer (one thread): 4 tcgen05.mma (K = 16)
//              per K-tile into one of four 128-column TMEM accumulators.
//   warp 13    streams the ternary operand: the codes are expanded to fp16 {0, +1, -1} once
//              per call (a stream-ordered temporary) and reach a four-stage ring of their own
//              by TMA in the MMA's swizzled layout, ahead of the K-tiles that use them.
//   warp 14    streams the activations: one TMA load per K-tile into a six-slot staging ring,
//              a 2D box of 128 consecutive input rows when the im2col rows are input rows
//              (1x1 stride-1 convolutions, GEMMs), otherwise an im2col box (the 128 output
//              positions' pixels at the K-tile's filter tap, zeros in the padding).
// The operand stages are released by the epilogue: the group's accumulator commit (one per
// group) is seen by epilogue thread 0, which frees the group's A and B stages, so no commit
// is spent on them.
// Every mbarrier wait is bounded; on expiry the kernel records FGQ_ERR_TIMEOUT, each role
// leaves its loop (uniformly within a role that uses named barriers), in-flight copies
// and MMAs are waited for, and TMEM is freed.
#include <cstdint>
#include <cstring>

#include "tc_common.cuh"

namespace fgq {
namespace {

using tc::encode_im2col;
using tc::encode_tiled;
using tc::im2col_fits;
using tc::make_map_2d;
using tc::make_map_im2col;
using tc::st_off;
using tc::sw128;
using tc::u8pair_to_h2;

constexpr int TC_BM = 128;        // filters per tile (MMA M, TMEM lanes)
constexpr int TC_BN = 128;        // positions per tile (MMA N)
constexpr int TC_KT = 64;         // reduction elements per K-tile
constexpr int TC_NO = 3;          // activation operand (B) ring depth
constexpr int TC_NAS = 4;         // ternary operand (A) ring depth
constexpr int TC_NS = 6;          // activation staging ring depth
constexpr int TC_NACC = 4;        // TMEM accumulator buffers
constexpr int TC_EPI_WARPS = 8;
constexpr int TC_LOAD_WARPS = 4;
constexpr int TC_LOADERS = 32 * TC_LOAD_WARPS;  // converter threads: one per tile row
static_assert(TC_LOADERS == TC_BN, "one converter thread per tile row");
constexpr int TC_LOAD_WARP0 = TC_EPI_WARPS;      // converters: warps 8 .. 8 + TC_LOAD_WARPS - 1
constexpr int TC_MMA_WARP = TC_EPI_WARPS + TC_LOAD_WARPS;  // warp 12
constexpr int TC_A_WARP = TC_MMA_WARP + 1;                 // warp 13: lane 0 streams the A boxes
constexpr int TC_ACT_WARP = TC_A_WARP + 1;                 // warp 14: lane 0 streams the activation boxes
constexpr int TC_THREADS = 32 * (TC_ACT_WARP + 1);
constexpr int TC_TMEM_COLS = TC_NACC * TC_BN;    // 512: all of TMEM
constexpr uint32_t TC_WAIT_LIMIT = 50000;        // polls of up to 20 us: about 1 s per wait
constexpr uint32_t TC_WAIT_SLEEP_NS = 20000;     // suspend hint of one poll
constexpr uint32_t TC_DRAIN_LIMIT = 1u << 20;    // polls of the final drains (never shortened)
constexpr uint32_t BAR_EPI = 2;                  // named barrier of the 256 epilogue threads

constexpr int OP_TILE = TC_BM * TC_KT * 2;            // 16 KB: one fp16 operand tile
constexpr int ST_STAGE = TC_BN * TC_KT;                // 8 KB raw activation bytes (8-bit)
constexpr int OUT_TILE = TC_BN * TC_BM * 4;            // 64 KB fp32 output tile
constexpr int SMEM_A = TC_NAS * OP_TILE;
constexpr int SMEM_B = TC_NO * OP_TILE;
constexpr int SMEM_BAR = 8 * (2 * TC_NAS + 2 * TC_NO + 2 * TC_NS + 2 * TC_NACC + 1) + 16;
constexpr int SMEM_MID = TC_NS * ST_STAGE + OUT_TILE;  // staging ring + fp32 output tile
constexpr int TC_SMEM = 1024 + SMEM_A + SMEM_B + SMEM_MID + SMEM_BAR;
static_assert(TC_SMEM <= 232448, "shared memory budget");

struct TcArgs {
  CUtensorMap a16_map;    // fp16 [M][Kp] expanded codes, box {64, 128 rows}, 128-byte swizzle
  CUtensorMap act_map;    // act_tma: 2D uint8 [pixels][row bytes], box {64 (or 32) bytes, 128 rows};
                          // otherwise the im2col map of the NHWC tensor, 128 pixels x 64 (32) bytes
  CUtensorMap out_map;    // fp32 [P][M], box {128 filters, 128 positions}; if out_tma
  const uint8_t* act;
  const float* alpha;
  const float* act_scale;
  float* out;
  int32_t* sums;    // SUMS: int32 group sums [M][ng][P]
  unsigned int* err;
  Geom g;
  int mtiles;       // filter tiles per conv group
  int ptiles;       // position tiles
  int ntiles;       // groups * mtiles * ptiles
  int ktiles;       // K-tiles per tile (= ng * G / 64)
  int kt_per_group; // G / 64
  int act_tma;      // 2D activation map (im2col rows are consecutive input rows); else im2col map
  int out_tma;      // output tile by TMA store (one conv group, M % 4 == 0)
  uint32_t wait_limit;     // polls per wait (each up to wait_sleep_ns)
  uint32_t wait_sleep_ns;
};

__device__ __forceinline__ void tile_coords(const TcArgs& a, int tile, int& gi, int& m0, int64_t& p0) {
  const int per_p = a.g.groups * a.mtiles;
  const int pt = tile / per_p;
  const int r = tile - pt * per_p;
  gi = r / a.mtiles;
  const int mt = r - gi * a.mtiles;
  m0 = gi * a.g.Mg + mt * TC_BM;
  p0 = (int64_t)pt * TC_BN;
}

// TMAP: the layer's im2col rows are contiguous input rows (2D box loads); otherwise the
// activation boxes come from an im2col map (one load per K-tile: 128 output positions at
// one filter tap and 64 channels, padding read as zeros).
template <int ABITS, bool SIGNED, bool TMAP, bool SUMS>
__global__ void __launch_bounds__(TC_THREADS, 1) tc_contract_kernel(const __grid_constant__ TcArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* abuf = smem;                             // TC_NAS A tiles
  uint8_t* bbuf = smem + SMEM_A;                    // TC_NO B tiles
  uint8_t* st = bbuf + SMEM_B;                      // TC_NS activation staging slots
  float* otile = reinterpret_cast<float*>(st + TC_NS * ST_STAGE);  // [128 positions][128 filters]
  uint64_t* bars = reinterpret_cast<uint64_t*>(st + SMEM_MID);
  uint64_t* a_full = bars;
  uint64_t* a_empty = bars + TC_NAS;
  uint64_t* op_full = bars + 2 * TC_NAS;
  uint64_t* op_empty = op_full + TC_NO;
  uint64_t* st_full = op_empty + TC_NO;
  uint64_t* st_empty = st_full + TC_NS;
  uint64_t* acc_full = st_empty + TC_NS;
  uint64_t* acc_empty = acc_full + TC_NACC;
  uint64_t* drain_bar = acc_empty + TC_NACC;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_bar + 1);
  volatile uint32_t* abort_flag = tmem_slot + 1;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const Geom& g = a.g;

  if (threadIdx.x == 0) {
    for (int i = 0; i < TC_NAS; ++i) {
      mbar_init(&a_full[i], 1);   // the A box's byte count
      mbar_init(&a_empty[i], 1);  // released by the epilogue (the group's MMAs completed)
    }
    for (int i = 0; i < TC_NO; ++i) {
      mbar_init(&op_full[i], TC_LOADERS);
      mbar_init(&op_empty[i], 1);  // released like a_empty
    }
    for (int i = 0; i < TC_NS; ++i) {
      mbar_init(&st_full[i], 1);
      mbar_init(&st_empty[i], TC_LOADERS);
    }
    for (int i = 0; i < TC_NACC; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], TC_EPI_WARPS);  // one arrival per epilogue warp
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == TC_MMA_WARP) {
    tmem_alloc(tmem_slot, TC_TMEM_COLS);
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

  // ------------------------------------------------------------------ activation boxes
  if (warp == TC_ACT_WARP && lane == 0) {
    const int total = my_tiles * a.ktiles;
    constexpr uint32_t TX_ACT = TC_BN * TC_KT * ABITS / 8;
    // per tile: conv group and first position; the filter tap (tr, ts) and channel offset
    // tc0 of the next K-tile advance incrementally
    int gi = 0, m0 = 0, tr = 0, ts = 0, tc0 = 0, kt = 0, tl = 0;
    int64_t p0 = 0;
    int n0 = 0, h0 = 0, w0 = 0;  // im2col: the tile's first window origin (input pixel coordinates)
    int issued = 0;
    bool ok = true;
    for (int j = 0; j < total; ++j) {
      if (kt == 0) {
        tile_coords(a, (int)blockIdx.x + tl * (int)gridDim.x, gi, m0, p0);
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
      const int slot = j % TC_NS;
      // the slot's previous contents (K-tile j - TC_NS) have been released by every converter
      if (j >= TC_NS &&
          !mbar_wait_or_abort(&st_empty[slot], ((j / TC_NS) & 1) ^ 1, a.wait_limit, abort_flag, a.wait_sleep_ns)) {
        ok = false;
        break;
      }
      uint8_t* sa = st + slot * ST_STAGE;
      const int cbyte = (gi * g.Cg + tc0) * ABITS / 8;  // a multiple of 32 bytes
      mbar_arrive_expect_tx(&st_full[slot], TX_ACT);
      if (TMAP)
        tma_load_2d(smem_u32(sa), &a.act_map, cbyte, (int)p0, &st_full[slot]);
      else
        tma_load_im2col_4d(smem_u32(sa), &a.act_map, cbyte, w0, h0, n0, (uint16_t)ts, (uint16_t)tr, &st_full[slot]);
      issued = j + 1;
      tc0 += TC_KT;
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
    // loads the converters may not have consumed: the last TC_NS issued, one per slot, each
    // the latest phase of its slot's barrier; none may outlive the CTA
    for (int j = issued - TC_NS < 0 ? 0 : issued - TC_NS; j < issued; ++j)
      mbar_wait_bounded(&st_full[j % TC_NS], (j / TC_NS) & 1, TC_DRAIN_LIMIT);
  }

  // ------------------------------------------------------------------ converters
  if (warp >= TC_LOAD_WARP0 && warp < TC_MMA_WARP) {
    const int tid = threadIdx.x - 32 * TC_LOAD_WARP0;
    const int t = tid & (TC_BN - 1);  // tile row converted by this thread
    const int total = my_tiles * a.ktiles;
    for (int j = 0; j < total; ++j) {
      if (*abort_flag) break;
      const int slot = j % TC_NS;
      const int os = j % TC_NO;
      if (!mbar_wait_or_abort(&st_full[slot], (j / TC_NS) & 1, a.wait_limit, abort_flag, a.wait_sleep_ns) ||
          !mbar_wait_or_abort(&op_empty[os], ((j / TC_NO) & 1) ^ 1, a.wait_limit, abort_flag, a.wait_sleep_ns)) {
        if (!*abort_flag) fail();
        break;
      }
      const uint8_t* sa = st + slot * ST_STAGE;
      uint8_t* Bt = bbuf + os * OP_TILE;
      // activations of row t -> fp16, 128-byte-swizzled K-major
      if (ABITS == 8) {
        const uint32_t bias2 = SIGNED ? 0x64806480u : 0x64006400u;  // 1152 or 1024 in both halves
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          uint4 v = *reinterpret_cast<const uint4*>(sa + st_off<8>(t, c));
          if (SIGNED) {
            v.x ^= 0x80808080u; v.y ^= 0x80808080u; v.z ^= 0x80808080u; v.w ^= 0x80808080u;
          }
          uint4 o0, o1;
          o0.x = u8pair_to_h2(v.x, 0x4140, bias2); o0.y = u8pair_to_h2(v.x, 0x4342, bias2);
          o0.z = u8pair_to_h2(v.y, 0x4140, bias2); o0.w = u8pair_to_h2(v.y, 0x4342, bias2);
          o1.x = u8pair_to_h2(v.z, 0x4140, bias2); o1.y = u8pair_to_h2(v.z, 0x4342, bias2);
          o1.z = u8pair_to_h2(v.w, 0x4140, bias2); o1.w = u8pair_to_h2(v.w, 0x4342, bias2);
          *reinterpret_cast<uint4*>(Bt + sw128(t, 2 * c)) = o0;
          *reinterpret_cast<uint4*>(Bt + sw128(t, 2 * c + 1)) = o1;
        }
      } else {
        const uint32_t bias2 = SIGNED ? 0x64086408u : 0x64006400u;  // 1032 or 1024
#pragma unroll
        for (int c = 0; c < 2; ++c) {
          const uint4 v = *reinterpret_cast<const uint4*>(sa + st_off<4>(t, c));
          const uint32_t w4[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            // 8 nibbles -> 8 bytes (element order preserved), then 8 fp16
            const uint32_t x = w4[q];
            const uint32_t lo = (x & 0x000f000fu) | ((x & 0x00f000f0u) << 4);                // e0 e1 e4 e5
            const uint32_t hi = ((x >> 8) & 0x000f000fu) | (((x >> 8) & 0x00f000f0u) << 4);  // e2 e3 e6 e7
            uint32_t b0 = (lo & 0xffffu) | ((hi & 0xffffu) << 16);                            // e0 e1 e2 e3
            uint32_t b1 = (lo >> 16) | (hi & 0xffff0000u);                                    // e4 e5 e6 e7
            if (SIGNED) {
              b0 ^= 0x08080808u;
              b1 ^= 0x08080808u;
            }
            uint4 o;
            o.x = u8pair_to_h2(b0, 0x4140, bias2); o.y = u8pair_to_h2(b0, 0x4342, bias2);
            o.z = u8pair_to_h2(b1, 0x4140, bias2); o.w = u8pair_to_h2(b1, 0x4342, bias2);
            *reinterpret_cast<uint4*>(Bt + sw128(t, 4 * c + q)) = o;
          }
        }
      }
      fence_proxy_async_smem();
      mbar_arrive(&op_full[os]);
      mbar_arrive(&st_empty[slot]);  // done reading this staging slot
    }
  }

  // ------------------------------------------------------------------ A boxes
  if (warp == TC_A_WARP && lane == 0) {
    const int total = my_tiles * a.ktiles;
    int armed = 0;
    bool ok = true;
    for (int j = 0; j < total; ++j) {
      const int as = j % TC_NAS;
      if (!mbar_wait_or_abort(&a_empty[as], ((j / TC_NAS) & 1) ^ 1, a.wait_limit, abort_flag, a.wait_sleep_ns)) {
        ok = false;
        break;
      }
      const int tl = j / a.ktiles;
      int gj, mj;
      int64_t pj;
      tile_coords(a, (int)blockIdx.x + tl * (int)gridDim.x, gj, mj, pj);
      mbar_arrive_expect_tx(&a_full[as], OP_TILE);
      tma_load_2d(smem_u32(abuf + as * OP_TILE), &a.a16_map, (j - tl * a.ktiles) * TC_KT, mj, &a_full[as]);
      armed = j + 1;
    }
    if (!ok && !*abort_flag) fail();
    // boxes the MMA issuer may not have consumed: the last TC_NAS armed ones, one per stage,
    // each the latest phase of its stage's barrier
    for (int j = armed - TC_NAS < 0 ? 0 : armed - TC_NAS; j < armed; ++j)
      mbar_wait_bounded(&a_full[j % TC_NAS], (j / TC_NAS) & 1, TC_DRAIN_LIMIT);
  }

  // ------------------------------------------------------------------ MMA issuer
  if (warp == TC_MMA_WARP && lane == 0) {
    const uint32_t idesc = idesc_f16_f32(TC_BM, TC_BN);
    int kt = 0, gc = 0;
    bool ok = true;
    for (int tl = 0; tl < my_tiles && ok; ++tl) {
      for (int grp = 0; grp < g.ng && ok; ++grp, ++gc) {
        const int b = gc % TC_NACC;
        if (!mbar_wait_or_abort(&acc_empty[b], ((gc / TC_NACC) & 1) ^ 1, a.wait_limit, abort_flag, a.wait_sleep_ns)) {
          if (!*abort_flag) fail();
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + (uint32_t)(b * TC_BN);
        for (int sub = 0; sub < a.kt_per_group; ++sub, ++kt) {
          const int os = kt % TC_NO, as = kt % TC_NAS;
          if (!mbar_wait_or_abort(&op_full[os], (kt / TC_NO) & 1, a.wait_limit, abort_flag, a.wait_sleep_ns) ||
              !mbar_wait_or_abort(&a_full[as], (kt / TC_NAS) & 1, a.wait_limit, abort_flag, a.wait_sleep_ns)) {
            if (!*abort_flag) fail();
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t ad = sdesc_k_sw128(smem_u32(abuf + as * OP_TILE));
          const uint64_t bd = sdesc_k_sw128(smem_u32(bbuf + os * OP_TILE));
#pragma unroll
          for (int k = 0; k < TC_KT / 16; ++k) {
            // advance 16 fp16 (32 bytes) along K inside the swizzled rows
            mma_f16(d, ad + 2 * k, bd + 2 * k, idesc, (sub > 0 || k > 0) ? 1u : 0u);
          }
        }
        if (ok) mma_commit(&acc_full[b]);
      }
    }
    // all MMAs issued by this thread are complete once the drain barrier flips
    mma_commit(drain_bar);
    mbar_wait_bounded(drain_bar, 0, TC_DRAIN_LIMIT);
  }

  // ------------------------------------------------------------------ epilogue
  if (warp < TC_EPI_WARPS) {
    const int quarter = warp & 3, half = warp >> 2;
    const int t = 32 * quarter + lane;  // TMEM lane = filter row of the tile
    const uint32_t tbase = tmem + ((uint32_t)(32 * quarter) << 16) + (uint32_t)(64 * half);
    const float sx = __ldg(a.act_scale);
    const bool leader = threadIdx.x == 0;
    int gc = 0;
    bool ok = true;
    for (int tl = 0; tl < my_tiles; ++tl) {
      int gi, m0;
      int64_t p0;
      tile_coords(a, (int)blockIdx.x + tl * (int)gridDim.x, gi, m0, p0);
      const int m = m0 + t;
      const bool mok = m < gi * g.Mg + g.Mg && m < g.M;
      const float* arow = a.alpha + (int64_t)(mok ? m : 0) * g.ng;
      float acc[64];
#pragma unroll
      for (int j = 0; j < 64; ++j) acc[j] = 0.0f;
      float al_next = mok ? __ldg(arow) : 0.0f;
      for (int grp = 0; grp < g.ng; ++grp, ++gc) {
        if (!ok) continue;  // after a failed wait: run out the tile, then leave with the others
        const int b = gc % TC_NACC;
        const float al = al_next;  // alpha of this group, loaded one group ahead
        if (mok && grp + 1 < g.ng) al_next = __ldg(arow + grp + 1);
        if (!mbar_wait_or_abort(&acc_full[b], (gc / TC_NACC) & 1, a.wait_limit, abort_flag, a.wait_sleep_ns)) {
          if (!*abort_flag) fail();
          ok = false;
          continue;
        }
        if (leader) {
          // the group's MMAs have completed: its K-tiles' A and B stages may be refilled
          for (int k = gc * a.kt_per_group; k < (gc + 1) * a.kt_per_group; ++k) {
            mbar_arrive(&a_empty[k % TC_NAS]);
            mbar_arrive(&op_empty[k % TC_NO]);
          }
        }
        tc_fence_after();
        uint32_t r[32];
        if (SUMS) {
          // the exact group sums of positions p0 + 64 half + j, filter m: s[m][grp][p]
          int32_t* srow = a.sums + ((int64_t)(mok ? m : 0) * g.ng + grp) * g.P;
          const int64_t pbase = p0 + 64 * half;
#pragma unroll
          for (int hh = 0; hh < 2; ++hh) {
            tmem_ld32(tbase + (uint32_t)(b * TC_BN + 32 * hh), r);
            tmem_ld_wait();
            if (hh == 1) {
              tc_fence_before();
              __syncwarp();
              if (lane == 0) mbar_arrive(&acc_empty[b]);
            }
            if (mok) {
#pragma unroll
              for (int j = 0; j < 32; ++j) {
                const int64_t p = pbase + 32 * hh + j;
                if (p < g.P) srow[p] = __float2int_rn(__uint_as_float(r[j]));
              }
            }
          }
          continue;
        }
        tmem_ld32(tbase + (uint32_t)(b * TC_BN), r);
        tmem_ld_wait();
#pragma unroll
        for (int j = 0; j < 32; ++j) acc[j] = fmaf(al, __uint_as_float(r[j]), acc[j]);
        tmem_ld32(tbase + (uint32_t)(b * TC_BN + 32), r);
        tmem_ld_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&acc_empty[b]);  // the buffer is free once the values are in registers
#pragma unroll
        for (int j = 0; j < 32; ++j) acc[32 + j] = fmaf(al, __uint_as_float(r[j]), acc[32 + j]);
      }
      if (named_bar_or(BAR_EPI, 32 * TC_EPI_WARPS, !ok)) break;  // leave together
      if (SUMS) continue;  // the group sums are stored already
      if (a.out_tma) {
        // the previous tile's store has finished reading the staging tile
        if (leader) bulk_wait_read_all();
        named_bar_sync(BAR_EPI, 32 * TC_EPI_WARPS);
        float* orow = otile + (64 * half) * TC_BM + t;
#pragma unroll
        for (int j = 0; j < 64; ++j) orow[j * TC_BM] = sx * acc[j];
        fence_proxy_async_smem();
        named_bar_sync(BAR_EPI, 32 * TC_EPI_WARPS);
        if (leader) {
          tma_store_2d(&a.out_map, m0, (int)p0, smem_u32(otile));
          bulk_commit();
        }
      } else if (mok) {
        const int64_t pbase = p0 + 64 * half;
        if (g.rq_out) {  // fused requantization: 8-bit codes instead of fp32
          const RqMul r = rq_mul(g.rq_scale, g.rq_signed);
#pragma unroll
          for (int j = 0; j < 64; ++j) {
            const int64_t p = pbase + j;
            if (p < g.P) g.rq_out[p * g.M + m] = rq_code(sx * acc[j], r);
          }
        } else {
#pragma unroll
          for (int j = 0; j < 64; ++j) {
            const int64_t p = pbase + j;
            if (p < g.P) a.out[p * g.M + m] = sx * acc[j];
          }
        }
      }
    }
    if (leader) bulk_wait_all();  // this thread's TMA stores are complete
  }

  tc_fence_before();
  __syncthreads();
  if (warp == TC_MMA_WARP) {
    tc_fence_after();
    tmem_dealloc(tmem, TC_TMEM_COLS);
  }
}

template <int ABITS, bool SIGNED, bool TMAP, bool SUMS>
fgq_status launch_tc(const TcArgs& args, int grid, cudaStream_t s) {
  if (!tc::smem_attr_once<tc_contract_kernel<ABITS, SIGNED, TMAP, SUMS>>(TC_SMEM)) return FGQ_ERR_CUDA;
  tc_contract_kernel<ABITS, SIGNED, TMAP, SUMS><<<grid, TC_THREADS, TC_SMEM, s>>>(args);
  return after_launch();
}

template <int ABITS, bool SIGNED>
fgq_status launch_tc_path(const TcArgs& args, int grid, cudaStream_t s) {
  if (args.sums)
    return args.act_tma ? launch_tc<ABITS, SIGNED, true, true>(args, grid, s)
                        : launch_tc<ABITS, SIGNED, false, true>(args, grid, s);
  return args.act_tma ? launch_tc<ABITS, SIGNED, true, false>(args, grid, s)
                      : launch_tc<ABITS, SIGNED, false, false>(args, grid, s);
}

// One block waits on an mbarrier that nothing arrives on; every wait is bounded, so the
// kernel always returns and records FGQ_ERR_TIMEOUT.
__global__ void wait_timeout_selftest_kernel(uint32_t max_iter, unsigned int* err) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_mbar_init();
  }
  __syncthreads();
  const bool ok = mbar_wait_bounded(&bar, 0, max_iter);
  if (!ok && threadIdx.x == 0) record_error(err, FGQ_ERR_TIMEOUT);
}

}  // namespace

bool tc_supports(const Geom& g) {
  if (g.G != 64 && g.G != 128) return false;
  if (g.Cg % TC_KT != 0) return false;        // every K-tile inside one filter tap (conv) or row (GEMM)
  if (g.C % 16 != 0) return false;            // 16-byte aligned activation rows
  if (g.P >= (int64_t)1 << 31) return false;  // positions decoded in 32 bits
  if (encode_tiled() == nullptr) return false;
  if (!(g.R == 1 && g.S == 1 && g.stride == 1 && g.pad == 0) &&
      (encode_im2col() == nullptr || !im2col_fits(g.R, g.S, g.stride, g.pad)))
    return false;
  return true;
}

fgq_status launch_tc_contract(const void* act, const Geom& g, const uint32_t* codes, const float* alpha,
                              const float* act_scale, float* out, int32_t* sums, unsigned int* err,
                              cudaStream_t s) {
  if (!tc_supports(g)) return FGQ_ERR_UNSUPPORTED;
  TcArgs a;
  memset(&a, 0, sizeof a);
  a.act = static_cast<const uint8_t*>(act);
  a.alpha = alpha;
  a.act_scale = act_scale;
  a.out = out;
  a.sums = sums;
  a.err = err;
  a.g = g;
  a.mtiles = (g.Mg + TC_BM - 1) / TC_BM;
  a.ptiles = (int)((g.P + TC_BN - 1) / TC_BN);
  a.ntiles = g.groups * a.mtiles * a.ptiles;
  a.kt_per_group = g.G / TC_KT;
  a.ktiles = g.ng * a.kt_per_group;
  // a test may shorten the waits (debug_wait_limit_us), never the final drains
  const int64_t lim_us = debug_wait_limit_us();
  a.wait_limit = lim_us < 0 ? TC_WAIT_LIMIT : (uint32_t)(lim_us / 20 + 1);
  a.wait_sleep_ns = lim_us < 0 ? TC_WAIT_SLEEP_NS : (uint32_t)(lim_us < 20 ? lim_us * 1000 : 20000);
  const int abits = (g.act_type == FGQ_U4 || g.act_type == FGQ_S4) ? 4 : 8;
  // expanded codes: fp16 [M][Kp] (Kp = 16 wrow), in a temporary from the stream-ordered pool
  cudaMemPool_t pool = scratch_pool();
  if (!pool) return FGQ_ERR_CUDA;
  const int64_t nwords = (int64_t)g.M * g.wrow;
  void* a16 = nullptr;
  if (cudaMallocFromPoolAsync(&a16, (size_t)nwords * 32, pool, s) != cudaSuccess) return FGQ_ERR_CUDA;
  fgq_status st = launch_expand_codes(codes, nwords, a16, s);
  if (st == FGQ_OK && !make_map_2d(&a.a16_map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, a16, (uint64_t)g.wrow * 16,
                                   (uint64_t)g.M, (uint64_t)g.wrow * 32, TC_KT, TC_BM, CU_TENSOR_MAP_SWIZZLE_128B))
    st = FGQ_ERR_CUDA;
  // im2col rows are consecutive input rows for a 1x1, stride-1, unpadded convolution or a GEMM
  const uint64_t row_bytes = (uint64_t)g.C * abits / 8;
  const CUtensorMapSwizzle act_sw = abits == 8 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_32B;
  bool act_ok;
  if (g.R == 1 && g.S == 1 && g.stride == 1 && g.pad == 0) {
    a.act_tma = 1;
    act_ok = make_map_2d(&a.act_map, CU_TENSOR_MAP_DATA_TYPE_UINT8, act, row_bytes, (uint64_t)g.B * g.H * g.W,
                         row_bytes, (uint32_t)(TC_KT * abits / 8), TC_BN, act_sw);
  } else {
    a.act_tma = 0;
    act_ok = make_map_im2col(&a.act_map, act, row_bytes, g.B, g.H, g.W, g.R, g.S, g.stride, g.pad,
                             (uint32_t)(TC_KT * abits / 8), TC_BN, act_sw);
  }
  if (st == FGQ_OK && !act_ok) st = FGQ_ERR_CUDA;
  if (g.groups == 1 && g.M % 4 == 0 && !g.rq_out && !sums) {
    a.out_tma = make_map_2d(&a.out_map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, out, (uint64_t)g.M, (uint64_t)g.P,
                            (uint64_t)g.M * 4, TC_BM, TC_BN, CU_TENSOR_MAP_SWIZZLE_NONE)
                    ? 1
                    : 0;
  }
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int grid = a.ntiles < sms ? a.ntiles : sms;
  const bool sgn = g.act_type == FGQ_S8 || g.act_type == FGQ_S4;
  if (st == FGQ_OK) {
    if (abits == 4)
      st = sgn ? launch_tc_path<4, true>(a, grid, s) : launch_tc_path<4, false>(a, grid, s);
    else
      st = sgn ? launch_tc_path<8, true>(a, grid, s) : launch_tc_path<8, false>(a, grid, s);
  }
  // the temporary returns to the pool once the work queued on s before this point is done
  if (cudaFreeAsync(a16, s) != cudaSuccess && st == FGQ_OK) st = FGQ_ERR_CUDA;
  return st;
}

fgq_status launch_wait_timeout_selftest(uint32_t max_iter, unsigned int* err, cudaStream_t s) {
  wait_timeout_selftest_kernel<<<1, 32, 0, s>>>(max_iter, err);
  return after_launch();
}

}  // namespace fgq
