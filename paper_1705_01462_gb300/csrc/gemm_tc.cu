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
// holds exactly s[m][g][p] for a 128-filter x 256-position tile; the epilogue multiplies
// it by alpha[m][g] and adds it into an fp32 register accumulator (one multiply per group,
// Section 4.1).  Two 256-column TMEM buffers let the MMAs of group g + 1 run while group g
// drains.  The group-sums variant (SUMS) stores each drained accumulator as the int32
// s[m][g][p] instead (the exact integers themselves, for verification).
//
// Both operands reach shared memory by TMA, already as MMA operands: the codes are expanded
// to {0, +1, -1} and the activations to their integer values once per call (stream-ordered
// temporaries written by one launch, prep64_kernel), fp16 for 8-bit activations and e4m3
// (kind::f8f6f4) for 4-bit ones, so every K-tile is two box loads into one ring stage and
// no thread converts operands inside the contraction.  An activation is read by R * S filter
// taps and M / 128 filter tiles; converting it once instead of at every use takes the
// conversion off the MMA's path.
//
// Warp roles (352 threads, one CTA per SM, persistent over tiles):
//   warps 0-7  epilogue: warp w reads TMEM lanes 32*(w%4).. (filter rows) and columns
//              128*(w/4).. (positions) of the drained buffer in four 32-column tcgen05.ld,
//              frees the buffer, and adds alpha * s into 128 fp32 registers.  At tile end
//              it stores the tile directly (32 lanes = 32 consecutive filters: one 128-byte
//              segment per position), requantized when asked.
//   warps 8, 9 the MMA issuers (one thread each; warp 8 also allocates TMEM): the even groups
//              into accumulator 0 and the odd groups into accumulator 1, 4 tcgen05.mma
//              (M = 128, N = 256, K = 16) per K-tile and one commit per group; while one
//              thread waits on its barriers, the other's MMAs keep the tensor pipe busy.
//   warp 10    the producer (one thread): per K-tile, the ternary box (64 reduction
//              elements x 128 filters) and the activation box (64 channels x 256 positions)
//              into one four-stage ring: a 2D box of consecutive input rows when the im2col
//              rows are input rows (1x1 stride-1 convolutions, GEMMs), otherwise an im2col
//              box (the 256 output positions' pixels at the K-tile's filter tap, zeros in
//              the padding).
// A stage is released by the epilogue: the group's accumulator commit (one per group) is
// seen by epilogue thread 0, which frees the group's stages, so no commit is spent on them.
// Every mbarrier wait is bounded; on expiry the kernel records FGQ_ERR_TIMEOUT, each role
// leaves its loop (uniformly within the epilogue, which uses named barriers), in-flight
// copies and MMAs are waited for, and TMEM is freed.
#include <cstdint>
#include <cstring>

#include "operand_prep.cuh"
#include "tc_common.cuh"

namespace fgq {
namespace {

using tc::encode_im2col;
using tc::encode_tiled;
using tc::im2col_fits;
using tc::make_map_2d;
using tc::make_map_im2col;

constexpr int TC_BM = 128;        // filters per tile (MMA M, TMEM lanes)
constexpr int TC_BN = 256;        // positions per tile (MMA N)
constexpr int TC_KT = 64;         // reduction elements per K-tile
constexpr int TC_NACC = 2;        // TMEM accumulator buffers
constexpr int TC_EPI_WARPS = 8;
constexpr int TC_MMA_WARP = TC_EPI_WARPS;       // warps 8 and 9: MMA issuers of even and odd groups
constexpr int TC_PROD_WARP = TC_EPI_WARPS + 2;  // warp 10: lane 0 streams both operands
constexpr int TC_THREADS = 32 * (TC_PROD_WARP + 1);
constexpr int TC_TMEM_COLS = TC_NACC * TC_BN;    // 512: all of TMEM
constexpr int TC_EPI_COLS = TC_BN / 2;           // positions per epilogue thread
constexpr uint32_t TC_WAIT_LIMIT = 50000;        // polls of up to 20 us: about 1 s per wait
constexpr uint32_t TC_WAIT_SLEEP_NS = 20000;     // suspend hint of one poll
constexpr uint32_t TC_DRAIN_LIMIT = 1u << 20;    // polls of the final drains (never shortened)
constexpr uint32_t BAR_EPI = 2;                  // named barrier of the 256 epilogue threads

constexpr int OUT_POS = 64;                      // positions per output box
constexpr int OUT_BOX = OUT_POS * TC_BM * 4;     // 32 KB fp32 [64 positions][128 filters]
constexpr int SMEM_OUT = 2 * OUT_BOX;            // one box per position half of the tile

// Operand plan of a variant.  fp16 operands (8-bit activations): 128-byte rows of 64
// elements, 128-byte swizzle, 4 MMAs of K = 16 per K-tile.  e4m3 operands (4-bit
// activations, F8): every 4-bit value and every code is exact in e4m3, so the K-tile is
// 64-byte rows with the 64-byte swizzle and 2 MMAs of K = 32 (kind::f8f6f4) -- half the bytes
// per K-tile in HBM, L2 and shared memory, twice the ring depth.
template <bool F8>
struct TcCfg {
  static constexpr int ES = F8 ? 1 : 2;                 // bytes per operand element
  static constexpr int A_TILE = TC_BM * TC_KT * ES;     // ternary operand
  static constexpr int B_TILE = TC_BN * TC_KT * ES;     // activation operand
  static constexpr int STAGE = A_TILE + B_TILE;
  static constexpr int NST = F8 ? 6 : 3;                // operand ring depth
  static constexpr int SMEM_BAR = 8 * (2 * NST + 2 * TC_NACC + 1) + 16;
  static constexpr int SMEM = 1024 + NST * STAGE + SMEM_OUT + SMEM_BAR;
};
static_assert(TcCfg<false>::SMEM <= 232448 && TcCfg<true>::SMEM <= 232448, "shared memory budget");
static_assert(TcCfg<false>::A_TILE % 1024 == 0 && TcCfg<false>::STAGE % 1024 == 0 &&
                  TcCfg<true>::A_TILE % 1024 == 0 && TcCfg<true>::STAGE % 1024 == 0,
              "swizzle atoms stay 1024-byte aligned");

struct TcArgs {
  CUtensorMap a16_map;    // expanded codes [M][Kp] (fp16, or e4m3 for F8), box {64, 128 rows}
  CUtensorMap act_map;    // expanded activations: act_tma: 2D [positions][C], box {64, 256 rows}; otherwise
                          // the im2col map of the NHWC tensor, 256 pixels x 64 channels
  CUtensorMap out_map;    // fp32 [P][M], box {128 filters, 64 positions}; if out_tma
  const float* alpha;
  const float* act_scale;
  float* out;
  int32_t* sums;    // SUMS: int32 group sums [M][ng][P]
  unsigned int* err;
  Geom g;
  int mtiles;       // filter tiles per conv group
  int ptiles;       // position tiles
  int ntiles;       // work items: groups * mtiles * ptiles tiles, each split into ksplit group ranges
  int ktiles;       // K-tiles of a whole tile (= ng * G / 64)
  int ksplit;       // group ranges per tile (1: whole tiles; > 1: partial sums added into the output)
  int gpk;          // groups per range
  int kt_per_group; // G / 64
  int act_tma;      // 2D activation map (one row per output position); else im2col map
  int out_tma;      // output boxes by TMA store (one conv group, M % 4 == 0, fp32 output)
  uint32_t wait_limit;     // polls per wait (each up to wait_sleep_ns)
  uint32_t wait_sleep_ns;
};

// Work item w: tile w / ksplit, groups [g0, g1) of range w % ksplit.  Tiles are numbered
// with the filter tiles of one position tile consecutive, so that CTAs running at the same
// time share activation boxes in L2.
__device__ __forceinline__ void item_coords(const TcArgs& a, int w, int& gi, int& m0, int64_t& p0, int& g0, int& g1) {
  const int tile = w / a.ksplit;
  const int ks = w - tile * a.ksplit;
  const int per_p = a.g.groups * a.mtiles;
  const int pt = tile / per_p;
  const int r = tile - pt * per_p;
  gi = r / a.mtiles;
  const int mt = r - gi * a.mtiles;
  m0 = gi * a.g.Mg + mt * TC_BM;
  p0 = (int64_t)pt * TC_BN;
  g0 = ks * a.gpk;
  g1 = g0 + a.gpk < a.g.ng ? g0 + a.gpk : a.g.ng;
}

// One launch prepares both operands of a call: blocks [0, code_blocks) expand the ternary
// codes (one 16-code word per thread and step), the others the activations (16 elements per
// thread and step); fp16 operands, or e4m3 for 4-bit activations (F8).
template <bool F8>
__global__ void __launch_bounds__(256) prep64_kernel(const uint32_t* __restrict__ codes, int64_t nwords,
                                                     uint4* __restrict__ a_op, const prep::ActSrc src,
                                                     uint4* __restrict__ x_op, int code_blocks) {
  pdl_wait();
  pdl_trigger();
  if ((int)blockIdx.x < code_blocks) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < nwords; i += (int64_t)code_blocks * blockDim.x) {
      if (F8) prep::codes_e4m3(codes, i, a_op);
      else prep::codes_f16(codes, i, a_op);
    }
  } else {
    const int64_t nb = (int64_t)gridDim.x - code_blocks;
    prep::act_expand<F8>(src, ((int64_t)blockIdx.x - code_blocks) * blockDim.x + threadIdx.x, nb * blockDim.x, x_op);
  }
}

// TMAP: the layer's im2col rows are contiguous input rows (2D box loads); otherwise the
// activation boxes come from an im2col map (one load per K-tile: 256 output positions at
// one filter tap and 64 channels, padding read as zeros).
template <bool TMAP, bool SUMS, bool F8>
__global__ void __launch_bounds__(TC_THREADS, 1) tc_contract_kernel(const __grid_constant__ TcArgs a) {
  using Cfg = TcCfg<F8>;
  constexpr int TC_NST = Cfg::NST;
  constexpr int STAGE = Cfg::STAGE;
  constexpr int A_TILE = Cfg::A_TILE;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  float* otile = reinterpret_cast<float*>(smem + TC_NST * STAGE);  // two [64 positions][128 filters] boxes
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + TC_NST * STAGE + SMEM_OUT);
  uint64_t* full = bars;                 // stage loaded (both boxes' bytes)
  uint64_t* empty = bars + TC_NST;       // stage free (released by the epilogue)
  uint64_t* acc_full = empty + TC_NST;
  uint64_t* acc_empty = acc_full + TC_NACC;
  uint64_t* drain_bar = acc_empty + TC_NACC;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_bar + 1);
  volatile uint32_t* abort_flag = tmem_slot + 1;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const Geom& g = a.g;

  if (threadIdx.x == 0) {
    for (int i = 0; i < TC_NST; ++i) {
      mbar_init(&full[i], 1);   // the producer's expect_tx, then the two boxes' bytes
      mbar_init(&empty[i], 1);  // released by the epilogue (the group's MMAs completed)
    }
    for (int i = 0; i < TC_NACC; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], TC_EPI_WARPS);  // one arrival per epilogue warp
    }
    mbar_init(drain_bar, TC_NACC);  // one commit per MMA issuer
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
  // the prologue above overlapped the previous kernel; global memory only from here on
  pdl_wait();
  pdl_trigger();
  const int my_tiles = (a.ntiles - (int)blockIdx.x + (int)gridDim.x - 1) / (int)gridDim.x;

  auto fail = [&]() {
    *abort_flag = 1;
    record_error(a.err, FGQ_ERR_TIMEOUT);
  };

  // ------------------------------------------------------------------ producer
  if (warp == TC_PROD_WARP && lane == 0) {
    const int kpt = g.Cg / TC_KT;  // K-tiles per filter tap
    int issued = 0;                // K-tiles issued by this CTA (the ring's sequence number)
    bool ok = true;
    for (int tl = 0; tl < my_tiles && ok; ++tl) {
      int gi, m0, g0, g1;
      int64_t p0;
      item_coords(a, (int)blockIdx.x + tl * (int)gridDim.x, gi, m0, p0, g0, g1);
      int n0 = 0, h0 = 0, w0 = 0;  // im2col: the tile's first window origin (input pixel coordinates)
      if (!TMAP) {
        const int pp = (int)p0;  // < P < 2^31
        const int wo = pp % g.Wo;
        const int q = pp / g.Wo;
        n0 = q / g.Ho;
        h0 = (q - n0 * g.Ho) * g.stride - g.pad;
        w0 = wo * g.stride - g.pad;
      }
      // the range's first K-tile and its filter tap (tr, ts) and channel offset tc0, which
      // then advance incrementally
      const int kt0 = g0 * a.kt_per_group, kt1 = g1 * a.kt_per_group;
      int tc0 = (kt0 % kpt) * TC_KT, ts = (kt0 / kpt) % g.S, tr = (kt0 / kpt) / g.S;
      for (int kt = kt0; kt < kt1; ++kt) {
        const int j = issued;
        const int s = j % TC_NST;
        // the stage's previous contents (K-tile j - TC_NST) have been consumed by the MMAs
        if (j >= TC_NST &&
            !mbar_wait_or_abort(&empty[s], ((j / TC_NST) & 1) ^ 1, a.wait_limit, abort_flag, a.wait_sleep_ns)) {
          ok = false;
          break;
        }
        uint8_t* sa = smem + s * STAGE;
        const int ch = gi * g.Cg + tc0;  // first channel: a multiple of 64 (128-byte aligned in fp16)
        mbar_arrive_expect_tx(&full[s], STAGE);
        tma_load_2d(smem_u32(sa), &a.a16_map, kt * TC_KT, m0, &full[s]);
        if (TMAP)
          tma_load_2d(smem_u32(sa + A_TILE), &a.act_map, ch, (int)p0, &full[s]);
        else
          tma_load_im2col_4d(smem_u32(sa + A_TILE), &a.act_map, ch, w0, h0, n0, (uint16_t)ts, (uint16_t)tr, &full[s]);
        issued = j + 1;
        tc0 += TC_KT;
        if (tc0 == g.Cg) {
          tc0 = 0;
          if (++ts == g.S) {
            ts = 0;
            ++tr;
          }
        }
      }
    }
    if (!ok && !*abort_flag) fail();
    // loads the MMA issuer may not have consumed: the last TC_NST issued, one per stage,
    // each the latest phase of its stage's barrier; none may outlive the CTA
    for (int j = issued - TC_NST < 0 ? 0 : issued - TC_NST; j < issued; ++j)
      mbar_wait_bounded(&full[j % TC_NST], (j / TC_NST) & 1, TC_DRAIN_LIMIT);
  }

  // ------------------------------------------------------------------ MMA issuers
  // Two threads issue the MMAs, one for the even and one for the odd groups, each into its
  // own TMEM accumulator: one thread's barrier waits and commit overlap the other's MMAs.
  if ((warp == TC_MMA_WARP || warp == TC_MMA_WARP + 1) && lane == 0) {
    const int b = warp - TC_MMA_WARP;  // accumulator = parity of the groups this thread issues
    const uint32_t idesc = idesc_f16_f32(TC_BM, TC_BN);
    int kt = 0, gc = 0;
    bool ok = true;
    for (int tl = 0; tl < my_tiles && ok; ++tl) {
      int gi_, m0_, g0, g1;
      int64_t p0_;
      item_coords(a, (int)blockIdx.x + tl * (int)gridDim.x, gi_, m0_, p0_, g0, g1);
      for (int grp = g0; grp < g1 && ok; ++grp, ++gc) {
        if ((gc & 1) != b) {
          kt += a.kt_per_group;  // the other issuer's group
          continue;
        }
        if (!mbar_wait_or_abort(&acc_empty[b], ((gc >> 1) & 1) ^ 1, a.wait_limit, abort_flag, a.wait_sleep_ns)) {
          if (!*abort_flag) fail();
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + (uint32_t)(b * TC_BN);
        for (int sub = 0; sub < a.kt_per_group; ++sub, ++kt) {
          const int s = kt % TC_NST;
          if (!mbar_wait_or_abort(&full[s], (kt / TC_NST) & 1, a.wait_limit, abort_flag, a.wait_sleep_ns)) {
            if (!*abort_flag) fail();
            ok = false;
            break;
          }
          tc_fence_after();
          if constexpr (F8) {
            const uint64_t ad = sdesc_k_sw64(smem_u32(smem + s * STAGE));
            const uint64_t bd = sdesc_k_sw64(smem_u32(smem + s * STAGE + A_TILE));
#pragma unroll
            for (int k = 0; k < TC_KT / 32; ++k)  // advance 32 e4m3 (32 bytes) along K
              mma_e4m3(d, ad + 2 * k, bd + 2 * k, idesc, (sub > 0 || k > 0) ? 1u : 0u);
          } else {
            const uint64_t ad = sdesc_k_sw128(smem_u32(smem + s * STAGE));
            const uint64_t bd = sdesc_k_sw128(smem_u32(smem + s * STAGE + A_TILE));
#pragma unroll
            for (int k = 0; k < TC_KT / 16; ++k)  // advance 16 fp16 (32 bytes) along K
              mma_f16(d, ad + 2 * k, bd + 2 * k, idesc, (sub > 0 || k > 0) ? 1u : 0u);
          }
        }
        if (ok) mma_commit(&acc_full[b]);
      }
    }
    // all MMAs issued by both threads are complete once the drain barrier flips
    mma_commit(drain_bar);
    mbar_wait_bounded(drain_bar, 0, TC_DRAIN_LIMIT);
  }

  // ------------------------------------------------------------------ epilogue
  if (warp < TC_EPI_WARPS) {
    const int quarter = warp & 3, half = warp >> 2;
    const int t = 32 * quarter + lane;  // TMEM lane = filter row of the tile
    const uint32_t tbase = tmem + ((uint32_t)(32 * quarter) << 16) + (uint32_t)(TC_EPI_COLS * half);
    const float sx = __ldg(a.act_scale);
    const bool leader = threadIdx.x == 0;
    int gc = 0;
    bool ok = true;
    for (int tl = 0; tl < my_tiles; ++tl) {
      int gi, m0, g0, g1;
      int64_t p0;
      item_coords(a, (int)blockIdx.x + tl * (int)gridDim.x, gi, m0, p0, g0, g1);
      const int m = m0 + t;
      const bool mok = m < gi * g.Mg + g.Mg && m < g.M;
      const int64_t pbase = p0 + TC_EPI_COLS * half;
      const float* arow = a.alpha + (int64_t)(mok ? m : 0) * g.ng;
      float acc[TC_EPI_COLS];
#pragma unroll
      for (int j = 0; j < TC_EPI_COLS; ++j) acc[j] = 0.0f;
      float al_next = mok ? __ldg(arow + g0) : 0.0f;
      for (int grp = g0; grp < g1; ++grp, ++gc) {
        if (!ok) continue;  // after a failed wait: run out the tile, then leave with the others
        const int b = gc & 1;
        const float al = al_next;  // alpha of this group, loaded one group ahead
        if (mok && grp + 1 < g1) al_next = __ldg(arow + grp + 1);
        if (!mbar_wait_or_abort(&acc_full[b], (gc >> 1) & 1, a.wait_limit, abort_flag, a.wait_sleep_ns)) {
          if (!*abort_flag) fail();
          ok = false;
          continue;
        }
        if (leader) {
          // the group's MMAs have completed: its K-tiles' stages may be refilled
          for (int k = gc * a.kt_per_group; k < (gc + 1) * a.kt_per_group; ++k) mbar_arrive(&empty[k % TC_NST]);
        }
        tc_fence_after();
        if constexpr (SUMS) {
          uint32_t r[32];
          // the exact group sums of positions pbase + j, filter m: s[m][grp][p]
          int32_t* srow = a.sums + ((int64_t)(mok ? m : 0) * g.ng + grp) * g.P;
#pragma unroll
          for (int c = 0; c < TC_EPI_COLS / 32; ++c) {
            tmem_ld32(tbase + (uint32_t)(b * TC_BN + 32 * c), r);
            tmem_ld_wait();
            if (c == TC_EPI_COLS / 32 - 1) {
              tc_fence_before();
              __syncwarp();
              if (lane == 0) mbar_arrive(&acc_empty[b]);
            }
            if (mok) {
#pragma unroll
              for (int j = 0; j < 32; ++j) {
                const int64_t p = pbase + 32 * c + j;
                if (p < g.P) srow[p] = __float2int_rn(__uint_as_float(r[j]));
              }
            }
          }
        } else {
        // 16 columns per load keep the 128 accumulators and the loaded values inside the
        // register budget of 10 warps (three of them on one SM sub-partition's 16K registers)
#pragma unroll
        for (int c = 0; c < TC_EPI_COLS / 16; ++c) {
          uint32_t r16[16];
          tmem_ld16(tbase + (uint32_t)(b * TC_BN + 16 * c), r16);
          tmem_ld_wait_regs16(r16);
          if (c == TC_EPI_COLS / 16 - 1) {
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&acc_empty[b]);  // the buffer is free once the values are in registers
          }
#pragma unroll
          for (int j = 0; j < 16; ++j) acc[16 * c + j] = fmaf(al, __uint_as_float(r16[j]), acc[16 * c + j]);
        }
        }
      }
      if (named_bar_or(BAR_EPI, 32 * TC_EPI_WARPS, !ok)) break;  // leave together
      if (SUMS) continue;  // the group sums are stored already
      if (a.out_tma) {
        // two rounds: the warps of position half h write positions 128 h + 64 k .. + 63 of
        // round k into box h, thread 0 stores both boxes (rows past P and filters past M are
        // clipped by the tensor map)
        float* ob = otile + half * (OUT_POS * TC_BM) + t;
#pragma unroll
        for (int k = 0; k < TC_EPI_COLS / OUT_POS; ++k) {
          if (leader) bulk_wait_read_all();  // the boxes' previous stores have read them
          named_bar_sync(BAR_EPI, 32 * TC_EPI_WARPS);
#pragma unroll
          for (int j = 0; j < OUT_POS; ++j) ob[j * TC_BM] = sx * acc[OUT_POS * k + j];
          fence_proxy_async_smem();
          named_bar_sync(BAR_EPI, 32 * TC_EPI_WARPS);
          if (leader) {
#pragma unroll
            for (int hh = 0; hh < 2; ++hh) {
              const int64_t pb = p0 + TC_EPI_COLS * hh + OUT_POS * k;
              if (pb < g.P) {
                if (a.ksplit > 1)  // a group range's partial sums: added into the (zeroed) output
                  tma_reduce_add_2d(&a.out_map, m0, (int)pb, smem_u32(otile + hh * (OUT_POS * TC_BM)));
                else
                  tma_store_2d(&a.out_map, m0, (int)pb, smem_u32(otile + hh * (OUT_POS * TC_BM)));
              }
            }
            bulk_commit();
          }
        }
        continue;
      }
      if (!mok) continue;
      // one 128-byte segment per position: the warp's 32 lanes are 32 consecutive filters
      if (g.rq_out) {  // fused requantization: 8-bit codes instead of fp32
        const RqMul r = rq_mul(g.rq_scale, g.rq_signed);
#pragma unroll
        for (int j = 0; j < TC_EPI_COLS; ++j) {
          const int64_t p = pbase + j;
          if (p < g.P) g.rq_out[p * g.M + m] = rq_code(sx * acc[j], r);
        }
      } else {
#pragma unroll
        for (int j = 0; j < TC_EPI_COLS; ++j) {
          const int64_t p = pbase + j;
          if (p < g.P) {
            if (a.ksplit > 1) atomicAdd(a.out + p * g.M + m, sx * acc[j]);
            else a.out[p * g.M + m] = sx * acc[j];
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

template <bool TMAP, bool SUMS, bool F8>
fgq_status launch_tc(const TcArgs& args, int grid, cudaStream_t s) {
  constexpr int smem = TcCfg<F8>::SMEM;
  if (!tc::smem_attr_once<tc_contract_kernel<TMAP, SUMS, F8>>(smem)) return FGQ_ERR_CUDA;
  return after_launch(launch_pdl(tc_contract_kernel<TMAP, SUMS, F8>, dim3(grid), dim3(TC_THREADS), smem, s, args));
}

template <bool F8>
fgq_status launch_tc_variant(const TcArgs& a, bool sums, int grid, cudaStream_t s) {
  if (sums) return a.act_tma ? launch_tc<true, true, F8>(a, grid, s) : launch_tc<false, true, F8>(a, grid, s);
  return a.act_tma ? launch_tc<true, false, F8>(a, grid, s) : launch_tc<false, false, F8>(a, grid, s);
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

namespace tc {

bool act_pointwise(const Geom& g) { return g.R == 1 && g.S == 1 && g.pad == 0; }

int64_t act16_elems(const Geom& g) {
  return act_pointwise(g) && g.stride > 1 ? g.P * g.C : (int64_t)g.B * g.H * g.W * g.C;
}

bool act16_map(CUtensorMap* m, const void* x16, const Geom& g, uint32_t pixels) {
  if (act_pointwise(g))
    return make_map_2d(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, x16, (uint64_t)g.C, (uint64_t)(act16_elems(g) / g.C),
                       (uint64_t)g.C * 2, 64, pixels, CU_TENSOR_MAP_SWIZZLE_128B);
  return make_map_im2col(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, x16, (uint64_t)g.C, 2, g.B, g.H, g.W, g.R, g.S, g.stride,
                         g.pad, 64, pixels, CU_TENSOR_MAP_SWIZZLE_128B);
}

bool act16_supported(const Geom& g) {
  if (g.C % 16 != 0 || g.Cg % 64 != 0) return false;
  if (encode_tiled() == nullptr) return false;
  return act_pointwise(g) || (encode_im2col() != nullptr && im2col_fits(g.R, g.S, g.stride, g.pad));
}

}  // namespace tc

using tc::act_pointwise;

bool tc_supports(const Geom& g) {
  if (g.G != 64 && g.G != 128) return false;
  if (g.P >= (int64_t)1 << 31) return false;  // positions decoded in 32 bits
  // every K-tile inside one filter tap (conv) or row (GEMM); 16-element expansion chunks;
  // activation boxes by 2D or im2col maps
  return tc::act16_supported(g);
}

fgq_status launch_tc_contract(const void* act, const Geom& g, const uint32_t* codes, const float* alpha,
                              const float* act_scale, float* out, int32_t* sums, unsigned int* err,
                              cudaStream_t s) {
  if (!tc_supports(g)) return FGQ_ERR_UNSUPPORTED;
  TcArgs a;
  memset(&a, 0, sizeof a);
  a.alpha = alpha;
  a.act_scale = act_scale;
  a.out = out;
  a.sums = sums;
  a.err = err;
  a.g = g;
  a.mtiles = (g.Mg + TC_BM - 1) / TC_BM;
  a.ptiles = (int)((g.P + TC_BN - 1) / TC_BN);
  a.kt_per_group = g.G / TC_KT;
  a.ktiles = g.ng * a.kt_per_group;
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  // A layer with fewer tiles than SMs and a long reduction (at least 64 K-tiles: 4096
  // products per output) splits each tile's groups into ranges of at least two groups whose
  // partial sums are added into the zeroed output (fp32 adds in L2), taking the count that
  // fills the device best (each count by more than 5% over the fewer ranges before it).
  // Shorter reductions lose more to zeroing the output and adding the partial sums than
  // they gain; outputs that are requantized or group sums keep whole tiles.
  const int tiles = g.groups * a.mtiles * a.ptiles;
  int ksplit = 1;
  if (tiles < sms && a.ktiles >= 64 && !sums && !g.rq_out) {
    double best = (double)tiles / sms;
    for (int k = 2; k <= debug_max_ksplit() && k <= g.ng / 2; ++k) {
      const int64_t items = (int64_t)tiles * k, waves = (items + sms - 1) / sms;
      const double eff = (double)items / (double)(waves * sms);
      if (eff > best * 1.05) {
        best = eff;
        ksplit = k;
      }
    }
  }
  a.gpk = (g.ng + ksplit - 1) / ksplit;
  a.ksplit = (g.ng + a.gpk - 1) / a.gpk;  // every range non-empty
  a.ntiles = tiles * a.ksplit;
  note_ksplit(a.ksplit);
  // a test may shorten the waits (debug_wait_limit_us), never the final drains
  const int64_t lim_us = debug_wait_limit_us();
  a.wait_limit = lim_us < 0 ? TC_WAIT_LIMIT : (uint32_t)(lim_us / 20 + 1);
  a.wait_sleep_ns = lim_us < 0 ? TC_WAIT_SLEEP_NS : (uint32_t)(lim_us < 20 ? lim_us * 1000 : 20000);
  // 4-bit activations run on e4m3 operands (exact), 8-bit ones on fp16 (exact)
  const bool f8 = g.act_type == FGQ_U4 || g.act_type == FGQ_S4;
  const int es = f8 ? 1 : 2;
  // temporaries from the stream-ordered pool: the codes expanded [M][Kp] (Kp = 16 wrow) and the
  // activations expanded NHWC (a strided 1x1 convolution: only the pixels it reads, [P][C])
  cudaMemPool_t pool = scratch_pool();
  if (!pool) return FGQ_ERR_CUDA;
  const int64_t nwords = (int64_t)g.M * g.wrow;
  const int64_t nact = tc::act16_elems(g);
  void* a16 = nullptr;
  void* x16 = nullptr;
  if (cudaMallocFromPoolAsync(&a16, (size_t)nwords * 16 * es, pool, s) != cudaSuccess) return FGQ_ERR_CUDA;
  if (cudaMallocFromPoolAsync(&x16, (size_t)nact * es, pool, s) != cudaSuccess) {
    cudaFreeAsync(a16, s);
    return FGQ_ERR_CUDA;
  }
  // both operands in one launch, the blocks split by the two jobs' sizes
  const prep::ActSrc src = prep::act_src(act, g);
  const int cb = prep::blocks_for(nwords), xb = prep::blocks_for(src.nchunks);
  fgq_status st = after_launch(
      f8 ? launch_pdl(prep64_kernel<true>, dim3(cb + xb), dim3(256), 0, s, codes, nwords, static_cast<uint4*>(a16),
                          src, static_cast<uint4*>(x16), cb)
         : launch_pdl(prep64_kernel<false>, dim3(cb + xb), dim3(256), 0, s, codes, nwords, static_cast<uint4*>(a16),
                          src, static_cast<uint4*>(x16), cb));
  const CUtensorMapDataType dt = f8 ? CU_TENSOR_MAP_DATA_TYPE_UINT8 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16;
  const CUtensorMapSwizzle sw = f8 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_128B;
  if (st == FGQ_OK && !make_map_2d(&a.a16_map, dt, a16, (uint64_t)g.wrow * 16, (uint64_t)g.M,
                                   (uint64_t)g.wrow * 16 * es, TC_KT, TC_BM, sw))
    st = FGQ_ERR_CUDA;
  a.act_tma = act_pointwise(g) ? 1 : 0;
  bool act_ok = true;
  if (st == FGQ_OK) {
    if (!f8)
      act_ok = tc::act16_map(&a.act_map, x16, g, TC_BN);
    else if (a.act_tma)
      act_ok = make_map_2d(&a.act_map, dt, x16, (uint64_t)g.C, (uint64_t)(nact / g.C), (uint64_t)g.C, TC_KT, TC_BN, sw);
    else
      act_ok = make_map_im2col(&a.act_map, dt, x16, (uint64_t)g.C, 1, g.B, g.H, g.W, g.R, g.S, g.stride, g.pad, TC_KT,
                               TC_BN, sw);
  }
  if (!act_ok) st = FGQ_ERR_CUDA;
  if (st == FGQ_OK && g.groups == 1 && g.M % 4 == 0 && !g.rq_out && !sums)
    a.out_tma = make_map_2d(&a.out_map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, out, (uint64_t)g.M, (uint64_t)g.P,
                            (uint64_t)g.M * 4, TC_BM, OUT_POS, CU_TENSOR_MAP_SWIZZLE_NONE)
                    ? 1
                    : 0;
  if (st == FGQ_OK && a.ksplit > 1 && cudaMemsetAsync(out, 0, (size_t)g.P * g.M * sizeof(float), s) != cudaSuccess)
    st = FGQ_ERR_CUDA;
  const int grid = a.ntiles < sms ? a.ntiles : sms;
  if (st == FGQ_OK)
    st = f8 ? launch_tc_variant<true>(a, sums != nullptr, grid, s) : launch_tc_variant<false>(a, sums != nullptr, grid, s);
  // the temporaries return to the pool once the work queued on s before this point is done
  if (cudaFreeAsync(x16, s) != cudaSuccess && st == FGQ_OK) st = FGQ_ERR_CUDA;
  if (cudaFreeAsync(a16, s) != cudaSuccess && st == FGQ_OK) st = FGQ_ERR_CUDA;
  return st;
}

fgq_status launch_wait_timeout_selftest(uint32_t max_iter, unsigned int* err, cudaStream_t s) {
  wait_timeout_selftest_kernel<<<1, 32, 0, s>>>(max_iter, err);
  return after_launch();
}

}  // namespace fgq
