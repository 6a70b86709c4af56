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
// Section 4.1).  Two TMEM buffers let group g+1's MMAs run while group g is drained.
//
// Warp roles (416 threads, one CTA per SM, persistent over tiles):
//   warps 0-7  epilogue: warp w reads TMEM lanes 32*(w%4).. (filter rows) and columns
//              64*(w/4).. (positions) of the drained buffer: one 64-column tcgen05.ld and
//              one wait per group, release of the buffer, then 64 FMAs with alpha into
//              fp32 registers; fp32 stores at tile end.
//   warps 8-11 loaders/converters: thread t owns activation row t (one output position,
//              implicit im2col) and code row t (one filter) of every K-tile; cp.async
//              copies raw bytes into a 6-deep staging ring, then the thread converts its
//              own rows to fp16 in the 128-byte-swizzled K-major layout the MMA reads.
//   warp 12    TMEM allocation and the MMA issuer (one thread): 4 tcgen05.mma (K = 16)
//              per K-tile into one of four 128-column TMEM accumulators.
// Every mbarrier wait is bounded; on expiry the kernel records FGQ_ERR_TIMEOUT, every
// role leaves its loop, in-flight copies and MMAs are waited for, and TMEM is freed.
#include <cstdint>

#include "fgq_device.cuh"
#include "ptx_sm100.cuh"

namespace fgq {
namespace {

constexpr int TC_BM = 128;        // filters per tile (MMA M, TMEM lanes)
constexpr int TC_BN = 128;        // positions per tile (MMA N)
constexpr int TC_KT = 64;         // reduction elements per K-tile
constexpr int TC_NO = 4;          // operand ring depth
constexpr int TC_NS = 6;          // staging ring depth
constexpr int TC_NACC = 4;        // TMEM accumulator buffers
constexpr int TC_EPI_WARPS = 8;
constexpr int TC_LOAD_WARP0 = TC_EPI_WARPS;      // loaders: warps 8-11
constexpr int TC_MMA_WARP = TC_EPI_WARPS + 4;    // warp 12
constexpr int TC_THREADS = 32 * (TC_MMA_WARP + 1);
constexpr int TC_TMEM_COLS = TC_NACC * TC_BN;    // 512: all of TMEM
constexpr uint32_t TC_WAIT_LIMIT = 1u << 22;

constexpr int OP_TILE = TC_BM * TC_KT * 2;            // 16 KB: one fp16 operand tile
constexpr int OP_STAGE = 2 * OP_TILE;                  // A (codes) + B (activations)
constexpr int ST_ACT = TC_BN * TC_KT;                  // 8 KB raw activation bytes (8-bit)
constexpr int ST_CODE = TC_BM * 16;                    // 2 KB raw code words
constexpr int ST_STAGE = ST_ACT + ST_CODE;
constexpr int SMEM_OP = TC_NO * OP_STAGE;
constexpr int SMEM_ST = TC_NS * ST_STAGE;
constexpr int SMEM_LUT = 256 * 8;                      // code byte -> 4 fp16
constexpr int SMEM_BAR = 8 * (2 * TC_NO + 2 * TC_NACC + 1) + 16;
constexpr int TC_SMEM = 1024 + SMEM_OP + SMEM_ST + SMEM_LUT + SMEM_BAR;

struct TcArgs {
  const uint8_t* act;
  const uint32_t* codes;
  const float* alpha;
  const float* act_scale;
  float* out;
  unsigned int* err;
  Geom g;
  int mtiles;       // filter tiles per conv group
  int ptiles;       // position tiles
  int ntiles;       // groups * mtiles * ptiles
  int ktiles;       // K-tiles per tile (= ng * G / 64)
  int kt_per_group; // G / 64
  uint32_t wait_limit;
};

// Byte offset of 16-byte chunk c (0..7) of row r in a 128B-swizzled K-major tile.
__device__ __forceinline__ uint32_t sw128(int r, int c) {
  return (uint32_t)((r >> 3) * 1024 + (r & 7) * 128 + ((c ^ (r & 7)) << 4));
}

__device__ __forceinline__ void tile_coords(const TcArgs& a, int tile, int& gi, int& m0, int64_t& p0) {
  const int per_p = a.g.groups * a.mtiles;
  const int pt = tile / per_p;
  const int r = tile - pt * per_p;
  gi = r / a.mtiles;
  const int mt = r - gi * a.mtiles;
  m0 = gi * a.g.Mg + mt * TC_BM;
  p0 = (int64_t)pt * TC_BN;
}

// fp16 pair (lo, hi) from two 8-bit lanes of x selected by sel (unsigned: 1024 + v - 1024).
__device__ __forceinline__ uint32_t u8pair_to_h2(uint32_t x, uint32_t sel, uint32_t bias2) {
  const uint32_t h = __byte_perm(x, 0x64646464u, sel);  // halves 1024 + v
  uint32_t r;
  asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(r) : "r"(h), "r"(bias2));
  return r;
}

template <int ABITS, bool SIGNED>
__global__ void __launch_bounds__(TC_THREADS, 1) tc_contract_kernel(const TcArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* op = smem;                       // TC_NO x {A tile, B tile}
  uint8_t* st = smem + SMEM_OP;             // TC_NS x {act bytes, code bytes}
  uint2* lut = reinterpret_cast<uint2*>(smem + SMEM_OP + SMEM_ST);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + SMEM_OP + SMEM_ST + SMEM_LUT);
  uint64_t* op_full = bars;
  uint64_t* op_empty = bars + TC_NO;
  uint64_t* acc_full = bars + 2 * TC_NO;
  uint64_t* acc_empty = bars + 2 * TC_NO + TC_NACC;
  uint64_t* drain_bar = bars + 2 * TC_NO + 2 * TC_NACC;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_bar + 1);
  volatile uint32_t* abort_flag = tmem_slot + 1;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const Geom& g = a.g;

  if (threadIdx.x == 0) {
    for (int i = 0; i < TC_NO; ++i) {
      mbar_init(&op_full[i], 128);
      mbar_init(&op_empty[i], 1);
    }
    for (int i = 0; i < TC_NACC; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], 32 * TC_EPI_WARPS);
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  // code byte (four 2-bit codes) -> four fp16 {0, +1, -1}
  for (int i = threadIdx.x; i < 256; i += blockDim.x) {
    uint32_t h[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const uint32_t c = (i >> (2 * e)) & 3u;
      h[e] = c == 1u ? 0x3C00u : (c == 3u ? 0xBC00u : 0u);
    }
    lut[i] = make_uint2(h[0] | (h[1] << 16), h[2] | (h[3] << 16));
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

  // ------------------------------------------------------------------ loaders/converters
  if (warp >= TC_LOAD_WARP0 && warp < TC_MMA_WARP) {
    const int t = threadIdx.x - 32 * TC_LOAD_WARP0;  // row owned in every tile
    const int total = my_tiles * a.ktiles;
    constexpr int ACT_BYTES = TC_KT * ABITS / 8;  // 64 (8-bit) or 32 (4-bit) bytes per row
    constexpr int ACT_CHUNKS = ACT_BYTES / 16;

    // per-tile state of this thread's rows (refreshed when the issued K-tile enters a new tile)
    int cur_tile = -1, gi = 0, m0 = 0, pb = 0, phb = 0, pwb = 0;
    bool pvalid = false;
    auto issue = [&](int j) {
      const int tl = j / a.ktiles;
      const int kk = j - tl * a.ktiles;
      if (tl != cur_tile) {
        cur_tile = tl;
        int64_t p0;
        tile_coords(a, (int)blockIdx.x + tl * (int)gridDim.x, gi, m0, p0);
        const int64_t p = p0 + t;
        pvalid = p < g.P;
        const int pp = pvalid ? (int)p : 0;
        const int wo = pp % g.Wo;
        const int q = pp / g.Wo;
        const int ho = q % g.Ho;
        pb = q / g.Ho;
        phb = ho * g.stride - g.pad;
        pwb = wo * g.stride - g.pad;
      }
      uint8_t* sa = st + (j % TC_NS) * ST_STAGE;
      const uint32_t sact = smem_u32(sa + t * ACT_BYTES);
      const uint32_t scode = smem_u32(sa + ST_ACT + t * 16);
      const int k0 = kk * TC_KT;
      const uint8_t* src = a.act;
      bool inside = false;
      if (pvalid) {
        const int tap = k0 / g.Cg;
        const int c0 = k0 - tap * g.Cg;
        const int r = tap / g.S, s = tap - r * g.S;
        const int hi = phb + r, wi = pwb + s;
        if (hi >= 0 && hi < g.H && wi >= 0 && wi < g.W) {
          const int64_t e = (((int64_t)pb * g.H + hi) * g.W + wi) * g.C + (int64_t)gi * g.Cg + c0;
          src = a.act + e * ABITS / 8;
          inside = true;
        }
      }
#pragma unroll
      for (int c = 0; c < ACT_CHUNKS; ++c)
        cp_async16(sact + 16 * c, inside ? (const void*)(src + 16 * c) : (const void*)a.act, inside ? 16u : 0u);
      const int m = m0 + t;
      const bool mok = m < gi * g.Mg + g.Mg && m < g.M;
      const uint32_t* csrc = mok ? a.codes + (int64_t)m * g.wrow + k0 / 16 : a.codes;
      cp_async16(scode, csrc, mok ? 16u : 0u);
    };

    bool ok = true;
    for (int j = 0; j < TC_NS - 1; ++j) {
      if (j < total) issue(j);
      cp_async_commit();
    }
    for (int j = 0; j < total && ok; ++j) {
      if (j + TC_NS - 1 < total) issue(j + TC_NS - 1);
      cp_async_commit();
      cp_async_wait<TC_NS - 1>();  // this thread's copies of K-tile j have landed
      const int os = j % TC_NO;
      if (!mbar_wait_or_abort(&op_empty[os], ((j / TC_NO) & 1) ^ 1, a.wait_limit, abort_flag)) {
        if (!*abort_flag) fail();
        ok = false;
        break;
      }
      const uint8_t* sa = st + (j % TC_NS) * ST_STAGE;
      uint8_t* A = op + os * OP_STAGE;
      uint8_t* Bt = A + OP_TILE;
      // activations -> fp16 row t of B
      if (ABITS == 8) {
        const uint4* src = reinterpret_cast<const uint4*>(sa + t * 64);
        const uint32_t bias2 = SIGNED ? 0x64806480u : 0x64006400u;  // 1152 or 1024 in both halves
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          uint4 v = src[c];
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
        const uint4* src = reinterpret_cast<const uint4*>(sa + t * 32);
        const uint32_t bias2 = SIGNED ? 0x64086408u : 0x64006400u;  // 1032 or 1024
#pragma unroll
        for (int c = 0; c < 2; ++c) {
          const uint4 v = src[c];
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
      // codes -> fp16 row t of A: 64 codes, 8 per 16-byte chunk, 4 per table lookup
      {
        const uint4 cv = *reinterpret_cast<const uint4*>(sa + ST_ACT + t * 16);
        const uint32_t cw[4] = {cv.x, cv.y, cv.z, cv.w};
#pragma unroll
        for (int c = 0; c < 8; ++c) {
          const uint32_t bits = (cw[c / 2] >> (16 * (c & 1))) & 0xffffu;  // 8 codes
          const uint2 lo = lut[bits & 0xffu], hi = lut[bits >> 8];
          *reinterpret_cast<uint4*>(A + sw128(t, c)) = make_uint4(lo.x, lo.y, hi.x, hi.y);
        }
      }
      fence_proxy_async_smem();
      mbar_arrive(&op_full[os]);
    }
    cp_async_wait_all();
  }

  // ------------------------------------------------------------------ MMA issuer
  if (warp == TC_MMA_WARP && lane == 0) {
    const uint32_t idesc = idesc_f16_f32(TC_BM, TC_BN);
    const uint32_t op_base = smem_u32(op);
    int kt = 0, gc = 0;
    bool ok = true;
    for (int tl = 0; tl < my_tiles && ok; ++tl) {
      for (int grp = 0; grp < g.ng && ok; ++grp, ++gc) {
        const int b = gc % TC_NACC;
        if (!mbar_wait_or_abort(&acc_empty[b], ((gc / TC_NACC) & 1) ^ 1, a.wait_limit, abort_flag)) {
          if (!*abort_flag) fail();
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + (uint32_t)(b * TC_BN);
        for (int sub = 0; sub < a.kt_per_group; ++sub, ++kt) {
          const int os = kt % TC_NO;
          if (!mbar_wait_or_abort(&op_full[os], (kt / TC_NO) & 1, a.wait_limit, abort_flag)) {
            if (!*abort_flag) fail();
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t abase = op_base + os * OP_STAGE;
          const uint64_t ad = sdesc_k_sw128(abase);
          const uint64_t bd = sdesc_k_sw128(abase + OP_TILE);
#pragma unroll
          for (int k = 0; k < TC_KT / 16; ++k) {
            // advance 16 fp16 (32 bytes) along K inside the swizzled rows
            mma_f16(d, ad + 2 * k, bd + 2 * k, idesc, (sub > 0 || k > 0) ? 1u : 0u);
          }
          mma_commit(&op_empty[os]);
        }
        if (ok) mma_commit(&acc_full[b]);
      }
    }
    // all MMAs issued by this thread are complete once the drain barrier flips
    mma_commit(drain_bar);
    mbar_wait_bounded(drain_bar, 0, a.wait_limit);
  }

  // ------------------------------------------------------------------ epilogue
  if (warp < TC_EPI_WARPS) {
    const int quarter = warp & 3, half = warp >> 2;
    const int t = 32 * quarter + lane;  // TMEM lane = filter row of the tile
    const uint32_t tbase = tmem + ((uint32_t)(32 * quarter) << 16) + (uint32_t)(64 * half);
    const float sx = __ldg(a.act_scale);
    int gc = 0;
    bool ok = true;
    for (int tl = 0; tl < my_tiles && ok; ++tl) {
      int gi, m0;
      int64_t p0;
      tile_coords(a, (int)blockIdx.x + tl * (int)gridDim.x, gi, m0, p0);
      const int m = m0 + t;
      const bool mok = m < gi * g.Mg + g.Mg && m < g.M;
      const float* arow = a.alpha + (int64_t)(mok ? m : 0) * g.ng;
      float acc[64];
#pragma unroll
      for (int j = 0; j < 64; ++j) acc[j] = 0.0f;
      for (int grp = 0; grp < g.ng; ++grp, ++gc) {
        const int b = gc % TC_NACC;
        const float al = mok ? __ldg(arow + grp) : 0.0f;
        if (!mbar_wait_or_abort(&acc_full[b], (gc / TC_NACC) & 1, a.wait_limit, abort_flag)) {
          if (!*abort_flag) fail();
          ok = false;
          break;
        }
        tc_fence_after();
        uint32_t r0[32], r1[32];
        tmem_ld32(tbase + (uint32_t)(b * TC_BN), r0);
        tmem_ld32(tbase + (uint32_t)(b * TC_BN + 32), r1);
        tmem_ld_wait();
        tc_fence_before();
        mbar_arrive(&acc_empty[b]);  // the buffer is free once the values are in registers
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          acc[j] = fmaf(al, __uint_as_float(r0[j]), acc[j]);
          acc[32 + j] = fmaf(al, __uint_as_float(r1[j]), acc[32 + j]);
        }
      }
      if (!ok) break;
      if (mok) {
        const int64_t pbase = p0 + 64 * half;
#pragma unroll
        for (int j = 0; j < 64; ++j) {
          const int64_t p = pbase + j;
          if (p < g.P) a.out[p * g.M + m] = sx * acc[j];
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == TC_MMA_WARP) {
    tc_fence_after();
    tmem_dealloc(tmem, TC_TMEM_COLS);
  }
}

template <int ABITS, bool SIGNED>
fgq_status launch_tc(const TcArgs& args, int grid, cudaStream_t s) {
  static bool attr_set = false;
  if (!attr_set) {
    if (cudaFuncSetAttribute(tc_contract_kernel<ABITS, SIGNED>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             TC_SMEM) != cudaSuccess)
      return FGQ_ERR_CUDA;
    attr_set = true;
  }
  tc_contract_kernel<ABITS, SIGNED><<<grid, TC_THREADS, TC_SMEM, s>>>(args);
  return after_launch();
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
  if (g.Cg % TC_KT != 0) return false;     // every K-tile inside one filter tap (conv) or row (GEMM)
  if (g.C % 16 != 0) return false;         // 16-byte aligned activation rows
  if (g.P >= (int64_t)1 << 31) return false;  // positions decoded in 32 bits
  return true;
}

fgq_status launch_tc_contract(const void* act, const Geom& g, const uint32_t* codes, const float* alpha,
                              const float* act_scale, float* out, int32_t* sums, unsigned int* err,
                              cudaStream_t s) {
  if (sums != nullptr || !tc_supports(g)) return FGQ_ERR_UNSUPPORTED;
  TcArgs a;
  a.act = static_cast<const uint8_t*>(act);
  a.codes = codes;
  a.alpha = alpha;
  a.act_scale = act_scale;
  a.out = out;
  a.err = err;
  a.g = g;
  a.mtiles = (g.Mg + TC_BM - 1) / TC_BM;
  a.ptiles = (int)((g.P + TC_BN - 1) / TC_BN);
  a.ntiles = g.groups * a.mtiles * a.ptiles;
  a.kt_per_group = g.G / TC_KT;
  a.ktiles = g.ng * a.kt_per_group;
  a.wait_limit = TC_WAIT_LIMIT;
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int grid = a.ntiles < sms ? a.ntiles : sms;
  const bool sgn = g.act_type == FGQ_S8 || g.act_type == FGQ_S4;
  const bool four = g.act_type == FGQ_U4 || g.act_type == FGQ_S4;
  if (four) return sgn ? launch_tc<4, true>(a, grid, s) : launch_tc<4, false>(a, grid, s);
  return sgn ? launch_tc<8, true>(a, grid, s) : launch_tc<8, false>(a, grid, s);
}

fgq_status launch_wait_timeout_selftest(uint32_t max_iter, unsigned int* err, cudaStream_t s) {
  wait_timeout_selftest_kernel<<<1, 32, 0, s>>>(max_iter, err);
  return after_launch();
}

}  // namespace fgq
