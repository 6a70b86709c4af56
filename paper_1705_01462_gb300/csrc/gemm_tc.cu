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
// Warp roles (288 threads, one CTA per SM, persistent over tiles):
//   warps 0-3  epilogue: thread t owns filter row t of the tile (TMEM lane t); per group
//              tcgen05.ld of the 128 columns, FMA with alpha, at tile end fp32 stores.
//   warps 4-7  loaders/converters: thread t owns activation row t (one output position,
//              implicit im2col) and code row t (one filter) of every K-tile; cp.async
//              copies raw bytes into a 6-deep staging ring, then the thread converts its
//              own rows to fp16 in the 128-byte-swizzled K-major layout the MMA reads.
//   warp 8     MMA issuer (one thread): 4 tcgen05.mma (K = 16) per K-tile.
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
constexpr int TC_NO = 3;          // operand ring depth
constexpr int TC_NS = 6;          // staging ring depth
constexpr int TC_THREADS = 288;
constexpr int TC_TMEM_COLS = 256; // two 128-column fp32 accumulators
constexpr uint32_t TC_WAIT_LIMIT = 1u << 22;

constexpr int OP_TILE = TC_BM * TC_KT * 2;            // 16 KB: one fp16 operand tile
constexpr int OP_STAGE = 2 * OP_TILE;                  // A (codes) + B (activations)
constexpr int ST_ACT = TC_BN * TC_KT;                  // 8 KB raw activation bytes (8-bit)
constexpr int ST_CODE = TC_BM * 16;                    // 2 KB raw code words
constexpr int ST_STAGE = ST_ACT + ST_CODE;
constexpr int SMEM_OP = TC_NO * OP_STAGE;
constexpr int SMEM_ST = TC_NS * ST_STAGE;
constexpr int SMEM_BAR = 8 * (2 * TC_NO + 4 + 1) + 16;
constexpr int TC_SMEM = 1024 + SMEM_OP + SMEM_ST + SMEM_BAR;

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
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + SMEM_OP + SMEM_ST);
  uint64_t* op_full = bars;
  uint64_t* op_empty = bars + TC_NO;
  uint64_t* acc_full = bars + 2 * TC_NO;
  uint64_t* acc_empty = bars + 2 * TC_NO + 2;
  uint64_t* drain_bar = bars + 2 * TC_NO + 4;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * TC_NO + 5);
  volatile uint32_t* abort_flag = tmem_slot + 1;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const Geom& g = a.g;

  if (threadIdx.x == 0) {
    for (int i = 0; i < TC_NO; ++i) {
      mbar_init(&op_full[i], 128);
      mbar_init(&op_empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], 128);
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 8) {
    tmem_alloc(tmem_slot, TC_TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  auto fail = [&]() {
    *abort_flag = 1;
    record_error(a.err, FGQ_ERR_TIMEOUT);
  };

  // ------------------------------------------------------------------ loaders/converters
  if (warp >= 4 && warp < 8) {
    const int t = threadIdx.x - 128;  // row owned in every tile
    const int my_tiles = (a.ntiles - (int)blockIdx.x + (int)gridDim.x - 1) / (int)gridDim.x;
    const int total = my_tiles * a.ktiles;
    constexpr int ACT_BYTES = TC_KT * ABITS / 8;  // 64 (8-bit) or 32 (4-bit) bytes per row
    constexpr int ACT_CHUNKS = ACT_BYTES / 16;

    // issue the copies of this CTA's j-th K-tile into staging slot j % TC_NS
    auto issue = [&](int j) {
      const int tl = j / a.ktiles;
      const int kk = j - tl * a.ktiles;
      int gi, m0;
      int64_t p0;
      tile_coords(a, (int)blockIdx.x + tl * (int)gridDim.x, gi, m0, p0);
      uint8_t* sa = st + (j % TC_NS) * ST_STAGE;
      const uint32_t sact = smem_u32(sa + t * ACT_BYTES);
      const uint32_t scode = smem_u32(sa + ST_ACT + t * 16);
      const int k0 = kk * TC_KT;
      // activation row: output position p0 + t, reduction elements k0 .. k0+63
      const int64_t p = p0 + t;
      const uint8_t* src = a.act;
      int valid_bytes = 0;
      if (p < g.P) {
        const int wo = (int)(p % g.Wo);
        const int64_t q = p / g.Wo;
        const int ho = (int)(q % g.Ho);
        const int b = (int)(q / g.Ho);
        const int tap = k0 / g.Cg;
        const int c0 = k0 - tap * g.Cg;
        const int r = tap / g.S, s = tap - (tap / g.S) * g.S;
        const int hi = ho * g.stride - g.pad + r, wi = wo * g.stride - g.pad + s;
        if (hi >= 0 && hi < g.H && wi >= 0 && wi < g.W) {
          const int64_t e = (((int64_t)b * g.H + hi) * g.W + wi) * g.C + (int64_t)gi * g.Cg + c0;
          src = a.act + e * ABITS / 8;
          const int remain = (g.Cg - c0) * ABITS / 8;  // bytes of this pixel's group channels left
          valid_bytes = remain < ACT_BYTES ? remain : ACT_BYTES;
        }
      }
#pragma unroll
      for (int c = 0; c < ACT_CHUNKS; ++c) {
        int nb = valid_bytes - 16 * c;
        nb = nb < 0 ? 0 : (nb > 16 ? 16 : nb);
        cp_async16(sact + 16 * c, nb ? (const void*)(src + 16 * c) : (const void*)a.act, (uint32_t)nb);
      }
      // code row: filter m0 + t, code words k0/16 .. k0/16 + 3
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
      if (!mbar_wait_or_abort(&op_empty[os], ((j / TC_NO) & 1) ^ 1, a.wait_limit, abort_flag) || *abort_flag) {
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
            uint32_t x = w4[q];
            uint32_t lo = (x & 0x000f000fu) | ((x & 0x00f000f0u) << 4);          // elements 0,1 / 4,5
            uint32_t hi = ((x >> 8) & 0x000f000fu) | (((x >> 8) & 0x00f000f0u) << 4);  // 2,3 / 6,7
            uint32_t b0 = (lo & 0xffffu) | ((hi & 0xffffu) << 16);                // bytes e0 e1 e2 e3
            uint32_t b1 = (lo >> 16) | (hi & 0xffff0000u);                        // bytes e4 e5 e6 e7
            if (SIGNED) { b0 ^= 0x08080808u; b1 ^= 0x08080808u; }
            uint4 o;
            o.x = u8pair_to_h2(b0, 0x4140, bias2); o.y = u8pair_to_h2(b0, 0x4342, bias2);
            o.z = u8pair_to_h2(b1, 0x4140, bias2); o.w = u8pair_to_h2(b1, 0x4342, bias2);
            *reinterpret_cast<uint4*>(Bt + sw128(t, 4 * c + q)) = o;
          }
        }
      }
      // codes -> fp16 row t of A: 64 codes, 8 per 16-byte chunk
      {
        const uint4 cv = *reinterpret_cast<const uint4*>(sa + ST_ACT + t * 16);
        const uint32_t cw[4] = {cv.x, cv.y, cv.z, cv.w};
#pragma unroll
        for (int c = 0; c < 8; ++c) {
          const uint32_t bits = (cw[c / 2] >> (16 * (c & 1))) & 0xffffu;  // 8 codes
          uint32_t h[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const uint32_t c0 = (bits >> (4 * e)) & 3u, c1 = (bits >> (4 * e + 2)) & 3u;
            const uint32_t lo = ((c0 & 1u) * 0x3C00u) | ((c0 & 2u) << 14);
            const uint32_t hi2 = ((c1 & 1u) * 0x3C00u) | ((c1 & 2u) << 14);
            h[e] = lo | (hi2 << 16);
          }
          *reinterpret_cast<uint4*>(A + sw128(t, c)) = make_uint4(h[0], h[1], h[2], h[3]);
        }
      }
      fence_proxy_async_smem();
      mbar_arrive(&op_full[os]);
    }
    cp_async_wait_all();
  }

  // ------------------------------------------------------------------ MMA issuer
  if (warp == 8 && lane == 0) {
    const uint32_t idesc = idesc_f16_f32(TC_BM, TC_BN);
    const int my_tiles = (a.ntiles - (int)blockIdx.x + (int)gridDim.x - 1) / (int)gridDim.x;
    const uint32_t op_base = smem_u32(op);
    int kt = 0, gc = 0;
    bool ok = true;
    for (int tl = 0; tl < my_tiles && ok; ++tl) {
      for (int grp = 0; grp < g.ng && ok; ++grp, ++gc) {
        const int b = gc & 1;
        if (!mbar_wait_or_abort(&acc_empty[b], ((gc >> 1) & 1) ^ 1, a.wait_limit, abort_flag) || *abort_flag) {
          if (!*abort_flag) fail();
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + (uint32_t)(b * TC_BN);
        for (int sub = 0; sub < a.kt_per_group; ++sub, ++kt) {
          const int os = kt % TC_NO;
          if (!mbar_wait_or_abort(&op_full[os], (kt / TC_NO) & 1, a.wait_limit, abort_flag) || *abort_flag) {
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
  if (warp < 4) {
    const int t = threadIdx.x;  // TMEM lane = filter row of the tile
    const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
    const float sx = __ldg(a.act_scale);
    const int my_tiles = (a.ntiles - (int)blockIdx.x + (int)gridDim.x - 1) / (int)gridDim.x;
    int gc = 0;
    bool ok = true;
    for (int tl = 0; tl < my_tiles && ok; ++tl) {
      int gi, m0;
      int64_t p0;
      tile_coords(a, (int)blockIdx.x + tl * (int)gridDim.x, gi, m0, p0);
      const int m = m0 + t;
      const bool mok = m < gi * g.Mg + g.Mg && m < g.M;
      const float* arow = a.alpha + (int64_t)(mok ? m : 0) * g.ng;
      float acc[TC_BN];
#pragma unroll
      for (int j = 0; j < TC_BN; ++j) acc[j] = 0.0f;
      for (int grp = 0; grp < g.ng; ++grp, ++gc) {
        const int b = gc & 1;
        const float al = mok ? __ldg(arow + grp) : 0.0f;
        if (!mbar_wait_or_abort(&acc_full[b], (gc >> 1) & 1, a.wait_limit, abort_flag) || *abort_flag) {
          if (!*abort_flag) fail();
          ok = false;
          break;
        }
        tc_fence_after();
#pragma unroll
        for (int c = 0; c < TC_BN / 32; ++c) {
          uint32_t r[32];
          tmem_ld32(tmem + lane_base + (uint32_t)(b * TC_BN + 32 * c), r);
          tmem_ld_wait();
#pragma unroll
          for (int j = 0; j < 32; ++j) acc[32 * c + j] = fmaf(al, __uint_as_float(r[j]), acc[32 * c + j]);
        }
        tc_fence_before();
        mbar_arrive(&acc_empty[b]);
      }
      if (!ok) break;
      if (mok) {
#pragma unroll
        for (int j = 0; j < TC_BN; ++j) {
          const int64_t p = p0 + j;
          if (p < g.P) a.out[p * g.M + m] = sx * acc[j];
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 8) {
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
