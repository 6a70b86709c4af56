// CUDA-core grouped ternary contraction (Eq. 2, 32-bit group accumulators of Section 4):
// the dispatcher over the tiled dp4a kernel (gemm_simt_kernel.cuh, instantiated per group
// size in gemm_simt_g*.cu) and the plain one-thread-per-output kernel used for G = 1 and 2.
#include <cstdint>

#include "gemm_simt_kernel.cuh"

namespace fgq {
namespace {

// Plain reference-style kernel for any G (used for G = 1 and 2): one thread per output.
__global__ void simple_contract_kernel(const uint8_t* __restrict__ act, const Geom g,
                                       const uint32_t* __restrict__ codes, const float* __restrict__ alpha,
                                       const float* __restrict__ act_scale, float* __restrict__ out,
                                       int32_t* __restrict__ sums) {
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= g.P * g.M) return;
  const int m = (int)(idx % g.M);
  const int64_t p = idx / g.M;
  const int gi = m / g.Mg;
  const PosInfo pi = pos_info(g, p);
  float acc = 0.0f;
  for (int gg = 0; gg < g.ng; ++gg) {
    int s = 0;
    for (int j = gg * g.G; j < (gg + 1) * g.G && j < g.Kred; ++j) {
      const uint32_t code = (codes[(int64_t)m * g.wrow + j / 16] >> (2 * (j % 16))) & 3u;
      if (code == 0) continue;
      int a = (int)act_byte(act, g.act_type, act_elem(g, pi, gi, j));
      if (g.act_type == FGQ_S8 || g.act_type == FGQ_S4) a = (int)(int8_t)(uint8_t)a;
      s += code == 1u ? a : -a;
    }
    if (sums) sums[((int64_t)m * g.ng + gg) * g.P + p] = s;
    else acc = fmaf(alpha[(int64_t)m * g.ng + gg], (float)s, acc);
  }
  if (sums) return;
  const float v = acc * act_scale[0];
  if (g.rq_out)
    g.rq_out[p * g.M + m] = rq_code(v, rq_mul(g.rq_scale, g.rq_signed));
  else
    out[p * g.M + m] = v;
}


bool launch_g(bool sa, bool sums, const void* act, const Geom& g, const void* w, const float* sc, const float* as,
              float* out, int32_t* sums_out, int mode, cudaStream_t s) {
  switch (g.G) {
    case 4: return simt_launch_g4(sa, sums, act, g, w, sc, as, out, sums_out, mode, s);
    case 8:
    case 16: return simt_launch_g8_16(sa, sums, act, g, w, sc, as, out, sums_out, mode, s);
    case 32:
    case 64: return simt_launch_g32_64(sa, sums, act, g, w, sc, as, out, sums_out, mode, s);
    case 128: return simt_launch_g128(sa, sums, act, g, w, sc, as, out, sums_out, mode, s);
  }
  return false;
}

}  // namespace

fgq_status launch_simt_contract(const void* act, const Geom& g, const void* weights, const float* scales,
                                int dense, const float* act_scale, float* out, int32_t* sums, cudaStream_t s) {
  if (g.P == 0 || g.M == 0) return FGQ_OK;
  const bool is4 = g.act_type == FGQ_U4 || g.act_type == FGQ_S4;
  const bool sa = g.act_type == FGQ_S8 || g.act_type == FGQ_S4;
  // gather mode: whole words inside one tap need Cg % 4 == 0 (and alignment of the words)
  int mode = 2;
  if (g.Cg % 4 == 0 && g.C % 4 == 0) mode = is4 ? 1 : 0;
  // 8-bit activations whose per-thread staging run (32 elements; 64 when G = 128) stays in
  // one tap and starts 16-byte aligned
  const int run = (g.G == 128) ? 64 : 32;
  if (!is4 && !dense && g.G >= 4 && g.Cg % run == 0 && g.C % 16 == 0) mode = 3;
  // byte gathers driven by a per-block (tap, channel) table while it fits in shared memory
  if (mode == 2 && g.Kp <= 8192) mode = 4;
  if (!dense && (g.G == 1 || g.G == 2)) {
    const int64_t n = g.P * g.M;
    simple_contract_kernel<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(
        static_cast<const uint8_t*>(act), g, static_cast<const uint32_t*>(weights), scales, act_scale, out, sums);
    return after_launch();
  }
  if (dense) {
    simt_launch_dense(sa, act, g, weights, scales, act_scale, out, mode, s);
    return after_launch();
  }
  if (!launch_g(sa, sums != nullptr, act, g, weights, scales, act_scale, out, sums, mode, s))
    return FGQ_ERR_UNSUPPORTED;
  return after_launch();
}

}  // namespace fgq
