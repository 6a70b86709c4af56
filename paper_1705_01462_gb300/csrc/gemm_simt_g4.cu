// Instantiations of the tiled dp4a contraction kernel for G = 4 and the dense 8-bit-weight mode.
#include "gemm_simt_kernel.cuh"

namespace fgq {

bool simt_launch_g4(bool sa, bool sums, const void* act, const Geom& g, const void* w, const float* sc, const float* as,
                    float* out, int32_t* sums_out, int mode, cudaStream_t s) {
  switch (g.G) {
    case 4:
      if (sums) sa ? launch_one<4, true, false, true>(act, g, w, sc, as, out, sums_out, mode, s)
                : launch_one<4, false, false, true>(act, g, w, sc, as, out, sums_out, mode, s);
      else sa ? launch_one<4, true, false, false>(act, g, w, sc, as, out, sums_out, mode, s)
              : launch_one<4, false, false, false>(act, g, w, sc, as, out, sums_out, mode, s);
      return true;
  }
  return false;
}

void simt_launch_dense(bool sa, const void* act, const Geom& g, const void* w, const float* sc, const float* as,
                       float* out, int mode, cudaStream_t s) {
  if (sa) launch_one<4, true, true, false>(act, g, w, sc, as, out, nullptr, mode, s);
  else launch_one<4, false, true, false>(act, g, w, sc, as, out, nullptr, mode, s);
}

}  // namespace fgq
