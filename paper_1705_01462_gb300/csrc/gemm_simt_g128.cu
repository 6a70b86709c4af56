// Instantiations of the tiled dp4a contraction kernel for G in {128}.
#include "gemm_simt_kernel.cuh"

namespace fgq {

bool simt_launch_g128(bool sa, bool sums, const void* act, const Geom& g, const void* w, const float* sc, const float* as,
                      float* out, int32_t* sums_out, int mode, cudaStream_t s) {
  switch (g.G) {
    case 128:
      if (sums) sa ? launch_one<128, true, false, true>(act, g, w, sc, as, out, sums_out, mode, s)
                : launch_one<128, false, false, true>(act, g, w, sc, as, out, sums_out, mode, s);
      else sa ? launch_one<128, true, false, false>(act, g, w, sc, as, out, sums_out, mode, s)
              : launch_one<128, false, false, false>(act, g, w, sc, as, out, sums_out, mode, s);
      return true;
  }
  return false;
}

}  // namespace fgq
