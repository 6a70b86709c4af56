// Tensor-core (tcgen05) grouped ternary contraction and the bounded-wait self test.
#include <cstdint>

#include "fgq_device.cuh"
#include "ptx_sm100.cuh"

namespace fgq {
namespace {

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

bool tc_supports(const Geom&) { return false; }

fgq_status launch_tc_contract(const void*, const Geom&, const uint32_t*, const float*, const float*, float*,
                              int32_t*, unsigned int*, cudaStream_t) {
  return FGQ_ERR_UNSUPPORTED;
}

fgq_status launch_wait_timeout_selftest(uint32_t max_iter, unsigned int* err, cudaStream_t s) {
  wait_timeout_selftest_kernel<<<1, 32, 0, s>>>(max_iter, err);
  return after_launch();
}

}  // namespace fgq
