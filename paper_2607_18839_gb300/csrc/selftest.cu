// selftest.cu -- exercises the bounded waits of the kernels without a fault:
// one warp waits on an mbarrier phase that nothing completes and on a
// shared-memory flag that nothing sets, each with a short limit, and records
// HPD_DEVERR_TIMEOUT in the workspace error word when a wait gives up.  The
// kernel then returns normally, so the context stays usable.
#include "common.cuh"
#include "sm100.cuh"

namespace hpd {
namespace {

using namespace sm100;

__global__ void __launch_bounds__(32, 1) wait_selftest_kernel(uint32_t *err, uint64_t limit_ns) {
  __shared__ __align__(8) uint64_t never;
  __shared__ int flag;
  const int lane = threadIdx.x & 31;
  if (lane == 0) {
    mbar_init(smem_u32(&never), 1);
    fence_mbar_init();
    flag = 0;
  }
  __syncwarp();
  // nothing arrives: the phase with parity 0 never completes
  if (!__all_sync(0xffffffffu, mbar_wait(smem_u32(&never), 0, nullptr, limit_ns)) && lane == 0)
    flag_error(err, HPD_DEVERR_TIMEOUT);
  // nothing sets the flag: a bounded spin gives up as well
  const uint64_t t0 = globaltimer();
  bool seen = false;
  for (uint32_t i = 0; !seen; ++i) {
    seen = *reinterpret_cast<volatile int *>(&flag) != 0;
    if (!seen && (i & 63u) == 63u && globaltimer() - t0 > limit_ns) break;
  }
  if (!__all_sync(0xffffffffu, seen) && lane == 0) atomicOr(err, HPD_DEVERR_TIMEOUT << 8);
}

}  // namespace

cudaError_t launch_wait_selftest(uint32_t *err, uint64_t limit_ns, cudaStream_t s) {
  wait_selftest_kernel<<<1, 32, 0, s>>>(err, limit_ns);
  return cudaGetLastError();
}

}  // namespace hpd
