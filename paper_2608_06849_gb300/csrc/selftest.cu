// Self-test of the bounded waits that every kernel of the library uses: one
// warp waits on an mbarrier that nothing ever arrives at, with a short
// limit. The wait gives up when the limit runs out, records the timeout in
// the error word and raises the CTA's abort flag, exactly as a kernel whose
// producer or MMA partner stalled would; the kernel then returns and the
// context stays usable. No GPU fault, trap or hang is involved.
#include "common.cuh"
#include "internal.h"

namespace aoh {
namespace {

__global__ void wait_selftest_kernel(uint32_t* err, uint64_t limit_ns, unsigned long long* elapsed_ns) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);  // one arrival that never comes
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  const uint64_t t0 = globaltimer_ns();
  const bool ok = wait_bar(&bar, 0, err, &abort_flag, limit_ns);
  const bool all = __all_sync(0xffffffffu, ok);
  if (threadIdx.x == 0) *elapsed_ns = all ? 0ull : (unsigned long long)(globaltimer_ns() - t0);
}

}  // namespace

cudaError_t launch_wait_selftest(uint32_t* err, uint64_t limit_ns, unsigned long long* elapsed_ns, cudaStream_t s) {
  wait_selftest_kernel<<<1, 32, 0, s>>>(err, limit_ns, elapsed_ns);
  return cudaGetLastError();
}

}  // namespace aoh
