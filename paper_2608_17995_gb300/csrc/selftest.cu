// selftest.cu — a test hook for the failure detection of the bounded waits.
//
// Every spin in the path's kernels is an mbarrier wait bounded by a wall-clock
// limit; on expiry it records AVITS_ERR_TIMEOUT in the status word and sets the
// CTA's abort flag, which ends the waits of the other roles.  This kernel runs
// exactly that code on barriers nothing ever arrives at, so the path can be
// checked on a GPU without a fault: warp 0 waits with the given limit, warp 1
// waits on another barrier with a hundred times that limit and must give up as
// soon as warp 0 raises the abort flag.  The kernel returns normally.
#include "avits_common.cuh"
#include "avits_internal.h"

namespace avits {
namespace {

__global__ void __launch_bounds__(64) wait_selftest_kernel(unsigned long long limit_ns,
                                                           long long* result, unsigned int* st) {
  __shared__ uint64_t bar[2];
  __shared__ int abort_flag;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    mbar_init(&bar[0], 1);
    mbar_init(&bar[1], 1);
    abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  if (lane == 0) {
    const unsigned long long t0 = globaltimer_ns();
    const bool ok = warp == 0 ? mbar_wait_bounded(&bar[0], 0, &abort_flag, st, limit_ns)
                              : mbar_wait_bounded(&bar[1], 0, &abort_flag, st, 100ull * limit_ns);
    result[2 * warp] = ok ? 1 : 0;
    result[2 * warp + 1] = (long long)(globaltimer_ns() - t0);
  }
  __syncthreads();
  if (threadIdx.x == 0) result[4] = abort_flag;
}

}  // namespace

cudaError_t launch_wait_selftest(unsigned long long limit_ns, long long* result,
                                 unsigned int* status, cudaStream_t s) {
  wait_selftest_kernel<<<1, 64, 0, s>>>(limit_ns, result, status);
  return cudaGetLastError();
}

}  // namespace avits
