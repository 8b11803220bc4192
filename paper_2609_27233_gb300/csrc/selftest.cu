// Self-test of the library's bounded waits (not part of the method): every
// wait on another agent (an mbarrier completed by TMA or tcgen05, a counter
// raised by another CTA) gives up after a time limit, records
// UMIM_ERR_TIMEOUT and lets the kernel return, so a stalled producer leaves
// an error status instead of a hung GPU.  This kernel waits, with the
// caller's limit, on something that never happens -- an mbarrier nobody
// arrives on, or a counter nobody raises -- and reports the outcome.
#include "common.cuh"

namespace umim {
namespace {

__global__ void selftest_wait_kernel(int which, uint64_t limit_ns, const int32_t *flags, uint64_t *elapsed,
                                     int32_t *status) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x != 0) return;
  const uint64_t t0 = globaltimer();
  const bool ok = which == 0 ? mbar_wait_for(&bar, 0, limit_ns)              // no arrival ever
                             : wait_count_for(flags, 1, flags + 1, limit_ns);   // counter stays 0
  if (elapsed) *elapsed = globaltimer() - t0;
  if (!ok) set_error(status, UMIM_ERR_TIMEOUT);
}

__global__ void selftest_bounds_kernel(int32_t *buf, int64_t n, int64_t index, int32_t *status) {
  if (in_bounds(index, n, status, kSiteSelftest)) buf[index] = 1;
}

}  // namespace

umim_status selftest_bounds_check(int32_t *buf, int64_t n, int64_t index, int32_t *status, cudaStream_t stream) {
  // without the check the store would go wherever index points
  if (!kDebugChecks) return UMIM_ERR_UNSUPPORTED;
  selftest_bounds_kernel<<<1, 1, 0, stream>>>(buf, n, index, status);
  return cudaGetLastError() == cudaSuccess ? UMIM_OK : UMIM_ERR_CUDA;
}

umim_status selftest_bounded_wait(int which, uint32_t limit_us, const int32_t *flags, uint64_t *elapsed,
                                  int32_t *status, cudaStream_t stream) {
  selftest_wait_kernel<<<1, 32, 0, stream>>>(which, (uint64_t)limit_us * 1000ull, flags, elapsed, status);
  return cudaGetLastError() == cudaSuccess ? UMIM_OK : UMIM_ERR_CUDA;
}

}  // namespace umim
