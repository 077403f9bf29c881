// Failure-detection self-test: one CTA waits on an mbarrier phase that
// nothing completes (an expected transaction count with no copy behind it),
// so the bounded wait every walk kernel uses gives up, records
// kErrWaitTimeout and returns.  No fault, trap or endless loop: the CTA
// exits normally and the context stays usable.
#include "walk.cuh"

namespace mlt {
namespace {

__global__ void __launch_bounds__(32) k_wait_selftest(unsigned* err, unsigned long long limit_ns) {
  __shared__ __align__(8) unsigned long long bar;
  const uint32_t b = walk::smem_u32(&bar);
  if (threadIdx.x == 0) {
    walk::mbar_init(b, 1);
    walk::fence_mbar_init();
  }
  __syncwarp();
  // the only arrival expects 16 bytes that no copy will deliver
  if (threadIdx.x == 0) walk::mbar_expect_tx(b, 16u);
  __syncwarp();
  const bool ok = walk::mbar_wait_bounded_ns(b, 0u, limit_ns);
  if (!__any_sync(0xFFFFFFFFu, ok) && threadIdx.x == 0) atomicOr(err, kErrWaitTimeout);
}

}  // namespace

cudaError_t launch_wait_selftest(unsigned* err, unsigned long long limit_ns, cudaStream_t st) {
  k_wait_selftest<<<1, 32, 0, st>>>(err, limit_ns);
  return cudaGetLastError();
}

}  // namespace mlt
