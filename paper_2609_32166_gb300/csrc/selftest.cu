// Self-test of the failure path every kernel's waits share: one thread
// waits on an mbarrier with the bounded wait of pf_ptx.cuh.  Unsignalled,
// nothing ever arrives, so the wait runs out after limit_ns, flags
// PF_DEVERR_TIMEOUT and the kernel returns normally (no trap, the context
// stays usable); signalled, the barrier's phase completes first.
#include "pf_internal.h"
#include "pf_ptx.cuh"

namespace pf {

namespace {

__global__ void selftest_wait_kernel(int32_t* err, unsigned long long limit_ns, int signal,
                                     int32_t* waited_ok) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x != 0) return;
  mbar_init(smem_u32(&bar), 1);
  fence_mbar_init();
  if (signal) mbar_arrive(smem_u32(&bar));
  const bool ok = mbar_wait_limit(smem_u32(&bar), 0, err, limit_ns);
  *waited_ok = ok ? 1 : 0;
}

}  // namespace

cudaError_t launch_selftest_wait(int32_t* err, unsigned long long limit_ns, int signal,
                                 int32_t* waited_ok, cudaStream_t s) {
  selftest_wait_kernel<<<1, 32, 0, s>>>(err, limit_ns, signal, waited_ok);
  return cudaGetLastError();
}

}  // namespace pf
