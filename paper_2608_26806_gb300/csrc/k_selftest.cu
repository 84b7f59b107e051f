// Check of the bounded-wait failure path: a wait on an mbarrier that nothing arrives
// on gives up after the requested time and is reported through the status word, the
// same way the pipeline kernels report a TMA copy or an MMA commit that never lands.
#include "avtp_tc.cuh"

namespace avtp {
namespace {

__global__ void __launch_bounds__(64) k_wait_selftest(DevStatus* st, uint64_t limit_ns, int arrive) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x == 0) {
    tc::mbar_init(&bar, 1);
    tc::fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    if (arrive) tc::mbar_arrive(&bar);
    if (!tc::mbar_wait(&bar, 0, limit_ns)) record_error(st, AVTP_ERR_TIMEOUT, 0);
  } else if (threadIdx.x >= 32) {
    const bool ok = tc::mbar_wait_warp(&bar, 0, limit_ns);
    if (!ok && threadIdx.x == 32) record_error(st, AVTP_ERR_TIMEOUT, 1);
  }
}

}  // namespace

cudaError_t launch_wait_selftest(uint64_t limit_ns, int arrive, void* ws, cudaStream_t s) {
  k_wait_selftest<<<1, 64, 0, s>>>(static_cast<DevStatus*>(ws), limit_ns, arrive);
  return cudaGetLastError();
}

}  // namespace avtp
