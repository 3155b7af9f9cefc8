// Self-test of the failure path that every TMA / tcgen05 / bulk-copy kernel of the library shares:
// a wait on an mbarrier phase is a bounded loop of try_wait polls, and a wait that gives up raises
// VARRATE_ERR_TIMEOUT in the device status word and lets the kernel return, so the context stays
// usable and the host learns of it from the status word (no trap, no fault, no endless loop).
//
// The kernel waits on an mbarrier whose phase nothing completes (no arrival, no copy in flight), so
// the wait always runs out after `polls` polls. No copy is in flight when it returns, so nothing can
// land in shared memory after the block has exited.
#include "common.cuh"
#include "kernels.h"
#include "varrate.h"

namespace vr {

namespace {

__global__ void wait_timeout_kernel(int32_t* __restrict__ dev_status, uint32_t polls) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) mbar_init(&bar, 1);   // one arrival expected; none ever comes
  fence_mbar_init();
  __syncthreads();
  const bool done = mbar_wait_bounded(&bar, 0u, polls);
  if (!done && threadIdx.x == 0) raise_status(dev_status, VARRATE_ERR_TIMEOUT);
}

}  // namespace

}  // namespace vr

extern "C" varrate_status varrate_selftest_wait_timeout(int32_t* dev_status, uint32_t polls, void* stream) {
  if (dev_status == nullptr || polls == 0 || polls > (1u << 24)) return VARRATE_ERR_ARG;
  if ((reinterpret_cast<uintptr_t>(dev_status) & 3u) != 0) return VARRATE_ERR_ARG;
  vr::wait_timeout_kernel<<<1, 32, 0, (cudaStream_t)stream>>>(dev_status, polls);
  return cudaGetLastError() == cudaSuccess ? VARRATE_OK : VARRATE_ERR_CUDA;
}
