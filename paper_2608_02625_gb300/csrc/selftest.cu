// Self-test of the bounded wait that every pipelined kernel of the library
// relies on (not a step of the method).
//
// The kernels' producer / consumer hand-offs wait on mbarriers through
// mbar_wait_for, which gives up after a wall-clock budget, records
// DLM_DEVERR_TIMEOUT in the device error word and returns, so a pipeline
// whose producer never arrives still ends and leaves the context usable.
// wait_timeout_kernel makes that happen on purpose, without a pipeline
// around it: one thread waits on a freshly initialised mbarrier on which
// nothing ever arrives, so only the budget can end the wait.
#include <cstdint>

#include "dlm_common.cuh"
#include "dlm_internal.h"

namespace dlm {
namespace {

__global__ void __launch_bounds__(32) wait_timeout_kernel(uint64_t budget_ns, int* err) {
  __shared__ uint64_t bar;
  __shared__ int abort;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);  // one arrival expected, none will come
    abort = 0;
    fence_mbar_init();
  }
  __syncthreads();
  // Phase 0 of a new barrier completes only on its arrival.
  if (threadIdx.x == 0) mbar_wait_for(&bar, 0, &abort, err, budget_ns);
}

}  // namespace
}  // namespace dlm

extern "C" int dlm_selftest_wait_timeout(int64_t budget_ns) {
  using dlm::fail;
  dlm::clear_error();
  if (budget_ns < 1000 || budget_ns > 1000000000LL)
    return fail(DLM_ERR_ARG, "budget_ns %lld outside [1e3, 1e9]", static_cast<long long>(budget_ns));
  int* err = dlm::device_error_word();
  if (!err) return fail(DLM_ERR_CUDA, "device error word unavailable on this device");
  dlm::wait_timeout_kernel<<<1, 32, 0, dlm::current_stream()>>>(static_cast<uint64_t>(budget_ns), err);
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return fail(DLM_ERR_CUDA, "wait_timeout_kernel launch: %s", cudaGetErrorString(e));
  return DLM_OK;
}
