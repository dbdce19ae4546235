// Step A3 -- the refine update (commit / edit / remask), one CTA per sequence.
// The per-sequence algorithm is in update_impl.cuh (Sec. 4.2; token editing
// with confident edits, Appendix C.4 / Table 11).
#include "update_impl.cuh"

namespace dlm {
namespace {

constexpr int kThreads = 512;

__global__ void __launch_bounds__(kThreads) refine_update_kernel(UpdateArgs a, int* err) {
  __shared__ UpdateShared<kThreads> sh;
  refine_sequence<kThreads, false>(a, blockIdx.x, err, sh);
}

}  // namespace

int launch_refine_update(const UpdateArgs& a, cudaStream_t stream) {
  if (a.B == 0) return DLM_OK;
  refine_update_kernel<<<a.B, kThreads, 0, stream>>>(a, device_error_word());
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return fail(DLM_ERR_CUDA, "refine_update launch: %s", cudaGetErrorString(e));
  return DLM_OK;
}

}  // namespace dlm
