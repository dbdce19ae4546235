// A recorded refine pass repeated on the GPU until no confident edit remains.
//
// The refiner runs passes until none of them changes a token any more or a
// pass budget is spent (early stop when no confident edits remain, Appendix
// C.4 / Table 11). The loop is a CUDA graph with a conditional WHILE node: its
// body is the caller's recorded pass (stream capture straight into the body
// graph) followed by loop_cond_kernel, which counts the pass and sets the
// node's condition from the pass's edit counts on the device, so a whole
// multi-pass refinement is one graph launch with no host round trip between
// passes.
#include <cstdint>

#include "dlm_internal.h"

namespace dlm {
namespace {

constexpr int kCondThreads = 256;

__global__ void loop_init_kernel(int32_t* steps) { *steps = 0; }

// Error-word bits that end the loop: a bounded wait that gave up, a NaN
// confidence, an input outside its contract -- the pass's outputs are then
// undefined. A clamped sequence or prompt length (DLM_DEVERR_LENGTH) does
// not: the kernels define the clamped result, so the pass is valid.
constexpr int kStopBits = ~DLM_DEVERR_LENGTH;

// Ends one pass: steps += 1; run another pass iff steps < max_steps, some
// sequence had an edit (n_edits[b] > 0) and no kernel has set a bit of
// kStopBits in the device error word.
__global__ void __launch_bounds__(kCondThreads)
    loop_cond_kernel(cudaGraphConditionalHandle handle, const int32_t* n_edits, int64_t batch, int32_t max_steps,
                     int32_t* steps, const int* err) {
  __shared__ int any_warp[kCondThreads / 32];
  int any = 0;
  for (int64_t b = threadIdx.x; b < batch; b += kCondThreads) any |= n_edits[b] > 0;
  any = __any_sync(0xffffffffu, any);
  if ((threadIdx.x & 31) == 0) any_warp[threadIdx.x >> 5] = any;
  __syncthreads();
  if (threadIdx.x == 0) {
    int edits = 0;
    for (int w = 0; w < kCondThreads / 32; ++w) edits |= any_warp[w];
    const int n = *steps + 1;
    *steps = n;
    const bool failed = (*reinterpret_cast<const volatile int*>(err) & kStopBits) != 0;
    cudaGraphSetConditional(handle, (n < max_steps && edits && !failed) ? 1u : 0u);
  }
}

// The loop being recorded on this thread (between dlm_loop_begin and dlm_loop_end).
struct Pending {
  cudaGraph_t graph = nullptr;
  cudaGraphConditionalHandle handle = 0;
  cudaStream_t stream = nullptr;
  int32_t* steps = nullptr;
};
thread_local Pending t_pending;

}  // namespace
}  // namespace dlm

struct dlm_loop {
  cudaGraph_t graph;
  cudaGraphExec_t exec;
};

extern "C" {

int dlm_loop_begin(int32_t* steps_out) {
  using dlm::fail;
  dlm::clear_error();
  cudaStream_t stream = dlm::current_stream();
  if (dlm::t_pending.graph) return fail(DLM_ERR_ARG, "a loop is already being recorded on this thread");
  if (!stream) return fail(DLM_ERR_ARG, "record a loop on a created stream (dlm_set_stream), not the legacy default");
  if (!steps_out) return fail(DLM_ERR_NULL, "steps_out is NULL");
  if (reinterpret_cast<uintptr_t>(steps_out) % 4 != 0) return fail(DLM_ERR_ALIGN, "steps_out not 4-byte aligned");
  cudaStreamCaptureStatus cs;
  cudaError_t e = cudaStreamIsCapturing(stream, &cs);
  if (e != cudaSuccess) return fail(DLM_ERR_CUDA, "cudaStreamIsCapturing: %s", cudaGetErrorString(e));
  if (cs != cudaStreamCaptureStatusNone) return fail(DLM_ERR_ARG, "the stream is already capturing");
  // Set-up that must not happen during the capture: the device addresses of
  // the error word and of the static step scratch (cudaGetSymbolAddress).
  if (!dlm::device_error_word()) return fail(DLM_ERR_CUDA, "device error word unavailable");
  int32_t* scratch = nullptr;
  if (const int st = dlm::static_step_scratch(&scratch)) return st;

  cudaGraph_t g = nullptr;
  if ((e = cudaGraphCreate(&g, 0)) != cudaSuccess)
    return fail(DLM_ERR_CUDA, "cudaGraphCreate: %s", cudaGetErrorString(e));
  auto bail = [&](const char* what) {
    cudaGraphDestroy(g);
    return fail(DLM_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
  };
  cudaGraphConditionalHandle handle;
  if ((e = cudaGraphConditionalHandleCreate(&handle, g, 1, cudaGraphCondAssignDefault)) != cudaSuccess)
    return bail("cudaGraphConditionalHandleCreate");
  // steps = 0, then WHILE (condition) { pass; loop_cond_kernel }.
  cudaKernelNodeParams kp = {};
  void* init_args[] = {&steps_out};
  kp.func = reinterpret_cast<void*>(dlm::loop_init_kernel);
  kp.gridDim = dim3(1);
  kp.blockDim = dim3(1);
  kp.kernelParams = init_args;
  cudaGraphNode_t n_init;
  if ((e = cudaGraphAddKernelNode(&n_init, g, nullptr, 0, &kp)) != cudaSuccess) return bail("adding the init node");
  cudaGraphNodeParams cp = {};
  cp.type = cudaGraphNodeTypeConditional;
  cp.conditional.handle = handle;
  cp.conditional.type = cudaGraphCondTypeWhile;
  cp.conditional.size = 1;
  cudaGraphNode_t n_while;
  if ((e = cudaGraphAddNode(&n_while, g, &n_init, nullptr, 1, &cp)) != cudaSuccess)
    return bail("adding the loop node");
  cudaGraph_t body = cp.conditional.phGraph_out[0];
  if ((e = cudaStreamBeginCaptureToGraph(stream, body, nullptr, nullptr, 0, cudaStreamCaptureModeThreadLocal)) !=
      cudaSuccess)
    return bail("cudaStreamBeginCaptureToGraph");
  dlm::t_pending.graph = g;
  dlm::t_pending.handle = handle;
  dlm::t_pending.stream = stream;
  dlm::t_pending.steps = steps_out;
  return DLM_OK;
}

int dlm_loop_end(const int32_t* n_edits, int64_t batch, int32_t max_steps, dlm_loop** loop) {
  using dlm::fail;
  dlm::clear_error();
  dlm::Pending pend = dlm::t_pending;
  if (!pend.graph) return fail(DLM_ERR_ARG, "no loop is being recorded on this thread");
  dlm::t_pending = dlm::Pending();
  int st = DLM_OK;
  if (!loop) st = fail(DLM_ERR_NULL, "loop is NULL");
  else if (batch < 0) st = fail(DLM_ERR_SHAPE, "batch < 0");
  else if (batch > 0 && !n_edits) st = fail(DLM_ERR_NULL, "n_edits is NULL");
  else if (reinterpret_cast<uintptr_t>(n_edits) % 4 != 0) st = fail(DLM_ERR_ALIGN, "n_edits not 4-byte aligned");
  else if (max_steps < 1) st = fail(DLM_ERR_ARG, "max_steps must be >= 1");
  if (st == DLM_OK) {
    dlm::loop_cond_kernel<<<1, dlm::kCondThreads, 0, pend.stream>>>(pend.handle, n_edits, batch, max_steps,
                                                                      pend.steps, dlm::device_error_word());
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) st = fail(DLM_ERR_CUDA, "loop condition launch: %s", cudaGetErrorString(e));
  }
  // The capture ends on every path, so the stream is usable again.
  cudaGraph_t captured = nullptr;
  cudaError_t e = cudaStreamEndCapture(pend.stream, &captured);
  if (st == DLM_OK && e != cudaSuccess)
    st = fail(DLM_ERR_CUDA, "the recorded pass could not be captured: %s", cudaGetErrorString(e));
  cudaGraphExec_t exec = nullptr;
  if (st == DLM_OK && (e = cudaGraphInstantiate(&exec, pend.graph, 0)) != cudaSuccess)
    st = fail(DLM_ERR_CUDA, "cudaGraphInstantiate: %s", cudaGetErrorString(e));
  if (st != DLM_OK) {
    cudaGraphDestroy(pend.graph);
    return st;
  }
  *loop = new dlm_loop{pend.graph, exec};
  return DLM_OK;
}

int dlm_loop_cancel(void) {
  dlm::clear_error();
  dlm::Pending pend = dlm::t_pending;
  if (!pend.graph) return DLM_OK;
  dlm::t_pending = dlm::Pending();
  cudaGraph_t captured = nullptr;
  cudaStreamEndCapture(pend.stream, &captured);
  cudaGetLastError();  // an invalidated capture reports its error here; nothing is kept
  cudaGraphDestroy(pend.graph);
  return DLM_OK;
}

int dlm_loop_launch(dlm_loop* loop) {
  using dlm::fail;
  dlm::clear_error();
  if (!loop) return fail(DLM_ERR_NULL, "loop is NULL");
  cudaError_t e = cudaGraphLaunch(loop->exec, dlm::current_stream());
  if (e != cudaSuccess) return fail(DLM_ERR_CUDA, "cudaGraphLaunch: %s", cudaGetErrorString(e));
  return DLM_OK;
}

int dlm_loop_destroy(dlm_loop* loop) {
  using dlm::fail;
  dlm::clear_error();
  if (!loop) return DLM_OK;
  cudaError_t e1 = cudaGraphExecDestroy(loop->exec);
  cudaError_t e2 = cudaGraphDestroy(loop->graph);
  delete loop;
  if (e1 != cudaSuccess || e2 != cudaSuccess)
    return fail(DLM_ERR_CUDA, "destroying the loop graph: %s", cudaGetErrorString(e1 != cudaSuccess ? e1 : e2));
  return DLM_OK;
}

}  // extern "C"
