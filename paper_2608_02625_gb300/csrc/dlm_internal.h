// Host-side interfaces between the C ABI layer (dlm_api.cu) and the kernel
// launchers. Arguments here are already validated.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "dlmrefine.h"

namespace dlm {

// Device address of the error word of the current device (set up once per device).
int* device_error_word();

// Budget of each bounded wait in the pipelined kernels (ns): 2 s, which no
// legitimate wait inside one launch approaches. Only DLM_CHECK_BOUNDS builds
// can change it (dlm_checked_set_wait_budget), to make waits run out in tests.
constexpr uint64_t kDefaultWaitBudgetNs = 2000000000ull;
uint64_t wait_budget_ns();
// Query tiles per attention work unit set on this thread (0: automatic).
int attn_tiles_per_unit();

// Device address of dlm_refine_step_static's scratch array on the current
// device (set up on first use; a status, with *out untouched, on failure).
int static_step_scratch(int32_t** out);

// Records a failure message for dlm_last_error() and returns `status`.
int fail(int status, const char* fmt, ...);
// Clears the calling thread's failure message (at the start of every entry point).
void clear_error();
// The calling thread's stream (dlm_set_stream).
cudaStream_t current_stream();

struct AttnArgs {
  const void* q;
  const void* k;
  const void* v;
  void* out;
  const int32_t* seq_lens;  // may be null: n_b = L
  const int32_t* prompt_lens;  // may be null: p_b = 0 (block masks only)
  int mask_mode, block;        // DLM_ATTN_* and the block size (block masks)
  int B, L, Hq, Hkv, D;
  // strides in elements, (b, l, h) order; the innermost stride is 1
  int64_t sq[3], sk[3], sv[3], so[3];
};

int launch_attn_tc_bf16(const AttnArgs& a, cudaStream_t stream);  // tcgen05 path
int launch_attn_f32(const AttnArgs& a, cudaStream_t stream);      // fp32 CUDA-core path

struct VocabArgs {
  const void* logits;
  int is_bf16;
  int64_t N, V, row_stride;  // row stride in elements
  int32_t* argmax;
  float* conf;
  float* lse;
  int* err;  // device error word (input checks of DLM_CHECK_BOUNDS builds)
};

int launch_vocab_confidence(const VocabArgs& a, cudaStream_t stream);


struct UpdateArgs {
  const int32_t* tokens;
  const uint8_t* mask;
  const int32_t* argmax;
  const float* conf;
  int32_t* new_tokens;
  uint8_t* new_mask;
  int32_t* n_edits;
  int64_t s_tokens, s_mask, s_argmax, s_conf, s_new_tokens, s_new_mask;  // sequence strides
  int B, L;
  float edit_threshold;
  int32_t remask_k;
  float remask_frac;
  int32_t mask_id;
  const int32_t* prompt_lens;
  const int32_t* seq_lens;
  // Remask ranking by the resulting token's probability when non-null: the
  // probability of each position's current token, [B, L] with sequence stride s_tok_prob.
  const float* tok_prob;
  int64_t s_tok_prob;
};

int launch_refine_update(const UpdateArgs& a, cudaStream_t stream);

// prob[r] = exp(logits[r, tokens[r]] - lse[r]) (0 for a token outside [0, V)).
int launch_token_prob(const VocabArgs& a, const int32_t* tokens, const float* lse, float* prob,
                      cudaStream_t stream);

// Fused vocabulary reduction + update (rows of sequence b are b * L .. b * L + L - 1;
// u.argmax / u.conf alias a.argmax / a.conf). counters: int32[B], zero on entry.
int launch_vocab_step(const VocabArgs& a, const UpdateArgs& u, int* counters, cudaStream_t stream);

// Vocabulary projection fused with the reduction: per row r of hidden [N, d]
// the argmax / conf / lse of hidden[r] . weight[v] over v < V.
struct LmArgs {
  const void* hidden;   // bf16 [N, d], row stride s_hidden elements
  const void* weight;   // bf16 [V, d], row stride s_weight elements
  int64_t N, V, d, s_hidden, s_weight;
  int32_t* argmax;
  float* conf;
  float* lse;
  void* workspace;      // lmhead_workspace_bytes(N)
};

constexpr int kLmMaxSplits = 64;
inline size_t lmhead_workspace_bytes(int64_t N) { return static_cast<size_t>(N) * kLmMaxSplits * 12; }
int lmhead_splits(int64_t N, int64_t V, int sms);
int launch_lmhead(const LmArgs& a, cudaStream_t stream);

}  // namespace dlm
