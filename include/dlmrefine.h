/*
 * libdlmrefine -- one bidirectional refine step of speculative correction
 * (draft-then-refine decoding for diffusion language models), on GB300.
 *
 * The refiner receives the fixed prompt plus a complete draft and revises any
 * response position with full-sequence bidirectional denoising passes
 * (Sec. 4.2). One pass on the hot path is three calls, in this order:
 *
 *   dlm_bidir_attn        non-causal GQA attention over all valid positions
 *   dlm_vocab_confidence  per position: argmax token, max softmax probability,
 *                         log-sum-exp over the vocabulary logits
 *   dlm_refine_update     commit masked positions, edit confident changes,
 *                         remask the k least confident positions
 *
 * Around them:
 *   dlm_refine_step          the last two in one launch (same results);
 *                            dlm_refine_step_static without a workspace
 *   dlm_lmhead_confidence    the vocabulary projection hidden x W^T fused with
 *                            the per-position reduction (logits never stored)
 *   dlm_attn_masked          block-causal / block-local attention (the
 *                            block-autoregressive pattern and local refinement)
 *   dlm_token_prob,          remask ranking by the probability of each
 *   dlm_refine_update_ranked position's resulting token (a second reading)
 *   dlm_loop_*               repeat a recorded pass on the GPU until no
 *                            confident edit remains (one graph launch)
 *
 * Conventions shared by every call
 * --------------------------------
 * - Tensors are passed as dlm_tensor descriptors: a DEVICE pointer of the
 *   current CUDA device, a dtype, the shape and the strides in elements.
 *   The caller owns every buffer; the library allocates no device memory and
 *   keeps no pointer after a call returns (a dlm_loop keeps the pointers of
 *   the calls it recorded). Its only device memory is static: the error word
 *   and the 16 KB scratch of dlm_refine_step_static.
 * - Calls are asynchronous on the stream set by dlm_set_stream for the calling
 *   thread (default: the legacy default stream). Outputs are valid once that
 *   stream has been synchronised. Arguments are validated on the host before
 *   any launch; a nonzero return means nothing was launched.
 * - Values that live in device memory (sequence and prompt lengths) cannot be
 *   checked on the host: the kernels clamp them into range and record
 *   DLM_DEVERR_LENGTH in the device error word (dlm_get_device_error).
 * - Return value: DLM_OK (0) or a negative dlm_status. dlm_last_error() gives
 *   a message for the most recent failure on the calling thread.
 */
#ifndef DLMREFINE_H_
#define DLMREFINE_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define DLM_VERSION_MAJOR 0
#define DLM_VERSION_MINOR 2
#define DLM_VERSION_PATCH 1

typedef enum dlm_dtype {
  DLM_BF16 = 1, /* bfloat16 */
  DLM_F32 = 2,  /* IEEE binary32 */
  DLM_I32 = 3,  /* int32 */
  DLM_U8 = 4    /* uint8 */
} dlm_dtype;

typedef enum dlm_status {
  DLM_OK = 0,
  DLM_ERR_NULL = -1,        /* a required pointer or descriptor is NULL */
  DLM_ERR_DTYPE = -2,       /* unsupported or mismatched dtype */
  DLM_ERR_SHAPE = -3,       /* rank or extents inconsistent */
  DLM_ERR_STRIDE = -4,      /* innermost dimension not contiguous, or an unsupported stride */
  DLM_ERR_ALIGN = -5,       /* base pointer or stride not aligned as required */
  DLM_ERR_ARG = -6,         /* a scalar argument out of range (NaN threshold, ...) */
  DLM_ERR_CUDA = -7,        /* a CUDA runtime call or launch failed */
  DLM_ERR_DEVICE = -8,      /* the device error word was set (dlm_get_device_error) */
  DLM_ERR_UNSUPPORTED = -9  /* no kernel for this device or configuration */
} dlm_status;

/* Bits of the device error word. */
#define DLM_DEVERR_LENGTH 0x1   /* a seq_len / prompt_len outside [0, L] was clamped */
#define DLM_DEVERR_TIMEOUT 0x2  /* a bounded wait in a kernel gave up; its outputs are undefined */
#define DLM_DEVERR_NAN 0x4      /* a NaN confidence reached the remask selection */
/* An input outside its contract was seen: a row of logits with a NaN entry or
 * with every entry -inf (dlm_vocab_confidence, dlm_refine_step), a token id
 * outside [0, V) (dlm_token_prob). Checked only by builds compiled with
 * DLM_CHECK_BOUNDS (python -m paper_2608_02625_gb300.build --check-bounds);
 * the default build leaves such outputs undefined, as documented per call. */
#define DLM_DEVERR_INPUT 0x8

typedef struct dlm_tensor {
  void* data;        /* device pointer; 16-byte aligned where a call requires it */
  int32_t dtype;     /* dlm_dtype */
  int32_t ndim;      /* 1..4 */
  int64_t shape[4];  /* extents, outermost first */
  int64_t stride[4]; /* strides in ELEMENTS, outermost first; stride[ndim-1] must be 1 */
} dlm_tensor;

/*
 * Parameters of the refine update (one pass).
 *   edit_threshold  tau: a filled response position whose argmax differs from
 *                   its token is edited iff conf >= tau (fp32 compare). Not NaN.
 *   remask_k        >= 0: remask min(remask_k, r_b) positions per sequence;
 *                   < 0: remask floor(remask_frac * r_b) (remask_frac in [0, 1]).
 *   mask_id         the token written at remasked positions.
 *   prompt_lens     device int32[B]: p_b, clamped into [0, n_b].
 *   seq_lens        device int32[B]: n_b, clamped into [0, L].
 * The response of sequence b is [p_b, n_b) and r_b = n_b - p_b.
 * The update only touches [p_b, n_b): to refine one window of a response
 * (the local 64-token refinement of Sec. 6.3 and the granular span schedules
 * of Appendix D.4), pass the window's bounds here (the attention keeps the
 * sequence's own lengths); positions outside the window are copied unchanged.
 */
typedef struct dlm_refine_params {
  float edit_threshold;
  int32_t remask_k;
  float remask_frac;
  int32_t mask_id;
  const int32_t* prompt_lens;
  const int32_t* seq_lens;
} dlm_refine_params;

/*
 * Step A1 -- non-causal GQA attention (Sec. 4.2: bidirectional correction
 * over the entire sequence; no causal or block mask, cf. Sec. 3.3).
 *
 *   out[b,i,h,:] = sum_{j<n_b} softmax_j(q[b,i,h,:] . k[b,j,g,:] / sqrt(D)) v[b,j,g,:]
 *   with g = floor(h * Hkv / Hq), for i < n_b; out[b,i,h,:] = 0 for i >= n_b.
 *
 *   q, out    [B, L, Hq, D]    BF16 or F32 (both the same dtype)
 *   k, v      [B, L, Hkv, D]   same dtype as q; Hq % Hkv == 0
 *   seq_lens  [B] I32          n_b; NULL means n_b = L for all b
 *   D in {64, 128}. Strides are free except that the innermost dimension is
 *   contiguous. BF16: tensor cores (tcgen05) with fp32 accumulation and
 *   softmax, every base pointer and every stride a multiple of 16 bytes.
 *   F32: fp32 throughout on the CUDA cores.
 * Key/value rows j >= n_b are never read into a result (they may hold any
 * bit pattern). out must not overlap q, k or v.
 */
int dlm_bidir_attn(const dlm_tensor* q, const dlm_tensor* k, const dlm_tensor* v,
                   const dlm_tensor* seq_lens, dlm_tensor* out);

/* Attention masks of dlm_attn_masked. */
#define DLM_ATTN_FULL 0          /* every valid key (dlm_bidir_attn) */
#define DLM_ATTN_BLOCK_CAUSAL 1  /* block-autoregressive attention (Sec. 3.3) */
#define DLM_ATTN_BLOCK_LOCAL 2   /* prompt + own block: local refinement (Sec. 5.3, 6.3) */

/*
 * dlm_bidir_attn over a subset of keys per query (the block-autoregressive
 * pattern the refiner replaces, Sec. 3.3, and the local 64-token refinement
 * of the causal ablation, Sec. 5.3 / 6.3). The response [p_b, n_b) is cut
 * into blocks of `block` positions starting at p_b; query i >= p_b of block
 * c = floor((i - p_b) / block) attends to
 *   DLM_ATTN_BLOCK_CAUSAL  keys j < min(n_b, p_b + (c + 1) * block)
 *                          (the prompt, earlier blocks and its own block);
 *   DLM_ATTN_BLOCK_LOCAL   keys j < p_b and keys of block c (j < n_b);
 * prompt queries i < p_b attend to keys j < p_b. DLM_ATTN_FULL is
 * dlm_bidir_attn. Rows i >= n_b are 0.
 *   prompt_lens  [B] I32 (p_b, clamped to [0, n_b]; a clamp sets
 *                DLM_DEVERR_LENGTH) or NULL (p_b = 0)
 *   mode         DLM_ATTN_*;  block >= 1 for the block masks
 *   other arguments as for dlm_bidir_attn (same dtypes, layouts, tolerances).
 */
int dlm_attn_masked(const dlm_tensor* q, const dlm_tensor* k, const dlm_tensor* v,
                    const dlm_tensor* seq_lens, const dlm_tensor* prompt_lens, int32_t mode,
                    int32_t block, dlm_tensor* out);

/*
 * Step A2 -- per-position reduction over the vocabulary (the confidences the
 * refine threshold of Table 10 and the confident edits of Appendix C.4 act on).
 *
 *   m         = max_v logits[r, v]
 *   argmax[r] = lowest v with logits[r, v] == m
 *   lse[r]    = m + ln sum_v exp(logits[r, v] - m)
 *   conf[r]   = exp(m - lse[r])          (the maximum softmax probability)
 *
 *   logits  [N, V] or [B, L, V]   BF16 or F32; innermost contiguous; rows may
 *                                 be strided (row stride in elements)
 *   argmax  N I32, conf N F32, lse N F32 (any rank with N elements, contiguous)
 * Math in fp32 with an fp32-accurate exp2; the argmax compare is exact.
 * Entries may be -inf; a NaN entry or a row of only -inf gives undefined
 * results for that row. V >= 1.
 */
int dlm_vocab_confidence(const dlm_tensor* logits, dlm_tensor* argmax, dlm_tensor* conf,
                         dlm_tensor* lse);

/*
 * Step A3 -- the refine update (prompt fixed, any response position revisable,
 * Sec. 4.2; token editing with confident edits, Appendix C.4 / Table 11).
 * For each sequence b, independently:
 *   1. prompt [0,p_b) and padding [n_b,L) are copied unchanged;
 *   2. response position i becomes unmasked and takes argmax[i] if it was
 *      masked (commit), argmax[i] if argmax[i] != tokens[i] and
 *      conf[i] >= edit_threshold (edit, counted), else tokens[i];
 *   3. k_b = remask_k >= 0 ? min(remask_k, r_b) : floor(remask_frac * r_b);
 *   4. the k_b response positions first in (conf ascending, index ascending)
 *      order are remasked: new_mask = 1, new_tokens = mask_id (-0.0 == +0.0);
 *   5. n_edits[b] = number of edits of step 2 (commits excluded; an edit that
 *      step 4 remasks still counts).
 *
 *   tokens, new_tokens  [B, L] I32      mask, new_mask  [B, L] U8
 *   argmax              [B, L] I32      conf            [B, L] F32
 *   n_edits             [B]    I32
 * Results are bit-exact: integer work and exact fp32 comparisons only.
 * new_tokens / new_mask may alias tokens / mask exactly (in-place update);
 * no other overlap is allowed. L <= 2^24.
 */
int dlm_refine_update(const dlm_tensor* tokens, const dlm_tensor* mask, const dlm_tensor* argmax,
                      const dlm_tensor* conf, const dlm_refine_params* params,
                      dlm_tensor* new_tokens, dlm_tensor* new_mask, dlm_tensor* n_edits);

/*
 * The vocabulary projection fused with step A2: for each row r of hidden,
 * the per-position reduction of dlm_vocab_confidence applied to
 *   logits[r, v] = sum_k hidden[r, k] * weight[v, k]      (v < V),
 * the refiner's output projection of its final hidden states (Sec. 4.2: every
 * revisable position's distribution over the vocabulary), without writing
 * the N x V logits to memory. tcgen05 MMAs (bf16 x bf16, fp32 accumulation);
 * the reduction reads the fp32 accumulators (no bf16 rounding of logits).
 *   hidden     [N, d] or [B, L, d] BF16, weight [V, d] BF16; d a multiple of
 *              64; base pointers and row strides multiples of 16 bytes
 *   argmax, conf, lse   N entries each (I32, F32, F32), contiguous
 *   workspace  >= dlm_lmhead_workspace_bytes(N) bytes of device memory,
 *              16-byte aligned, owned by the caller (no initial contents
 *              needed); calls sharing it must not overlap on the GPU.
 * Accuracy: the logits carry fp32 accumulation error (a few 1e-5 relative to
 * sum_k |hidden[r,k] weight[v,k]|); an argmax can differ from exact
 * arithmetic only where two logits are that close. The width d is a
 * parameter: the paper does not give the refiner's dimensions.
 */
int dlm_lmhead_confidence(const dlm_tensor* hidden, const dlm_tensor* weight, dlm_tensor* argmax,
                          dlm_tensor* conf, dlm_tensor* lse, void* workspace, size_t workspace_bytes);
/* Bytes of workspace dlm_lmhead_confidence needs for `rows` rows. */
size_t dlm_lmhead_workspace_bytes(int64_t rows);

/*
 * Probability of a given token of each row under the row's softmax:
 *   prob[r] = exp(logits[r, tokens[r]] - lse[r]),   0 if tokens[r] is outside [0, V).
 * With lse from dlm_vocab_confidence and tokens[r] the current token of a
 * position, this is the probability the refiner assigns to keeping it; it
 * feeds the remask ranking of dlm_refine_update_ranked.
 *   logits  as for dlm_vocab_confidence;  tokens N I32, lse N F32, prob N F32
 *   (any rank with N elements, contiguous). fp32: one gathered logit per row.
 */
int dlm_token_prob(const dlm_tensor* logits, const dlm_tensor* tokens, const dlm_tensor* lse,
                   dlm_tensor* prob);

/*
 * dlm_refine_update with the remask ranking of a second reading of the paper's
 * editing rule (Appendix C.4 / Table 11 do not fix which probability ranks the
 * positions to remask): step 4 orders the response positions by the
 * probability of the token each holds after step 2 -- conf[i] where that
 * token is the argmax (commit, edit, or a kept token equal to the argmax),
 * tok_prob[i] (the kept token's probability, dlm_token_prob) elsewhere --
 * ascending, index ascending. Steps 1-3 and 5 are those of dlm_refine_update.
 *   tok_prob  [B, L] F32 (innermost contiguous); the other arguments as for
 *             dlm_refine_update. Bit-exact (exact fp32 compares only).
 */
int dlm_refine_update_ranked(const dlm_tensor* tokens, const dlm_tensor* mask, const dlm_tensor* argmax,
                             const dlm_tensor* conf, const dlm_tensor* tok_prob,
                             const dlm_refine_params* params, dlm_tensor* new_tokens,
                             dlm_tensor* new_mask, dlm_tensor* n_edits);

/*
 * Steps A2 and A3 fused in one launch (the per-position reduction of the
 * confidences of Table 10 / Appendix C.4 feeding the update of Sec. 4.2).
 * Computes exactly what dlm_vocab_confidence(logits, argmax, conf, lse)
 * followed by dlm_refine_update(tokens, mask, argmax, conf, params,
 * new_tokens, new_mask, n_edits) computes: argmax, conf and lse are written
 * as by the first call, and the update reads them back. The CTA that finishes
 * the last row of sequence b runs the update of b, so the update of one
 * sequence overlaps the vocabulary stream of the others and no second launch
 * is needed.
 *
 *   logits  [B * L, V] or [B, L, V]   BF16 or F32, as for dlm_vocab_confidence
 *   argmax, conf, lse                 [B, L] contiguous (I32, F32, F32)
 *   other tensors and params          as for dlm_refine_update
 *   workspace                         device memory of at least
 *                                     dlm_refine_step_workspace_bytes(B) bytes,
 *                                     4-byte aligned, owned by the caller
 * The workspace holds one row counter per sequence. It must be zero before
 * its first use (e.g. cudaMemsetAsync); each completed call leaves it zero
 * again, so it can be reused by later calls without clearing. Calls that
 * share a workspace must not overlap on the GPU (they would race on the
 * counters): issue them on one stream. new_tokens / new_mask may alias
 * tokens / mask exactly; no other overlap among the tensors is allowed.
 */
int dlm_refine_step(const dlm_tensor* logits, const dlm_tensor* tokens, const dlm_tensor* mask,
                    const dlm_refine_params* params, dlm_tensor* argmax, dlm_tensor* conf,
                    dlm_tensor* lse, dlm_tensor* new_tokens, dlm_tensor* new_mask,
                    dlm_tensor* n_edits, void* workspace, size_t workspace_bytes);
/* Bytes of workspace dlm_refine_step needs for a batch of `batch` sequences. */
size_t dlm_refine_step_workspace_bytes(int64_t batch);

/* Largest batch dlm_refine_step_static accepts (its static scratch: 16 KB). */
#define DLM_STATIC_STEP_MAX_BATCH 4096

/*
 * dlm_refine_step without a workspace argument; the paper has no counterpart
 * (it is a deployment convenience of this library, not part of the method).
 * For callers that cannot allocate device memory: a serving engine whose
 * allocator reserves nearly all of HBM up front (a cudaMalloc outside its pool
 * fails or fragments it), a latency-critical loop that cannot take
 * cudaMalloc's implicit device synchronisation, or a plugin interface with a
 * fixed signature and no slot for a workspace.
 *
 * Computes exactly what dlm_refine_step computes, with the same arguments
 * minus the workspace. The per-sequence counters live in a static device
 * array of DLM_STATIC_STEP_MAX_BATCH int32 inside the library, which every
 * device that loads the library holds until the process exits. The call
 * allocates nothing (no cudaMalloc, cudaFree or allocating library routine).
 *
 * - The first call on a device sets up that device: it takes the array's
 *   device address with cudaGetSymbolAddress, with that device current.
 *   Make that first call before any stream capture on the device;
 *   dlm_loop_begin does this set-up itself, so a recorded pass may use it.
 * - Each call clears the counters it uses (an asynchronous memset on the
 *   call's stream) and then launches the fused kernel.
 * - All calls on one device share the array: calls that overlap on the GPU
 *   (different streams, or different host threads) race on it and give
 *   undefined results. Issue them on one stream.
 * - B > DLM_STATIC_STEP_MAX_BATCH returns DLM_ERR_SHAPE with nothing
 *   launched; use dlm_refine_step with a workspace for larger batches.
 */
int dlm_refine_step_static(const dlm_tensor* logits, const dlm_tensor* tokens, const dlm_tensor* mask,
                           const dlm_refine_params* params, dlm_tensor* argmax, dlm_tensor* conf,
                           dlm_tensor* lse, dlm_tensor* new_tokens, dlm_tensor* new_mask,
                           dlm_tensor* n_edits);

/*
 * Multi-pass refinement as one graph launch, with the early stop on the device
 * (passes repeat until no confident edit remains, Appendix C.4 / Table 11).
 *
 *   int32_t* steps;                  // device int32: passes run by a launch
 *   dlm_loop_begin(steps);           // start recording one pass
 *   ... the pass: the caller's model forward, dlm_bidir_attn,
 *       dlm_refine_step (or the two separate calls) on the same stream ...
 *   dlm_loop_end(n_edits, B, max_steps, &loop);
 *   dlm_loop_launch(loop);           // runs the recorded pass repeatedly
 *   dlm_loop_destroy(loop);
 *
 * dlm_loop_begin starts a stream capture (thread-local mode) on the calling
 * thread's stream, which must be a created stream (not the legacy default):
 * calls issued on it until dlm_loop_end are recorded, not run. The recorded
 * pass must read its inputs from and write its outputs to fixed device
 * buffers (in-place token update: new_tokens / new_mask aliasing tokens /
 * mask), because every repetition replays the same launches.
 *
 * dlm_loop_end builds a CUDA graph: steps = 0, then WHILE { pass; steps += 1;
 * continue iff steps < max_steps and n_edits[b] > 0 for some b < B and the
 * device error word holds no bit other than DLM_DEVERR_LENGTH }: a clamped
 * length has a defined result, every other bit leaves the pass's outputs
 * undefined and ends the loop. n_edits is the [B] int32 edit count written
 * by the recorded pass. The test runs on the GPU after each pass, so there is
 * no host round trip between passes. Validation failures and capture errors
 * end the capture and return an error; dlm_loop_cancel ends an unfinished
 * recording. A loop may be launched any number of times (on the calling
 * thread's stream); each launch restarts steps at 0. The loop keeps device
 * pointers of the recorded calls: their buffers must outlive it.
 */
typedef struct dlm_loop dlm_loop;
int dlm_loop_begin(int32_t* steps_out);
int dlm_loop_end(const int32_t* n_edits, int64_t batch, int32_t max_steps, dlm_loop** loop);
int dlm_loop_cancel(void);
int dlm_loop_launch(dlm_loop* loop);
int dlm_loop_destroy(dlm_loop* loop);

/* Sets the CUDA stream (a cudaStream_t) used by later calls on this thread. */
int dlm_set_stream(void* stream);
/* The stream currently set for this thread. */
void* dlm_get_stream(void);

/* Work granularity of the BF16 attention kernels (dlm_bidir_attn,
 * dlm_attn_masked) for later calls on this thread; no effect on results.
 * A work unit is one or two 128-row query tiles of one sequence and key/value
 * head, run by one CTA. tiles = 2: two tiles per unit, which share each
 * key/value tile the CTA loads (the faster choice unless every single tile
 * fits on the SMs at once); 1: one tile per unit (a single short sequence:
 * every tile runs at once); 0: automatic, the default (1 when twice the
 * number of tile pairs is at most the SM count, else 2). Returns DLM_ERR_ARG
 * for any other value, leaving the setting unchanged. */
int dlm_set_attn_tiles_per_unit(int tiles);

/* Static description of a status code. */
const char* dlm_status_string(int status);
/* Message for the most recent failure on this thread ("" if none). */
const char* dlm_last_error(void);
/* MAJOR * 10000 + MINOR * 100 + PATCH. */
int dlm_version(void);

/*
 * Self-test of the bounded waits; a diagnostic of this library, with no
 * counterpart in the paper. Every pipelined kernel waits for its producers
 * with a wait that gives up after a wall-clock budget, records
 * DLM_DEVERR_TIMEOUT in the device error word and ends the kernel, so that a
 * stalled pipeline cannot hang the GPU. This call launches, on the calling
 * thread's stream, a one-thread kernel that waits through that same code, for
 * budget_ns nanoseconds (1e3 .. 1e9), on a barrier on which nothing ever
 * arrives. Once it has run, dlm_get_device_error reports DLM_DEVERR_TIMEOUT
 * (a recorded refine loop whose pass makes this call stops after that pass).
 * Returns DLM_ERR_ARG, with nothing launched, for a budget outside the range.
 */
int dlm_selftest_wait_timeout(int64_t budget_ns);

/*
 * Reads the device error word of the current device into *bits (DLM_DEVERR_*),
 * clearing it if clear != 0. Synchronises the current device. Returns DLM_OK,
 * or DLM_ERR_CUDA if the device could not be read.
 */
int dlm_get_device_error(int32_t* bits, int clear);

#ifdef __cplusplus
}
#endif

#endif /* DLMREFINE_H_ */
