// Step A3 -- the refine update of one sequence, executed by one thread block.
//
// Sec. 4.2: the prompt stays fixed while any response position may be
// revised; the per-pass rule is token editing with confident edits
// (Appendix C.4, Table 11). For sequence b (response [p_b, n_b)):
//   pass 1  elementwise over [0, L): copy prompt/padding, commit masked
//           response positions to argmax, edit filled ones whose argmax
//           differs and whose conf >= tau; count edits (block reduction);
//   pass 2  radix select over the response keys: the k_b-th smallest of
//           key(conf) (an order-preserving map of the fp32 bits, -0 -> +0),
//           4 passes of 8 bits with warp-aggregated shared-memory histograms
//           (with a.tok_prob, key of the probability of the token each
//           position holds after pass 1: conf where that is the argmax, the
//           given probability of the kept token elsewhere);
//   pass 3  remask keys below the k-th key, and the lowest-index positions
//           whose key equals it (an ordered block scan), up to k_b in total.
// Responses of at most 4 keys per thread compute each key once, in pass 1,
// and keep it in shared memory for passes 2 and 3; longer ones re-read the
// predictions in each pass.
// Integer work and exact fp32 compares only: results are bit-exact.
// Used by the stand-alone update kernel (update.cu) and by the fused
// vocabulary + update kernel (vocab.cu), whose last row block of a sequence
// runs it.
#pragma once

#include <cmath>
#include <cstdint>

#include "dlm_common.cuh"
#include "dlm_internal.h"

namespace dlm {

template <int kThreads>
struct UpdateShared {
  static constexpr int kKeyCap = 4 * kThreads;  // response positions whose keys are kept here
  int hist[256];
  int warp_sums[kThreads / 32];
  int sel_digit, sel_before;
  uint32_t keys[kKeyCap];  // ranking key of response position p + j (responses of at most kKeyCap)
};

// Order-preserving map of an fp32 value to uint32 (smaller value -> smaller
// key), with -0.0 mapped like +0.0.
__device__ __forceinline__ uint32_t conf_key(float c) {
  uint32_t u = __float_as_uint(c);
  if (u == 0x80000000u) u = 0u;
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__device__ __forceinline__ bool is_nan_bits(uint32_t u) {
  return (u & 0x7F800000u) == 0x7F800000u && (u & 0x007FFFFFu) != 0u;
}

// Inclusive prefix sum over the block of `v` (one value per thread); returns
// the inclusive prefix for this thread and the block total in *total.
template <int kThreads>
__device__ __forceinline__ int block_inclusive_scan(int v, int* warp_sums, int* total) {
  constexpr int kWarps = kThreads / 32;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_sums[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int w = lane < kWarps ? warp_sums[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      int y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    if (lane < kWarps) warp_sums[lane] = w;  // inclusive over warps
  }
  __syncthreads();
  int before = warp > 0 ? warp_sums[warp - 1] : 0;
  *total = warp_sums[kWarps - 1];
  __syncthreads();  // warp_sums is reused by the next call
  return before + x;
}

// Reads of predictions written earlier in the same launch by other blocks go
// around L1 (kFresh); otherwise plain loads.
template <bool kFresh, typename T>
__device__ __forceinline__ T load_pred(const T* p) {
  if constexpr (kFresh) return __ldcg(p);
  else return *p;
}

// Runs the update of sequence b with the whole block (blockDim.x == kThreads).
// Every thread of the block must call it.
template <int kThreads, bool kFresh>
__device__ void refine_sequence(const UpdateArgs& a, int b, int* err, UpdateShared<kThreads>& sh) {
  const int tid = threadIdx.x;
  const int L = a.L;

  int n = a.seq_lens ? a.seq_lens[b] : L;
  int p = a.prompt_lens ? a.prompt_lens[b] : 0;
  bool clamped = false;
  if (n < 0 || n > L) { n = n < 0 ? 0 : L; clamped = true; }
  if (p < 0 || p > n) { p = p < 0 ? 0 : n; clamped = true; }
  if (clamped && tid == 0) set_device_error(err, DLM_DEVERR_LENGTH);
  const int r = n - p;

  const int32_t* tok = a.tokens + b * a.s_tokens;
  const uint8_t* msk = a.mask + b * a.s_mask;
  const int32_t* am = a.argmax + b * a.s_argmax;
  const float* cf = a.conf + b * a.s_conf;
  int32_t* ntok = a.new_tokens + b * a.s_new_tokens;
  uint8_t* nmsk = a.new_mask + b * a.s_new_mask;
  const float* tp = a.tok_prob ? a.tok_prob + b * a.s_tok_prob : nullptr;
  // Ranking value of response position i once pass 1 has written new_tokens.
  auto rank_value = [&](int i) -> float {
    if (tp && ntok[i] != load_pred<kFresh>(am + i)) return tp[i];
    return load_pred<kFresh>(cf + i);
  };

  // ---- pass 1: copy / commit / edit (read and write of position i by one
  // thread, so new_* may alias tokens/mask). Responses of at most kKeyCap
  // positions also keep each position's ranking key in shared memory, so
  // that the selection below reads the predictions once.
  const bool cached = r <= UpdateShared<kThreads>::kKeyCap;
  bool saw_nan = false;
  int edits = 0;
  for (int i = tid; i < L; i += kThreads) {
    int t = tok[i];
    uint8_t m = msk[i];
    if (i >= p && i < n) {
      const int pred = load_pred<kFresh>(am + i);
      const float c = load_pred<kFresh>(cf + i);
      if (m) {
        t = pred;
      } else if (pred != t && c >= a.edit_threshold) {
        t = pred;
        ++edits;
      }
      m = 0;
      if (cached) {
        const float v = (tp && t != pred) ? tp[i] : c;
        saw_nan |= is_nan_bits(__float_as_uint(v));
        sh.keys[i - p] = conf_key(v);
      }
    }
    ntok[i] = t;
    nmsk[i] = m;
  }
  int total_edits;
  block_inclusive_scan<kThreads>(edits, sh.warp_sums, &total_edits);
  if (tid == 0) a.n_edits[b] = total_edits;

  // ---- k_b
  long long k;
  if (a.remask_k >= 0) {
    k = a.remask_k;
  } else {
    k = static_cast<long long>(floor(static_cast<double>(a.remask_frac) * static_cast<double>(r)));
  }
  if (k > r) k = r;
  if (k <= 0) return;
  __syncthreads();  // pass-1 writes precede the remask writes below

  if (k == r) {
    for (int i = p + tid; i < n; i += kThreads) {
      ntok[i] = a.mask_id;
      nmsk[i] = 1;
    }
    return;
  }

  // ---- pass 2: radix select of the k-th smallest key (1-based rank `need`)
  // The key of response position i (pass 1's copy when cached).
  auto key_of = [&](int i) -> uint32_t {
    if (cached) return sh.keys[i - p];
    const float c = rank_value(i);
    saw_nan |= is_nan_bits(__float_as_uint(c));
    return conf_key(c);
  };
  uint32_t prefix = 0, pmask = 0;
  int need = static_cast<int>(k);
  for (int shift = 24; shift >= 0; shift -= 8) {
    for (int i = tid; i < 256; i += kThreads) sh.hist[i] = 0;
    __syncthreads();
    for (int base = p; base < n; base += kThreads) {
      int i = base + tid;
      bool active = false;
      uint32_t digit = 0;
      if (i < n) {
        const uint32_t key = key_of(i);
        if ((key & pmask) == prefix) {
          active = true;
          digit = (key >> shift) & 0xFFu;
        }
      }
      // Warp-aggregated histogram update: one atomic per distinct digit.
      unsigned act = __ballot_sync(0xffffffffu, active);
      if (active) {
        unsigned same = __match_any_sync(act, digit);
        int leader = __ffs(same) - 1;
        if ((tid & 31) == leader) atomicAdd(&sh.hist[digit], __popc(same));
      }
    }
    __syncthreads();
    // One warp finds the digit whose cumulative count first reaches `need`.
    if (tid < 32) {
      int c[8];
      int s = 0;
#pragma unroll
      for (int j = 0; j < 8; ++j) { c[j] = sh.hist[tid * 8 + j]; s += c[j]; }
      int incl = s;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (tid >= o) incl += y;
      }
      int excl = incl - s;
      if (excl < need && need <= incl) {
        int run = excl;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          if (run < need && need <= run + c[j]) { sh.sel_digit = tid * 8 + j; sh.sel_before = run; }
          run += c[j];
        }
      }
    }
    __syncthreads();
    prefix |= static_cast<uint32_t>(sh.sel_digit) << shift;
    pmask |= 0xFFu << shift;
    need -= sh.sel_before;
    __syncthreads();  // sel_* are rewritten by the next pass
  }
  if (__syncthreads_or(saw_nan) && tid == 0) set_device_error(err, DLM_DEVERR_NAN);
  const uint32_t kth = prefix;  // every key < kth is remasked, plus `need` keys == kth

  // ---- pass 3: remask, equal keys in index order
  int taken = 0;
  for (int base = p; base < n; base += kThreads) {
    int i = base + tid;
    uint32_t key = i < n ? key_of(i) : 0xFFFFFFFFu;
    bool eq = i < n && key == kth;
    int total;
    int incl = block_inclusive_scan<kThreads>(eq ? 1 : 0, sh.warp_sums, &total);
    bool sel = (i < n) && (key < kth || (eq && taken + incl <= need));
    if (sel) {
      ntok[i] = a.mask_id;
      nmsk[i] = 1;
    }
    taken += total;
  }
}

}  // namespace dlm
