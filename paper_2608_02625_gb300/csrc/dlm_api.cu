// libdlmrefine C ABI: argument validation, stream and error state, dispatch.
//
// Every entry point validates its descriptors on the host and returns a
// negative dlm_status before any launch when something is wrong. Values that
// live in device memory (lengths) are clamped by the kernels, which record it
// in the per-device error word read by dlm_get_device_error.
#include <atomic>
#include <cstdarg>
#include <cmath>
#include <cstdint>
#include <cstdio>
#include <cstring>
#include <mutex>

#include "dlm_internal.h"
#include "dlmrefine.h"

namespace {

// The device error word. Kernels receive its device address (taken once per
// device with cudaGetSymbolAddress) as an argument.
__device__ int g_dlm_device_error;

thread_local cudaStream_t t_stream = nullptr;
thread_local int t_attn_tpu = 0;  // query tiles per attention work unit (0: automatic)
thread_local char t_last_error[512] = "";

constexpr int kMaxDevices = 64;
std::mutex g_err_mu;
int* g_err_addr[kMaxDevices] = {};

std::atomic<uint64_t> g_wait_budget_ns{dlm::kDefaultWaitBudgetNs};

int64_t elem_size(int dtype) {
  switch (dtype) {
    case DLM_BF16: return 2;
    case DLM_F32: return 4;
    case DLM_I32: return 4;
    case DLM_U8: return 1;
    default: return 0;
  }
}

int64_t numel(const dlm_tensor* t) {
  int64_t n = 1;
  for (int i = 0; i < t->ndim; ++i) n *= t->shape[i];
  return n;
}

// Checks pointer, dtype, rank, non-negative extents and a contiguous innermost
// dimension. `name` appears in the error message.
int check_tensor(const dlm_tensor* t, const char* name, int dtype_mask, int ndim_lo, int ndim_hi) {
  using dlm::fail;
  if (!t) return fail(DLM_ERR_NULL, "%s: descriptor is NULL", name);
  if (elem_size(t->dtype) == 0 || !((1 << t->dtype) & dtype_mask))
    return fail(DLM_ERR_DTYPE, "%s: unsupported dtype %d", name, t->dtype);
  if (t->ndim < ndim_lo || t->ndim > ndim_hi)
    return fail(DLM_ERR_SHAPE, "%s: rank %d not in [%d, %d]", name, t->ndim, ndim_lo, ndim_hi);
  for (int i = 0; i < t->ndim; ++i) {
    if (t->shape[i] < 0) return fail(DLM_ERR_SHAPE, "%s: negative extent", name);
    if (t->shape[i] > 0x7FFFFFFFLL) return fail(DLM_ERR_SHAPE, "%s: extent too large", name);
  }
  if (numel(t) > 0) {
    if (!t->data) return fail(DLM_ERR_NULL, "%s: data pointer is NULL", name);
    if (t->shape[t->ndim - 1] > 1 && t->stride[t->ndim - 1] != 1)
      return fail(DLM_ERR_STRIDE, "%s: innermost dimension must be contiguous", name);
    for (int i = 0; i < t->ndim; ++i)
      if (t->stride[i] < 0) return fail(DLM_ERR_STRIDE, "%s: negative stride", name);
    if (reinterpret_cast<uintptr_t>(t->data) % static_cast<uintptr_t>(elem_size(t->dtype)) != 0)
      return fail(DLM_ERR_ALIGN, "%s: data pointer not aligned to its element size", name);
  }
  return DLM_OK;
}

bool is_dense(const dlm_tensor* t) {
  int64_t expect = 1;
  for (int i = t->ndim - 1; i >= 0; --i) {
    if (t->shape[i] > 1 && t->stride[i] != expect) return false;
    expect *= t->shape[i];
  }
  return true;
}

// Byte range [lo, hi) touched by a strided tensor.
void byte_span(const dlm_tensor* t, uintptr_t* lo, uintptr_t* hi) {
  int64_t last = 0;
  for (int i = 0; i < t->ndim; ++i)
    if (t->shape[i] > 0) last += (t->shape[i] - 1) * t->stride[i];
  *lo = reinterpret_cast<uintptr_t>(t->data);
  *hi = *lo + static_cast<uintptr_t>((last + 1) * elem_size(t->dtype));
}

bool overlaps(const dlm_tensor* a, const dlm_tensor* b) {
  if (numel(a) == 0 || numel(b) == 0) return false;
  uintptr_t alo, ahi, blo, bhi;
  byte_span(a, &alo, &ahi);
  byte_span(b, &blo, &bhi);
  return alo < bhi && blo < ahi;
}

bool same_view(const dlm_tensor* a, const dlm_tensor* b) {
  if (a->data != b->data || a->ndim != b->ndim || a->dtype != b->dtype) return false;
  for (int i = 0; i < a->ndim; ++i)
    if (a->shape[i] != b->shape[i] || (a->shape[i] > 1 && a->stride[i] != b->stride[i])) return false;
  return true;
}

constexpr int kMaskBF16F32 = (1 << DLM_BF16) | (1 << DLM_F32);

}  // namespace

namespace dlm {

int fail(int status, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(t_last_error, sizeof(t_last_error), fmt, ap);
  va_end(ap);
  return status;
}

void clear_error() { t_last_error[0] = '\0'; }

cudaStream_t current_stream() { return t_stream; }

uint64_t wait_budget_ns() { return g_wait_budget_ns.load(std::memory_order_relaxed); }

int attn_tiles_per_unit() { return t_attn_tpu; }

int* device_error_word() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lock(g_err_mu);
  if (!g_err_addr[dev]) {
    void* ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_dlm_device_error) != cudaSuccess) return nullptr;
    g_err_addr[dev] = static_cast<int*>(ptr);
  }
  return g_err_addr[dev];
}

}  // namespace dlm

namespace {

// Every kernel records device-side failures in the error word; refuse to launch without it.
int require_error_word() {
  if (!dlm::device_error_word()) return dlm::fail(DLM_ERR_CUDA, "device error word unavailable on this device");
  return DLM_OK;
}

}  // namespace

extern "C" {

int dlm_version(void) { return DLM_VERSION_MAJOR * 10000 + DLM_VERSION_MINOR * 100 + DLM_VERSION_PATCH; }

const char* dlm_status_string(int status) {
  switch (status) {
    case DLM_OK: return "ok";
    case DLM_ERR_NULL: return "null pointer";
    case DLM_ERR_DTYPE: return "unsupported or mismatched dtype";
    case DLM_ERR_SHAPE: return "inconsistent shape";
    case DLM_ERR_STRIDE: return "unsupported stride";
    case DLM_ERR_ALIGN: return "misaligned pointer or stride";
    case DLM_ERR_ARG: return "scalar argument out of range";
    case DLM_ERR_CUDA: return "CUDA error";
    case DLM_ERR_DEVICE: return "device-side error recorded";
    case DLM_ERR_UNSUPPORTED: return "unsupported device or configuration";
    default: return "unknown status";
  }
}

const char* dlm_last_error(void) { return t_last_error; }

int dlm_set_stream(void* stream) {
  t_stream = static_cast<cudaStream_t>(stream);
  return DLM_OK;
}

void* dlm_get_stream(void) { return t_stream; }

int dlm_set_attn_tiles_per_unit(int tiles) {
  if (tiles < 0 || tiles > 2) return dlm::fail(DLM_ERR_ARG, "dlm_set_attn_tiles_per_unit: %d is not 0, 1 or 2", tiles);
  t_attn_tpu = tiles;
  return DLM_OK;
}

int dlm_get_device_error(int32_t* bits, int clear) {
  if (!bits) return dlm::fail(DLM_ERR_NULL, "dlm_get_device_error: bits is NULL");
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return dlm::fail(DLM_ERR_CUDA, "device synchronize: %s", cudaGetErrorString(e));
  int v = 0;
  e = cudaMemcpyFromSymbol(&v, g_dlm_device_error, sizeof(int));
  if (e != cudaSuccess) return dlm::fail(DLM_ERR_CUDA, "read error word: %s", cudaGetErrorString(e));
  if (clear) {
    const int zero = 0;
    e = cudaMemcpyToSymbol(g_dlm_device_error, &zero, sizeof(int));
    if (e != cudaSuccess) return dlm::fail(DLM_ERR_CUDA, "clear error word: %s", cudaGetErrorString(e));
  }
  *bits = v;
  return DLM_OK;
}

}  // extern "C"

namespace {

int attn_impl(const dlm_tensor* q, const dlm_tensor* k, const dlm_tensor* v, const dlm_tensor* seq_lens,
              const dlm_tensor* prompt_lens, int32_t mode, int32_t block, dlm_tensor* out) {
  using dlm::fail;
  int st;
  if (mode != DLM_ATTN_FULL && mode != DLM_ATTN_BLOCK_CAUSAL && mode != DLM_ATTN_BLOCK_LOCAL)
    return fail(DLM_ERR_ARG, "unknown attention mask mode %d", mode);
  if (mode != DLM_ATTN_FULL && block < 1) return fail(DLM_ERR_ARG, "block must be >= 1 for a block mask");
  if ((st = check_tensor(q, "q", kMaskBF16F32, 4, 4))) return st;
  if ((st = check_tensor(k, "k", kMaskBF16F32, 4, 4))) return st;
  if ((st = check_tensor(v, "v", kMaskBF16F32, 4, 4))) return st;
  if ((st = check_tensor(out, "out", kMaskBF16F32, 4, 4))) return st;
  if (k->dtype != q->dtype || v->dtype != q->dtype || out->dtype != q->dtype)
    return fail(DLM_ERR_DTYPE, "q, k, v and out must share one dtype");
  const int64_t B = q->shape[0], L = q->shape[1], Hq = q->shape[2], D = q->shape[3];
  const int64_t Hkv = k->shape[2];
  for (int i = 0; i < 4; ++i)
    if (out->shape[i] != q->shape[i]) return fail(DLM_ERR_SHAPE, "out must have the shape of q");
  for (int i = 0; i < 4; ++i)
    if (v->shape[i] != k->shape[i]) return fail(DLM_ERR_SHAPE, "v must have the shape of k");
  if (k->shape[0] != B || k->shape[1] != L || k->shape[3] != D)
    return fail(DLM_ERR_SHAPE, "k must be [B, L, Hkv, D] with the B, L, D of q");
  if (D != 64 && D != 128) return fail(DLM_ERR_SHAPE, "head_dim %lld not supported (64 or 128)", (long long)D);
  if (B * L > 0 && (Hkv < 1 || Hq < Hkv || Hq % Hkv != 0))
    return fail(DLM_ERR_SHAPE, "Hq (%lld) must be a positive multiple of Hkv (%lld)", (long long)Hq, (long long)Hkv);
  if (L > (1 << 24)) return fail(DLM_ERR_SHAPE, "L too large");
  if (seq_lens) {
    if ((st = check_tensor(seq_lens, "seq_lens", 1 << DLM_I32, 1, 1))) return st;
    if (seq_lens->shape[0] != B) return fail(DLM_ERR_SHAPE, "seq_lens must have B entries");
  }
  if (prompt_lens) {
    if ((st = check_tensor(prompt_lens, "prompt_lens", 1 << DLM_I32, 1, 1))) return st;
    if (prompt_lens->shape[0] != B) return fail(DLM_ERR_SHAPE, "prompt_lens must have B entries");
    if (overlaps(out, prompt_lens)) return fail(DLM_ERR_ARG, "out overlaps an input");
  }
  if (overlaps(out, q) || overlaps(out, k) || overlaps(out, v))
    return fail(DLM_ERR_ARG, "out overlaps an input");
  if (B == 0 || L == 0 || Hq == 0) return DLM_OK;
  dlm::AttnArgs a;
  a.q = q->data;
  a.k = k->data;
  a.v = v->data;
  a.out = out->data;
  a.seq_lens = seq_lens ? static_cast<const int32_t*>(seq_lens->data) : nullptr;
  a.prompt_lens = prompt_lens && mode != DLM_ATTN_FULL ? static_cast<const int32_t*>(prompt_lens->data) : nullptr;
  a.mask_mode = mode;
  a.block = mode != DLM_ATTN_FULL ? block : 1;
  a.B = static_cast<int>(B);
  a.L = static_cast<int>(L);
  a.Hq = static_cast<int>(Hq);
  a.Hkv = static_cast<int>(Hkv);
  a.D = static_cast<int>(D);
  for (int i = 0; i < 3; ++i) {
    a.sq[i] = q->stride[i];
    a.sk[i] = k->stride[i];
    a.sv[i] = v->stride[i];
    a.so[i] = out->stride[i];
  }
  if (q->dtype == DLM_BF16) {
    const dlm_tensor* ts[4] = {q, k, v, out};
    for (const dlm_tensor* t : ts) {
      if (reinterpret_cast<uintptr_t>(t->data) % 16 != 0)
        return fail(DLM_ERR_ALIGN, "bf16 attention needs 16-byte aligned base pointers");
      for (int i = 0; i < 3; ++i)
        if ((t->stride[i] * 2) % 16 != 0 || t->stride[i] * 2 >= (1LL << 40))
          return fail(DLM_ERR_ALIGN, "bf16 attention needs strides that are multiples of 16 bytes");
    }
    if ((st = require_error_word())) return st;
    return dlm::launch_attn_tc_bf16(a, t_stream);
  }
  if ((st = require_error_word())) return st;
  return dlm::launch_attn_f32(a, t_stream);
}

}  // namespace

extern "C" {

int dlm_bidir_attn(const dlm_tensor* q, const dlm_tensor* k, const dlm_tensor* v, const dlm_tensor* seq_lens,
                   dlm_tensor* out) {
  t_last_error[0] = '\0';
  return attn_impl(q, k, v, seq_lens, nullptr, DLM_ATTN_FULL, 1, out);
}

int dlm_attn_masked(const dlm_tensor* q, const dlm_tensor* k, const dlm_tensor* v, const dlm_tensor* seq_lens,
                    const dlm_tensor* prompt_lens, int32_t mode, int32_t block, dlm_tensor* out) {
  t_last_error[0] = '\0';
  return attn_impl(q, k, v, seq_lens, prompt_lens, mode, block, out);
}

}  // extern "C"

namespace {

// Validates a logits descriptor ([N, V] or [B, L, V], evenly strided rows)
// and fills the logits fields of *a.
int prepare_logits(const dlm_tensor* logits, dlm::VocabArgs* a) {
  using dlm::fail;
  int st;
  if ((st = check_tensor(logits, "logits", kMaskBF16F32, 2, 3))) return st;
  const int nd = logits->ndim;
  const int64_t V = logits->shape[nd - 1];
  int64_t N = 1;
  for (int i = 0; i < nd - 1; ++i) N *= logits->shape[i];
  int64_t row_stride = logits->stride[nd - 2];
  if (nd == 3 && logits->shape[1] > 1 && logits->shape[0] > 1 &&
      logits->stride[0] != logits->shape[1] * logits->stride[1])
    return fail(DLM_ERR_STRIDE, "logits rows must be evenly strided ([B, L, V] with stride[0] = L * stride[1])");
  if (N > 0 && V < 1) return fail(DLM_ERR_SHAPE, "V must be >= 1");
  if (N > 1 && row_stride < V) return fail(DLM_ERR_STRIDE, "logits rows overlap");
  a->logits = logits->data;
  a->is_bf16 = logits->dtype == DLM_BF16;
  a->N = N;
  a->V = V;
  a->row_stride = N > 1 ? row_stride : V;
  a->err = dlm::device_error_word();
  return DLM_OK;
}

// Validates the arguments of the vocabulary reduction and fills *a.
int prepare_vocab(const dlm_tensor* logits, dlm_tensor* argmax, dlm_tensor* conf, dlm_tensor* lse,
                  dlm::VocabArgs* a) {
  using dlm::fail;
  int st;
  if ((st = prepare_logits(logits, a))) return st;
  if ((st = check_tensor(argmax, "argmax", 1 << DLM_I32, 1, 3))) return st;
  if ((st = check_tensor(conf, "conf", 1 << DLM_F32, 1, 3))) return st;
  if ((st = check_tensor(lse, "lse", 1 << DLM_F32, 1, 3))) return st;
  const int64_t N = a->N;
  const dlm_tensor* outs[3] = {argmax, conf, lse};
  for (const dlm_tensor* t : outs) {
    if (numel(t) != N) return fail(DLM_ERR_SHAPE, "argmax, conf and lse must have one entry per logits row");
    if (!is_dense(t)) return fail(DLM_ERR_STRIDE, "argmax, conf and lse must be contiguous");
    if (overlaps(t, logits)) return fail(DLM_ERR_ARG, "outputs overlap logits");
  }
  if (overlaps(argmax, conf) || overlaps(argmax, lse) || overlaps(conf, lse))
    return fail(DLM_ERR_ARG, "outputs overlap each other");
  a->argmax = static_cast<int32_t*>(argmax->data);
  a->conf = static_cast<float*>(conf->data);
  a->lse = static_cast<float*>(lse->data);
  return DLM_OK;
}

// Validates the arguments of the refine update and fills *a.
int prepare_update(const dlm_tensor* tokens, const dlm_tensor* mask, const dlm_tensor* argmax, const dlm_tensor* conf,
                   const dlm_refine_params* params, dlm_tensor* new_tokens, dlm_tensor* new_mask, dlm_tensor* n_edits,
                   dlm::UpdateArgs* a) {
  using dlm::fail;
  int st;
  if ((st = check_tensor(tokens, "tokens", 1 << DLM_I32, 2, 2))) return st;
  if ((st = check_tensor(mask, "mask", 1 << DLM_U8, 2, 2))) return st;
  if ((st = check_tensor(argmax, "argmax", 1 << DLM_I32, 2, 2))) return st;
  if ((st = check_tensor(conf, "conf", 1 << DLM_F32, 2, 2))) return st;
  if ((st = check_tensor(new_tokens, "new_tokens", 1 << DLM_I32, 2, 2))) return st;
  if ((st = check_tensor(new_mask, "new_mask", 1 << DLM_U8, 2, 2))) return st;
  if ((st = check_tensor(n_edits, "n_edits", 1 << DLM_I32, 1, 1))) return st;
  if (!params) return fail(DLM_ERR_NULL, "params is NULL");
  const int64_t B = tokens->shape[0], L = tokens->shape[1];
  const dlm_tensor* bl[6] = {tokens, mask, argmax, conf, new_tokens, new_mask};
  for (const dlm_tensor* t : bl)
    if (t->shape[0] != B || t->shape[1] != L) return fail(DLM_ERR_SHAPE, "all [B, L] tensors must share B and L");
  if (n_edits->shape[0] != B) return fail(DLM_ERR_SHAPE, "n_edits must have B entries");
  if (L > (1 << 24)) return fail(DLM_ERR_SHAPE, "L too large (max 2^24)");
  if (B > 0 && (!params->prompt_lens || !params->seq_lens))
    return fail(DLM_ERR_NULL, "params: prompt_lens / seq_lens is NULL");
  if (reinterpret_cast<uintptr_t>(params->prompt_lens) % 4 != 0 || reinterpret_cast<uintptr_t>(params->seq_lens) % 4 != 0)
    return fail(DLM_ERR_ALIGN, "params: prompt_lens / seq_lens not 4-byte aligned");
  if (std::isnan(params->edit_threshold)) return fail(DLM_ERR_ARG, "edit_threshold is NaN");
  if (params->remask_k < 0 && !(params->remask_frac >= 0.f && params->remask_frac <= 1.f))
    return fail(DLM_ERR_ARG, "remask_frac must be in [0, 1] when remask_k < 0");
  // Outputs may alias their own input exactly; every other overlap is refused.
  if (!same_view(new_tokens, tokens) && overlaps(new_tokens, tokens))
    return fail(DLM_ERR_ARG, "new_tokens partially overlaps tokens");
  if (!same_view(new_mask, mask) && overlaps(new_mask, mask))
    return fail(DLM_ERR_ARG, "new_mask partially overlaps mask");
  const dlm_tensor* ins[4] = {tokens, mask, argmax, conf};
  const dlm_tensor* outs[3] = {new_tokens, new_mask, n_edits};
  for (int o = 0; o < 3; ++o)
    for (int i = 0; i < 4; ++i) {
      if ((o == 0 && i == 0) || (o == 1 && i == 1)) continue;
      if (overlaps(outs[o], ins[i])) return fail(DLM_ERR_ARG, "an output overlaps an input");
    }
  if (overlaps(new_tokens, new_mask) || overlaps(new_tokens, n_edits) || overlaps(new_mask, n_edits))
    return fail(DLM_ERR_ARG, "outputs overlap each other");
  a->tokens = static_cast<const int32_t*>(tokens->data);
  a->mask = static_cast<const uint8_t*>(mask->data);
  a->argmax = static_cast<const int32_t*>(argmax->data);
  a->conf = static_cast<const float*>(conf->data);
  a->new_tokens = static_cast<int32_t*>(new_tokens->data);
  a->new_mask = static_cast<uint8_t*>(new_mask->data);
  a->n_edits = static_cast<int32_t*>(n_edits->data);
  a->s_tokens = tokens->stride[0];
  a->s_mask = mask->stride[0];
  a->s_argmax = argmax->stride[0];
  a->s_conf = conf->stride[0];
  a->s_new_tokens = new_tokens->stride[0];
  a->s_new_mask = new_mask->stride[0];
  a->B = static_cast<int>(B);
  a->L = static_cast<int>(L);
  a->edit_threshold = params->edit_threshold;
  a->remask_k = params->remask_k;
  a->remask_frac = params->remask_frac;
  a->mask_id = params->mask_id;
  a->prompt_lens = params->prompt_lens;
  a->seq_lens = params->seq_lens;
  a->tok_prob = nullptr;
  a->s_tok_prob = 0;
  return DLM_OK;
}

// Validates the fused step's arguments (both parts plus their coupling).
int prepare_step(const dlm_tensor* logits, const dlm_tensor* tokens, const dlm_tensor* mask,
                 const dlm_refine_params* params, dlm_tensor* argmax, dlm_tensor* conf, dlm_tensor* lse,
                 dlm_tensor* new_tokens, dlm_tensor* new_mask, dlm_tensor* n_edits, dlm::VocabArgs* va,
                 dlm::UpdateArgs* ua) {
  using dlm::fail;
  int st;
  if ((st = prepare_vocab(logits, argmax, conf, lse, va))) return st;
  if ((st = prepare_update(tokens, mask, argmax, conf, params, new_tokens, new_mask, n_edits, ua))) return st;
  if (va->N != static_cast<int64_t>(ua->B) * ua->L)
    return fail(DLM_ERR_SHAPE, "logits must have one row per (sequence, position): B * L rows");
  if (logits->ndim == 3 && (logits->shape[0] != ua->B || logits->shape[1] != ua->L))
    return fail(DLM_ERR_SHAPE, "3-D logits must be [B, L, V]");
  if (!is_dense(argmax) || !is_dense(conf)) return fail(DLM_ERR_STRIDE, "argmax and conf must be contiguous [B, L]");
  const dlm_tensor* ins[3] = {tokens, mask, logits};
  const dlm_tensor* outs[6] = {argmax, conf, lse, new_tokens, new_mask, n_edits};
  for (int o = 0; o < 6; ++o)
    for (int i = 0; i < 3; ++i) {
      if ((o == 3 && i == 0) || (o == 4 && i == 1)) continue;  // in-place update allowed
      if (overlaps(outs[o], ins[i])) return fail(DLM_ERR_ARG, "an output overlaps an input");
    }
  for (int o = 0; o < 3; ++o)
    for (int q = 3; q < 6; ++q)
      if (overlaps(outs[o], outs[q])) return fail(DLM_ERR_ARG, "outputs overlap each other");
  return DLM_OK;
}

}  // namespace

extern "C" {

int dlm_vocab_confidence(const dlm_tensor* logits, dlm_tensor* argmax, dlm_tensor* conf, dlm_tensor* lse) {
  t_last_error[0] = '\0';
  dlm::VocabArgs a;
  int st = prepare_vocab(logits, argmax, conf, lse, &a);
  if (st != DLM_OK || a.N == 0) return st;
  if ((st = require_error_word())) return st;
  return dlm::launch_vocab_confidence(a, t_stream);
}

int dlm_refine_update(const dlm_tensor* tokens, const dlm_tensor* mask, const dlm_tensor* argmax,
                      const dlm_tensor* conf, const dlm_refine_params* params, dlm_tensor* new_tokens,
                      dlm_tensor* new_mask, dlm_tensor* n_edits) {
  t_last_error[0] = '\0';
  dlm::UpdateArgs a;
  int st = prepare_update(tokens, mask, argmax, conf, params, new_tokens, new_mask, n_edits, &a);
  if (st != DLM_OK || a.B == 0) return st;
  if ((st = require_error_word())) return st;
  return dlm::launch_refine_update(a, t_stream);
}

int dlm_token_prob(const dlm_tensor* logits, const dlm_tensor* tokens, const dlm_tensor* lse, dlm_tensor* prob) {
  using dlm::fail;
  t_last_error[0] = '\0';
  int st;
  dlm::VocabArgs a = {};
  if ((st = prepare_logits(logits, &a))) return st;
  if ((st = check_tensor(tokens, "tokens", 1 << DLM_I32, 1, 3))) return st;
  if ((st = check_tensor(lse, "lse", 1 << DLM_F32, 1, 3))) return st;
  if ((st = check_tensor(prob, "prob", 1 << DLM_F32, 1, 3))) return st;
  const int64_t N = a.N;
  if (numel(tokens) != N || numel(lse) != N || numel(prob) != N)
    return fail(DLM_ERR_SHAPE, "tokens, lse and prob must have one entry per logits row");
  if (!is_dense(tokens) || !is_dense(lse) || !is_dense(prob))
    return fail(DLM_ERR_STRIDE, "tokens, lse and prob must be contiguous");
  if (overlaps(prob, logits) || overlaps(prob, tokens) || overlaps(prob, lse))
    return fail(DLM_ERR_ARG, "prob overlaps an input");
  if (N == 0) return DLM_OK;
  if ((st = require_error_word())) return st;
  return dlm::launch_token_prob(a, static_cast<const int32_t*>(tokens->data), static_cast<const float*>(lse->data),
                                static_cast<float*>(prob->data), t_stream);
}

int dlm_refine_update_ranked(const dlm_tensor* tokens, const dlm_tensor* mask, const dlm_tensor* argmax,
                             const dlm_tensor* conf, const dlm_tensor* tok_prob, const dlm_refine_params* params,
                             dlm_tensor* new_tokens, dlm_tensor* new_mask, dlm_tensor* n_edits) {
  using dlm::fail;
  t_last_error[0] = '\0';
  dlm::UpdateArgs a;
  int st = prepare_update(tokens, mask, argmax, conf, params, new_tokens, new_mask, n_edits, &a);
  if (st != DLM_OK) return st;
  if ((st = check_tensor(tok_prob, "tok_prob", 1 << DLM_F32, 2, 2))) return st;
  if (tok_prob->shape[0] != a.B || tok_prob->shape[1] != a.L)
    return fail(DLM_ERR_SHAPE, "tok_prob must be [B, L]");
  const dlm_tensor* outs[3] = {new_tokens, new_mask, n_edits};
  for (const dlm_tensor* o : outs)
    if (overlaps(o, tok_prob)) return fail(DLM_ERR_ARG, "an output overlaps tok_prob");
  if (a.B == 0) return DLM_OK;
  if ((st = require_error_word())) return st;
  a.tok_prob = static_cast<const float*>(tok_prob->data);
  a.s_tok_prob = tok_prob->stride[0];
  return dlm::launch_refine_update(a, t_stream);
}

size_t dlm_lmhead_workspace_bytes(int64_t rows) { return rows > 0 ? dlm::lmhead_workspace_bytes(rows) : 0; }

int dlm_lmhead_confidence(const dlm_tensor* hidden, const dlm_tensor* weight, dlm_tensor* argmax, dlm_tensor* conf,
                          dlm_tensor* lse, void* workspace, size_t workspace_bytes) {
  using dlm::fail;
  t_last_error[0] = '\0';
  int st;
  if ((st = check_tensor(hidden, "hidden", 1 << DLM_BF16, 2, 3))) return st;
  if ((st = check_tensor(weight, "weight", 1 << DLM_BF16, 2, 2))) return st;
  if ((st = check_tensor(argmax, "argmax", 1 << DLM_I32, 1, 3))) return st;
  if ((st = check_tensor(conf, "conf", 1 << DLM_F32, 1, 3))) return st;
  if ((st = check_tensor(lse, "lse", 1 << DLM_F32, 1, 3))) return st;
  const int nd = hidden->ndim;
  const int64_t d = hidden->shape[nd - 1];
  int64_t N = 1;
  for (int i = 0; i < nd - 1; ++i) N *= hidden->shape[i];
  const int64_t V = weight->shape[0];
  const int64_t s_hidden = hidden->stride[nd - 2];
  if (nd == 3 && hidden->shape[0] > 1 && hidden->shape[1] > 1 && hidden->stride[0] != hidden->shape[1] * s_hidden)
    return fail(DLM_ERR_STRIDE, "3-D hidden must be [B, L, d] with evenly strided rows");
  if (weight->shape[1] != d) return fail(DLM_ERR_SHAPE, "weight must be [V, d] with the d of hidden");
  if (d < 64 || d % 64 != 0) return fail(DLM_ERR_SHAPE, "d must be a positive multiple of 64 (got %lld)", (long long)d);
  if (V < 1 && N > 0) return fail(DLM_ERR_SHAPE, "V must be >= 1");
  if (N > 0x7FFFFFFFLL || V > 0x7FFFFFFFLL) return fail(DLM_ERR_SHAPE, "N and V must be < 2^31");
  const dlm_tensor* mats[2] = {hidden, weight};
  for (const dlm_tensor* t : mats) {
    if (numel(t) == 0) continue;
    if (reinterpret_cast<uintptr_t>(t->data) % 16 != 0) return fail(DLM_ERR_ALIGN, "hidden / weight not 16-byte aligned");
    for (int i = 0; i < t->ndim - 1; ++i)
      if ((t->stride[i] * 2) % 16 != 0) return fail(DLM_ERR_ALIGN, "hidden / weight strides must be multiples of 16 bytes");
  }
  const dlm_tensor* outs[3] = {argmax, conf, lse};
  for (const dlm_tensor* t : outs) {
    if (numel(t) != N) return fail(DLM_ERR_SHAPE, "argmax, conf and lse must have one entry per row of hidden");
    if (!is_dense(t)) return fail(DLM_ERR_STRIDE, "argmax, conf and lse must be contiguous");
    if (overlaps(t, hidden) || overlaps(t, weight)) return fail(DLM_ERR_ARG, "an output overlaps an input");
  }
  if (overlaps(argmax, conf) || overlaps(argmax, lse) || overlaps(conf, lse))
    return fail(DLM_ERR_ARG, "outputs overlap each other");
  if (N == 0) return DLM_OK;
  if (!workspace) return fail(DLM_ERR_NULL, "workspace is NULL");
  if (reinterpret_cast<uintptr_t>(workspace) % 16 != 0) return fail(DLM_ERR_ALIGN, "workspace not 16-byte aligned");
  const size_t need = dlm::lmhead_workspace_bytes(N);
  if (workspace_bytes < need) return fail(DLM_ERR_ARG, "workspace too small: %zu bytes, %zu needed", workspace_bytes, need);
  const uintptr_t wlo = reinterpret_cast<uintptr_t>(workspace), whi = wlo + need;
  const dlm_tensor* all[5] = {hidden, weight, argmax, conf, lse};
  for (const dlm_tensor* t : all) {
    uintptr_t lo, hi;
    byte_span(t, &lo, &hi);
    if (numel(t) > 0 && lo < whi && wlo < hi) return fail(DLM_ERR_ARG, "workspace overlaps a tensor");
  }
  if ((st = require_error_word())) return st;
  dlm::LmArgs a;
  a.hidden = hidden->data;
  a.weight = weight->data;
  a.N = N;
  a.V = V;
  a.d = d;
  a.s_hidden = N > 1 ? s_hidden : d;
  a.s_weight = V > 1 ? weight->stride[0] : d;
  a.argmax = static_cast<int32_t*>(argmax->data);
  a.conf = static_cast<float*>(conf->data);
  a.lse = static_cast<float*>(lse->data);
  a.workspace = workspace;
  return dlm::launch_lmhead(a, t_stream);
}

size_t dlm_refine_step_workspace_bytes(int64_t batch) {
  return batch > 0 ? static_cast<size_t>(batch) * sizeof(int32_t) : 0;
}

int dlm_refine_step(const dlm_tensor* logits, const dlm_tensor* tokens, const dlm_tensor* mask,
                    const dlm_refine_params* params, dlm_tensor* argmax, dlm_tensor* conf, dlm_tensor* lse,
                    dlm_tensor* new_tokens, dlm_tensor* new_mask, dlm_tensor* n_edits, void* workspace,
                    size_t workspace_bytes) {
  using dlm::fail;
  t_last_error[0] = '\0';
  dlm::VocabArgs va;
  dlm::UpdateArgs ua;
  int st = prepare_step(logits, tokens, mask, params, argmax, conf, lse, new_tokens, new_mask, n_edits, &va, &ua);
  if (st != DLM_OK) return st;
  if (ua.B == 0 || va.N == 0) return DLM_OK;
  if (!workspace) return fail(DLM_ERR_NULL, "workspace is NULL");
  if (reinterpret_cast<uintptr_t>(workspace) % 4 != 0) return fail(DLM_ERR_ALIGN, "workspace not 4-byte aligned");
  if (workspace_bytes < dlm_refine_step_workspace_bytes(ua.B))
    return fail(DLM_ERR_ARG, "workspace too small: %zu bytes, %zu needed", workspace_bytes,
                dlm_refine_step_workspace_bytes(ua.B));
  const uintptr_t wlo = reinterpret_cast<uintptr_t>(workspace);
  const uintptr_t whi = wlo + dlm_refine_step_workspace_bytes(ua.B);
  const dlm_tensor* all[9] = {logits, tokens, mask, argmax, conf, lse, new_tokens, new_mask, n_edits};
  for (const dlm_tensor* t : all) {
    uintptr_t lo, hi;
    byte_span(t, &lo, &hi);
    if (numel(t) > 0 && lo < whi && wlo < hi) return fail(DLM_ERR_ARG, "workspace overlaps a tensor");
  }
  if ((st = require_error_word())) return st;
  return dlm::launch_vocab_step(va, ua, static_cast<int*>(workspace), t_stream);
}

}  // extern "C"

// ---------------------------------------------------------------------------
// dlm_refine_step_static: the fused step with library-owned scratch memory.
//
// For callers that cannot allocate device memory themselves: a serving engine
// whose allocator reserves nearly all of HBM for weights and KV cache up front
// (a cudaMalloc outside that pool fails or fragments it), a latency-critical
// loop that cannot afford cudaMalloc's implicit device synchronisation, or a
// plugin interface whose fixed signature has no slot for a workspace. Instead
// of a caller-provided workspace, the per-sequence arrival counters live in
// the file-scope array below: DLM_STATIC_STEP_MAX_BATCH int32 values (16 KB),
// held by every device that loads the library until the process exits.
//
// On the host, g_dlm_step_scratch is only a stand-in for the device symbol:
// its device address is taken once per device, with that device current, by
// cudaGetSymbolAddress on the first call on that device, and that address is
// what the kernel receives. Every call on a device shares the array and finds
// the last call's contents there, so each call clears the counters it uses
// (cudaMemsetAsync on the caller's stream) before the launch; two calls that
// overlap on the GPU race on the counters.
// ---------------------------------------------------------------------------
static __device__ __align__(256) int32_t g_dlm_step_scratch[DLM_STATIC_STEP_MAX_BATCH];

namespace {

std::mutex g_scratch_mu;
int32_t* g_scratch_addr[kMaxDevices] = {};

}  // namespace

namespace dlm {

// Device address of g_dlm_step_scratch on the current device (set up on first use).
int static_step_scratch(int32_t** out) {
  using dlm::fail;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(DLM_ERR_CUDA, "cudaGetDevice: %s", cudaGetErrorString(e));
  if (dev < 0 || dev >= kMaxDevices) return fail(DLM_ERR_UNSUPPORTED, "device ordinal %d out of range", dev);
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (!g_scratch_addr[dev]) {
    void* ptr = nullptr;
    e = cudaGetSymbolAddress(&ptr, g_dlm_step_scratch);
    if (e != cudaSuccess)
      return fail(DLM_ERR_CUDA, "cudaGetSymbolAddress(static step scratch): %s", cudaGetErrorString(e));
    g_scratch_addr[dev] = static_cast<int32_t*>(ptr);
  }
  *out = g_scratch_addr[dev];
  return DLM_OK;
}

}  // namespace dlm

extern "C" {

int dlm_refine_step_static(const dlm_tensor* logits, const dlm_tensor* tokens, const dlm_tensor* mask,
                           const dlm_refine_params* params, dlm_tensor* argmax, dlm_tensor* conf, dlm_tensor* lse,
                           dlm_tensor* new_tokens, dlm_tensor* new_mask, dlm_tensor* n_edits) {
  using dlm::fail;
  t_last_error[0] = '\0';
  dlm::VocabArgs va;
  dlm::UpdateArgs ua;
  int st = prepare_step(logits, tokens, mask, params, argmax, conf, lse, new_tokens, new_mask, n_edits, &va, &ua);
  if (st != DLM_OK) return st;
  if (ua.B == 0 || va.N == 0) return DLM_OK;
  if (ua.B > DLM_STATIC_STEP_MAX_BATCH)
    return fail(DLM_ERR_SHAPE, "batch %d exceeds the static scratch maximum of %d sequences (use dlm_refine_step)",
                ua.B, DLM_STATIC_STEP_MAX_BATCH);
  if ((st = require_error_word())) return st;
  int32_t* counters = nullptr;
  if ((st = dlm::static_step_scratch(&counters))) return st;
  cudaError_t e = cudaMemsetAsync(counters, 0, static_cast<size_t>(ua.B) * sizeof(int32_t), t_stream);
  if (e != cudaSuccess) return fail(DLM_ERR_CUDA, "clearing the static step scratch: %s", cudaGetErrorString(e));
  return dlm::launch_vocab_step(va, ua, counters, t_stream);
}

}  // extern "C"

#ifdef DLM_CHECK_BOUNDS
#include "dlmrefine_checked.h"

extern "C" int dlm_checked_fill_static_scratch(int32_t byte_value) {
  using dlm::fail;
  t_last_error[0] = '\0';
  if (byte_value < 0 || byte_value > 255) return fail(DLM_ERR_ARG, "byte_value %d outside 0..255", byte_value);
  int32_t* scratch = nullptr;
  if (const int st = dlm::static_step_scratch(&scratch)) return st;
  const cudaError_t e = cudaMemsetAsync(scratch, byte_value, sizeof(g_dlm_step_scratch), t_stream);
  if (e != cudaSuccess) return fail(DLM_ERR_CUDA, "filling the static step scratch: %s", cudaGetErrorString(e));
  return DLM_OK;
}

extern "C" int dlm_checked_set_wait_budget(int64_t budget_ns) {
  t_last_error[0] = '\0';
  if (budget_ns < 100 || budget_ns > static_cast<int64_t>(dlm::kDefaultWaitBudgetNs))
    return dlm::fail(DLM_ERR_ARG, "budget_ns %lld outside [100, 2e9]", static_cast<long long>(budget_ns));
  g_wait_budget_ns.store(static_cast<uint64_t>(budget_ns), std::memory_order_relaxed);
  return DLM_OK;
}
#endif  // DLM_CHECK_BOUNDS
