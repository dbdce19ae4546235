// Step A1, fp32 path -- non-causal GQA attention on the CUDA cores.
//
// Sec. 4.2: every valid position attends to every valid position (the block
// masks of dlm_attn_masked restrict each query to its key ranges). fp32
// inputs call for fp32 arithmetic throughout (TF32 tensor cores would not hold
// a 1e-5 error bound), so this path is a plain online-softmax loop: one warp
// per query row, lanes split the head dimension, a key's score is a warp
// reduction, and the running maximum / sum / output are rescaled with expf.
#include <cmath>
#include <cstdint>

#include "dlm_common.cuh"
#include "dlm_internal.h"

namespace dlm {
namespace {

constexpr int kWarpsPerBlock = 8;

template <int D>
__global__ void __launch_bounds__(kWarpsPerBlock * 32) attn_f32_kernel(AttnArgs a, float scale, int* err) {
  constexpr int kPer = D / 32;
  const int lane = threadIdx.x & 31;
  const int i = blockIdx.x * kWarpsPerBlock + (threadIdx.x >> 5);
  const int h = blockIdx.y;
  const int b = blockIdx.z;
  if (i >= a.L) return;
  int n = a.seq_lens ? a.seq_lens[b] : a.L;
  if (n < 0 || n > a.L) {
    if (lane == 0) set_device_error(err, DLM_DEVERR_LENGTH);
    n = n < 0 ? 0 : a.L;
  }
  const int g = (h * a.Hkv) / a.Hq;
  float* o = static_cast<float*>(a.out) + b * a.so[0] + i * a.so[1] + h * a.so[2];
  if (i >= n) {
#pragma unroll
    for (int t = 0; t < kPer; ++t) o[lane + 32 * t] = 0.f;
    return;
  }
  const float* qp = static_cast<const float*>(a.q) + b * a.sq[0] + i * a.sq[1] + h * a.sq[2];
  const float* kb = static_cast<const float*>(a.k) + b * a.sk[0] + g * a.sk[2];
  const float* vb = static_cast<const float*>(a.v) + b * a.sv[0] + g * a.sv[2];
  float q[kPer], acc[kPer];
#pragma unroll
  for (int t = 0; t < kPer; ++t) {
    q[t] = qp[lane + 32 * t] * scale;
    acc[t] = 0.f;
  }
  int p = 0;
  if (a.mask_mode != DLM_ATTN_FULL && a.prompt_lens) {
    p = a.prompt_lens[b];
    if (p < 0 || p > n) {
      if (lane == 0) set_device_error(err, DLM_DEVERR_LENGTH);
      p = p < 0 ? 0 : n;
    }
  }
  const KeyRanges kr = key_ranges(a.mask_mode, a.block, i, n, p);
  float m = -INFINITY, l = 0.f;
  for (int j = 0; j < kr.hi2; ++j) {
    if (j == kr.hi1 && kr.lo2 > j) j = kr.lo2;   // skip the keys between the two ranges
    if (j >= kr.hi2) break;
    const float* kj = kb + j * a.sk[1];
    float s = 0.f;
#pragma unroll
    for (int t = 0; t < kPer; ++t) s = fmaf(q[t], kj[lane + 32 * t], s);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
    const float m_new = fmaxf(m, s);
    const float corr = expf(m - m_new);  // 0 on the first key (m = -inf)
    const float pj = expf(s - m_new);
    l = l * corr + pj;
    const float* vj = vb + j * a.sv[1];
#pragma unroll
    for (int t = 0; t < kPer; ++t) acc[t] = fmaf(pj, vj[lane + 32 * t], acc[t] * corr);
    m = m_new;
  }
  const float inv = 1.0f / l;
#pragma unroll
  for (int t = 0; t < kPer; ++t) o[lane + 32 * t] = acc[t] * inv;
}

}  // namespace

int launch_attn_f32(const AttnArgs& a, cudaStream_t stream) {
  if (a.B == 0 || a.L == 0) return DLM_OK;
  dim3 grid((a.L + kWarpsPerBlock - 1) / kWarpsPerBlock, a.Hq, a.B);
  const float scale = 1.0f / sqrtf(static_cast<float>(a.D));
  if (a.D == 64) {
    attn_f32_kernel<64><<<grid, kWarpsPerBlock * 32, 0, stream>>>(a, scale, device_error_word());
  } else {
    attn_f32_kernel<128><<<grid, kWarpsPerBlock * 32, 0, stream>>>(a, scale, device_error_word());
  }
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return fail(DLM_ERR_CUDA, "attn_f32 launch: %s", cudaGetErrorString(e));
  return DLM_OK;
}

}  // namespace dlm
