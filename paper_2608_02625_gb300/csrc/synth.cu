// libdlmsynth: the device twin of the seeded input generator (synth.py).
// Input generation only -- none of the refine step's arithmetic lives here.
#include <cuda_runtime.h>

#include <cstdint>

#include "dlmsynth.h"

namespace {

constexpr uint64_t kGolden = 0x9E3779B97F4A7C15ull;
constexpr int kIhMean = 393210;

__device__ __forceinline__ uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

__device__ __forceinline__ uint64_t draw(uint64_t key, uint64_t i) { return mix64(key + i * kGolden); }

__device__ __forceinline__ int lane_sum(uint64_t d) {
  return static_cast<int>((d & 0xFFFF) + ((d >> 16) & 0xFFFF) + ((d >> 32) & 0xFFFF) + (d >> 48));
}

__device__ __forceinline__ float normal(uint64_t key, uint64_t e, float c) {
  const int s = lane_sum(draw(key, 3 * e)) + lane_sum(draw(key, 3 * e + 1)) + lane_sum(draw(key, 3 * e + 2));
  return __fmul_rn(__int2float_rn(s - kIhMean), c);
}

__device__ __forceinline__ uint16_t to_bf16_bits(float x) {
  const uint32_t u = __float_as_uint(x);
  return static_cast<uint16_t>((u + 0x7FFFu + ((u >> 16) & 1u)) >> 16);
}

__device__ __forceinline__ int64_t uniform_int(uint64_t d, int64_t n) {
  return static_cast<int64_t>(((d >> 32) * static_cast<uint64_t>(n)) >> 32);
}

__device__ __forceinline__ void store(void* out, int dtype, int64_t off, float x) {
  if (dtype == 1) static_cast<uint16_t*>(out)[off] = to_bf16_bits(x);
  else static_cast<float*>(out)[off] = x;
}

__global__ void normal_kernel(void* out, int dtype, int64_t count, uint64_t key, int64_t e0, float c) {
  for (int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; e < count;
       e += static_cast<int64_t>(gridDim.x) * blockDim.x)
    store(out, dtype, e, normal(key, static_cast<uint64_t>(e0 + e), c));
}

__global__ void logits_kernel(void* out, int dtype, int64_t first_row, int64_t rows, int64_t V, int64_t row_stride,
                              uint64_t key, float c, const float* zipf, uint64_t key_shift) {
  const int64_t total = rows * V;
  for (int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; e < total;
       e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t lr = e / V, v = e - lr * V;
    const int64_t r = first_row + lr;
    float x = normal(key, static_cast<uint64_t>(r) * static_cast<uint64_t>(V) + v, c);
    if (zipf) {
      const int64_t sh = uniform_int(draw(key_shift, static_cast<uint64_t>(r)), V);
      x = __fadd_rn(zipf[(v + sh) % V], x);
    }
    store(out, dtype, lr * row_stride + v, x);
  }
}

__global__ void peaks_kernel(void* out, int dtype, int64_t first_row, int64_t rows, int64_t V, int64_t row_stride,
                             uint64_t key_peak, uint64_t peak_thresh, uint64_t current_thresh, float base,
                             float width, const int32_t* tokens, const uint8_t* mask) {
  const int64_t lr = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x;
  if (lr >= rows) return;
  const uint64_t r = static_cast<uint64_t>(first_row + lr);
  if ((draw(key_peak, 4 * r) >> 32) >= peak_thresh) return;
  int64_t t = uniform_int(draw(key_peak, 4 * r + 2), V);
  if (tokens && mask && mask[lr] == 0 && (draw(key_peak, 4 * r + 1) >> 32) < current_thresh) t = tokens[lr];
  const float u = __fmul_rn(static_cast<float>(draw(key_peak, 4 * r + 3) >> 40), 5.9604644775390625e-08f);
  const float val = __fadd_rn(__fmul_rn(u, width), base);
  store(out, dtype, lr * row_stride + t, val);
}

int grid_for(int64_t n) {
  int64_t g = (n + 255) / 256;
  return static_cast<int>(g < 1 ? 1 : (g > 1048576 ? 1048576 : g));
}

}  // namespace

extern "C" {

int dlm_synth_normal(void* out, int dtype, int64_t count, uint64_t key, int64_t e0, float scale_c, void* stream) {
  if (count <= 0) return 0;
  if (!out || (dtype != 1 && dtype != 2)) return -1;
  normal_kernel<<<grid_for(count), 256, 0, static_cast<cudaStream_t>(stream)>>>(out, dtype, count, key, e0, scale_c);
  return cudaGetLastError() == cudaSuccess ? 0 : -7;
}

int dlm_synth_logits(void* out, int dtype, int64_t first_row, int64_t rows, int64_t V, int64_t row_stride,
                     uint64_t key_logit, float scale_c, const float* zipf_table, uint64_t key_shift,
                     uint64_t key_peak, uint64_t peak_thresh, uint64_t current_thresh, float peak_base,
                     float peak_width, const int32_t* tokens, const uint8_t* mask, void* stream) {
  if (rows <= 0 || V <= 0) return 0;
  if (!out || (dtype != 1 && dtype != 2) || row_stride < V) return -1;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  logits_kernel<<<grid_for(rows * V), 256, 0, s>>>(out, dtype, first_row, rows, V, row_stride, key_logit, scale_c,
                                                   zipf_table, key_shift);
  if (peak_thresh > 0)
    peaks_kernel<<<static_cast<int>((rows + 255) / 256), 256, 0, s>>>(out, dtype, first_row, rows, V, row_stride,
                                                                     key_peak, peak_thresh, current_thresh,
                                                                     peak_base, peak_width, tokens, mask);
  return cudaGetLastError() == cudaSuccess ? 0 : -7;
}

}  // extern "C"
