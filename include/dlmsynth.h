/*
 * libdlmsynth -- seeded synthetic inputs for libdlmrefine, generated on the GPU.
 *
 * Input generation only: this library holds none of the refine step's
 * arithmetic. It is the device twin of paper_2608_02625_gb300/synth.py and
 * produces the same bits for the same (key, element index), so tensors of
 * tens of GB are generated in HBM at full speed while any slice can be
 * regenerated on the host.
 *
 * Definitions (shared with the host module):
 *   mix64      SplitMix64's output function (Steele, Lea & Flood, OOPSLA 2014)
 *   draw(k, i) mix64(k + i * 0x9E3779B97F4A7C15) (mod 2^64)
 *   normal     element e: the 12 16-bit lanes of draw(k, 3e), draw(k, 3e+1),
 *              draw(k, 3e+2) summed, minus 393210, converted to fp32 (exact)
 *              and multiplied once (round to nearest) by scale_c, where
 *              scale_c = fp32(sigma) * 2^-16
 *   bf16       round to nearest even of the fp32 value
 * All pointers are device pointers of the current device; calls are
 * asynchronous on `stream` (a cudaStream_t). Return 0 or a negative code.
 */
#ifndef DLMSYNTH_H_
#define DLMSYNTH_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* dtype: 1 = bf16, 2 = fp32 (the dlm_dtype codes). out[e] = normal(key, e0 + e), e < count. */
int dlm_synth_normal(void* out, int dtype, int64_t count, uint64_t key, int64_t e0, float scale_c,
                     void* stream);

/*
 * Logits of `rows` positions (row r = first_row + local row), row-major with
 * row stride `row_stride` elements:
 *   x[r, v] = base(r, v) + normal(key_logit, r * V + v)
 *   base(r, v) = 0, or zipf_table[(v + shift_r) % V] when zipf_table != NULL,
 *   with shift_r = uniform_int(draw(key_shift, r), V).
 * Then, for rows with hi32(draw(key_peak, 4r)) < peak_thresh: the token
 *   t = uniform_int(draw(key_peak, 4r+2), V), replaced by tokens[r] when
 *   tokens != NULL, mask[r] == 0 and hi32(draw(key_peak, 4r+1)) < current_thresh,
 * gets the value peak_base + peak_width * unit(draw(key_peak, 4r+3)), where
 * unit(d) = (d >> 40) * 2^-24, multiply then add, each rounded to nearest.
 * uniform_int(d, n) = (hi32(d) * n) >> 32.
 */
int dlm_synth_logits(void* out, int dtype, int64_t first_row, int64_t rows, int64_t V, int64_t row_stride,
                     uint64_t key_logit, float scale_c, const float* zipf_table, uint64_t key_shift,
                     uint64_t key_peak, uint64_t peak_thresh, uint64_t current_thresh, float peak_base,
                     float peak_width, const int32_t* tokens, const uint8_t* mask, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* DLMSYNTH_H_ */
