/*
 * Test hooks exported only by DLM_CHECK_BOUNDS builds of libdlmrefine
 * (python -m paper_2608_02625_gb300.build --check-bounds --out DIR); the
 * default build does not have them. None of them is part of the method.
 */
#ifndef DLMREFINE_CHECKED_H_
#define DLMREFINE_CHECKED_H_

#include "dlmrefine.h"

#ifdef __cplusplus
extern "C" {
#endif

/*
 * Fills every byte of dlm_refine_step_static's static scratch array on the
 * current device with `byte_value` (0..255), asynchronously on the calling
 * thread's stream. A test sets it to a nonzero pattern to check that each
 * static call clears the counters it uses before it counts. Returns
 * DLM_ERR_ARG for a value outside 0..255.
 */
int dlm_checked_fill_static_scratch(int32_t byte_value);

/*
 * Sets the budget of every bounded wait in the attention and fused
 * projection kernels launched afterwards by this library (default 2e9 ns;
 * 100 .. 2e9 accepted, DLM_ERR_ARG otherwise). With a budget of a few hundred
 * ns the waits of a real pipeline run out: the kernel records
 * DLM_DEVERR_TIMEOUT, lets the copies and MMAs it issued land, frees its
 * tensor memory and returns, leaving its outputs undefined. Calls made after
 * setting the budget back to 2e9 are unaffected. A checked build times every
 * wait, also one that completes at its first try, against the GPU's global
 * timer, whose resolution is about a microsecond: waits shorter than that may
 * not run out.
 */
int dlm_checked_set_wait_budget(int64_t budget_ns);

#ifdef __cplusplus
}
#endif

#endif /* DLMREFINE_CHECKED_H_ */
