/*
 * cm_testing.h - testing hooks of libcm: failure injection for the bounded waits, and
 * the violation count of bounds-checked builds.
 *
 * The render kernel waits on its own TMA copies through mbarriers; every such wait
 * gives up after about one second of device time, records the failure in the
 * context and lets the kernel return, so a lost copy can never hang the GPU. This
 * call exercises that path without any fault: it renders like cm_render, except that
 * the first work item of one warp never has its copy issued, so that warp's wait runs
 * out. The render's output is incomplete; cm_context_check on the same stream then
 * returns CM_ERR_TIMEOUT, and the context stays usable. Not for production use.
 */
#ifndef CM_TESTING_H_
#define CM_TESTING_H_

#include "cm.h"

#ifdef __cplusplus
extern "C" {
#endif

/* cm_render with one withheld TMA load (warp 0 of CTA 0, its first item). Arguments as
 * for cm_render. Takes about two seconds of device time (the timed-out wait, then the
 * bounded wait for the withheld stage before the warp returns). */
cm_status cm_testing_render_withheld_load(const cm_set *set, void *k_out, void *v_out,
                                          int64_t capacity_tokens, cm_stream_t stream);

/* Bounds-checked builds of the library (compiled with -DCM_DEBUG_BOUNDS; build.py --bounds
 * writes libcm_bounds.so) test every global access of the render and content-address
 * kernels against the buffer it belongs to (a fragment, an output, a level of the hash
 * tree, the norm key, a paged block table and the lower end of a paged pool, whose size
 * the library is not told); an access outside it is counted and not made, so a wrong index
 * cannot fault. This call synchronises `device` and returns the number of such accesses on
 * it since the previous call (then zeroes it), and *out_enabled = 1 in a bounds-checked
 * build, 0 otherwise (where the count is always 0). CM_ERR_INVALID_ARG for NULL outputs;
 * CM_ERR_CUDA if the device cannot be selected or synchronised. */
cm_status cm_testing_bounds_violations(int32_t device, uint64_t *out_count, int32_t *out_enabled);

#ifdef __cplusplus
}  /* extern "C" */
#endif

#endif  /* CM_TESTING_H_ */
