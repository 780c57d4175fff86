/*
 * cm_testing.h - failure-injection hook of libcm, for tests of the bounded waits.
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

#ifdef __cplusplus
}  /* extern "C" */
#endif

#endif  /* CM_TESTING_H_ */
