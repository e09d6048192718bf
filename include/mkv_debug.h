/*
 * mkv_debug.h -- test hooks of the MomentKV library (no counterpart in the
 * paper).  They exist so that tests can drive the library's failure handling
 * on a GPU without faulting or hanging it: every device-side wait in the
 * kernels is bounded, and on running out records MKV_ERR_TIMEOUT in the
 * workspace's error word, waits (with the full limit) for the CTA's copies
 * and tensor-core operations in flight, and returns.  Production code does
 * not call these.  Both settings are process-wide, apply to launches made
 * after the call, and are not thread-safe with respect to launches on other
 * host threads.
 */
#ifndef MKV_DEBUG_H
#define MKV_DEBUG_H

#include <stdint.h>

#include "mkv.h"

#ifdef __cplusplus
extern "C" {
#endif

/*
 * Poll limit of the kernels' pipeline waits (tile copies and tensor-core
 * commits in mkv_compress and mkv_decode_step / mkv_decode_evict_step /
 * mkv_decode_step_noalloc).  polls < 0 restores the default (over a second
 * of polling); polls = 0 makes the first such wait of every CTA give up at
 * once, so the call records MKV_ERR_TIMEOUT and its outputs are undefined.
 * The eviction kernels have no such waits (their CTAs synchronise through
 * hardware cluster barriers), so mkv_evict_append is unaffected.  Returns
 * the previous limit (as a count of polls).
 */
MKV_API int64_t mkv_debug_set_poll_limit(int64_t polls);

/*
 * on = 1: mkv_decode_step and its variants merge the split-K partial states
 * through global memory (a ticket taken by the last CTA of a unit) instead
 * of in one thread-block cluster, as they do when a cluster of the split
 * count cannot be co-scheduled.  on = 0 restores the default.  Returns the
 * previous setting.
 */
MKV_API int32_t mkv_debug_force_ticket_merge(int32_t on);

#ifdef __cplusplus
}
#endif

#endif /* MKV_DEBUG_H */
