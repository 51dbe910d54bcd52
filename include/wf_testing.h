/* Test-only controls of libwf.  Not part of the library's interface: they
 * exist so that tests can drive the failure path of the tensor-core kernels'
 * bounded waits without faulting or hanging a GPU.
 *
 * The fused step kernel (wf_step) and the tensor-core sparse attention
 * (wf_sparse_attn for bf16 / head_dim 128) wait on mbarriers for copies,
 * tensor-core completion and cluster exchanges.  Every wait is bounded; when
 * one gives up, the kernel sets the status word that wf_workspace_status()
 * (or wf_noalloc_status()) reports as WF_ERR_TIMEOUT, stops issuing work,
 * drains what it already issued (copies in flight, tensor-core operations,
 * remote stores into its shared memory), frees its tensor memory and
 * returns; the outputs of that call are undefined and nothing outside them
 * is written.
 */
#ifndef WF_TESTING_H
#define WF_TESTING_H

#include "wf.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Controls for the launches that follow (process-wide, any thread):
 * - stall != 0: the first wait of each CTA (the fused kernel's tensor-core
 *   issuing thread, before its first MMA; the tensor-core attention's wait on
 *   its score MMAs) waits on a barrier that nothing completes, so it gives up
 *   after wait_limit_cycles and the kernel takes its failure path.
 * - wait_limit_cycles: the bound of every wait that can give up, in SM clock
 *   cycles; 0 restores the default (2^31 cycles, about one second).  Waits
 *   that drain work already issued keep the default bound.
 * Returns WF_ERR_INVALID_ARG for a negative limit. */
wf_status wf_testing_set_wait_failure(int stall, long long wait_limit_cycles);

#ifdef __cplusplus
}
#endif
#endif /* WF_TESTING_H */
