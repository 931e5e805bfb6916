/*
 * commitkv_testing.h — test support of libcommitkv.so (not part of the hot
 * path).
 *
 * The greedy joint test (Section 3.3, Eq. 11) runs as one cooperative kernel
 * whose blocks meet at a grid barrier once per candidate; every wait at that
 * barrier is bounded (about one second), after which the kernel records
 * COMMITKV_ERR_TIMEOUT in the workspace status word and returns, leaving the
 * CUDA context usable.  This entry point makes that wait run out on purpose:
 * it launches `blocks` blocks at the same barrier code but tells it to
 * expect blocks + 1 arrivals, so the wait can only end by its limit.
 *
 *   workspace  an initialised CommitKV workspace (>= 256 bytes).
 *   blocks     1..64 co-resident blocks.
 * Returns COMMITKV_OK if the kernel was launched; the timeout is then read
 * with commitkv_workspace_status (expected: COMMITKV_ERR_TIMEOUT).
 */
#ifndef COMMITKV_TESTING_H
#define COMMITKV_TESTING_H

#include "commitkv.h"

#ifdef __cplusplus
extern "C" {
#endif

commitkv_status commitkv_test_barrier_timeout(void *workspace, size_t workspace_bytes,
                                              int32_t blocks, cudaStream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* COMMITKV_TESTING_H */
