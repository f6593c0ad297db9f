/*
 * ccq_diag.h -- diagnostic entry point of libccq.so (not part of the CCQ
 * computation; the paper has no counterpart).  It checks the tensor-core
 * operand layouts the CCQ kernels are built from.
 */
#ifndef CCQ_DIAG_H_
#define CCQ_DIAG_H_

#include "ccq.h"

#ifdef __cplusplus
extern "C" {
#endif

/*
 * A B on one CTA through the same shared-memory tiles, descriptors and
 * tcgen05.mma sequence as the CCQ kernels.
 *   A  device bf16 [M][K] row-major;  B device bf16 [K][N] row-major;
 *   D  device fp32 [128][N] row-major.  M = 128: the accumulator, TMEM lane i
 *      holding row i.  M = 64: rows 0..63 of D = A B read back with the
 *      16-lane split load the kernels use (rows 64..127 are not written).
 *   M in {64, 128}; N in {64, 128}; K in {64, 128}; a_mn / b_mn = 1 stage that
 *   operand MN-major in shared memory, 0 = K-major.
 * Asynchronous on `stream`; CCQ_ERR_UNSUPPORTED for other shapes.
 */
CCQ_API ccq_status ccq_diag_mma(const void *A, const void *B, float *D, int M, int N, int K,
                                int a_mn, int b_mn, void *stream);

/*
 * Exercises the kernels' failure path without a fault: one CTA waits on an
 * mbarrier that nothing arrives on, with the same bounded wait every CCQ kernel
 * uses (about one second of SM clock).  The wait gives up, records
 * CCQ_ERR_TIMEOUT in the device status word and the kernel returns normally,
 * so the context stays usable; ccq_device_status() then reports (and clears)
 * the timeout.  Asynchronous on `stream`.
 */
CCQ_API ccq_status ccq_diag_wait_timeout(void *stream);

#ifdef __cplusplus
}
#endif

#endif /* CCQ_DIAG_H_ */
