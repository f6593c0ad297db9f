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
 * D = A B on one CTA through the same shared-memory tiles, descriptors and
 * tcgen05.mma sequence as the CCQ kernels.
 *   A  device bf16 [128][K] row-major;  B device bf16 [K][N] row-major;
 *   D  device fp32 [128][N] row-major (written).
 *   N in {64, 128}; K in {64, 128}; a_mn / b_mn = 1 stage that operand
 *   MN-major in shared memory, 0 = K-major.
 * Asynchronous on `stream`; CCQ_ERR_UNSUPPORTED for other shapes.
 */
CCQ_API ccq_status ccq_diag_mma(const void *A, const void *B, float *D, int N, int K, int a_mn,
                                int b_mn, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* CCQ_DIAG_H_ */
