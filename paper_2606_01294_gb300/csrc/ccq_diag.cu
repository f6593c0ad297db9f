// ccq_diag.cu -- layout self-test of the tensor-core building blocks.
//
// One CTA stages A (M x K, M in {64, 128}) and B (K x N) from global memory into the same
// 128-byte-swizzled T64 tiles the CCQ kernels use -- K-major or MN-major for
// each operand -- issues the tcgen05.mma sequence over K with the kernels'
// descriptors, and dumps all 128 TMEM lanes x N columns of the accumulator
// (lanes the MMA does not write read back as NaN) through tcgen05.ld.  The C ABI
// entry point ccq_diag_mma (include/ccq_diag.h) lets tests check every
// descriptor form against a plain matrix product.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/ccq_diag.h"
#include "ccq_internal.h"
#include "sm100_ptx.cuh"

namespace ccq {
namespace {

// A tile set: K-major -> tiles [128 rows (m)][64 k] for each 64-wide K block
// (tile bytes 16K); MN-major -> tiles [K rows][64 m] for each 64-wide M block
// (tile bytes K*128).  B likewise with N in place of M.
__global__ void __launch_bounds__(128, 1)
diag_mma_kernel(const __nv_bfloat16 *A, const __nv_bfloat16 *Bm, float *D, int M, int N, int K,
                int a_mn, int b_mn, int *status) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = smem_align1024(smem_raw);
    const uint32_t sb = smem_addr(sm);
    uint8_t *sa = sm;               // up to 32K
    uint8_t *sbm = sm + 32768;      // up to 32K
    uint64_t *bar = reinterpret_cast<uint64_t *>(sm + 65536);
    uint32_t *slot = reinterpret_cast<uint32_t *>(sm + 65536 + 8);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(sm + 65536 + 12);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    if (tid == 0) {
        mbar_init(bar, 1);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 0) tmem_alloc(slot, 128);
    // stage A (logical [M][K] row-major in global)
    for (int e = tid; e < M * K; e += 128) {
        const int m = e / K, k = e % K;
        uint32_t off;
        if (!a_mn) off = (k >> 6) * (M * 128) + t64_offset(m, k & 63);
        else off = (m >> 6) * (K * 128) + t64_offset(k, m & 63);
        *reinterpret_cast<__nv_bfloat16 *>(sa + off) = A[e];
    }
    // stage B (logical [K][N] row-major in global)
    for (int e = tid; e < K * N; e += 128) {
        const int k = e / N, n = e % N;
        uint32_t off;
        if (!b_mn) off = (k >> 6) * (N * 128) + t64_offset(n, k & 63);
        else off = (n >> 6) * (K * 128) + t64_offset(k, n & 63);
        *reinterpret_cast<__nv_bfloat16 *>(sbm + off) = Bm[e];
    }
    fence_proxy_async_smem();
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *slot;
    {
        // mark every TMEM lane / column first, so lanes the MMA does not write show NaN
        float nanv[32];
        for (int i = 0; i < 32; ++i) nanv[i] = __int_as_float(0x7fc00000);
        for (int c = 0; c < N; c += 32)
            tmem_st32(tbase + (static_cast<uint32_t>(32 * warp) << 16) + c, nanv);
        tmem_wait_st();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (tid == 0) {
        const uint32_t idesc = make_idesc(M, N, a_mn, b_mn);
        for (int k16 = 0; k16 < K / 16; ++k16) {
            const uint64_t ad = a_mn ? desc_mnmajor(sb, K * 128, k16)
                                     : desc_kmajor(sb + (k16 >> 2) * (M * 128), k16 & 3);
            const uint64_t bd = b_mn ? desc_mnmajor(sb + 32768, K * 128, k16)
                                     : desc_kmajor(sb + 32768 + (k16 >> 2) * (N * 128), k16 & 3);
            mma_bf16(tbase, ad, bd, idesc, k16 != 0);
        }
        mma_commit(bar);
    }
    mbar_wait(bar, 0, abort_flag, status);
    tc_fence_after();
    if (M == 128 || N == 0) {
        const int row = 32 * warp + lane;
        for (int c = 0; c < N; c += 32) {
            float x[32];
            tmem_ld32(tbase + (static_cast<uint32_t>(32 * warp) << 16) + c, x);
            for (int i = 0; i < 32; ++i) D[row * N + c + i] = x[i];
        }
    } else {
        // M = 64: rows 16w..16w+15 of warp w, read with the 16-lane split load;
        // D rows 64..127 are left untouched
        const int row = 16 * warp + (lane & 15), half = lane >> 4;
        const uint32_t ta = tbase + (static_cast<uint32_t>(32 * warp) << 16);
        float x[32];
        if (N == 64) {
            tmem_ld16x2_32<32>(ta, x);
            for (int i = 0; i < 32; ++i) D[row * N + 32 * half + i] = x[i];
        } else {
            tmem_ld16x2_32<64>(ta, x);
            for (int i = 0; i < 32; ++i) D[row * N + 64 * half + i] = x[i];
            tmem_ld16x2_32<64>(ta + 32, x);
            for (int i = 0; i < 32; ++i) D[row * N + 64 * half + 32 + i] = x[i];
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tbase, 128);
    }
}

// Waits (bounded) on a barrier that no thread or copy ever completes.
__global__ void diag_wait_kernel(int *status) {
    __shared__ uint64_t bar;
    __shared__ int abort_flag;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        abort_flag = 0;
        fence_barrier_init();
    }
    __syncthreads();
    mbar_wait(&bar, 0, &abort_flag, status);
}

}  // namespace
}  // namespace ccq

extern "C" CCQ_API ccq_status ccq_diag_wait_timeout(void *stream) {
    int *status = ccq::device_status_word();
    if (!status) return CCQ_ERR_CUDA;
    ccq::diag_wait_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(status);
    return cudaGetLastError() == cudaSuccess ? CCQ_OK : CCQ_ERR_CUDA;
}

extern "C" CCQ_API ccq_status ccq_diag_mma(const void *A, const void *B, float *D, int M, int N,
                                           int K, int a_mn, int b_mn, void *stream) {
    if (!A || !B || !D) return CCQ_ERR_INVALID_ARG;
    if ((M != 64 && M != 128) || (N != 64 && N != 128) || (K != 64 && K != 128) ||
        (a_mn | b_mn) > 1 || a_mn < 0 || b_mn < 0)
        return CCQ_ERR_UNSUPPORTED;
    int *status = ccq::device_status_word();
    if (!status) return CCQ_ERR_CUDA;
    const int smem = 65536 + 64 + 1024;
    if (cudaFuncSetAttribute(ccq::diag_mma_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) !=
        cudaSuccess)
        return CCQ_ERR_CUDA;
    ccq::diag_mma_kernel<<<1, 128, smem, static_cast<cudaStream_t>(stream)>>>(
        static_cast<const __nv_bfloat16 *>(A), static_cast<const __nv_bfloat16 *>(B), D, M, N, K,
        a_mn, b_mn, status);
    return cudaGetLastError() == cudaSuccess ? CCQ_OK : CCQ_ERR_CUDA;
}
