// ccq_gdn_bwd_tc.cuh -- the tensor-core product of the CCQ-Gated-DeltaNet backward's per-chunk
// kernels (gdn_bwd_local_kernel and gdn_bwd_kv_kernel, instantiated with TC = true for bf16
// inputs).
//
// Those kernels keep their operands as fp32 tiles in shared memory (row strides D + 1 and 65) and
// evaluate some thirty small products a chunk,
//   out(m, n) = sum_{k<K} A[m ars + k acs] B[k brs + n bcs],   M in {64, 128}, N in {64, 128},
// the same contract as tile_mm.  tc_mm runs one on the tensor core: the CTA's 512 threads convert
// the operands kTcSliceK reduction steps at a time into bf16 MN-major slices (SK K-rows of 64 M-
// or N-columns, 128-byte swizzled; one 16-byte chunk of eight consecutive M or N a thread), one
// thread issues the slice's K = 16 tcgen05.mma into an fp32 TMEM accumulator, and (with more than
// one staging buffer) the next slice is converted while they run.  Then every thread reads its share of
// the accumulator (one row, N/8 or N/4 consecutive columns) and hands it to the epilogue.  The
// operand strides are odd in shared memory, so the lanes of a warp (32 consecutive K-rows of one
// 8-row group) convert without bank conflicts.  Operands may also be in global memory.
//
// Rounding: operands to bf16 (round to nearest even), accumulation in fp32 -- the precision of the
// forward's tensor-core products.
#pragma once

#include <cuda_bf16.h>
#include <stdint.h>

#ifdef __CUDACC__
#include "sm100_ptx.cuh"
#endif

namespace ccq {
namespace gbwd {

// Per-CTA state of the tensor-core products: two staging buffers and their commit barriers, the
// TMEM accumulator (128 columns), the give-up flag of the bounded waits and the status word.
struct TcEng {
    uint8_t *stage;
    int stride;  // bytes of one staging buffer
    int nbuf;    // staging buffers (1 to 4), used in turn
    uint64_t *bar;  // [nbuf] commit barriers
    uint32_t *tmem_slot;
    volatile int *abort;
    int *status;
    uint32_t tmem;
    uint32_t used, par;  // bit b: buffer b has a commit; the parity of its last commit
    int next;            // the buffer the next slice goes to
    float *host_acc;     // host builds: the accumulator ([128][128] fp32)
};

// Reduction steps per staged slice (16, 32 or 64; M = 128 products take 16), and the staging
// buffers of the local and the kv kernel.  Measured on the backward (B=4, H=16, T=4096):
// 16-deep slices in two buffers 7.82 ms, in three or four 7.83 ms, 32-deep in two 7.45 ms, and
// (after the non-product phases were reworked) 32-deep in two 6.89 ms, 64-deep in one 6.33 ms:
// each slice costs a conversion pass and a block barrier, the MMA round trip hardly shows.
constexpr int kTcSliceK = 64;
constexpr int kTcBufLocal = 1, kTcBufKv = 1;

// Bytes of one staging slice of an M x N product: an SK x 64 bf16 tile per 64 rows or columns.
constexpr int tc_stage_bytes(int M, int N, int SK) { return (M / 64 + N / 64) * SK * 128; }
// Shared memory the engine adds behind a kernel's own: 1024-byte alignment, the staging buffers,
// the barriers, the TMEM address and the give-up flag.
constexpr int tc_smem_bytes(int stage, int nbuf) { return 1024 + nbuf * stage + 64; }
constexpr int kTcCols = 128;

#ifdef __CUDACC__

// Set up (all threads): `region` is the first byte behind the kernel's own shared memory.
__device__ __forceinline__ void tc_setup(TcEng &e, uint8_t *region, int stage_bytes, int nbuf, int *status) {
    e.stage = smem_align1024(region);
    e.stride = stage_bytes;
    e.nbuf = nbuf;
    uint8_t *misc = e.stage + nbuf * stage_bytes;
    e.bar = reinterpret_cast<uint64_t *>(misc);
    e.tmem_slot = reinterpret_cast<uint32_t *>(misc + 32);
    e.abort = reinterpret_cast<volatile int *>(misc + 36);
    e.status = status;
    e.used = e.par = 0;
    e.next = 0;
    if (threadIdx.x == 0) {
        for (int b = 0; b < nbuf; ++b) mbar_init(&e.bar[b], 1);
        *e.abort = 0;
        fence_barrier_init();
    }
    if (threadIdx.x < 32) tmem_alloc(e.tmem_slot, kTcCols);
    __syncthreads();
    tc_fence_after();
    e.tmem = *e.tmem_slot;
}

// Tear down (all threads, uniform control flow): after a give-up, wait (bounded) for the
// products still in flight, then free the TMEM.
__device__ __forceinline__ void tc_teardown(TcEng &e) {
    if (threadIdx.x == 0 && *e.abort) {
        for (int b = 0; b < e.nbuf; ++b)
            if ((e.used >> b) & 1u) mbar_drain(&e.bar[b], (e.par >> b) & 1u);
    }
    tc_fence_before();
    __syncthreads();
    if (threadIdx.x < 32) {
        tc_fence_after();
        tmem_dealloc(e.tmem, kTcCols);
    }
}

// Wait until the last product issued from buffer b has completed.
__device__ __forceinline__ void tc_wait_buf(TcEng &e, int b) {
    if ((e.used >> b) & 1u) mbar_wait(&e.bar[b], (e.par >> b) & 1u, e.abort, e.status);
}

// 16 fp32 columns of the thread's TMEM lane quadrant as two half-warps: threads 0-15 lanes 0-15 at
// columns [c, c + NR), threads 16-31 the same lanes at [c + NR, c + 2 NR).
template <int NR>
__device__ __forceinline__ void tmem_ld16x2(uint32_t taddr, float (&v)[NR]);
template <>
__device__ __forceinline__ void tmem_ld16x2<8>(uint32_t taddr, float (&v)[8]) {
    uint32_t r[8];
    asm volatile("tcgen05.ld.sync.aligned.16x32bx2.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8], 8;"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
                   "=r"(r[7])
                 : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 8; ++i) v[i] = __uint_as_float(r[i]);
}
template <>
__device__ __forceinline__ void tmem_ld16x2<16>(uint32_t taddr, float (&v)[16]) {
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.16x32bx2.x16.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16], 16;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// Convert reduction steps [k0, k0 + SK) of A (M x K) and B (N x K) into the MN-major SK x 64
// tiles of buffer buf: A's M/64 tiles first, then B's N/64.  Item it (one 16-byte chunk) is K-row
// k of the 8-row group mc of its operand: for SK >= 32 a warp takes 32 consecutive K-rows of one
// group, for SK = 16 its two halves take groups 16 rows apart.
template <int M, int N, int SK>
__device__ __forceinline__ void tc_stage(uint8_t *buf, const float *A, int ars, int acs, const float *B, int brs,
                                         int bcs, int k0) {
    constexpr int kA = M / 8 * SK, kItems = (M + N) / 8 * SK, kTile = SK * 128;
    for (int it = static_cast<int>(threadIdx.x); it < kItems; it += static_cast<int>(blockDim.x)) {
        const bool isA = it < kA;
        const int j = isA ? it : it - kA;
        int k, mc;
        if constexpr (SK >= 32) {
            k = j & (SK - 1);
            mc = j / SK;
        } else {
            const int p = j >> 5;
            k = j & 15;
            mc = (p & 1) + ((p >> 1) << 2) + 2 * ((j >> 4) & 1);
        }
        const float *src = isA ? A + static_cast<long long>(k0 + k) * acs + static_cast<long long>(8 * mc) * ars
                               : B + static_cast<long long>(k0 + k) * brs + static_cast<long long>(8 * mc) * bcs;
        const int st = isA ? ars : bcs;
        float f[8];
#pragma unroll
        for (int x = 0; x < 8; ++x) f[x] = src[static_cast<long long>(x) * st];
        uint4 u;
        u.x = pack_bf16(f[0], f[1]);
        u.y = pack_bf16(f[2], f[3]);
        u.z = pack_bf16(f[4], f[5]);
        u.w = pack_bf16(f[6], f[7]);
        uint8_t *dst = buf + (isA ? 0 : (M / 64) * kTile) + (mc >> 3) * kTile + t64_chunk(k, mc & 7);
        *reinterpret_cast<uint4 *>(dst) = u;
    }
}

// Stage and issue an M x N x K product into the TMEM accumulator (every thread of the 512-thread
// CTA calls it, operands complete and visible): on top of what the accumulator holds when acc
// (products chained this way sum), else in its place.  Nothing is read back; the operand tiles may
// be overwritten as soon as it returns.
template <int M, int N, int K>
__device__ __forceinline__ void tc_mma(TcEng &e, const float *A, int ars, int acs, const float *B, int brs, int bcs,
                                       bool acc) {
    constexpr int SK = M == 128 ? 16 : kTcSliceK;  // e.stride >= tc_stage_bytes(M, N, SK)
    static_assert((M == 64 || M == 128) && (N == 64 || N == 128) && K % SK == 0 && K > 0, "tc_mm shape");
    constexpr int kTile = SK * 128;
    constexpr uint32_t kIdesc = make_idesc(M, N, 1, 1);
#pragma unroll 1
    for (int ks = 0; ks < K / SK; ++ks) {
        const int b = e.next;
        e.next = e.next + 1 == e.nbuf ? 0 : e.next + 1;
        uint8_t *buf = e.stage + b * e.stride;
        tc_wait_buf(e, b);
        tc_stage<M, N, SK>(buf, A, ars, acs, B, brs, bcs, SK * ks);
        fence_proxy_async_smem();
        __syncthreads();
        if (threadIdx.x == 0 && !*e.abort) {
            tc_fence_after();
            const uint32_t sa = smem_addr(buf);
#pragma unroll
            for (int k16 = 0; k16 < SK / 16; ++k16)
                mma_bf16(e.tmem, make_desc(sa + 2048 * k16, kTile, 1024),
                         make_desc(sa + (M / 64) * kTile + 2048 * k16, kTile, 1024), kIdesc,
                         (acc || ks > 0 || k16 > 0) ? 1u : 0u);
            mma_commit(&e.bar[b]);
        }
        e.par = ((e.used >> b) & 1u) ? (e.par ^ (1u << b)) : (e.par & ~(1u << b));
        e.used |= 1u << b;
    }
}

// Wait for the products issued so far and hand the M x N accumulator to the epilogue:
// ep(i, j0, v) receives row i, columns [j0, j0 + NV) in v[NV], NV = M N / 512; each output is
// handed over once.  Returns after every thread's epilogue (a block barrier).
template <int M, int N, typename Ep>
__device__ __forceinline__ void tc_read(TcEng &e, Ep ep) {
    constexpr int kNV = M * N / 512;
    for (int b = 0; b < e.nbuf; ++b) tc_wait_buf(e, b);
    tc_fence_after();
    {
        const int warp = static_cast<int>(threadIdx.x >> 5), lane = static_cast<int>(threadIdx.x & 31);
        const int q = warp & 3, cg = warp >> 2;
        const uint32_t tq = e.tmem + (static_cast<uint32_t>(32 * q) << 16) + static_cast<uint32_t>(cg * (N / 4));
        float v[kNV];
        if constexpr (M == 64) {
            // rows 16q..16q+15 sit in TMEM lanes 32q..32q+15
            tmem_ld16x2<kNV>(tq, v);
            ep(16 * q + (lane & 15), cg * (N / 4) + (lane >> 4) * kNV, v);
        } else {
            if constexpr (kNV == 32) tmem_ld32(tq, v);
            else tmem_ld16(tq, v);
            ep(32 * q + lane, cg * (N / 4), v);
        }
    }
    tc_fence_before();
    __syncthreads();
}

// The element-wise form of tc_read: ep(i, j, value), as tile_mm calls it.
template <int M, int N, typename Ep>
__device__ __forceinline__ void tc_read_elem(TcEng &e, Ep ep) {
    constexpr int kNV = M * N / 512;
    tc_read<M, N>(e, [&](int i, int j0, const float (&v)[kNV]) {
#pragma unroll
        for (int c = 0; c < kNV; ++c) ep(i, j0 + c, v[c]);
    });
}

// One product read back at once: ep as for tc_read.
template <int M, int N, int K, typename Ep>
__device__ __forceinline__ void tc_mm_rows(TcEng &e, const float *A, int ars, int acs, const float *B, int brs,
                                           int bcs, Ep ep) {
    tc_mma<M, N, K>(e, A, ars, acs, B, brs, bcs, false);
    tc_read<M, N>(e, ep);
}

// The same with an element-wise epilogue ep(i, j, value), as tile_mm calls it.
template <int M, int N, int K, typename Ep>
__device__ __forceinline__ void tc_mm(TcEng &e, const float *A, int ars, int acs, const float *B, int brs, int bcs,
                                      Ep ep) {
    constexpr int kNV = M * N / 512;
    tc_mm_rows<M, N, K>(e, A, ars, acs, B, brs, bcs, [&](int i, int j0, const float (&v)[kNV]) {
#pragma unroll
        for (int c = 0; c < kNV; ++c) ep(i, j0 + c, v[c]);
    });
}

#else  // host builds (the CPU check of the kernels): the same contract, computed in place

// A product on the host: operands rounded to bf16 (nearest even) as the staging rounds them,
// sums in fp32 in order of increasing k (the tensor core's order within a slice is not
// specified; either is a valid fp32 sum of the same bf16 products).
inline float tc_host_bf16(float x) { return __bfloat162float(__float2bfloat16_rn(x)); }

template <typename X>
void tc_setup(TcEng &e, uint8_t *, int, int, X *) {
    static thread_local float acc[128 * 128];
    e.host_acc = acc;
}
template <typename X>
void tc_teardown(X &) {}
template <int M, int N, int K>
void tc_mma(TcEng &e, const float *A, int ars, int acs, const float *B, int brs, int bcs, bool acc) {
    for (int m = 0; m < M; ++m)
        for (int n = 0; n < N; ++n) {
            float s = acc ? e.host_acc[m * N + n] : 0.f;
            for (int k = 0; k < K; ++k)
                s += tc_host_bf16(A[m * ars + k * acs]) * tc_host_bf16(B[k * brs + n * bcs]);
            e.host_acc[m * N + n] = s;
        }
}
template <int M, int N, typename Ep>
void tc_read(TcEng &e, Ep ep) {
    constexpr int kNV = M * N / 512;
    for (int i = 0; i < M; ++i)
        for (int j0 = 0; j0 < N; j0 += kNV) {
            float v[kNV];
            for (int c = 0; c < kNV; ++c) v[c] = e.host_acc[i * N + j0 + c];
            ep(i, j0, v);
        }
}
template <int M, int N, typename Ep>
void tc_read_elem(TcEng &e, Ep ep) {
    for (int i = 0; i < M; ++i)
        for (int j = 0; j < N; ++j) ep(i, j, e.host_acc[i * N + j]);
}
template <int M, int N, int K, typename Ep>
void tc_mm_rows(TcEng &e, const float *A, int ars, int acs, const float *B, int brs, int bcs, Ep ep) {
    tc_mma<M, N, K>(e, A, ars, acs, B, brs, bcs, false);
    tc_read<M, N>(e, ep);
}
template <int M, int N, int K, typename Ep>
void tc_mm(TcEng &e, const float *A, int ars, int acs, const float *B, int brs, int bcs, Ep ep) {
    tc_mma<M, N, K>(e, A, ars, acs, B, brs, bcs, false);
    tc_read_elem<M, N>(e, ep);
}

#endif

}  // namespace gbwd
}  // namespace ccq
