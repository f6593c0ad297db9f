// ccq_gdn_bwd_state_tc.cu -- the reverse state pass of the CCQ-Gated-DeltaNet backward on
// sm_103a tensor cores, for Dk = Dv = 128 (bf16 inputs).
//
// The pass carries the adjoint dH of the delta-rule state backwards through the chunks of one
// sequence and head (the chunkwise reverse mode of the write rule, Sec. 2.2 with the WY/UT
// form of the chunk; the only quantity that crosses chunks sequentially).  Per chunk r, last
// to first, with Kbar the chunk's normalised keys, Tt = (I + A)^{-1} its UT factor, gc the
// cumulative log decay inside the chunk, E = e^{gc}, ed = e^{gc_last - gc}, and the two
// terms the per-chunk kernel computed without dH -- X1 = P^T D (64 x Dv) and
// Y1 = (diag(E) Qc)^T D (Dk x Dv):
//   dU  = X1 + diag(ed) Kbar dH                       (MMA1, 64 x 64 per column half, K = Dk)
//   dR' = diag(E beta) Tt^T dU                        (MMA2, K = 64)
//   dH <- e^{gc_last} dH + Y1 - Kbar^T dR'            (MMA3 accumulating into TMEM, K = 64)
// and stores dH_{r+1} (the adjoint of the state leaving chunk r) for the per-chunk key/value
// kernel; after chunk 0, dH is dS0.  The delta rule acts on the value columns of the state
// independently, so each (sequence, head) runs as two CTAs, one per half of the value columns.
//
// Layout: dH lives in TMEM as fp32 (128 lanes = key dim, 64 columns = this CTA's value
// columns); every MMA operand is a bf16 tile in 128-byte-swizzled shared memory: Kbar
// [64 tokens][128] (K-major for MMA1, MN-major for MMA3), the bf16 copy of dH [128][64]
// (MN-major B of MMA1), Tt [64 l][64 i] (MN-major A of MMA2), dU and -dR' [64][64] (MN-major
// B of MMA2 and MMA3).  The fp32 inputs of a chunk (raw k, X1, Y1 by TMA; Tt by a bulk copy)
// are double-buffered and loaded two chunks ahead.  256 threads: thread (row, th) holds TMEM
// lane `row` (key dim) and columns 32 th .. 32 th + 31 of dH; the 64-row epilogues run on
// warps 0-3 (rows 16 w + (lane % 16), column half lane / 16).
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "ccq_gdn_bwd.h"
#include "ccq_gdn_bwd_kernels.cuh"
#include "ccq_internal.h"
#include "sm100_ptx.cuh"

namespace ccq {

namespace {

constexpr int kC = 64, kD = 128, kThreads = 256;
// per input buffer
constexpr uint32_t B_K = 0;        // 16K  raw k, then kbar: two T64 tiles (key dims 0-63, 64-127)
constexpr uint32_t B_X1 = 16384;   // 16K  X1 columns of this half: two [64][32] fp32 swizzled boxes
constexpr uint32_t B_Y1 = 32768;   // 32K  Y1 columns of this half: two [128][32] fp32 swizzled boxes
constexpr uint32_t B_TT = 65536;   // 16K  Tt [64][64] fp32, row-major
constexpr uint32_t BUF_BYTES = 81920;
constexpr uint32_t OFF_TB = 2 * BUF_BYTES;   // 163840: bf16 Tt [64 l][64 i]
constexpr uint32_t OFF_DHB = OFF_TB + 8192;  // 172032: bf16 dH [128][64]
constexpr uint32_t OFF_DUB = OFF_DHB + 16384;  // 188416: bf16 dU [64][64]
constexpr uint32_t OFF_DRB = OFF_DUB + 8192;   // 196608: bf16 -dR' [64][64]
constexpr uint32_t OFF_MISC = OFF_DRB + 8192;  // 204800
constexpr uint32_t M_GC = 0, M_ED = 256, M_EB = 512, M_EL = 768, M_BAR = 832, M_TMEM = 896, M_ABORT = 900;
constexpr uint32_t kMisc = 1280;
constexpr uint32_t kSmem = OFF_MISC + kMisc + 1024;
static_assert(kSmem <= 232448, "exceeds the 227 KB per-CTA limit");
enum { BAR_IN0 = 0, BAR_IN1 = 1, BAR_M1 = 2, BAR_M2 = 3, BAR_M3 = 4, kBars = 5 };
constexpr uint32_t TM_DH = 0, TM_A1 = 64, TM_A2 = 128, kTmemCols = 256;

constexpr uint32_t ID_M1 = make_idesc(64, 64, 0, 1);   // Kbar (K-major) x dH (MN-major)
constexpr uint32_t ID_M2 = make_idesc(64, 64, 1, 1);   // Tt^T (MN-major) x dU (MN-major)
constexpr uint32_t ID_M3 = make_idesc(128, 64, 1, 1);  // Kbar^T (MN-major) x -dR' (MN-major)

__device__ __forceinline__ void tma_load_2d(void *dst, const CUtensorMap *m, uint64_t *bar, int c0, int c1) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];" ::"r"(smem_addr(dst)),
        "l"(reinterpret_cast<uint64_t>(m)), "r"(c0), "r"(c1), "r"(smem_addr(bar))
        : "memory");
}

// eight fp32 values as one swizzled 16-byte chunk of bf16 (row r, chunk c of a T64 tile)
__device__ __forceinline__ void put_bf16x8(uint8_t *tile, int r, int c, const float *w) {
    *reinterpret_cast<uint4 *>(tile + t64_chunk(r, c)) =
        make_uint4(pack_bf16(w[0], w[1]), pack_bf16(w[2], w[3]), pack_bf16(w[4], w[5]), pack_bf16(w[6], w[7]));
}

__global__ void __launch_bounds__(kThreads, 1)
gdn_bwd_state_tc_kernel(const __grid_constant__ CUtensorMap map_k, const __grid_constant__ CUtensorMap map_x1,
                        const __grid_constant__ CUtensorMap map_y1, const gbwd::GdnBwdArgs a, int *status) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = smem_align1024(smem_raw);
    const uint32_t sb = smem_addr(sm);
    uint8_t *misc = sm + OFF_MISC;
    float *gcs = reinterpret_cast<float *>(misc + M_GC);  // E_i = e^{gc_i}
    float *eds = reinterpret_cast<float *>(misc + M_ED);  // e^{gc_last - gc_i}
    float *ebs = reinterpret_cast<float *>(misc + M_EB);  // E_i beta_i
    float *els = reinterpret_cast<float *>(misc + M_EL);  // e^{gc_last}
    uint64_t *bar = reinterpret_cast<uint64_t *>(misc + M_BAR);
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(misc + M_TMEM);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(misc + M_ABORT);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int row = tid & (kD - 1), th = tid >> 7;
    const int half = blockIdx.x & 1, bh = blockIdx.x >> 1, b = bh / a.H, h = bh % a.H;
    const int T = a.T, NC = a.NC;
    const size_t chunk0 = static_cast<size_t>(bh) * NC;

    if (tid == 0) {
        for (int i = 0; i < kBars; ++i) mbar_init(&bar[i], 1);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 0) tmem_alloc(tmem_slot, kTmemCols);
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *tmem_slot;
    const uint32_t tq = tbase + (static_cast<uint32_t>(32 * (warp & 3)) << 16);

    auto issue = [&](int r, int buf) {  // the fp32 inputs of chunk r into buffer buf
        uint8_t *base = sm + buf * BUF_BYTES;
        uint64_t *bb = &bar[BAR_IN0 + buf];
        const size_t ci = chunk0 + r;
        mbar_arrive_expect_tx(bb, BUF_BYTES);
        tma_load_4d(base + B_K, &map_k, bb, 0, h, r * kC, b);
        tma_load_4d(base + B_K + 8192, &map_k, bb, 64, h, r * kC, b);
        for (int q = 0; q < 2; ++q) {
            tma_load_2d(base + B_X1 + 8192 * q, &map_x1, bb, 64 * half + 32 * q, static_cast<int>(ci * kC));
            tma_load_2d(base + B_Y1 + 16384 * q, &map_y1, bb, 64 * half + 32 * q, static_cast<int>(ci * kD));
        }
        bulk_load(base + B_TT, a.tt + ci * kC * kC, kC * kC * 4, bb);
    };
    {
        // dH <- dS_T (this CTA's value columns), or zero
        const float *src = a.dST ? a.dST + (static_cast<size_t>(bh) * kD + row) * kD + 64 * half + 32 * th : nullptr;
        float x[32];
#pragma unroll
        for (int e = 0; e < 32; ++e) x[e] = src ? src[e] : 0.f;
        tmem_st32(tq + TM_DH + 32 * th, x);
        tmem_wait_st();
    }
    if (tid == 0) {
        issue(NC - 1, 0);
        if (NC > 1) issue(NC - 2, 1);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();

    for (int it = 0; it < NC; ++it) {
        const int r = NC - 1 - it, buf = it & 1;
        const size_t ci = chunk0 + r;
        uint8_t *base = sm + buf * BUF_BYTES;
        const uint32_t bsb = sb + buf * BUF_BYTES;
        if (it > 0) {
            // chunk r+1's three products are done: dH is updated, the shared tiles and buffer
            // buf ^ 1 are free; load chunk r-1 into that buffer
            mbar_wait(&bar[BAR_M3], (it - 1) & 1, abort_flag, status);
            tc_fence_after();
            if (tid == 0 && !*abort_flag && r >= 1) issue(r - 1, buf ^ 1);
        }
        mbar_wait(&bar[BAR_IN0 + buf], (it >> 1) & 1, abort_flag, status);
        // ---- prep: gates (warp 7), kbar in place, Tt to bf16
        if (warp == 7) {
            const int t0 = r * kC + 2 * lane;
            const size_t r0 = (static_cast<size_t>(b) * T + (t0 < T ? t0 : 0)) * a.H + h;
            const size_t r1 = (static_cast<size_t>(b) * T + (t0 + 1 < T ? t0 + 1 : 0)) * a.H + h;
            const float g0 = t0 < T ? a.g[r0] : 0.f, g1 = t0 + 1 < T ? a.g[r1] : 0.f;
            const float b0 = t0 < T ? a.beta[r0] : 0.f, b1 = t0 + 1 < T ? a.beta[r1] : 0.f;
            float p = g0 + g1;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const float y = __shfl_up_sync(0xffffffffu, p, o);
                if (lane >= o) p += y;
            }
            const float gc0 = p - g1, gc1 = p;
            const float glast = __shfl_sync(0xffffffffu, p, 31);
            const float e0 = expf(gc0), e1 = expf(gc1);
            gcs[2 * lane] = e0;
            gcs[2 * lane + 1] = e1;
            eds[2 * lane] = expf(glast - gc0);
            eds[2 * lane + 1] = expf(glast - gc1);
            ebs[2 * lane] = e0 * b0;
            ebs[2 * lane + 1] = e1 * b1;
            if (lane == 0) *els = expf(glast);
        }
        {
            // kbar = k / |k| in place: four threads per row, each one 32-column quarter
            const int j = tid >> 2, part = tid & 3;
            uint8_t *kt = base + B_K + (part >> 1) * 8192;
            uint4 kv[4];
            float ss = 0.f;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                kv[q] = *reinterpret_cast<const uint4 *>(kt + t64_chunk(j, 4 * (part & 1) + q));
                float f[8];
                unpack_bf16x8(kv[q], f);
#pragma unroll
                for (int e = 0; e < 8; ++e) ss = fmaf(f[e], f[e], ss);
            }
            ss += __shfl_xor_sync(0xffffffffu, ss, 1);
            ss += __shfl_xor_sync(0xffffffffu, ss, 2);
            const float rk = a.l2norm ? rsqrtf(fmaxf(ss, 1e-12f)) : 1.f;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                float f[8];
                unpack_bf16x8(kv[q], f);
#pragma unroll
                for (int e = 0; e < 8; ++e) f[e] *= rk;
                put_bf16x8(kt, j, 4 * (part & 1) + q, f);
            }
            // Tt rows to bf16: row l = tid / 4, columns 16 (tid % 4) .. + 15
            const float *tt = reinterpret_cast<const float *>(base + B_TT) + j * kC + 16 * part;
            float w[16];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const float4 v = *reinterpret_cast<const float4 *>(tt + 4 * q);
                w[4 * q] = v.x; w[4 * q + 1] = v.y; w[4 * q + 2] = v.z; w[4 * q + 3] = v.w;
            }
            put_bf16x8(sm + OFF_TB, j, 2 * part, w);
            put_bf16x8(sm + OFF_TB, j, 2 * part + 1, w + 8);
        }
        __syncthreads();
        // ---- dH_{r+1}: stored for the key/value kernel, copied to bf16 for MMA1, then
        // e^{gc_last} dH + Y1 in place (MMA3 subtracts Kbar^T dR' from it)
        {
            float x[32];
            tmem_ld32(tq + TM_DH + 32 * th, x);
            float4 *dst = reinterpret_cast<float4 *>(a.dh + (ci * kD + row) * kD + 64 * half + 32 * th);
#pragma unroll
            for (int e = 0; e < 8; ++e) dst[e] = make_float4(x[4 * e], x[4 * e + 1], x[4 * e + 2], x[4 * e + 3]);
#pragma unroll
            for (int q = 0; q < 4; ++q) put_bf16x8(sm + OFF_DHB, row, 4 * th + q, x + 8 * q);
            const float el = *els;
            const uint8_t *y1 = base + B_Y1 + 16384 * th;
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                const float4 yv = *reinterpret_cast<const float4 *>(y1 + t64_chunk(row, q));
                x[4 * q] = fmaf(el, x[4 * q], yv.x);
                x[4 * q + 1] = fmaf(el, x[4 * q + 1], yv.y);
                x[4 * q + 2] = fmaf(el, x[4 * q + 2], yv.z);
                x[4 * q + 3] = fmaf(el, x[4 * q + 3], yv.w);
            }
            tmem_st32(tq + TM_DH + 32 * th, x);
        }
        tmem_wait_st();
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        if (tid == 0 && !*abort_flag) {
            tc_fence_after();
            // MMA1: Kbar dH (M = 64 tokens, N = 64 columns, K = 128 key dims)
            const uint64_t dK = make_desc(bsb + B_K, 16, 1024);
            const uint64_t dH = make_desc(sb + OFF_DHB, 8192, 1024);
            for (int k = 0; k < 8; ++k)
                mma_bf16(tbase + TM_A1, dK + (k >> 2) * 512 + (k & 3) * 2, dH + k * 128, ID_M1, k != 0);
            mma_commit(&bar[BAR_M1]);
        }
        // ---- dU = X1 + diag(ed) Kbar dH (warps 0-3: row i, columns 32 hf .. + 31)
        mbar_wait(&bar[BAR_M1], it & 1, abort_flag, status);
        tc_fence_after();
        if (warp < 4) {
            const int i = 16 * warp + (lane & 15), hf = lane >> 4;
            float v[32];
            tmem_ld16x2_32<32>(tq + TM_A1, v);
            const float ed = eds[i];
            const uint8_t *x1 = base + B_X1 + 8192 * hf;
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                const float4 xv = *reinterpret_cast<const float4 *>(x1 + t64_chunk(i, q));
                v[4 * q] = fmaf(ed, v[4 * q], xv.x);
                v[4 * q + 1] = fmaf(ed, v[4 * q + 1], xv.y);
                v[4 * q + 2] = fmaf(ed, v[4 * q + 2], xv.z);
                v[4 * q + 3] = fmaf(ed, v[4 * q + 3], xv.w);
            }
#pragma unroll
            for (int q = 0; q < 4; ++q) put_bf16x8(sm + OFF_DUB, i, 4 * hf + q, v + 8 * q);
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        if (tid == 0 && !*abort_flag) {
            tc_fence_after();
            // MMA2: Tt^T dU (M = 64, N = 64, K = 64)
            const uint64_t dT = make_desc(sb + OFF_TB, 8192, 1024);
            const uint64_t dU = make_desc(sb + OFF_DUB, 8192, 1024);
            for (int k = 0; k < 4; ++k) mma_bf16(tbase + TM_A2, dT + k * 128, dU + k * 128, ID_M2, k != 0);
            mma_commit(&bar[BAR_M2]);
        }
        // ---- -dR' = -diag(E beta) Tt^T dU
        mbar_wait(&bar[BAR_M2], it & 1, abort_flag, status);
        tc_fence_after();
        if (warp < 4) {
            const int i = 16 * warp + (lane & 15), hf = lane >> 4;
            float v[32];
            tmem_ld16x2_32<32>(tq + TM_A2, v);
            const float nb = -ebs[i];
#pragma unroll
            for (int e = 0; e < 32; ++e) v[e] *= nb;
#pragma unroll
            for (int q = 0; q < 4; ++q) put_bf16x8(sm + OFF_DRB, i, 4 * hf + q, v + 8 * q);
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        if (tid == 0 && !*abort_flag) {
            tc_fence_after();
            // MMA3: dH += Kbar^T (-dR') (M = 128 key dims, N = 64, K = 64 tokens)
            const uint64_t dKm = make_desc(bsb + B_K, 8192, 1024);
            const uint64_t dR = make_desc(sb + OFF_DRB, 8192, 1024);
            for (int k = 0; k < 4; ++k) mma_bf16(tbase + TM_DH, dKm + k * 128, dR + k * 128, ID_M3, 1);
            mma_commit(&bar[BAR_M3]);
        }
    }
    // dS0 = dH after chunk 0
    mbar_wait(&bar[BAR_M3], (NC - 1) & 1, abort_flag, status);
    tc_fence_after();
    if (a.dS0) {
        float x[32];
        tmem_ld32(tq + TM_DH + 32 * th, x);
        float4 *dst = reinterpret_cast<float4 *>(a.dS0 + (static_cast<size_t>(bh) * kD + row) * kD + 64 * half + 32 * th);
#pragma unroll
        for (int e = 0; e < 8; ++e) dst[e] = make_float4(x[4 * e], x[4 * e + 1], x[4 * e + 2], x[4 * e + 3]);
    }
    if (tid == 0 && *abort_flag) {
        // after a give-up, wait (bounded) for the loads still in flight
        for (int it = (NC > 2 ? NC - 2 : 0); it < NC; ++it) mbar_drain(&bar[BAR_IN0 + (it & 1)], (it >> 1) & 1);
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tbase, kTmemCols);
    }
}

}  // namespace

// The fp32 [rows][128] workspace arrays X1 ([chunks * 64][128]) and Y1 ([chunks * 128][128]) as
// 2-D tensor maps with 32-column (128-byte) swizzled boxes.
static bool f32_rows_map(CUtensorMap *map, const float *base, long long rows, int box_rows) {
    return make_f32_rows_map(map, base, rows, 128, 32, box_rows);
}

cudaError_t launch_gdn_dstate_tc(const gbwd::GdnBwdArgs &a, const void *k, cudaStream_t s) {
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(gdn_bwd_state_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(kSmem));
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    const long long chunks = static_cast<long long>(a.B) * a.H * a.NC;
    CUtensorMap mk, mx, my;
    if (!make_token_map(&mk, k, 2, a.B, a.T, a.H, 128, 64, true) || !f32_rows_map(&mx, a.x1, chunks * kC, kC) ||
        !f32_rows_map(&my, a.y1, chunks * kD, kD))
        return cudaErrorInvalidValue;
    int *status = device_status_word();
    if (!status) return cudaErrorInvalidValue;
    gdn_bwd_state_tc_kernel<<<a.B * a.H * 2, kThreads, kSmem, s>>>(mk, mx, my, a, status);
    return cudaGetLastError();
}

}  // namespace ccq
