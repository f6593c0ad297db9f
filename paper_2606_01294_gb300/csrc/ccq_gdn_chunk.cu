// ccq_gdn_chunk.cu -- chunkwise CCQ-Gated-DeltaNet forward on sm_103a tensor cores.
//
// The gated delta rule S_t = alpha_t S_{t-1}(I - beta_t kbar_t kbar_t^T) + beta_t v_t kbar_t^T
// (the Gated DeltaNet write, Sec. 2.2) is kept as H = S^T [Dk][Dv].  Inside a 64-token
// chunk with start state H0, gc_i the in-chunk cumulative log-decay and gc_m its value at
// the chunk midpoint (token 31), unrolling the recurrence gives (chunkwise form):
//   A_ij = beta_i e^{gc_i - gc_j} kbar_i . kbar_j   (j < i),   Tt = (I + A)^{-1}
//   U    = Tt diag(beta) V - Tt diag(beta e^{gc - gc_m}) Kbar (e^{gc_m} H0)  =  Ut - W Hm
//   o_i  = scale [ e^{gc_i - gc_m} q_clean_i Hm + sum_{j<=i} e^{gc_i - gc_j}(q_clean_i . kbar_j) U_j ]
//   H_C  = e^{gc_C - gc_m} [ Hm + sum_j e^{gc_m - gc_j} kbar_j U_j^T ]
// with Hm = e^{gc_m} H0.  Ut and W depend only on the chunk's own inputs, so they are
// computed for every chunk in parallel by gdn_wy_kernel (into a caller workspace);
// gdn_chunk_kernel then walks the chunks of each (batch, head) sequentially with the
// same warp-specialised structure as the GLA kernel and the same CCQ read (App. B):
//
//   group A  G2  Sc  = Q Kbar^T          D2  WH = W Hm
//   (epilogue: W' of the CCQ mean fold;  U = Ut - WH -> bf16 U tile)
//   group B  G1  P   = Q S^K             G3  P += W' Kbar
//   (epilogue: q_clean e^{gc - gc_m} into the Q tile)
//   group C  D4  QK  = Qc Kbar^T         D3  O  = Qc Hm
//   group S  D6  X  += Kd^T U            G8  S^K += Kbar^T Kbar      (Kd = kbar e^{gc_m - gc})
//   (epilogue: Pm_ij = [j<=i] QK_ij e^{gc_m - gc_j})
//   group D  D5  O  += Pm U
//   (epilogue: o = scale O, TMA store)
// X = e^{gc_m - gc_C} H_{r+1} stays in TMEM; the scalar e^{gc_C - gc_m} is applied at the
// next snapshot.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "ccq_internal.h"
#include "sm100_ptx.cuh"

namespace ccq {

namespace {

constexpr int kC = 64;
constexpr int kD = 128;
constexpr float kLog2e = 1.4426950408889634f;

__device__ __forceinline__ void store_row_chunk(uint8_t *tile, int row, int chunk, const float *w) {
    uint4 u;
    u.x = pack_bf16(w[0], w[1]);
    u.y = pack_bf16(w[2], w[3]);
    u.z = pack_bf16(w[4], w[5]);
    u.w = pack_bf16(w[6], w[7]);
    *reinterpret_cast<uint4 *>(tile + t64_chunk(row, chunk)) = u;
}

// ============================================================================ WY kernel
//
// One CTA (128 threads) per (batch, head, chunk).  Writes Ut and W as bf16 rows
// [((b*H + h)*NC + r)*64 + i][0..127] of the workspace.

constexpr uint32_t WY_K = 0;        // 16K  k raw -> kbar; later staging of W
constexpr uint32_t WY_V = 16384;    // 16K  v; later staging of Ut
constexpr uint32_t WY_A = 32768;    // 64 x 68 fp32: A; after the inversion the two bf16 tiles:
constexpr uint32_t WY_TB = 32768;   //   8K  bf16 Tt diag(beta)               ([64][64] T64 tile)
constexpr uint32_t WY_TG = 40960;   //   8K  bf16 Tt diag(beta e^{gc - gc_m})
constexpr uint32_t WY_T = 50176;    // 64 x 68 fp32: Tt
constexpr uint32_t WY_Y = 67584;    // 3 x 256 fp32: block products
constexpr uint32_t WY_MISC = 70656; // gc, beta, factors, rk, barrier
constexpr uint32_t WY_SMEM = WY_MISC + 2048 + 1024;  // 73.7 KB: three CTAs per SM
constexpr int kAS = 68;             // padded fp32 row stride of A and Tt

__global__ void __launch_bounds__(128, 3)
gdn_wy_kernel(const __grid_constant__ CUtensorMap map_k, const __grid_constant__ CUtensorMap map_v,
              const __grid_constant__ CUtensorMap map_ut, const __grid_constant__ CUtensorMap map_w,
              const ChunkArgs a, int NC) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = smem_align1024(smem_raw);
    const uint32_t sb = smem_addr(sm);
    float *A = reinterpret_cast<float *>(sm + WY_A);
    float *Tt = reinterpret_cast<float *>(sm + WY_T);
    float *Y = reinterpret_cast<float *>(sm + WY_Y);
    float *gcs = reinterpret_cast<float *>(sm + WY_MISC);        // [64] cumulative log decay
    float *bet = gcs + 64;                                        // [64] beta
    float *epos = gcs + 128;                                      // [64] e^{gc - gc_m}
    float *eneg = gcs + 192;                                      // [64] e^{gc_m - gc}
    float *rk = gcs + 256;                                        // [64] 1/|k|
    uint64_t *bar = reinterpret_cast<uint64_t *>(sm + WY_MISC + 1536);
    uint32_t *tslot = reinterpret_cast<uint32_t *>(sm + WY_MISC + 1560);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(sm + WY_MISC + 1564);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int item = blockIdx.x;
    const int r = item % NC, bh = item / NC, b = bh / a.H, h = bh % a.H;
    const int T = a.T, H = a.H;
    const int c0 = r * kC;
    int *status = a.status;

    if (tid == 0) {
        for (int i = 0; i < 3; ++i) mbar_init(&bar[i], 1);
        *abort_flag = 0;
        fence_barrier_init();
        mbar_arrive_expect_tx(&bar[0], 4 * 8192);
        tma_load_4d(sm + WY_K, &map_k, &bar[0], 0, h, c0, b);
        tma_load_4d(sm + WY_K + 8192, &map_k, &bar[0], 64, h, c0, b);
        tma_load_4d(sm + WY_V, &map_v, &bar[0], 0, h, c0, b);
        tma_load_4d(sm + WY_V + 8192, &map_v, &bar[0], 64, h, c0, b);
    }
    if (warp == 0) tmem_alloc(tslot, 128);
    if (tid < 64) {
        const int t = c0 + tid;
        const size_t row = (static_cast<size_t>(b) * T + t) * H + h;
        gcs[tid] = t < T ? a.g[row] : 0.f;
        bet[tid] = t < T ? a.beta[row] : 0.f;
    }
    __syncthreads();
    tc_fence_after();
    const uint32_t tb = *tslot;
    const uint32_t tq = tb + (static_cast<uint32_t>(32 * warp) << 16);

    // ---- cumulative decay (warp 2: two values per lane, shuffle scan) and the k row norms
    if (warp == 2) {
        const float x0 = gcs[2 * lane], x1 = gcs[2 * lane + 1];
        float p = x0 + x1;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const float y = __shfl_up_sync(0xffffffffu, p, o);
            if (lane >= o) p += y;
        }
        gcs[2 * lane] = p - x1;
        gcs[2 * lane + 1] = p;
    }
    mbar_wait(&bar[0], 0, abort_flag, status);
    if (tid < 64) {
        float ss = 0.f;
#pragma unroll
        for (int t64 = 0; t64 < 2; ++t64)
#pragma unroll
            for (int cc = 0; cc < 8; ++cc) {
                float f[8];
                unpack_bf16x8(*reinterpret_cast<const uint4 *>(sm + WY_K + t64 * 8192 + t64_chunk(tid, cc)), f);
#pragma unroll
                for (int e = 0; e < 8; ++e) ss = fmaf(f[e], f[e], ss);
            }
        rk[tid] = a.l2norm ? rsqrtf(fmaxf(ss, 1e-12f)) : 1.f;
    }
    __syncthreads();
    if (tid < 64) {
        const float gm = gcs[31];
        epos[tid] = fast_exp2((gcs[tid] - gm) * kLog2e);
        eneg[tid] = fast_exp2((gm - gcs[tid]) * kLog2e);
    }
    // ---- kbar in place (row j = tid/2, column half tid%2)
    {
        const int j = tid >> 1, hf = tid & 1;
        const float s = rk[j];
        uint8_t *tile = sm + WY_K + hf * 8192;
#pragma unroll
        for (int cc = 0; cc < 8; ++cc) {
            float f[8];
            unpack_bf16x8(*reinterpret_cast<const uint4 *>(tile + t64_chunk(j, cc)), f);
#pragma unroll
            for (int e = 0; e < 8; ++e) f[e] *= s;
            store_row_chunk(tile, j, cc, f);
        }
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    // ---- KK = Kbar Kbar^T (M = 64: rows 16w..16w+15 in lanes 32w..32w+15)
    if (tid == 0 && !*abort_flag) {
        tc_fence_after();
        const uint64_t dk = make_desc(sb + WY_K, 16, 1024);
        for (int k = 0; k < 8; ++k) {
            const uint64_t ko = (k >> 2) * 512 + (k & 3) * 2;
            mma_bf16(tb, dk + ko, dk + ko, make_idesc(64, 64, 0, 0), k != 0);
        }
        mma_commit(&bar[1]);
    }
    mbar_wait(&bar[1], 0, abort_flag, status);
    tc_fence_after();
    {
        // A_ij = beta_i e^{gc_i - gc_j} KK_ij for j < i
        const int i = 16 * warp + (lane & 15), hf = lane >> 4;
        float kk[32];
        tmem_ld16x2_32<32>(tq, kk);
        const float ri = bet[i] * epos[i];
#pragma unroll
        for (int q4 = 0; q4 < 8; ++q4) {
            float w[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int j = 32 * hf + 4 * q4 + e;
                w[e] = (j < i) ? ri * eneg[j] * kk[4 * q4 + e] : 0.f;
            }
            *reinterpret_cast<float4 *>(A + i * kAS + 32 * hf + 4 * q4) = make_float4(w[0], w[1], w[2], w[3]);
        }
    }
    __syncthreads();
    // ---- Tt = (I + A)^{-1}: the four 16 x 16 diagonal blocks by forward substitution
    if (tid < 64) {
        const int bb = tid >> 4, c = tid & 15, o = 16 * bb;
        float x[16];
#pragma unroll
        for (int rr = 0; rr < 16; ++rr) {
            float s = 0.f;
#pragma unroll
            for (int j = 0; j < rr; ++j) s = fmaf(A[(o + rr) * kAS + o + j], x[j], s);
            x[rr] = (rr < c) ? 0.f : ((rr == c) ? 1.f : -s);
        }
#pragma unroll
        for (int rr = 0; rr < 16; ++rr) Tt[(o + rr) * kAS + o + c] = x[rr];
    }
    __syncthreads();
    // off-diagonal blocks, by distance from the diagonal:
    //   Tt_IJ = -Tt_II sum_{K=J}^{I-1} A_IK Tt_KJ
    // 16 threads per 16 x 16 block, each a 4 x 4 sub-tile with float4 shared loads
    for (int dist = 1; dist < 4; ++dist) {
        const int nblk = 4 - dist;
        const int blk = tid >> 4, t = tid & 15, r0 = 4 * (t >> 2), c0 = 4 * (t & 3);
        const int J = blk, I = blk + dist;
        if (blk < nblk) {
            float acc[4][4] = {};
            for (int K = J; K < I; ++K) {
#pragma unroll
                for (int m = 0; m < 16; m += 4) {
                    float4 av[4], tv[4];
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        av[u] = *reinterpret_cast<const float4 *>(A + (16 * I + r0 + u) * kAS + 16 * K + m);
                        tv[u] = *reinterpret_cast<const float4 *>(Tt + (16 * K + m + u) * kAS + 16 * J + c0);
                    }
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        const float a4[4] = {av[u].x, av[u].y, av[u].z, av[u].w};
#pragma unroll
                        for (int mm = 0; mm < 4; ++mm) {
                            acc[u][0] = fmaf(a4[mm], tv[mm].x, acc[u][0]);
                            acc[u][1] = fmaf(a4[mm], tv[mm].y, acc[u][1]);
                            acc[u][2] = fmaf(a4[mm], tv[mm].z, acc[u][2]);
                            acc[u][3] = fmaf(a4[mm], tv[mm].w, acc[u][3]);
                        }
                    }
                }
            }
#pragma unroll
            for (int u = 0; u < 4; ++u)
                *reinterpret_cast<float4 *>(Y + blk * 256 + (r0 + u) * 16 + c0) =
                    make_float4(acc[u][0], acc[u][1], acc[u][2], acc[u][3]);
        }
        __syncthreads();
        if (blk < nblk) {
            float acc[4][4] = {};
#pragma unroll
            for (int m = 0; m < 16; m += 4) {
                float4 av[4], yv[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    av[u] = *reinterpret_cast<const float4 *>(Tt + (16 * I + r0 + u) * kAS + 16 * I + m);
                    yv[u] = *reinterpret_cast<const float4 *>(Y + blk * 256 + (m + u) * 16 + c0);
                }
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const float a4[4] = {av[u].x, av[u].y, av[u].z, av[u].w};
#pragma unroll
                    for (int mm = 0; mm < 4; ++mm) {
                        acc[u][0] = fmaf(a4[mm], yv[mm].x, acc[u][0]);
                        acc[u][1] = fmaf(a4[mm], yv[mm].y, acc[u][1]);
                        acc[u][2] = fmaf(a4[mm], yv[mm].z, acc[u][2]);
                        acc[u][3] = fmaf(a4[mm], yv[mm].w, acc[u][3]);
                    }
                }
            }
#pragma unroll
            for (int u = 0; u < 4; ++u)
                *reinterpret_cast<float4 *>(Tt + (16 * I + r0 + u) * kAS + 16 * J + c0) =
                    make_float4(-acc[u][0], -acc[u][1], -acc[u][2], -acc[u][3]);
        }
        __syncthreads();
    }
    // zero the blocks above the diagonal, then the two scaled bf16 copies
    {
        const int i = tid >> 1, hf = tid & 1;
#pragma unroll
        for (int q4 = 0; q4 < 4; ++q4) {
            float wb[8], wg[8];
            const float4 t0 = *reinterpret_cast<const float4 *>(Tt + i * kAS + 32 * hf + 8 * q4);
            const float4 t1 = *reinterpret_cast<const float4 *>(Tt + i * kAS + 32 * hf + 8 * q4 + 4);
            const float tr[8] = {t0.x, t0.y, t0.z, t0.w, t1.x, t1.y, t1.z, t1.w};
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                const int j = 32 * hf + 8 * q4 + e;
                const float t = (j <= i) ? tr[e] : 0.f;  // A is dead: its space takes the tiles
                wb[e] = t * bet[j];
                wg[e] = wb[e] * epos[j];
            }
            store_row_chunk(sm + WY_TB, i, 4 * hf + q4, wb);
            store_row_chunk(sm + WY_TG, i, 4 * hf + q4, wg);
        }
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    // ---- Ut = Tt diag(beta) V, then W = Tt diag(beta e^{gc-gc_m}) Kbar  (M = 64, N = 128, K = 64)
    const size_t out_row = static_cast<size_t>(item) * kC;
    for (int pass = 0; pass < 2; ++pass) {
        if (tid == 0 && !*abort_flag) {
            tc_fence_after();
            const uint64_t da = make_desc(sb + (pass == 0 ? WY_TB : WY_TG), 16, 1024);
            const uint64_t dbm = make_desc(sb + (pass == 0 ? WY_V : WY_K), 8192, 1024);
            for (int k = 0; k < 4; ++k)
                mma_bf16(tb, da + k * 2, dbm + k * 128, make_idesc(64, 128, 0, 1), k != 0);
            mma_commit(&bar[2]);
        }
        mbar_wait(&bar[2], pass, abort_flag, status);
        tc_fence_after();
        {
            const int i = 16 * warp + (lane & 15), hf = lane >> 4;
            uint8_t *stage = sm + (pass == 0 ? WY_V : WY_K) + hf * 8192;  // operand no longer read
#pragma unroll
            for (int h2 = 0; h2 < 2; ++h2) {
                float x[32];
                tmem_ld16x2_32<64>(tq + 32 * h2, x);
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) store_row_chunk(stage, i, 4 * h2 + q4, x + 8 * q4);
            }
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        if (tid == 0 && !*abort_flag) {
            const CUtensorMap *m = pass == 0 ? &map_ut : &map_w;
            uint8_t *stage = sm + (pass == 0 ? WY_V : WY_K);
            asm volatile(
                "cp.async.bulk.tensor.2d.global.shared::cta.tile.bulk_group [%0, {%2, %3}], [%1];" ::"l"(
                    reinterpret_cast<uint64_t>(m)),
                "r"(smem_addr(stage)), "r"(0), "r"(static_cast<int>(out_row))
                : "memory");
            asm volatile(
                "cp.async.bulk.tensor.2d.global.shared::cta.tile.bulk_group [%0, {%2, %3}], [%1];" ::"l"(
                    reinterpret_cast<uint64_t>(m)),
                "r"(smem_addr(stage + 8192)), "r"(64), "r"(static_cast<int>(out_row))
                : "memory");
            tma_store_commit();
        }
    }
    if (tid == 0) tma_store_wait_read();  // shared memory must outlive the stores' reads
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tb, 128);
    }
}


// ============================================================================ main kernel

constexpr int kThreads = 384;
constexpr uint32_t SLOT_BYTES = 49152;
constexpr uint32_t SO_Q = 0;        // raw q, then q_clean e^{gc - gc_m}; finally the output staging
constexpr uint32_t SO_K = 16384;    // raw k, then kbar
constexpr uint32_t SO_KD = 32768;   // kbar e^{gc_m - gc}
constexpr uint32_t OFF_UT = 98304;  // 16K  Ut of the chunk (workspace)
constexpr uint32_t OFF_WW = 114688; // 16K  W of the chunk (workspace)
constexpr uint32_t OFF_UB = 131072; // 16K  U (bf16, rows j)
constexpr uint32_t OFF_WM = 147456; // 8K   W' of the CCQ fold, then Pm
constexpr uint32_t OFF_SK = 155648; // 32K  bf16 S^K
constexpr uint32_t OFF_HB = 188416; // 32K  bf16 Hm = e^{gc_m} H
constexpr uint32_t OFF_MISC = 221184;
constexpr uint32_t MS_BYTES = 2560;
constexpr uint32_t MS_RQ = 0, MS_MQ = 256, MS_LAM = 512, MS_RK = 768, MS_EP = 1024, MS_EN = 1280,
                   MS_SCAL = 1536, MS_MST = 2048;  // SCAL: [0] e^{gc_m}, [1] e^{gc_C - gc_m}, [2..65] gc
constexpr uint32_t M_DMPREV = 5120;  // [128]
constexpr uint32_t M_CV = 5632;      // [64]
constexpr uint32_t M_BAR = 5888;     // 14 mbarriers
constexpr uint32_t M_TMEM = 6016;
constexpr uint32_t M_ABORT = 6020;
constexpr uint32_t kMiscBytes = 6144;
constexpr uint32_t kSmemBytes = OFF_MISC + kMiscBytes + 1024;
static_assert(kSmemBytes <= 232448, "exceeds the 227 KB per-CTA limit");
static_assert(MS_SCAL + 66 * 4 <= MS_MST, "scalar area overlaps");

enum {
    BAR_IN0 = 0, BAR_IN1 = 1, BAR_WU = 2, BAR_GA = 3, BAR_GB = 4, BAR_GC = 5, BAR_GD = 6,
    BAR_PREP0 = 7, BAR_PREP1 = 8, BAR_SNAP = 9, BAR_GS = 10, BAR_GC2 = 11, kNumBars = 12
};

constexpr uint32_t TM_S = 0, TM_SK = 128, TM_PO = 256, TM_SA = 384, kTmemCols = 512;
constexpr uint32_t ID_64x64_KK = make_idesc(64, 64, 0, 0);
constexpr uint32_t ID_64x128_KK = make_idesc(64, 128, 0, 0);
constexpr uint32_t ID_64x128_KM = make_idesc(64, 128, 0, 1);
constexpr uint32_t ID_128x128_MM = make_idesc(128, 128, 1, 1);

__device__ __forceinline__ void tma_load_2d(void *dst, const CUtensorMap *m, uint64_t *bar, int c0, int c1) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];" ::"r"(smem_addr(dst)),
        "l"(reinterpret_cast<uint64_t>(m)), "r"(c0), "r"(c1), "r"(smem_addr(bar))
        : "memory");
}

__global__ void __launch_bounds__(kThreads, 1)
gdn_chunk_kernel(const __grid_constant__ CUtensorMap map_q, const __grid_constant__ CUtensorMap map_k,
                 const __grid_constant__ CUtensorMap map_ut, const __grid_constant__ CUtensorMap map_w,
                 const __grid_constant__ CUtensorMap map_o, const ChunkArgs a) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = smem_align1024(smem_raw);
    const uint32_t sb = smem_addr(sm);
    uint8_t *misc = sm + OFF_MISC;
    float *dmprev = reinterpret_cast<float *>(misc + M_DMPREV);
    float *cv = reinterpret_cast<float *>(misc + M_CV);
    uint64_t *bar = reinterpret_cast<uint64_t *>(misc + M_BAR);
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(misc + M_TMEM);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(misc + M_ABORT);
    auto slot_f = [&](int s, uint32_t off) {
        return reinterpret_cast<float *>(misc + s * MS_BYTES + off);
    };

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int wg = tid >> 7, wt = tid & 127;
    const int bh = blockIdx.x, b = bh / a.H, h = bh % a.H;
    const int T = a.T, H = a.H;
    const int NC = (T + kC - 1) / kC;
    const int64_t t0 = a.t0 ? a.t0[b] : 0;
    int *status = a.status;
    const int wrow0 = bh * NC * kC;  // first workspace row of this (b, h)

    if (tid == 0) {
        for (int i = 0; i < kNumBars; ++i) mbar_init(&bar[i], 1);
        *abort_flag = 0;
        fence_barrier_init();
        tma_prefetch_desc(&map_q);
        tma_prefetch_desc(&map_k);
        tma_prefetch_desc(&map_ut);
        tma_prefetch_desc(&map_w);
        tma_prefetch_desc(&map_o);
    }
    if (warp == 0) tmem_alloc(tmem_slot, kTmemCols);
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *tmem_slot;
    const uint32_t tq = tbase + (static_cast<uint32_t>(32 * (warp & 3)) << 16);

    auto issue_in = [&](int r) {
        const int s = r & 1;
        uint8_t *base = sm + s * SLOT_BYTES;
        uint64_t *bb = &bar[BAR_IN0 + s];
        mbar_arrive_expect_tx(bb, 4 * 8192);
        tma_load_4d(base + SO_Q, &map_q, bb, 0, h, r * kC, b);
        tma_load_4d(base + SO_Q + 8192, &map_q, bb, 64, h, r * kC, b);
        tma_load_4d(base + SO_K, &map_k, bb, 0, h, r * kC, b);
        tma_load_4d(base + SO_K + 8192, &map_k, bb, 64, h, r * kC, b);
    };
    auto issue_wu = [&](int r) {
        uint64_t *bb = &bar[BAR_WU];
        const int row = wrow0 + r * kC;
        mbar_arrive_expect_tx(bb, 4 * 8192);
        tma_load_2d(sm + OFF_UT, &map_ut, bb, 0, row);
        tma_load_2d(sm + OFF_UT + 8192, &map_ut, bb, 64, row);
        tma_load_2d(sm + OFF_WW, &map_w, bb, 0, row);
        tma_load_2d(sm + OFF_WW + 8192, &map_w, bb, 64, row);
    };

    if (wg == 2) {
        const size_t bhs = static_cast<size_t>(bh);
        const int row = 32 * (warp & 3) + lane;
        for (int m = 0; m < 2; ++m) {
            const float *src = m == 0 ? a.S0 : a.C0;
            const uint32_t col0 = m == 0 ? TM_S : TM_SK;
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                float x[32];
                if (src) {
                    const float4 *p4 = reinterpret_cast<const float4 *>(src + (bhs * kD + row) * kD + 32 * c);
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        const float4 f = p4[e];
                        x[4 * e] = f.x; x[4 * e + 1] = f.y; x[4 * e + 2] = f.z; x[4 * e + 3] = f.w;
                    }
                } else {
#pragma unroll
                    for (int e = 0; e < 32; ++e) x[e] = 0.f;
                }
                tmem_st32(tq + col0 + 32 * c, x);
            }
        }
        tmem_wait_st();
    } else if (wg == 1) {
        slot_f(0, MS_MST)[wt] = a.m0 ? a.m0[static_cast<size_t>(bh) * kD + wt] : 0.f;
        dmprev[wt] = 0.f;
    } else if (tid == 0) {
        issue_in(0);
        issue_wu(0);
    }
    tc_fence_before();
    __syncthreads();

    if (wg == 0) {
        // =============================================================== WG0: the chain
        const int i = 16 * warp + (lane & 15);
        const int hf = lane >> 4;
        const uint64_t dWm = make_desc(sb + OFF_WM, 16, 1024);
        const uint64_t dSK = make_desc(sb + OFF_SK, 16, 1024);
        const uint64_t dHB = make_desc(sb + OFF_HB, 16384, 1024);
        const uint64_t dWW = make_desc(sb + OFF_WW, 16, 1024);
        const uint64_t dUBm = make_desc(sb + OFF_UB, 8192, 1024);
        for (int r = 0; r < NC; ++r) {
            const int s = r & 1;
            const uint32_t sp = (r >> 1) & 1, par = r & 1;
            uint8_t *slot = sm + s * SLOT_BYTES;
            const uint32_t ss = sb + s * SLOT_BYTES;
            const int c0 = r * kC;
            const float ti = static_cast<float>(t0 + c0 + i + 1);
            const uint64_t dQ = make_desc(ss + SO_Q, 16, 1024);
            const uint64_t dK = make_desc(ss + SO_K, 16, 1024);
            const uint64_t dKm = make_desc(ss + SO_K, 8192, 1024);
            const uint64_t dKDm = make_desc(ss + SO_KD, 8192, 1024);
            mbar_wait(&bar[BAR_PREP0 + s], sp, abort_flag, status);
            mbar_wait(&bar[BAR_SNAP], par, abort_flag, status);
            if (tid == 0 && !*abort_flag) {
                if (r + 1 < NC) {
                    tma_store_wait_read();
                    issue_in(r + 1);
                }
                mbar_wait(&bar[BAR_WU], par, abort_flag, status);
                tc_fence_after();
                // group A: G2 Sc = Q Kbar^T; D2 WH = W Hm
                for (int k = 0; k < 8; ++k) {
                    const uint64_t ko = (k >> 2) * 512 + (k & 3) * 2;
                    mma_bf16(tbase + TM_SA, dQ + ko, dK + ko, ID_64x64_KK, k != 0);
                }
                for (int k = 0; k < 8; ++k)
                    mma_bf16(tbase + TM_PO, dWW + (k >> 2) * 512 + (k & 3) * 2, dHB + k * 128, ID_64x128_KM,
                             k != 0);
                mma_commit(&bar[BAR_GA]);
            }
            mbar_wait(&bar[BAR_GA], par, abort_flag, status);
            tc_fence_after();
            const float rqi = slot_f(s, MS_RQ)[i];
            {
                // W' of the CCQ mean fold (as in the GLA kernel)
                float sc[32];
                tmem_ld16x2_32<32>(tq + TM_SA, sc);
                float part = 0.f;
#pragma unroll
                for (int jj = 0; jj < 32; ++jj)
                    if (32 * hf + jj <= i) part += sc[jj];
                part += __shfl_xor_sync(0xffffffffu, part, 16);
                const float cq = slot_f(s, MS_MQ)[i] + rqi * part;
                const float c = a.centered ? cq / ti : 0.f;
                if (hf == 0) cv[i] = c;
                const float cn = c / rqi;
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) {
                    float w[8];
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        const int j = 32 * hf + 8 * q4 + e;
                        w[e] = (j <= i) ? sc[8 * q4 + e] - cn : 0.f;
                    }
                    store_row_chunk(sm + OFF_WM, i, 4 * hf + q4, w);
                }
                // U = Ut - W Hm  -> bf16 U tile (row i)
                uint8_t *ut = sm + OFF_UT + hf * 8192;
                uint8_t *ub = sm + OFF_UB + hf * 8192;
#pragma unroll
                for (int h2 = 0; h2 < 2; ++h2) {
                    float x[32];
                    tmem_ld16x2_32<64>(tq + TM_PO + 32 * h2, x);
#pragma unroll
                    for (int q4 = 0; q4 < 4; ++q4) {
                        const int cc = 4 * h2 + q4;
                        float u8[8];
                        unpack_bf16x8(*reinterpret_cast<const uint4 *>(ut + t64_chunk(i, cc)), u8);
#pragma unroll
                        for (int e = 0; e < 8; ++e) u8[e] -= x[8 * q4 + e];
                        store_row_chunk(ub, i, cc, u8);
                    }
                }
            }
            fence_proxy_async_smem();
            tc_fence_before();
            named_bar(1, 128);
            if (tid == 0 && !*abort_flag) {
                if (r + 1 < NC) issue_wu(r + 1);  // Ut and W of this chunk are consumed
                tc_fence_after();
                // group B: G1 P = Q S^K; G3 P += W' Kbar
                for (int k = 0; k < 8; ++k)
                    mma_bf16(tbase + TM_PO, dQ + (k >> 2) * 512 + (k & 3) * 2,
                             dSK + (k >> 2) * 1024 + (k & 3) * 2, ID_64x128_KK, k != 0);
                for (int k = 0; k < 4; ++k) mma_bf16(tbase + TM_PO, dWm + k * 2, dKm + k * 128, ID_64x128_KM, 1);
                mma_commit(&bar[BAR_GB]);
            }
            // ---- q_clean (Eq. clean) scaled by e^{gc_i - gc_m}, into the Q tile
            {
                uint8_t *qt = slot + SO_Q + hf * 8192;
                const float *Mst = slot_f(s, MS_MST) + 64 * hf;
                uint4 qraw[8];
#pragma unroll
                for (int cc = 0; cc < 8; ++cc) qraw[cc] = *reinterpret_cast<const uint4 *>(qt + t64_chunk(i, cc));
                const float lt = slot_f(s, MS_LAM)[i] / ti;
                const float ep = slot_f(s, MS_EP)[i];
                mbar_wait(&bar[BAR_GB], par, abort_flag, status);
                tc_fence_after();
                const float cm = lt * cv[i];
#pragma unroll
                for (int h2 = 0; h2 < 2; ++h2) {
                    float p[32];
                    tmem_ld16x2_32<64>(tq + TM_PO + 32 * h2, p);
#pragma unroll
                    for (int q4 = 0; q4 < 4; ++q4) {
                        const int cc = 4 * h2 + q4;
                        float qr[8], out[8];
                        unpack_bf16x8(qraw[cc], qr);
                        const float4 m0 = *reinterpret_cast<const float4 *>(Mst + 8 * cc);
                        const float4 m1 = *reinterpret_cast<const float4 *>(Mst + 8 * cc + 4);
                        const float mv[8] = {m0.x, m0.y, m0.z, m0.w, m1.x, m1.y, m1.z, m1.w};
#pragma unroll
                        for (int e = 0; e < 8; ++e)
                            out[e] = ep * fmaf(rqi, fmaf(-lt, p[8 * q4 + e], qr[e]), cm * mv[e]);
                        store_row_chunk(qt, i, cc, out);
                    }
                }
            }
            fence_proxy_async_smem();
            tc_fence_before();
            named_bar(1, 128);
            if (tid == 0 && !*abort_flag) {
                tc_fence_after();
                // group C: D4 QK = Qc Kbar^T; D3 O = Qc Hm
                for (int k = 0; k < 8; ++k) {
                    const uint64_t ko = (k >> 2) * 512 + (k & 3) * 2;
                    mma_bf16(tbase + TM_SA, dQ + ko, dK + ko, ID_64x64_KK, k != 0);
                }
                mma_commit(&bar[BAR_GC]);
                for (int k = 0; k < 8; ++k)
                    mma_bf16(tbase + TM_PO, dQ + (k >> 2) * 512 + (k & 3) * 2, dHB + k * 128, ID_64x128_KM,
                             k != 0);
                mma_commit(&bar[BAR_GC2]);
                // group S: D6 X += Kd^T U; G8 S^K += Kbar^T Kbar
                for (int k = 0; k < 4; ++k) mma_bf16(tbase + TM_S, dKDm + k * 128, dUBm + k * 128, ID_128x128_MM, 1);
                for (int k = 0; k < 4; ++k) mma_bf16(tbase + TM_SK, dKm + k * 128, dKm + k * 128, ID_128x128_MM, 1);
                mma_commit(&bar[BAR_GS]);
            }
            // ---- Pm_ij = [j<=i] QK_ij e^{gc_m - gc_j}
            mbar_wait(&bar[BAR_GC], par, abort_flag, status);
            tc_fence_after();
            {
                const float *en = slot_f(s, MS_EN) + 32 * hf;
                float sc[32];
                tmem_ld16x2_32<32>(tq + TM_SA, sc);
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) {
                    const float4 e0 = *reinterpret_cast<const float4 *>(en + 8 * q4);
                    const float4 e1 = *reinterpret_cast<const float4 *>(en + 8 * q4 + 4);
                    const float ev[8] = {e0.x, e0.y, e0.z, e0.w, e1.x, e1.y, e1.z, e1.w};
                    float w[8];
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        const int j = 32 * hf + 8 * q4 + e;
                        w[e] = (j <= i) ? sc[8 * q4 + e] * ev[e] : 0.f;
                    }
                    store_row_chunk(sm + OFF_WM, i, 4 * hf + q4, w);
                }
            }
            fence_proxy_async_smem();
            tc_fence_before();
            named_bar(1, 128);
            if (tid == 0 && !*abort_flag) {
                tc_fence_after();
                // group D: D5 O += Pm U
                for (int k = 0; k < 4; ++k) mma_bf16(tbase + TM_PO, dWm + k * 2, dUBm + k * 128, ID_64x128_KM, 1);
                mma_commit(&bar[BAR_GD]);
            }
            mbar_wait(&bar[BAR_GD], par, abort_flag, status);
            tc_fence_after();
            {
                uint8_t *ot = slot + SO_Q + hf * 8192;
#pragma unroll
                for (int h2 = 0; h2 < 2; ++h2) {
                    float x[32];
                    tmem_ld16x2_32<64>(tq + TM_PO + 32 * h2, x);
#pragma unroll
                    for (int e = 0; e < 32; ++e) x[e] *= a.scale;
#pragma unroll
                    for (int q4 = 0; q4 < 4; ++q4) store_row_chunk(ot, i, 4 * h2 + q4, x + 8 * q4);
                }
            }
            fence_proxy_async_smem();
            tc_fence_before();
            named_bar(1, 128);
            if (tid == 0 && !*abort_flag) {
                tma_store_4d(&map_o, slot + SO_Q, 0, h, c0, b);
                tma_store_4d(&map_o, slot + SO_Q + 8192, 64, h, c0, b);
                tma_store_commit();
            }
        }
        if (tid == 0) tma_store_wait_all();
    } else if (wg == 1) {
        // =============================================================== WG1: prep
        float lam_reg = 0.f, g_reg = 0.f;
        if (wt < 64) lam_reg = (wt < T) ? a.lambda[(static_cast<size_t>(b) * T + wt) * H + h] : 0.f;
        else g_reg = (wt - 64 < T) ? a.g[(static_cast<size_t>(b) * T + (wt - 64)) * H + h] : 0.f;
        for (int r = 0; r < NC; ++r) {
            const int s = r & 1;
            const uint32_t sp = (r >> 1) & 1;
            uint8_t *slot = sm + s * SLOT_BYTES;
            float *Mst = slot_f(s, MS_MST);
            float *scal = slot_f(s, MS_SCAL);
            mbar_wait(&bar[BAR_IN0 + s], sp, abort_flag, status);
            if (r > 0) Mst[wt] = slot_f(s ^ 1, MS_MST)[wt] + dmprev[wt];
            if (wt < 64) {
                slot_f(s, MS_LAM)[wt] = lam_reg;
                const int tn = (r + 1) * kC + wt;
                lam_reg = (tn < T) ? a.lambda[(static_cast<size_t>(b) * T + tn) * H + h] : 0.f;
            } else {
                scal[2 + wt - 64] = g_reg;
                const int tn = (r + 1) * kC + wt - 64;
                g_reg = (tn < T) ? a.g[(static_cast<size_t>(b) * T + tn) * H + h] : 0.f;
            }
            named_bar(2, 128);
            // row norms and M . qbar; in-chunk cumulative decay (one thread)
            {
                const int j = wt & 63;
                const bool isq = wt < 64;
                const uint8_t *base = slot + (isq ? SO_Q : SO_K);
                float ss = 0.f, md = 0.f;
#pragma unroll
                for (int t64 = 0; t64 < 2; ++t64) {
#pragma unroll
                    for (int cc = 0; cc < 8; ++cc) {
                        float f[8];
                        unpack_bf16x8(*reinterpret_cast<const uint4 *>(base + t64 * 8192 + t64_chunk(j, cc)), f);
                        const float4 m0 = *reinterpret_cast<const float4 *>(Mst + 64 * t64 + 8 * cc);
                        const float4 m1 = *reinterpret_cast<const float4 *>(Mst + 64 * t64 + 8 * cc + 4);
                        const float mv[8] = {m0.x, m0.y, m0.z, m0.w, m1.x, m1.y, m1.z, m1.w};
#pragma unroll
                        for (int e = 0; e < 8; ++e) {
                            ss = fmaf(f[e], f[e], ss);
                            if (isq) md = fmaf(f[e], mv[e], md);
                        }
                    }
                }
                const float rn = a.l2norm ? rsqrtf(fmaxf(ss, 1e-12f)) : 1.f;
                if (isq) {
                    slot_f(s, MS_RQ)[j] = rn;
                    slot_f(s, MS_MQ)[j] = md * rn;
                } else {
                    slot_f(s, MS_RK)[j] = rn;
                }
                if (wt == 127) {
                    float run = 0.f;
                    for (int t = 0; t < 64; ++t) {
                        run += scal[2 + t];
                        scal[2 + t] = run;
                    }
                }
            }
            named_bar(2, 128);
            if (wt < 64) {
                const float gm = scal[2 + 31];
                slot_f(s, MS_EP)[wt] = fast_exp2((scal[2 + wt] - gm) * kLog2e);
                slot_f(s, MS_EN)[wt] = fast_exp2((gm - scal[2 + wt]) * kLog2e);
                if (wt == 0) {
                    scal[0] = fast_exp2(gm * kLog2e);
                    scal[1] = fast_exp2((scal[2 + 63] - gm) * kLog2e);
                }
            }
            named_bar(2, 128);
            // kbar (in place) and Kd = kbar e^{gc_m - gc}: thread = (row, column half)
            {
                const int j = wt >> 1, hf = wt & 1;
                const float rkj = slot_f(s, MS_RK)[j], enj = slot_f(s, MS_EN)[j];
                uint8_t *kt = slot + SO_K + hf * 8192;
                uint8_t *kd = slot + SO_KD + hf * 8192;
#pragma unroll
                for (int cc = 0; cc < 8; ++cc) {
                    float f[8], g8[8];
                    unpack_bf16x8(*reinterpret_cast<const uint4 *>(kt + t64_chunk(j, cc)), f);
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        f[e] *= rkj;
                        g8[e] = f[e] * enj;
                    }
                    store_row_chunk(kt, j, cc, f);
                    store_row_chunk(kd, j, cc, g8);
                }
            }
            fence_proxy_async_smem();
            named_bar(2, 128);
            // key sum of the chunk, per key dim (from the bf16 kbar tile)
            {
                const int d = wt;
                const uint8_t *kt = slot + SO_K + (d >> 6) * 8192;
                float sum = 0.f;
                for (int j = 0; j < 64; ++j)
                    sum += __bfloat162float(*reinterpret_cast<const __nv_bfloat16 *>(kt + t64_offset(j, d & 63)));
                dmprev[d] = sum;
            }
            named_bar(2, 128);
            if (wt == 0) mbar_arrive(&bar[BAR_PREP0 + s]);
        }
        if (NC > 0 && a.mT) {
            const int sl = (NC - 1) & 1;
            a.mT[static_cast<size_t>(bh) * kD + wt] = slot_f(sl, MS_MST)[wt] + dmprev[wt];
        }
    } else {
        // =============================================================== WG2: states
        const int row = 32 * (warp & 3) + lane;
        for (int r = 0; r < NC; ++r) {
            const int s = r & 1;
            const uint32_t sp = (r >> 1) & 1;
            if (r > 0) mbar_wait(&bar[BAR_GS], (r - 1) & 1, abort_flag, status);
            mbar_wait(&bar[BAR_PREP0 + s], sp, abort_flag, status);
            tc_fence_after();
            const float hs = (r > 0 ? slot_f(s ^ 1, MS_SCAL)[1] : 1.f) * slot_f(s, MS_SCAL)[0];
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                float x[32];
                tmem_ld32(tq + TM_S + 32 * c, x);
#pragma unroll
                for (int e = 0; e < 32; ++e) x[e] *= hs;
                uint8_t *tile = sm + OFF_HB + (c >> 1) * 16384;
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) store_row_chunk(tile, row, 4 * (c & 1) + q4, x + 8 * q4);
                tmem_st32(tq + TM_S + 32 * c, x);
            }
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                float x[32];
                tmem_ld32(tq + TM_SK + 32 * c, x);
                uint8_t *tile = sm + OFF_SK + (c >> 1) * 16384;
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) store_row_chunk(tile, row, 4 * (c & 1) + q4, x + 8 * q4);
            }
            tmem_wait_st();
            fence_proxy_async_smem();
            tc_fence_before();
            named_bar(3, 128);
            if (wt == 0) mbar_arrive(&bar[BAR_SNAP]);
        }
        if (NC > 0) {
            mbar_wait(&bar[BAR_GS], (NC - 1) & 1, abort_flag, status);
            tc_fence_after();
            const float fs = slot_f((NC - 1) & 1, MS_SCAL)[1];
            const size_t bhs = static_cast<size_t>(bh);
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                float x[32];
                tmem_ld32(tq + TM_S + 32 * c, x);
                if (a.ST) {
                    float4 *dst = reinterpret_cast<float4 *>(a.ST + (bhs * kD + row) * kD + 32 * c);
#pragma unroll
                    for (int e = 0; e < 8; ++e)
                        dst[e] = make_float4(fs * x[4 * e], fs * x[4 * e + 1], fs * x[4 * e + 2], fs * x[4 * e + 3]);
                }
                tmem_ld32(tq + TM_SK + 32 * c, x);
                if (a.CT) {
                    float4 *dst = reinterpret_cast<float4 *>(a.CT + (bhs * kD + row) * kD + 32 * c);
#pragma unroll
                    for (int e = 0; e < 8; ++e) dst[e] = make_float4(x[4 * e], x[4 * e + 1], x[4 * e + 2], x[4 * e + 3]);
                }
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tbase, kTmemCols);
    }
}

}  // namespace

cudaError_t launch_gdn_wy(const ChunkArgs &a, const GdnMaps &m, cudaStream_t s) {
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(gdn_wy_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(WY_SMEM));
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    const int NC = (a.T + kC - 1) / kC;
    gdn_wy_kernel<<<a.B * a.H * NC, 128, WY_SMEM, s>>>(m.k, m.v, m.ut, m.w, a, NC);
    return cudaGetLastError();
}

}  // namespace ccq

namespace ccq {

cudaError_t launch_gdn_chunk(const ChunkArgs &a, const GdnMaps &m, cudaStream_t s) {
    cudaError_t e = launch_gdn_wy(a, m, s);
    if (e != cudaSuccess) return e;
    static bool attr_set = false;
    if (!attr_set) {
        e = cudaFuncSetAttribute(gdn_chunk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 static_cast<int>(kSmemBytes));
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    gdn_chunk_kernel<<<a.B * a.H, kThreads, kSmemBytes, s>>>(m.q, m.k, m.ut, m.w, m.o, a);
    return cudaGetLastError();
}

size_t gdn_workspace_bytes(int B, int T, int H) {
    const size_t nc = static_cast<size_t>((T + kC - 1) / kC);
    return 2 * static_cast<size_t>(B) * H * nc * kC * kD * sizeof(__nv_bfloat16);
}

}  // namespace ccq
