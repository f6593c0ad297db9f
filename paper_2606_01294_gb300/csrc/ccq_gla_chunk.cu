// ccq_gla_chunk.cu -- chunkwise CCQ-GLA forward on sm_103a tensor cores.
//
// One CTA per (batch, head) walks the chunks of Algorithm 1 (chunk C = 64,
// Dk = Dv = 128).  The two recurrent states live in tensor memory as fp32
// accumulators for the whole sequence:
//   S   [Dk lanes][Dv cols]  the GLA state (transposed, S[a][e])
//   SK  [Dk lanes][Dk cols]  the undecayed key second-moment sum S^K (App. B)
// and every product of the chunk is a tcgen05.mma with bf16 operands staged
// in 128-byte-swizzled shared-memory tiles (TMA-loaded for q, k, v):
//
//   G2  Sc   = Qbar Kbar^T                    (CCQ intra-chunk scores)
//   G1  P    = Qbar S^K                       (CCQ inter-chunk read, P^prev)
//   G8  S^K += Kbar^T Kbar                    (second-moment update)
//   G3  P   += W' Kbar,  W'_ij = [j<=i](Sc_ij - c_i)   (P^intra with the mean fold)
//   G4  A    = Qg Kg^T                        (gated GLA scores)
//   G6  O    = Qg (Diag(e^{Gmid}) S)          (GLA inter-chunk read)
//   G5  O   += [j<=i] A  V                    (GLA intra-chunk read)
//   G7  S    = Diag(e^{Gtot}) S + Ku^T V      (GLA state update)
//
// The CCQ mean term is folded into the intra product: with
// cq_i = CumK_i . qbar_i = M . qbar_i + sum_{j<=i} Sc_ij and c_i = cq_i / t_i,
//   D (P^prev + P^intra) - MeanCorr = (P_i - c_i M) / t_i          (App. B)
// where P_i = S^K qbar_i + sum_{j<=i} (Sc_ij - c_i) kbar_j.  Then
//   q_clean_i = qbar_i - lambda_i (P_i - c_i M) / t_i               (Eq. clean)
// and the GLA chunk form reads with q_clean scaled by exp(G_i - Gmid) and keys
// scaled by exp(Gmid - G_j), Gmid the cumulative gate at the chunk midpoint
// (halves the exponent range), the state snapshot scaled by exp(Gmid).
//
// Rows past T load as zeros through the tensor maps: zero keys add nothing to
// any sum and zero gates leave the cumulative gate unchanged, so the ragged
// tail needs no special arithmetic; only its output rows are not stored.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "ccq_internal.h"
#include "sm100_ptx.cuh"

namespace ccq {

namespace {

constexpr int kC = 64;         // chunk length
constexpr int kD = 128;        // Dk = Dv
constexpr int kThreads = 256;  // 8 warps (two warpgroups)

// ---- shared memory map (bytes from the 1024-aligned base)
constexpr uint32_t OFF_Q = 0;        // 16K  q raw -> qbar -> q_clean*e^{G-Gmid} ([64][128], 2 T64 tiles of 8K)
constexpr uint32_t OFF_K = 16384;    // 16K  k raw -> kbar
constexpr uint32_t OFF_V = 32768;    // 16K  v
constexpr uint32_t OFF_KG = 49152;   // 16K  kbar * e^{Gmid - G}
constexpr uint32_t OFF_KU = 65536;   // 16K  kbar * e^{Gtot - G}
constexpr uint32_t OFF_W = 81920;    // 8K   W' then masked A ([64][64], one T64 tile)
constexpr uint32_t OFF_SK = 90112;   // 32K  bf16 snapshot of S^K ([128][128], 2 T64 tiles of 16K)
constexpr uint32_t OFF_S = 122880;   // 32K  bf16 snapshot of e^{Gmid} S ([128][128], 2 T64 tiles of 16K)
constexpr uint32_t OFF_G = 155648;   // 32K  raw gates, plain [64][128] (bf16 or fp32)
constexpr uint32_t OFF_EG = 188416;  // 17K  e^{G - Gmid} bf16, [64][kEgStride]
constexpr int kEgStride = 136;       // padded row (272 B) -> conflict-free row reads
constexpr uint32_t OFF_MISC = OFF_EG + 64 * kEgStride * 2;  // 205824
// misc (fp32 unless noted)
constexpr uint32_t M_M = 0;           // [128] key sum M (chunk start)
constexpr uint32_t M_DM = 512;        // [2][128] partial key sums of the chunk
constexpr uint32_t M_GP = 1536;       // [2][128] partial gate sums
constexpr uint32_t M_EGT = 2560;      // [128] e^{Gtot}
constexpr uint32_t M_EGM = 3072;      // [128] e^{Gmid}
constexpr uint32_t M_RQ = 3584;       // [64] 1/|q_i|
constexpr uint32_t M_RK = 3840;       // [64] 1/|k_j|
constexpr uint32_t M_MQ = 4096;       // [64] M . qbar_i
constexpr uint32_t M_LAM = 4352;      // [64] lambda_i
constexpr uint32_t M_CV = 4608;       // [64] c_i
constexpr uint32_t M_PART = 4864;     // [2][64] masked row sums of Sc
constexpr uint32_t M_BAR = 5376;      // 5 mbarriers (8 B each)
constexpr uint32_t M_TMEM = 5424;     // u32 TMEM base
constexpr uint32_t M_ABORT = 5428;    // int abort flag
constexpr uint32_t kMiscBytes = 5504;
constexpr uint32_t kSmemBytes = OFF_MISC + kMiscBytes + 1024;  // + alignment slack

static_assert(OFF_MISC == 205824, "smem map");
static_assert(kSmemBytes <= 232448, "exceeds the 227 KB per-CTA limit");

// ---- tensor memory columns
constexpr uint32_t TM_S = 0;     // 128 cols
constexpr uint32_t TM_SK = 128;  // 128 cols
constexpr uint32_t TM_PO = 256;  // 128 cols: P, then O
constexpr uint32_t TM_SA = 384;  // 64 cols: Sc, then A
constexpr uint32_t kTmemCols = 512;

// ---- instruction descriptors
constexpr uint32_t ID_N64_KK = make_idesc(128, 64, 0, 0);
constexpr uint32_t ID_N128_KK = make_idesc(128, 128, 0, 0);
constexpr uint32_t ID_N128_KM = make_idesc(128, 128, 0, 1);
constexpr uint32_t ID_N128_MM = make_idesc(128, 128, 1, 1);

enum { BAR_Q = 0, BAR_K = 1, BAR_V = 2, BAR_G = 3, BAR_MMA = 4 };

__device__ __forceinline__ float bf(const uint8_t *p) {
    return __bfloat162float(*reinterpret_cast<const __nv_bfloat16 *>(p));
}
__device__ __forceinline__ void st_bf(uint8_t *p, float x) {
    *reinterpret_cast<__nv_bfloat16 *>(p) = __float2bfloat16_rn(x);
}

__global__ void __launch_bounds__(kThreads, 1)
gla_chunk_kernel(const __grid_constant__ CUtensorMap map_q, const __grid_constant__ CUtensorMap map_k,
                 const __grid_constant__ CUtensorMap map_v, const __grid_constant__ CUtensorMap map_g,
                 const ChunkArgs a) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                              ~static_cast<uintptr_t>(1023));
    const uint32_t sb = smem_addr(sm);
    uint8_t *misc = sm + OFF_MISC;
    float *Mv = reinterpret_cast<float *>(misc + M_M);
    float *dm = reinterpret_cast<float *>(misc + M_DM);
    float *gp = reinterpret_cast<float *>(misc + M_GP);
    float *egt = reinterpret_cast<float *>(misc + M_EGT);
    float *egm = reinterpret_cast<float *>(misc + M_EGM);
    float *rq = reinterpret_cast<float *>(misc + M_RQ);
    float *rk = reinterpret_cast<float *>(misc + M_RK);
    float *mq = reinterpret_cast<float *>(misc + M_MQ);
    float *lam = reinterpret_cast<float *>(misc + M_LAM);
    float *cv = reinterpret_cast<float *>(misc + M_CV);
    float *part = reinterpret_cast<float *>(misc + M_PART);
    uint64_t *bar = reinterpret_cast<uint64_t *>(misc + M_BAR);
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(misc + M_TMEM);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(misc + M_ABORT);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int bh = blockIdx.x, b = bh / a.H, h = bh % a.H;
    const int T = a.T, H = a.H;
    const int NC = (T + kC - 1) / kC;
    const bool gate_f32 = a.gate_dtype != 0;
    const uint32_t g_bytes = gate_f32 ? kC * kD * 4 : kC * kD * 2;

    // lane quarter (TMEM lanes 32*lq..) and column half of this warp
    const int lq = warp & 3, ch = warp >> 2;
    const int row = 32 * lq + lane;  // TMEM lane: state row a, or chunk row i

    if (tid == 0) {
        for (int i = 0; i < 5; ++i) mbar_init(&bar[i], 1);
        *abort_flag = 0;
        fence_barrier_init();
        tma_prefetch_desc(&map_q);
        tma_prefetch_desc(&map_k);
        tma_prefetch_desc(&map_v);
        tma_prefetch_desc(&map_g);
    }
    if (warp == 0) tmem_alloc(tmem_slot, kTmemCols);
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *tmem_slot;
    const uint32_t tl = tbase + (static_cast<uint32_t>(32 * lq) << 16);  // this warp's lane base

    // ---- initial states into TMEM, M into shared memory
    {
        const size_t bhs = static_cast<size_t>(bh);
        float x[32];
#pragma unroll
        for (int half = 0; half < 2; ++half) {
            const int c0 = 64 * ch + 32 * half;
            if (a.S0) {
                const float4 *src = reinterpret_cast<const float4 *>(a.S0 + (bhs * kD + row) * kD + c0);
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    float4 f = src[i];
                    x[4 * i] = f.x; x[4 * i + 1] = f.y; x[4 * i + 2] = f.z; x[4 * i + 3] = f.w;
                }
            } else {
#pragma unroll
                for (int i = 0; i < 32; ++i) x[i] = 0.f;
            }
            tmem_st32(tl + TM_S + c0, x);
            if (a.C0) {
                const float4 *src = reinterpret_cast<const float4 *>(a.C0 + (bhs * kD + row) * kD + c0);
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    float4 f = src[i];
                    x[4 * i] = f.x; x[4 * i + 1] = f.y; x[4 * i + 2] = f.z; x[4 * i + 3] = f.w;
                }
            } else {
#pragma unroll
                for (int i = 0; i < 32; ++i) x[i] = 0.f;
            }
            tmem_st32(tl + TM_SK + c0, x);
        }
        if (tid < kD) Mv[tid] = a.m0 ? a.m0[bhs * kD + tid] : 0.f;
        tmem_wait_st();
    }
    int64_t tpos = a.t0 ? a.t0[b] : 0;  // tokens before the current chunk

    auto issue_q = [&](int r) {
        mbar_arrive_expect_tx(&bar[BAR_Q], 2 * 8192);
        tma_load_4d(sm + OFF_Q, &map_q, &bar[BAR_Q], 0, h, r * kC, b);
        tma_load_4d(sm + OFF_Q + 8192, &map_q, &bar[BAR_Q], 64, h, r * kC, b);
    };
    auto issue_k = [&](int r) {
        mbar_arrive_expect_tx(&bar[BAR_K], 2 * 8192);
        tma_load_4d(sm + OFF_K, &map_k, &bar[BAR_K], 0, h, r * kC, b);
        tma_load_4d(sm + OFF_K + 8192, &map_k, &bar[BAR_K], 64, h, r * kC, b);
    };
    auto issue_v = [&](int r) {
        mbar_arrive_expect_tx(&bar[BAR_V], 2 * 8192);
        tma_load_4d(sm + OFF_V, &map_v, &bar[BAR_V], 0, h, r * kC, b);
        tma_load_4d(sm + OFF_V + 8192, &map_v, &bar[BAR_V], 64, h, r * kC, b);
    };
    auto issue_g = [&](int r) {
        mbar_arrive_expect_tx(&bar[BAR_G], g_bytes);
        tma_load_4d(sm + OFF_G, &map_g, &bar[BAR_G], 0, h, r * kC, b);
    };
    if (tid == 0 && NC > 0) {
        issue_q(0);
        issue_k(0);
        issue_v(0);
        issue_g(0);
    }
    // lambda of the next chunk is prefetched into a register by warps 2-3
    float lam_next = 0.f;
    if (tid >= 64 && tid < 128) {
        const int i = tid - 64;
        lam_next = (i < T) ? a.lambda[(static_cast<size_t>(b) * T + i) * H + h] : 0.f;
    }
    tc_fence_before();
    __syncthreads();

    uint32_t mma_par = 0;
    for (int r = 0; r < NC; ++r) {
        const int c0 = r * kC;
        const int n = min(kC, T - c0);
        const uint32_t tpar = static_cast<uint32_t>(r & 1);
        const float tf = static_cast<float>(tpos);

        // ================= P1a: row norms, M . qbar, lambda
        mbar_wait(&bar[BAR_Q], tpar, abort_flag, a.status);
        mbar_wait(&bar[BAR_K], tpar, abort_flag, a.status);
        if (tid < 128) {
            const bool isq = tid < 64;
            const int i = tid & 63;
            const uint8_t *base = sm + (isq ? OFF_Q : OFF_K);
            float ss = 0.f, mdot = 0.f;
#pragma unroll
            for (int t64 = 0; t64 < 2; ++t64) {
#pragma unroll
                for (int cc = 0; cc < 8; ++cc) {
                    const uint4 u = *reinterpret_cast<const uint4 *>(base + t64 * 8192 + t64_chunk(i, cc));
                    float f[8];
                    unpack_bf16x8(u, f);
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        ss = fmaf(f[e], f[e], ss);
                        mdot = fmaf(f[e], Mv[64 * t64 + 8 * cc + e], mdot);
                    }
                }
            }
            const float rn = a.l2norm ? rsqrtf(fmaxf(ss, 1e-12f)) : 1.f;
            if (isq) {
                rq[i] = rn;
                mq[i] = mdot * rn;
            } else {
                rk[i] = rn;
            }
            if (tid >= 64) lam[i] = lam_next;
        }
        __syncthreads();

        // ================= P1b: gate cumsum (per key dim), normalised and gated operand tiles
        mbar_wait(&bar[BAR_G], tpar, abort_flag, a.status);
        {
            const int d = tid & 127, th = tid >> 7;  // key dim, token half
            float gl[32];
            float run = 0.f;
#pragma unroll
            for (int jj = 0; jj < 32; ++jj) {
                const int j = 32 * th + jj;
                const float g = gate_f32 ? reinterpret_cast<const float *>(sm + OFF_G)[j * kD + d]
                                         : bf(sm + OFF_G + (j * kD + d) * 2);
                run += g;
                gl[jj] = run;
            }
            gp[th * kD + d] = run;
            __syncthreads();  // all raw gates read; partial sums visible
            if (tid == 0 && r + 1 < NC) issue_g(r + 1);
            const float gmid = gp[d];               // cumulative gate after token 31
            const float gtot = gp[d] + gp[kD + d];  // after token 63 (zero-filled past T)
            const float off = th ? gmid : 0.f;
            if (th == 0) {
                egt[d] = __expf(gtot);
                egm[d] = __expf(gmid);
            }
            const int tile = d >> 6, dc = d & 63;
            float dmp = 0.f;
#pragma unroll
            for (int jj = 0; jj < 32; ++jj) {
                const int j = 32 * th + jj;
                const float G = gl[jj] + off;
                const uint32_t o = tile * 8192 + t64_offset(j, dc);
                const float kb = bf(sm + OFF_K + o) * rk[j];
                const float qb = bf(sm + OFF_Q + o) * rq[j];
                st_bf(sm + OFF_K + o, kb);
                st_bf(sm + OFF_Q + o, qb);
                st_bf(sm + OFF_KG + o, kb * __expf(gmid - G));
                st_bf(sm + OFF_KU + o, kb * __expf(gtot - G));
                st_bf(sm + OFF_EG + (j * kEgStride + d) * 2, __expf(G - gmid));
                dmp += kb;
            }
            dm[th * kD + d] = dmp;
        }
        fence_proxy_async_smem();
        __syncthreads();

        // ================= P1c: snapshot S (scaled by e^{Gmid}) and S^K to bf16; decay S in TMEM
        tc_fence_after();
        {
            const float sgm = egm[row], sgt = egt[row];
#pragma unroll
            for (int half = 0; half < 2; ++half) {
                const uint32_t col = 64 * ch + 32 * half;
                float x[32];
                tmem_ld32(tl + TM_S + col, x);
                uint8_t *dst = sm + OFF_S + ch * 16384;
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) {
                    uint4 u;
                    u.x = pack_bf16(x[8 * q4 + 0] * sgm, x[8 * q4 + 1] * sgm);
                    u.y = pack_bf16(x[8 * q4 + 2] * sgm, x[8 * q4 + 3] * sgm);
                    u.z = pack_bf16(x[8 * q4 + 4] * sgm, x[8 * q4 + 5] * sgm);
                    u.w = pack_bf16(x[8 * q4 + 6] * sgm, x[8 * q4 + 7] * sgm);
                    *reinterpret_cast<uint4 *>(dst + t64_chunk(row, 4 * half + q4)) = u;
                }
#pragma unroll
                for (int i = 0; i < 32; ++i) x[i] *= sgt;
                tmem_st32(tl + TM_S + col, x);
                tmem_ld32(tl + TM_SK + col, x);
                dst = sm + OFF_SK + ch * 16384;
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) {
                    uint4 u;
                    u.x = pack_bf16(x[8 * q4 + 0], x[8 * q4 + 1]);
                    u.y = pack_bf16(x[8 * q4 + 2], x[8 * q4 + 3]);
                    u.z = pack_bf16(x[8 * q4 + 4], x[8 * q4 + 5]);
                    u.w = pack_bf16(x[8 * q4 + 6], x[8 * q4 + 7]);
                    *reinterpret_cast<uint4 *>(dst + t64_chunk(row, 4 * half + q4)) = u;
                }
            }
            tmem_wait_st();
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();

        // ================= P2: G2 (Sc), G1 (P = Qbar S^K), G8 (S^K += Kbar^T Kbar)
        if (tid == 0 && !*abort_flag) {
            tc_fence_after();
            for (int kb = 0; kb < 2; ++kb)
                for (int k16 = 0; k16 < 4; ++k16)
                    mma_bf16(tbase + TM_SA, desc_kmajor(sb + OFF_Q + kb * 8192, k16),
                             desc_kmajor(sb + OFF_K + kb * 8192, k16), ID_N64_KK, (kb | k16) != 0);
            for (int kb = 0; kb < 2; ++kb)
                for (int k16 = 0; k16 < 4; ++k16)
                    mma_bf16(tbase + TM_PO, desc_kmajor(sb + OFF_Q + kb * 8192, k16),
                             desc_kmajor(sb + OFF_SK + kb * 16384, k16), ID_N128_KK, (kb | k16) != 0);
            for (int k16 = 0; k16 < 4; ++k16)
                mma_bf16(tbase + TM_SK, desc_mnmajor(sb + OFF_K, 8192, k16),
                         desc_mnmajor(sb + OFF_K, 8192, k16), ID_N128_MM, 1);
            mma_commit(&bar[BAR_MMA]);
        }

        // ================= P3: masked row sums of Sc -> c_i; W'
        mbar_wait(&bar[BAR_MMA], mma_par, abort_flag, a.status);
        mma_par ^= 1;
        tc_fence_after();
        const bool rows_warp = lq < 2;  // warps 0,1,4,5 own chunk rows 0..63
        float sc[32];
        if (rows_warp) {
            tmem_ld32(tl + TM_SA + 32 * ch, sc);
            float s = 0.f;
#pragma unroll
            for (int jj = 0; jj < 32; ++jj)
                if (32 * ch + jj <= row) s += sc[jj];
            part[ch * 64 + row] = s;
        }
        __syncthreads();
        if (rows_warp) {
            const float ti = tf + static_cast<float>(row + 1);
            const float cq = mq[row] + part[row] + part[64 + row];
            const float c = a.centered ? cq / ti : 0.f;
            if (ch == 0) cv[row] = c;
#pragma unroll
            for (int q4 = 0; q4 < 4; ++q4) {
                float w[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const int j = 32 * ch + 8 * q4 + e;
                    w[e] = (j <= row) ? sc[8 * q4 + e] - c : 0.f;
                }
                uint4 u;
                u.x = pack_bf16(w[0], w[1]);
                u.y = pack_bf16(w[2], w[3]);
                u.z = pack_bf16(w[4], w[5]);
                u.w = pack_bf16(w[6], w[7]);
                *reinterpret_cast<uint4 *>(sm + OFF_W + t64_chunk(row, 4 * ch + q4)) = u;
            }
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();

        // ================= P4: G3 (P += W' Kbar)
        if (tid == 0 && !*abort_flag) {
            tc_fence_after();
            for (int k16 = 0; k16 < 4; ++k16)
                mma_bf16(tbase + TM_PO, desc_kmajor(sb + OFF_W, k16), desc_mnmajor(sb + OFF_K, 8192, k16),
                         ID_N128_KM, 1);
            mma_commit(&bar[BAR_MMA]);
        }
        // lambda prefetch for the next chunk (warps 2-3 are idle here)
        if (tid >= 64 && tid < 128) {
            const int i = tid - 64, tn = c0 + kC + i;
            lam_next = (tn < T) ? a.lambda[(static_cast<size_t>(b) * T + tn) * H + h] : 0.f;
        }

        // ================= P5: q_clean (Eq. clean), scaled by e^{G - Gmid}, into the Q tile
        mbar_wait(&bar[BAR_MMA], mma_par, abort_flag, a.status);
        mma_par ^= 1;
        tc_fence_after();
        if (tid == 0 && r + 1 < NC && !*abort_flag) issue_k(r + 1);  // Kbar no longer read
        if (rows_warp) {
            const float ti = tf + static_cast<float>(row + 1);
            const float inv_t = 1.f / ti;
            const float c = cv[row], lm = lam[row];
            uint8_t *qt = sm + OFF_Q + ch * 8192;
            const uint8_t *eg = sm + OFF_EG + (row * kEgStride + 64 * ch) * 2;
#pragma unroll
            for (int half = 0; half < 2; ++half) {
                float p[32];
                tmem_ld32(tl + TM_PO + 64 * ch + 32 * half, p);
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) {
                    const int cc = 4 * half + q4;
                    uint4 *qp = reinterpret_cast<uint4 *>(qt + t64_chunk(row, cc));
                    float qb[8], e8[8];
                    unpack_bf16x8(*qp, qb);
                    unpack_bf16x8(*reinterpret_cast<const uint4 *>(eg + 16 * cc), e8);
                    float out[8];
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        const float corr = (p[8 * q4 + e] - c * Mv[64 * ch + 8 * cc + e]) * inv_t;
                        out[e] = (qb[e] - lm * corr) * e8[e];
                    }
                    uint4 u;
                    u.x = pack_bf16(out[0], out[1]);
                    u.y = pack_bf16(out[2], out[3]);
                    u.z = pack_bf16(out[4], out[5]);
                    u.w = pack_bf16(out[6], out[7]);
                    *qp = u;
                }
            }
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();

        // ================= P6: G4 (A = Qg Kg^T), G6 (O = Qg Ssnap)
        if (tid == 0 && !*abort_flag) {
            tc_fence_after();
            for (int kb = 0; kb < 2; ++kb)
                for (int k16 = 0; k16 < 4; ++k16)
                    mma_bf16(tbase + TM_SA, desc_kmajor(sb + OFF_Q + kb * 8192, k16),
                             desc_kmajor(sb + OFF_KG + kb * 8192, k16), ID_N64_KK, (kb | k16) != 0);
            for (int k16 = 0; k16 < 8; ++k16)
                mma_bf16(tbase + TM_PO, desc_kmajor(sb + OFF_Q + (k16 >> 2) * 8192, k16 & 3),
                         desc_mnmajor(sb + OFF_S, 16384, k16), ID_N128_KM, k16 != 0);
            mma_commit(&bar[BAR_MMA]);
        }

        // ================= P7: causal mask of A -> bf16 tile
        mbar_wait(&bar[BAR_MMA], mma_par, abort_flag, a.status);
        mma_par ^= 1;
        tc_fence_after();
        if (tid == 0 && r + 1 < NC && !*abort_flag) issue_q(r + 1);  // Q tile no longer read
        if (rows_warp) {
            tmem_ld32(tl + TM_SA + 32 * ch, sc);
#pragma unroll
            for (int q4 = 0; q4 < 4; ++q4) {
                float w[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const int j = 32 * ch + 8 * q4 + e;
                    w[e] = (j <= row) ? sc[8 * q4 + e] : 0.f;
                }
                uint4 u;
                u.x = pack_bf16(w[0], w[1]);
                u.y = pack_bf16(w[2], w[3]);
                u.z = pack_bf16(w[4], w[5]);
                u.w = pack_bf16(w[6], w[7]);
                *reinterpret_cast<uint4 *>(sm + OFF_W + t64_chunk(row, 4 * ch + q4)) = u;
            }
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();

        // ================= P8: G5 (O += A V), G7 (S += Ku^T V)
        if (tid == 0 && !*abort_flag) {
            mbar_wait(&bar[BAR_V], tpar, abort_flag, a.status);
            tc_fence_after();
            for (int k16 = 0; k16 < 4; ++k16)
                mma_bf16(tbase + TM_PO, desc_kmajor(sb + OFF_W, k16), desc_mnmajor(sb + OFF_V, 8192, k16),
                         ID_N128_KM, 1);
            for (int k16 = 0; k16 < 4; ++k16)
                mma_bf16(tbase + TM_S, desc_mnmajor(sb + OFF_KU, 8192, k16),
                         desc_mnmajor(sb + OFF_V, 8192, k16), ID_N128_MM, 1);
            mma_commit(&bar[BAR_MMA]);
        }

        // ================= P9: o = scale * O; M += chunk key sum; t += n
        mbar_wait(&bar[BAR_MMA], mma_par, abort_flag, a.status);
        mma_par ^= 1;
        tc_fence_after();
        if (tid == 0 && r + 1 < NC && !*abort_flag) issue_v(r + 1);  // V no longer read
        if (rows_warp) {
            const bool valid = row < n;
            __nv_bfloat16 *dst = a.o + ((static_cast<size_t>(b) * T + c0 + row) * H + h) * kD + 64 * ch;
#pragma unroll
            for (int half = 0; half < 2; ++half) {
                float x[32];
                tmem_ld32(tl + TM_PO + 64 * ch + 32 * half, x);
                if (valid) {
#pragma unroll
                    for (int q4 = 0; q4 < 4; ++q4) {
                        uint4 u;
                        u.x = pack_bf16(a.scale * x[8 * q4 + 0], a.scale * x[8 * q4 + 1]);
                        u.y = pack_bf16(a.scale * x[8 * q4 + 2], a.scale * x[8 * q4 + 3]);
                        u.z = pack_bf16(a.scale * x[8 * q4 + 4], a.scale * x[8 * q4 + 5]);
                        u.w = pack_bf16(a.scale * x[8 * q4 + 6], a.scale * x[8 * q4 + 7]);
                        reinterpret_cast<uint4 *>(dst)[4 * half + q4] = u;
                    }
                }
            }
        } else {
            const int d = 32 * (lq - 2) + 64 * ch + lane;  // warps 2,3,6,7 cover dims 0..127
            Mv[d] += dm[d] + dm[kD + d];
        }
        tpos += n;
        tc_fence_before();
        __syncthreads();
    }

    // ---- final states
    tc_fence_after();
    {
        const size_t bhs = static_cast<size_t>(bh);
#pragma unroll
        for (int half = 0; half < 2; ++half) {
            const int c0 = 64 * ch + 32 * half;
            float x[32];
            tmem_ld32(tl + TM_S + c0, x);
            if (a.ST) {
                float4 *dst = reinterpret_cast<float4 *>(a.ST + (bhs * kD + row) * kD + c0);
#pragma unroll
                for (int i = 0; i < 8; ++i) dst[i] = make_float4(x[4 * i], x[4 * i + 1], x[4 * i + 2], x[4 * i + 3]);
            }
            tmem_ld32(tl + TM_SK + c0, x);
            if (a.CT) {
                float4 *dst = reinterpret_cast<float4 *>(a.CT + (bhs * kD + row) * kD + c0);
#pragma unroll
                for (int i = 0; i < 8; ++i) dst[i] = make_float4(x[4 * i], x[4 * i + 1], x[4 * i + 2], x[4 * i + 3]);
            }
        }
        if (a.mT && tid < kD) a.mT[bhs * kD + tid] = Mv[tid];
        if (a.tT && h == 0 && tid == 0) a.tT[b] = tpos;
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tbase, kTmemCols);
    }
}

}  // namespace

cudaError_t launch_gla_chunk(const ChunkArgs &a, const ChunkMaps &m, cudaStream_t s) {
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(gla_chunk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(kSmemBytes));
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    gla_chunk_kernel<<<a.B * a.H, kThreads, kSmemBytes, s>>>(m.q, m.k, m.v, m.g, a);
    return cudaGetLastError();
}

}  // namespace ccq
