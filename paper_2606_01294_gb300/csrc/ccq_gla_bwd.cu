// ccq_gla_bwd.cu -- chunkwise CCQ-GLA backward on sm_103a tensor cores.
//
// Reverse mode of the chunkwise forward (Algorithm 1 with the GLA write,
// Eqs. clean/read, the undecayed running sums of Section 3.2).  The paper
// times a backward but gives none; the adjoint below is derived from those
// definitions and checked against the oracle's reverse mode, which is itself
// pinned by finite differences.
//
// Per chunk r (tokens i, positions t_i, qbar/kbar the unit rows, G the
// in-chunk cumulative log gate, Gmid its value after token 31, Gc after token
// 63, S_r / S^K_r / M_r the forward states at the chunk start, EG = e^{G-Gmid},
// Kd = kbar e^{Gmid-G}, Sx_r = e^{Gmid} S_r):
//   z_i    = Sigma_{t_i} qbar_i = (Zi_i - c1_i M_r) / t_i,  Zi = Qbar S^K + W2 Kbar,
//            c1_i = m_i . qbar_i / t_i,  W2_ij = [j<=i](qbar_i . kbar_j - c1_i)
//   qc_i   = qbar_i - lambda_i z_i                             (Eq. clean)
//   dqc_i  = scale S_{t_i} do_i = scale EG_i (dO Sx_r^T + P1 Kd)_i,  P1_ij = [j<=i] do_i . v_j
//   dlambda_i = -z_i . dqc_i
//   dz'_i  = -lambda_i dqc_i / t_i   (adjoint of z_i, divided by t_i)
//   dqbar_i = dqc_i + C_{t_i} dz'_i - m_i (m_i . dz'_i) / t_i = dqc_i + u_i - cz_i M_r,
//            u = DZ S^K + W3 Kbar,  cz_i = m_i . dz'_i / t_i,  W3_ij = [j<=i](dz'_i . kbar_j - cz_i)
//   carried backwards over chunks (no decay):
//            DC = dC_T + sum dz'_t qbar_t^T      (adjoint of the second-moment sum)
//            Dm = dm_T - sum (c1_t dz'_t + cz_t qbar_t)   (adjoint of the key sum)
//   dkbar_j (CCQ part) = (DC_{r+1} + DC_{r+1}^T) kbar_j + Dm_{r+1} + (W2^T DZ + W3^T Qbar)_j
//   GLA adjoint with q_clean as the query (QG = scale qc EG):
//            dS_r  = Diag(e^{Gc}) dS_{r+1} + Diag(e^{Gmid}) QG^T dO
//            dkbar_j (write part) = e^{Gmid-G_j} (V dSs^T + P1^T QG)_j,  dSs = Diag(e^{Gc-Gmid}) dS_{r+1}
//            dv_j  = (Kd dSs + SA dO)_j,  SA_jt = [t>=j] Kd_j . QG_t
//            dG_t  = qc_t dqc_t - kbar_t dkbar_t(write);  dgk_t = sum_{s>=t} dG_s + rowsum(dS_T S_T),
//            evaluated per chunk as sum_{s>=t in chunk r} dG_s + rowsum(dS_{r+1} S_{r+1})
//   l2 normalisation: dq = (dqbar - qbar (qbar . dqbar)) / |q|, likewise dk.
//
// Everything per chunk depends only on the forward's chunk-start states (the
// checkpoints ccq_gla_chunk.cu writes) and on the three carried adjoints
// (dS, DC, Dm) at the chunk's end, so the backward is three launches:
//   gla_bwd_q_kernel     one CTA per chunk (parallel): z, qc, dqc, dq, dlambda,
//                        the chunk-local CCQ part of dkbar (W2^T DZ + W3^T Qbar),
//                        and the chunk's inputs to the carried sums (QG, DZ
//                        scaled by 1/|q|, the Dm increment, the gate factors).
//   gla_bwd_state_kernel two CTAs per sequence and head (one per column half of
//                        dS and DC), chunks last to first: carries dS (kept as
//                        e^{-Gmid} dS, like the forward's deferred state scaling)
//                        and DC in TMEM and Dm, and writes, per chunk, the states
//                        carried into it (bf16 tile images of Diag(e^{Gc-Gmid})
//                        dS_{r+1} and DC_{r+1}, Dm_{r+1}) and the gate carry
//                        rowsum(dS_{r+1} S_{r+1}) as two column-half sums.
//   gla_bwd_kv_kernel    one CTA per chunk (parallel): dk (write part, the
//                        CCQ inter term K (DC + DC^T), Dm), dv, dgk.
// 64-row products are M = 64 MMAs whose rows 16q..16q+15 sit in TMEM lanes
// 32q..32q+15, so in the chunk-parallel kernels (256 compute threads, two warps
// per lane quadrant, plus a warp that issues the input copies) thread (warp w,
// lane l) owns row 16 (w % 4) + l % 16, column half l / 16 of a 64-column load,
// and -- for 128-column products -- the 32-column slice w / 4 of each half; in
// the state pass (256 threads) thread t owns state row t % 128 and the 32-column
// slice t / 128 of its CTA's column half.
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
constexpr int kThreads = 256;     // the state pass: two warps per TMEM lane quadrant
constexpr int kThreadsPar = 256;  // the chunk-parallel kernels: two warps per TMEM lane quadrant,
constexpr int kLoadWarp = kThreadsPar / 32;       // then one warp that issues the input copies
constexpr int kThreadsLoad = kThreadsPar + 32;
// Barrier of the kThreadsPar compute threads (the load warp leaves once its copies are issued).
__device__ __forceinline__ void compute_sync() { named_bar(1, kThreadsPar); }
constexpr float kLog2e = 1.4426950408889634f;

constexpr uint32_t ID_64x64_KK = make_idesc(64, 64, 0, 0);
constexpr uint32_t ID_64x128_KK = make_idesc(64, 128, 0, 0);
constexpr uint32_t ID_64x128_KM = make_idesc(64, 128, 0, 1);
constexpr uint32_t ID_64x128_MM = make_idesc(64, 128, 1, 1);
constexpr uint32_t ID_128x128_MM = make_idesc(128, 128, 1, 1);
constexpr uint32_t ID_128x64_MK = make_idesc(128, 64, 1, 0);

__device__ __forceinline__ void store_row_chunk(uint8_t *tile, int row, int chunk, const float *w) {
    uint4 u;
    u.x = pack_bf16(w[0], w[1]);
    u.y = pack_bf16(w[2], w[3]);
    u.z = pack_bf16(w[4], w[5]);
    u.w = pack_bf16(w[6], w[7]);
    *reinterpret_cast<uint4 *>(tile + t64_chunk(row, chunk)) = u;
}

__device__ __forceinline__ void load_row_chunk(const uint8_t *tile, int row, int chunk, float (&f)[8]) {
    unpack_bf16x8(*reinterpret_cast<const uint4 *>(tile + t64_chunk(row, chunk)), f);
}

// Chunk preparation of the chunk-parallel kernels (all 256 threads).  Normalises
// the k rows (and the q rows when q_tile is set) of the chunk in place -- two
// threads per row for q and k, four for k alone -- and turns the raw gates
// landed at kd_tile (a plain [64][128] array, bf16 or fp32; the fp32 one also
// covers eg_tile) into the tiles Kd = kbar e^{Gmid-G} and EG = e^{G-Gmid} (G the
// in-chunk cumulative log gate over token quarters, gq4 a [4][128] scratch; Gmid
// its value after token 31).  Outputs per row: rq (1/|q|), mq (M_r . qbar),
// rk (1/|k|); per key dim (when non-null): f = e^{Gc-Gmid}, emid = e^{Gmid}.
__device__ void prep_chunk(uint8_t *q_tile, uint8_t *k_tile, uint8_t *kd_tile, uint8_t *eg_tile,
                              bool gate_f32, bool l2norm, const float *Mr, float *rq, float *mq, float *rk,
                              float *gq4, float *f, float *emid, int pt) {
    {
        const int tpr = q_tile ? 2 : 4;  // threads per row
        const int rr = pt / tpr, part = pt % tpr;
        const bool isq = q_tile != nullptr && rr < 64;
        const int j = rr & 63;
        uint8_t *base = isq ? q_tile : k_tile;
        const int cpp = 16 / tpr;  // 16-byte chunks of the row per thread
        uint4 raw[8];              // the row's chunks, loaded once
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            if (u < cpp) {
                const int cidx = part * cpp + u, t64 = cidx >> 3, cc = cidx & 7;
                raw[u] = *reinterpret_cast<const uint4 *>(base + t64 * 8192 + t64_chunk(j, cc));
            }
        }
        uint64_t s2 = 0, m2 = 0;
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            if (u < cpp) {
                const int cidx = part * cpp + u, t64 = cidx >> 3, cc = cidx & 7;
                const uint32_t w[4] = {raw[u].x, raw[u].y, raw[u].z, raw[u].w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const uint64_t x2 = f2_from_bf16x2(w[e]);
                    s2 = f2_fma(x2, x2, s2);
                    if (isq) m2 = f2_fma(x2, f2_make(Mr[64 * t64 + 8 * cc + 2 * e], Mr[64 * t64 + 8 * cc + 2 * e + 1]), m2);
                }
            }
        }
        const float2 sv = f2_split(s2), mv = f2_split(m2);
        float ss = sv.x + sv.y, md = mv.x + mv.y;
        ss += __shfl_xor_sync(0xffffffffu, ss, 1);
        md += __shfl_xor_sync(0xffffffffu, md, 1);
        if (tpr == 4) {
            ss += __shfl_xor_sync(0xffffffffu, ss, 2);
            md += __shfl_xor_sync(0xffffffffu, md, 2);
        }
        const float rn = l2norm ? rsqrtf(fmaxf(ss, 1e-12f)) : 1.f;
        if (l2norm) {
            const uint64_t rn2 = f2_make(rn, rn);
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                if (u < cpp) {
                    const int cidx = part * cpp + u, t64 = cidx >> 3, cc = cidx & 7;
                    *reinterpret_cast<uint4 *>(base + t64 * 8192 + t64_chunk(j, cc)) =
                        make_uint4(bf16x2_from_f2(f2_mul(f2_from_bf16x2(raw[u].x), rn2)),
                                   bf16x2_from_f2(f2_mul(f2_from_bf16x2(raw[u].y), rn2)),
                                   bf16x2_from_f2(f2_mul(f2_from_bf16x2(raw[u].z), rn2)),
                                   bf16x2_from_f2(f2_mul(f2_from_bf16x2(raw[u].w), rn2)));
                }
            }
        }
        if (part == 0) {
            if (isq) {
                rq[j] = rn;
                mq[j] = md * rn;
            } else {
                rk[j] = rn;
            }
        }
    }
    compute_sync();
    const int p = pt & 63, qt = pt >> 6, d0 = 2 * p;
    uint64_t g2[16];  // cumulative gates of dims d0, d0 + 1 as fp32 pairs
    uint64_t r2 = 0;
#pragma unroll
    for (int jj = 0; jj < 16; ++jj) {
        const int j = 16 * qt + jj;
        const uint64_t x2 = gate_f32 ? *reinterpret_cast<const uint64_t *>(kd_tile + (j * kD + d0) * 4)
                                     : f2_from_bf16x2(*reinterpret_cast<const uint32_t *>(kd_tile + (j * kD + d0) * 2));
        r2 = f2_add(r2, x2);
        g2[jj] = r2;
    }
    const float2 rv = f2_split(r2);
    const float r0 = rv.x, r1 = rv.y;
    gq4[qt * kD + d0] = r0;
    gq4[qt * kD + d0 + 1] = r1;
    compute_sync();  // every raw gate read, quarter sums visible
    float off0 = 0.f, off1 = 0.f;
#pragma unroll
    for (int q = 0; q < 3; ++q)
        if (q < qt) {
            off0 += gq4[q * kD + d0];
            off1 += gq4[q * kD + d0 + 1];
        }
    const float gm0 = gq4[d0] + gq4[kD + d0], gm1 = gq4[d0 + 1] + gq4[kD + d0 + 1];  // Gmid
    const uint64_t o2 = f2_make((off0 - gm0) * kLog2e, (off1 - gm1) * kLog2e);
    const uint64_t l2e = f2_make(kLog2e, kLog2e);
    if (qt == 3) {
        if (f) {
            f[d0] = fast_exp2((off0 + r0 - gm0) * kLog2e);
            f[d0 + 1] = fast_exp2((off1 + r1 - gm1) * kLog2e);
        }
        if (emid) {
            emid[d0] = fast_exp2(gm0 * kLog2e);
            emid[d0 + 1] = fast_exp2(gm1 * kLog2e);
        }
    }
    const uint32_t tcol = (d0 >> 6) * 8192;
    uint32_t kraw[16];  // every k pair before any tile store
#pragma unroll
    for (int jj = 0; jj < 16; ++jj)
        kraw[jj] = *reinterpret_cast<const uint32_t *>(k_tile + tcol + t64_offset(16 * qt + jj, d0 & 63));
#pragma unroll
    for (int jj = 0; jj < 16; ++jj) {
        const int j = 16 * qt + jj;
        const uint32_t off = tcol + t64_offset(j, d0 & 63);
        const float2 x = f2_split(f2_fma(g2[jj], l2e, o2));
        *reinterpret_cast<uint32_t *>(kd_tile + off) =
            bf16x2_from_f2(f2_mul(f2_from_bf16x2(kraw[jj]), f2_make(fast_exp2(-x.x), fast_exp2(-x.y))));
        *reinterpret_cast<uint32_t *>(eg_tile + off) = pack_bf16(fast_exp2(x.x), fast_exp2(x.y));
    }
    fence_proxy_async_smem();
    compute_sync();
}

// Masked row of a 64 x 64 score tile: w_j = [j <= i] (sc_j - c) for the 32
// columns [32 hf, 32 hf + 32) this thread holds; also returns the masked sum.
__device__ __forceinline__ void masked_row(uint8_t *tile, int i, int hf, const float (&sc)[32], float c) {
#pragma unroll
    for (int q4 = 0; q4 < 4; ++q4) {
        float w[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const int j = 32 * hf + 8 * q4 + e;
            w[e] = (j <= i) ? sc[8 * q4 + e] - c : 0.f;
        }
        store_row_chunk(tile, i, 4 * hf + q4, w);
    }
}

__device__ __forceinline__ float masked_sum(int i, int hf, const float (&sc)[32]) {
    float pa[4] = {0.f, 0.f, 0.f, 0.f};  // four chains of eight
#pragma unroll
    for (int jj = 0; jj < 32; ++jj)
        if (32 * hf + jj <= i) pa[jj & 3] += sc[jj];
    const float part = (pa[0] + pa[1]) + (pa[2] + pa[3]);
    return part + __shfl_xor_sync(0xffffffffu, part, 16);
}

// =====================================================================================
// gla_bwd_q_kernel: one CTA per (sequence, head, chunk)
// =====================================================================================
namespace qk {
constexpr uint32_t OFF_Q = 0;        // qbar; then dq (staged for the store)
constexpr uint32_t OFF_K = 16384;    // kbar; then the chunk-local CCQ part of dkbar (staged)
constexpr uint32_t OFF_V = 32768;    // v; then QG (staged)
constexpr uint32_t OFF_DO = 49152;   // do; then DZ
constexpr uint32_t OFF_KD = 65536;   // raw gates land here (fp32: KD + EG); then Kd; then DZ / |q| (staged)
constexpr uint32_t OFF_EG = 81920;   // EG
constexpr uint32_t OFF_SK = 98304;   // S^K_r      } one checkpoint record,
constexpr uint32_t OFF_SX = 131072;  // Sx_r       } one bulk copy; then dqc (16K) + qc*dqc (16K)
constexpr uint32_t OFF_W2 = 163840;  // W2
constexpr uint32_t OFF_P1 = 172032;  // P1, then W3
constexpr uint32_t OFF_BC = 180224;  // [64][64] K-major B operand of the Dm increment: row 0 = -c1, then -cz
constexpr uint32_t OFF_MISC = 188416;
constexpr uint32_t M_MR = 0, M_RQ = 512, M_LAM = 768, M_ITAU = 1024, M_MQ = 1280, M_C1 = 1536, M_MDZ = 1792,
                   M_CZ = 2048, M_RK = 2304, M_F = 2560, M_EM = 3072, M_GQ4 = 3584, M_RED = 5632,
                   M_BAR = 6656, M_TMEM = 6704, M_ABORT = 6708;
constexpr uint32_t kMisc = 6784;
constexpr uint32_t kSmem = OFF_MISC + kMisc + 1024;
static_assert(kSmem <= 232448, "exceeds the 227 KB per-CTA limit");
static_assert(OFF_SX == OFF_SK + 32768, "a checkpoint record lands as one block");
enum { BAR_IN = 0, BAR_INB, BAR_R1, BAR_R2, BAR_R3, BAR_R4, kBars };
static_assert(M_BAR + 8 * kBars <= M_TMEM, "barriers reach the TMEM slot");
constexpr uint32_t TM_SC = 0, TM_T1 = 64, TM_Z = 128, TM_DQ = 256;
}  // namespace qk

__global__ void __launch_bounds__(kThreadsLoad, 1)
gla_bwd_q_kernel(const __grid_constant__ CUtensorMap map_q, const __grid_constant__ CUtensorMap map_k,
                 const __grid_constant__ CUtensorMap map_v, const __grid_constant__ CUtensorMap map_do,
                 const __grid_constant__ CUtensorMap map_g, const __grid_constant__ CUtensorMap map_dq,
                 const __grid_constant__ CUtensorMap map_qg, const __grid_constant__ CUtensorMap map_dkc,
                 const __grid_constant__ CUtensorMap map_gq, const __grid_constant__ CUtensorMap map_dzr,
                 const BwdArgs a) {
    using namespace qk;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = smem_align1024(smem_raw);
    const uint32_t sb = smem_addr(sm);
    uint8_t *misc = sm + OFF_MISC;
    float *Mr = reinterpret_cast<float *>(misc + M_MR);
    float *rqv = reinterpret_cast<float *>(misc + M_RQ);
    float *lamv = reinterpret_cast<float *>(misc + M_LAM);
    float *itauv = reinterpret_cast<float *>(misc + M_ITAU);
    float *mqv = reinterpret_cast<float *>(misc + M_MQ);
    float *c1v = reinterpret_cast<float *>(misc + M_C1);
    float *mdzv = reinterpret_cast<float *>(misc + M_MDZ);
    float *czv = reinterpret_cast<float *>(misc + M_CZ);
    float *rkv = reinterpret_cast<float *>(misc + M_RK);
    float *fv = reinterpret_cast<float *>(misc + M_F);
    float *emv = reinterpret_cast<float *>(misc + M_EM);
    float *gq4 = reinterpret_cast<float *>(misc + M_GQ4);
    float *red = reinterpret_cast<float *>(misc + M_RED);  // [2 groups][2][64] row partial sums
    uint64_t *bar = reinterpret_cast<uint64_t *>(misc + M_BAR);
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(misc + M_TMEM);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(misc + M_ABORT);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int qd = warp & 3, grp = warp >> 2;  // TMEM lane quadrant, warp group
    const int T = a.T, H = a.H, NC = (T + kC - 1) / kC;
    const int bh = blockIdx.x / NC, r = blockIdx.x % NC, b = bh / H, h = bh % H;
    const int c0 = r * kC;
    const bool gate_f32 = a.gate_dtype != 0;
    const uint32_t g_bytes = gate_f32 ? kC * kD * 4 : kC * kD * 2;
    const int64_t tseq0 = a.t0 ? a.t0[b] : 0;
    const uint8_t *rec = a.ckpt + static_cast<size_t>(bh) * ckpt_head_bytes(T) + static_cast<size_t>(r) * kCkptChunkBytes;
    float *cvec = a.chunk_vec + static_cast<size_t>(blockIdx.x) * 3 * kD;  // f, e^{Gmid}, Dm increment
    int *status = a.status;

    // The load warp issues the copies: first what the row norms and the gate prefix need
    // (q, k, gates, M_r), then, once the compute threads are released, the rest, which
    // lands while that preparation runs.  Issuing stalls as the copy engine fills, so no
    // compute thread waits for it.
    if (warp == kLoadWarp && lane == 0) {
        for (int i = 0; i < kBars; ++i) mbar_init(&bar[i], 1);
        *abort_flag = 0;
        fence_barrier_init();
        uint64_t *ba = &bar[BAR_IN], *bb = &bar[BAR_INB];
        mbar_arrive_expect_tx(ba, 2 * 16384 + g_bytes + 512);
        mbar_arrive_expect_tx(bb, 2 * 16384 + 65536);
        tma_load_4d(sm + OFF_Q, &map_q, ba, 0, h, c0, b);
        tma_load_4d(sm + OFF_Q + 8192, &map_q, ba, 64, h, c0, b);
        tma_load_4d(sm + OFF_K, &map_k, ba, 0, h, c0, b);
        tma_load_4d(sm + OFF_K + 8192, &map_k, ba, 64, h, c0, b);
        tma_load_4d(sm + OFF_KD, &map_g, ba, 0, h, c0, b);
        bulk_load(misc + M_MR, rec + 65536, 512, ba);
    }
    if (warp == 0) tmem_alloc(tmem_slot, 512);
    if (tid < kThreadsPar)
        for (int e = tid; e < 8192 / 16; e += kThreadsPar)
            reinterpret_cast<uint4 *>(sm + OFF_BC)[e] = make_uint4(0u, 0u, 0u, 0u);
    if (tid < kC) {
        const int n = c0 + tid;
        lamv[tid] = n < T ? a.lambda[(static_cast<size_t>(b) * T + n) * H + h] : 0.f;
        itauv[tid] = 1.f / static_cast<float>(tseq0 + n + 1);
    }
    __syncthreads();
    if (warp == kLoadWarp) {
        if (lane == 0) {
            uint64_t *bb = &bar[BAR_INB];
            tma_load_4d(sm + OFF_V, &map_v, bb, 0, h, c0, b);
            tma_load_4d(sm + OFF_V + 8192, &map_v, bb, 64, h, c0, b);
            tma_load_4d(sm + OFF_DO, &map_do, bb, 0, h, c0, b);
            tma_load_4d(sm + OFF_DO + 8192, &map_do, bb, 64, h, c0, b);
            bulk_load(sm + OFF_SK, rec, 65536, bb);
            // the chunk one wave later finds its inputs in L2
            const int nx = blockIdx.x + a.wave;
            if (a.wave > 0 && nx < static_cast<int>(gridDim.x)) {
                const int bh2 = nx / NC, r2 = nx % NC, b2 = bh2 / H, h2 = bh2 % H, c2 = r2 * kC;
                tma_prefetch_l2_4d(&map_q, 0, h2, c2, b2);
                tma_prefetch_l2_4d(&map_q, 64, h2, c2, b2);
                tma_prefetch_l2_4d(&map_k, 0, h2, c2, b2);
                tma_prefetch_l2_4d(&map_k, 64, h2, c2, b2);
                tma_prefetch_l2_4d(&map_v, 0, h2, c2, b2);
                tma_prefetch_l2_4d(&map_v, 64, h2, c2, b2);
                tma_prefetch_l2_4d(&map_do, 0, h2, c2, b2);
                tma_prefetch_l2_4d(&map_do, 64, h2, c2, b2);
                tma_prefetch_l2_4d(&map_g, 0, h2, c2, b2);
                bulk_prefetch_l2(a.ckpt + static_cast<size_t>(bh2) * ckpt_head_bytes(T) + static_cast<size_t>(r2) * kCkptChunkBytes,
                                 static_cast<uint32_t>(kCkptChunkBytes));
            }
        }
        return;
    }
    tc_fence_after();
    const uint32_t tbase = *tmem_slot;
    const uint32_t tq = tbase + (static_cast<uint32_t>(32 * qd) << 16);

    const int i = 16 * qd + (lane & 15);  // chunk row of this thread in the M = 64 products
    const int hf = lane >> 4;             // column half of a 64-column load; group grp takes the
                                          // 32-column slice h2 = grp of each 128-column product
    // descriptors (K-major: advance 32 B per K16 slice, 8 KB / 16 KB per 64-wide K block;
    // MN-major: advance 2 KB per 16 K rows)
    const uint64_t dQ = make_desc(sb + OFF_Q, 16, 1024), dQm = make_desc(sb + OFF_Q, 8192, 1024);
    const uint64_t dK = make_desc(sb + OFF_K, 16, 1024), dKm = make_desc(sb + OFF_K, 8192, 1024);
    const uint64_t dV = make_desc(sb + OFF_V, 16, 1024);
    const uint64_t dDO = make_desc(sb + OFF_DO, 16, 1024), dDOm = make_desc(sb + OFF_DO, 8192, 1024);
    const uint64_t dKDm = make_desc(sb + OFF_KD, 8192, 1024);
    const uint64_t dSK = make_desc(sb + OFF_SK, 16, 1024), dSX = make_desc(sb + OFF_SX, 16, 1024);
    const uint64_t dW2 = make_desc(sb + OFF_W2, 16, 1024), dW2m = make_desc(sb + OFF_W2, 8192, 1024);
    const uint64_t dP1 = make_desc(sb + OFF_P1, 16, 1024), dP1m = make_desc(sb + OFF_P1, 8192, 1024);
    const uint64_t dBC = make_desc(sb + OFF_BC, 16, 1024);

    mbar_wait(&bar[BAR_IN], 0, abort_flag, status);
    prep_chunk(sm + OFF_Q, sm + OFF_K, sm + OFF_KD, sm + OFF_EG, gate_f32, a.l2norm, Mr, rqv, mqv, rkv, gq4,
               fv, emv, tid);
    mbar_wait(&bar[BAR_INB], 0, abort_flag, status);
    tc_fence_before();
    if (tid == 0 && !*abort_flag) {
        tc_fence_after();
        for (int k = 0; k < 8; ++k) {  // Sc = Qbar Kbar^T, T1 = dO V^T
            const uint64_t ko = (k >> 2) * 512 + (k & 3) * 2;
            mma_bf16(tbase + TM_SC, dQ + ko, dK + ko, ID_64x64_KK, k != 0);
        }
        for (int k = 0; k < 8; ++k) {
            const uint64_t ko = (k >> 2) * 512 + (k & 3) * 2;
            mma_bf16(tbase + TM_T1, dDO + ko, dV + ko, ID_64x64_KK, k != 0);
        }
        for (int k = 0; k < 8; ++k) {  // Zi = Qbar S^K, Dq = dO Sx^T
            const uint64_t ka = (k >> 2) * 512 + (k & 3) * 2, kb = (k >> 2) * 1024 + (k & 3) * 2;
            mma_bf16(tbase + TM_Z, dQ + ka, dSK + kb, ID_64x128_KK, k != 0);
        }
        for (int k = 0; k < 8; ++k) {
            const uint64_t ka = (k >> 2) * 512 + (k & 3) * 2, kb = (k >> 2) * 1024 + (k & 3) * 2;
            mma_bf16(tbase + TM_DQ, dDO + ka, dSX + kb, ID_64x128_KK, k != 0);
        }
        mma_commit(&bar[BAR_R1]);
    }
    // ---- E1: c1, W2, P1
    mbar_wait(&bar[BAR_R1], 0, abort_flag, status);
    tc_fence_after();
    if (grp == 0) {
        float sc[32];
        tmem_ld16x2_32<32>(tq + TM_SC, sc);
        const float part = masked_sum(i, hf, sc);
        const float c1 = a.centered ? (mqv[i] + part) * itauv[i] : 0.f;
        if (hf == 0) {
            c1v[i] = c1;
            *reinterpret_cast<__nv_bfloat16 *>(sm + OFF_BC + t64_offset(0, i)) = __float2bfloat16_rn(-c1);
        }
        masked_row(sm + OFF_W2, i, hf, sc, c1);
    } else {
        float t1[32];
        tmem_ld16x2_32<32>(tq + TM_T1, t1);
        masked_row(sm + OFF_P1, i, hf, t1, 0.f);
    }
    fence_proxy_async_smem();
    tc_fence_before();
    compute_sync();
    if (tid == 0 && !*abort_flag) {
        tc_fence_after();
        for (int k = 0; k < 4; ++k)  // Zi += W2 Kbar, Dq += P1 Kd
            mma_bf16(tbase + TM_Z, dW2 + k * 2, dKm + k * 128, ID_64x128_KM, 1);
        for (int k = 0; k < 4; ++k)
            mma_bf16(tbase + TM_DQ, dP1 + k * 2, dKDm + k * 128, ID_64x128_KM, 1);
        mma_commit(&bar[BAR_R2]);
    }
    // ---- E2: z, q_clean, dqc, dlambda; tiles QG, DZ, DZ / |q|, dqc, qc*dqc
    mbar_wait(&bar[BAR_R2], 0, abort_flag, status);
    tc_fence_after();
    {
        const float lam = lamv[i], itau = itauv[i], c1 = c1v[i], rq = rqv[i];
        const float nl = -lam * itau;
        const float *Mh = Mr + 64 * hf;
        const uint8_t *qbt = sm + OFF_Q + hf * 8192;
        const uint8_t *egt = sm + OFF_EG + hf * 8192;
        float dl = 0.f, mdz = 0.f;
        {
            // fp32 pairs over consecutive columns
            const int h2 = grp;
            float zi[32], dqa[32];
            tmem_ld16x2_32<64>(tq + TM_Z + 32 * h2, zi);
            tmem_ld16x2_32<64>(tq + TM_DQ + 32 * h2, dqa);
            const uint64_t nc1 = f2_make(-c1, -c1), itau2 = f2_make(itau, itau), nlam2 = f2_make(-lam, -lam);
            const uint64_t sc2 = f2_make(a.scale, a.scale), nl2 = f2_make(nl, nl), rq2 = f2_make(rq, rq);
            uint64_t dl2 = 0, mdz2 = 0;  // sum of z dqc (negated at the end), sum of m d
#pragma unroll
            for (int q4 = 0; q4 < 4; ++q4) {
                const int cc = 4 * h2 + q4;
                const uint4 qraw = *reinterpret_cast<const uint4 *>(qbt + t64_chunk(i, cc));
                const uint4 eraw = *reinterpret_cast<const uint4 *>(egt + t64_chunk(i, cc));
                const ulonglong2 mlo = *reinterpret_cast<const ulonglong2 *>(Mh + 8 * cc);
                const ulonglong2 mhi = *reinterpret_cast<const ulonglong2 *>(Mh + 8 * cc + 4);
                const uint32_t qw[4] = {qraw.x, qraw.y, qraw.z, qraw.w};
                const uint32_t ew[4] = {eraw.x, eraw.y, eraw.z, eraw.w};
                const uint64_t mp[4] = {mlo.x, mlo.y, mhi.x, mhi.y};
                uint32_t qg[4], dz[4], dzr[4], dqv[4], gq[4];
#pragma unroll
                for (int w = 0; w < 4; ++w) {
                    const int e = 8 * q4 + 2 * w;
                    const uint64_t eg2 = f2_from_bf16x2(ew[w]);
                    const uint64_t z2 = f2_mul(f2_fma(nc1, mp[w], f2_make(zi[e], zi[e + 1])), itau2);
                    const uint64_t qc2 = f2_fma(nlam2, z2, f2_from_bf16x2(qw[w]));
                    const uint64_t dqc2 = f2_mul(f2_mul(sc2, eg2), f2_make(dqa[e], dqa[e + 1]));
                    const uint64_t d2 = f2_mul(nl2, dqc2);
                    dl2 = f2_fma(z2, dqc2, dl2);
                    mdz2 = f2_fma(mp[w], d2, mdz2);
                    qg[w] = bf16x2_from_f2(f2_mul(f2_mul(sc2, qc2), eg2));
                    dz[w] = bf16x2_from_f2(d2);
                    dzr[w] = bf16x2_from_f2(f2_mul(d2, rq2));
                    dqv[w] = bf16x2_from_f2(dqc2);
                    gq[w] = bf16x2_from_f2(f2_mul(qc2, dqc2));
                }
                const uint32_t off = t64_chunk(i, cc);
                *reinterpret_cast<uint4 *>(sm + OFF_V + hf * 8192 + off) = make_uint4(qg[0], qg[1], qg[2], qg[3]);
                *reinterpret_cast<uint4 *>(sm + OFF_DO + hf * 8192 + off) = make_uint4(dz[0], dz[1], dz[2], dz[3]);
                *reinterpret_cast<uint4 *>(sm + OFF_KD + hf * 8192 + off) = make_uint4(dzr[0], dzr[1], dzr[2], dzr[3]);
                *reinterpret_cast<uint4 *>(sm + OFF_SX + hf * 8192 + off) = make_uint4(dqv[0], dqv[1], dqv[2], dqv[3]);
                *reinterpret_cast<uint4 *>(sm + OFF_SX + 16384 + hf * 8192 + off) = make_uint4(gq[0], gq[1], gq[2], gq[3]);
            }
            const float2 dlv = f2_split(dl2), mdv = f2_split(mdz2);
            dl = -(dlv.x + dlv.y);
            mdz = mdv.x + mdv.y;
        }
        dl += __shfl_xor_sync(0xffffffffu, dl, 16);
        mdz += __shfl_xor_sync(0xffffffffu, mdz, 16);
        if (hf == 0) {
            red[grp * 128 + i] = dl;
            red[grp * 128 + 64 + i] = mdz;
        }
        compute_sync();
        if (grp == 0 && hf == 0) {
            dl = red[i] + red[128 + i];
            mdzv[i] = red[64 + i] + red[192 + i];
            const int n = c0 + i;
            if (n < T && a.dlambda) a.dlambda[(static_cast<size_t>(b) * T + n) * H + h] = dl;
        }
    }
    fence_proxy_async_smem();
    tc_fence_before();
    compute_sync();
    if (tid == 0 && !*abort_flag) {
        tma_store_4d(&map_qg, sm + OFF_V, 0, h, c0, b);
        tma_store_4d(&map_qg, sm + OFF_V + 8192, 64, h, c0, b);
        tma_store_4d(&map_gq, sm + OFF_SX + 16384, 0, h, c0, b);
        tma_store_4d(&map_gq, sm + OFF_SX + 16384 + 8192, 64, h, c0, b);
        tma_store_4d(&map_dzr, sm + OFF_KD, 0, h, c0, b);
        tma_store_4d(&map_dzr, sm + OFF_KD + 8192, 64, h, c0, b);
        tma_store_commit();
        tc_fence_after();
        for (int k = 0; k < 8; ++k) {  // T3 = DZ Kbar^T
            const uint64_t ko = (k >> 2) * 512 + (k & 3) * 2;
            mma_bf16(tbase + TM_SC, dDO + ko, dK + ko, ID_64x64_KK, k != 0);
        }
        for (int k = 0; k < 8; ++k) {  // u = DZ S^K
            const uint64_t ka = (k >> 2) * 512 + (k & 3) * 2, kb = (k >> 2) * 1024 + (k & 3) * 2;
            mma_bf16(tbase + TM_Z, dDO + ka, dSK + kb, ID_64x128_KK, k != 0);
        }
        for (int k = 0; k < 4; ++k)  // dkc = W2^T DZ
            mma_bf16(tbase + TM_DQ, dW2m + k * 128, dDOm + k * 128, ID_64x128_MM, k != 0);
        for (int k = 0; k < 4; ++k)  // Dm increment, first half: DZ^T (-c1)
            mma_bf16(tbase + TM_T1, dDOm + k * 128, dBC + k * 2, ID_128x64_MK, k != 0);
        mma_commit(&bar[BAR_R3]);
    }
    // ---- E3: cz, W3
    mbar_wait(&bar[BAR_R3], 0, abort_flag, status);
    tc_fence_after();
    if (grp == 0) {
        float t3[32];
        tmem_ld16x2_32<32>(tq + TM_SC, t3);
        const float part = masked_sum(i, hf, t3);
        const float cz = a.centered ? (mdzv[i] + part) * itauv[i] : 0.f;
        if (hf == 0) {
            czv[i] = cz;
            *reinterpret_cast<__nv_bfloat16 *>(sm + OFF_BC + t64_offset(0, i)) = __float2bfloat16_rn(-cz);
        }
        masked_row(sm + OFF_P1, i, hf, t3, cz);
    }
    fence_proxy_async_smem();
    tc_fence_before();
    compute_sync();
    if (tid == 0 && !*abort_flag) {
        tc_fence_after();
        for (int k = 0; k < 4; ++k)  // u += W3 Kbar
            mma_bf16(tbase + TM_Z, dP1 + k * 2, dKm + k * 128, ID_64x128_KM, 1);
        for (int k = 0; k < 4; ++k)  // dkc += W3^T Qbar
            mma_bf16(tbase + TM_DQ, dP1m + k * 128, dQm + k * 128, ID_64x128_MM, 1);
        for (int k = 0; k < 4; ++k)  // Dm increment, second half: Qbar^T (-cz)
            mma_bf16(tbase + TM_T1, dQm + k * 128, dBC + k * 2, ID_128x64_MK, 1);
        mma_commit(&bar[BAR_R4]);
    }
    // ---- E4: dq, the chunk-local CCQ part of dkbar, the chunk's vectors
    mbar_wait(&bar[BAR_R4], 0, abort_flag, status);
    tc_fence_after();
    if (grp == 0) {
        float x[32];
        tmem_ld32(tq + TM_T1, x);  // lane tid, column 0: the Dm increment of this chunk
        cvec[tid] = fv[tid];
        cvec[kD + tid] = emv[tid];
        cvec[2 * kD + tid] = x[0];
    }
    {
        const float cz = czv[i], rq = rqv[i];
        const float *Mh = Mr + 64 * hf;
        uint8_t *qbt = sm + OFF_Q + hf * 8192;
        const uint8_t *dqt = sm + OFF_SX + hf * 8192;
        const int h2 = grp;
        uint64_t dqb[16];  // fp32 pairs over consecutive columns
        float dot;
        {
            float u[32];
            tmem_ld16x2_32<64>(tq + TM_Z + 32 * h2, u);
            const uint64_t ncz = f2_make(-cz, -cz);
            uint64_t dot2 = 0;
#pragma unroll
            for (int q4 = 0; q4 < 4; ++q4) {
                const int cc = 4 * h2 + q4;
                const uint4 draw = *reinterpret_cast<const uint4 *>(dqt + t64_chunk(i, cc));
                const uint4 qraw = *reinterpret_cast<const uint4 *>(qbt + t64_chunk(i, cc));
                const ulonglong2 mlo = *reinterpret_cast<const ulonglong2 *>(Mh + 8 * cc);
                const ulonglong2 mhi = *reinterpret_cast<const ulonglong2 *>(Mh + 8 * cc + 4);
                const uint32_t dw[4] = {draw.x, draw.y, draw.z, draw.w};
                const uint32_t qw[4] = {qraw.x, qraw.y, qraw.z, qraw.w};
                const uint64_t mp[4] = {mlo.x, mlo.y, mhi.x, mhi.y};
#pragma unroll
                for (int w = 0; w < 4; ++w) {
                    const int e = 8 * q4 + 2 * w;
                    const uint64_t v = f2_fma(ncz, mp[w], f2_add(f2_from_bf16x2(dw[w]), f2_make(u[e], u[e + 1])));
                    dqb[4 * q4 + w] = v;
                    dot2 = f2_fma(f2_from_bf16x2(qw[w]), v, dot2);
                }
            }
            const float2 dv = f2_split(dot2);
            dot = dv.x + dv.y;
        }
        dot += __shfl_xor_sync(0xffffffffu, dot, 16);
        if (hf == 0) red[grp * 128 + i] = dot;
        // the dkc tile: this group's 32-column slice
        uint8_t *kt = sm + OFF_K + hf * 8192;
        {
            float x[32];
            tmem_ld16x2_32<64>(tq + TM_DQ + 32 * h2, x);
#pragma unroll
            for (int q4 = 0; q4 < 4; ++q4) store_row_chunk(kt, i, 4 * h2 + q4, x + 8 * q4);
        }
        compute_sync();
        dot = red[i] + red[128 + i];
        const uint64_t ndot = f2_make(-dot, -dot), rq2 = f2_make(rq, rq);
#pragma unroll
        for (int q4 = 0; q4 < 4; ++q4) {
            const int cc = 4 * h2 + q4;
            const uint4 qraw = *reinterpret_cast<const uint4 *>(qbt + t64_chunk(i, cc));
            const uint32_t qw[4] = {qraw.x, qraw.y, qraw.z, qraw.w};
            uint32_t ow[4];
#pragma unroll
            for (int w = 0; w < 4; ++w) {
                const uint64_t v = dqb[4 * q4 + w];
                ow[w] = bf16x2_from_f2(a.l2norm ? f2_mul(rq2, f2_fma(ndot, f2_from_bf16x2(qw[w]), v)) : v);
            }
            *reinterpret_cast<uint4 *>(qbt + t64_chunk(i, cc)) = make_uint4(ow[0], ow[1], ow[2], ow[3]);
        }
    }
    fence_proxy_async_smem();
    tc_fence_before();
    compute_sync();
    if (tid == 0 && !*abort_flag) {
        tma_store_4d(&map_dq, sm + OFF_Q, 0, h, c0, b);
        tma_store_4d(&map_dq, sm + OFF_Q + 8192, 64, h, c0, b);
        tma_store_4d(&map_dkc, sm + OFF_K, 0, h, c0, b);
        tma_store_4d(&map_dkc, sm + OFF_K + 8192, 64, h, c0, b);
        tma_store_commit();
        tma_store_wait_read();  // shared memory outlives the stores' reads
    }
    tc_fence_before();
    compute_sync();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tbase, 512);
    }
}

// =====================================================================================
// gla_bwd_state_kernel: two CTAs per (sequence, head) (column halves), chunks last to first
// =====================================================================================
namespace st {
// per input buffer: QG, DZ/|q| (16 KB each), this CTA's column half of dO and raw q (8 KB each)
constexpr uint32_t BUF_BYTES = 49152;
constexpr uint32_t B_QG = 0, B_DZ = 16384, B_DO = 32768, B_Q = 40960;
constexpr uint32_t OFF_SX = 2 * BUF_BYTES;      // 98304: column half of Sx_r (checkpoint, for the gate carry)
constexpr uint32_t OFF_IMG = OFF_SX + 16384;    // 114688: column halves of the images written per chunk:
                                                //   Diag(e^{Gc-Gmid}) dS_{r+1} (16 KB), DC_{r+1} (16 KB)
constexpr uint32_t OFF_MISC = OFF_IMG + 32768;  // 147456
constexpr uint32_t M_DM = 0, M_CARRY = 512, M_BAR = 1536, M_TMEM = 1568, M_ABORT = 1572;
constexpr uint32_t kMisc = 1600;
constexpr uint32_t kSmem = OFF_MISC + kMisc + 1024;
static_assert(kSmem <= 232448, "exceeds the 227 KB per-CTA limit");
enum { BAR_IN0 = 0, BAR_IN1, BAR_SX, BAR_MMA, kBars };
constexpr uint32_t TM_X = 0, TM_DC = 64;
constexpr uint32_t ID_128x64_MM = make_idesc(128, 64, 1, 1);
}  // namespace st

// Two CTAs per (sequence, head), one per column half ch of dS and DC (both updates split
// by columns), two warps per TMEM lane quadrant: thread (row, th) holds state row `row`,
// columns 64 ch + 32 th .. + 31.  Per chunk r (last to first) the chain is: read X (the
// state after chunk r+1's update), its gate carry against Sx_{r+1} (a partial row sum over
// this CTA's columns; the consumer adds the two), rescale to Diag(e^{Gc-Gmid}) dS_{r+1} (the
// image, and X in place), the DC image, then the two updates of chunk r.
__global__ void __launch_bounds__(kThreads, 1)
gla_bwd_state_kernel(const __grid_constant__ CUtensorMap map_qg, const __grid_constant__ CUtensorMap map_do,
                     const __grid_constant__ CUtensorMap map_dzr, const __grid_constant__ CUtensorMap map_q,
                     const BwdArgs a) {
    using namespace st;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = smem_align1024(smem_raw);
    const uint32_t sb = smem_addr(sm);
    uint8_t *misc = sm + OFF_MISC;
    float *Dm = reinterpret_cast<float *>(misc + M_DM);
    float *carry = reinterpret_cast<float *>(misc + M_CARRY);  // [2 thread halves][128] partial row sums
    uint64_t *bar = reinterpret_cast<uint64_t *>(misc + M_BAR);
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(misc + M_TMEM);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(misc + M_ABORT);

    const int tid = threadIdx.x, warp = tid >> 5;
    const int row = tid & (kD - 1), th = tid >> 7;
    const int ch = blockIdx.x & 1, c = 2 * ch + th;  // column half of the state; 32-column unit
    const int bh = blockIdx.x >> 1, b = bh / a.H, h = bh % a.H;
    const int T = a.T, NC = (T + kC - 1) / kC;
    const uint8_t *ck = a.ckpt + static_cast<size_t>(bh) * ckpt_head_bytes(T);
    const size_t chunk0 = static_cast<size_t>(bh) * NC;  // flat index of this sequence's chunk 0
    int *status = a.status;

    if (tid == 0) {
        for (int i = 0; i < kBars; ++i) mbar_init(&bar[i], 1);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 0) tmem_alloc(tmem_slot, 128);
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *tmem_slot;
    const uint32_t tq = tbase + (static_cast<uint32_t>(32 * (warp & 3)) << 16);
    {
        // X <- dS_T, DC <- dC_T, Dm <- dm_T; the gate carry of the last chunk is rowsum(dS_T * S_T)
        const size_t grow = static_cast<size_t>(bh) * kD + row;
        const float *dst_row = a.dST ? a.dST + grow * kD : nullptr;
        const float *dct_row = a.dCT ? a.dCT + grow * kD : nullptr;
        const float *st_row = reinterpret_cast<const float *>(ck + static_cast<size_t>(NC) * kCkptChunkBytes) + row * kD;
        float cs = 0.f;
        {
            float x[32], y[32];
#pragma unroll
            for (int e = 0; e < 32; ++e) {
                x[e] = dst_row ? dst_row[32 * c + e] : 0.f;
                if (dst_row) cs = fmaf(x[e], st_row[32 * c + e], cs);
                y[e] = dct_row ? dct_row[32 * c + e] : 0.f;
            }
            tmem_st32(tq + TM_X + 32 * th, x);
            tmem_st32(tq + TM_DC + 32 * th, y);
        }
        tmem_wait_st();
        carry[th * kD + row] = cs;
        if (th == 0) Dm[row] = a.dmT ? a.dmT[grow] : 0.f;
    }
    auto issue = [&](int r, int buf) {
        const int tg = r * kC;
        uint8_t *base = sm + buf * BUF_BYTES;
        uint64_t *bb = &bar[BAR_IN0 + buf];
        mbar_arrive_expect_tx(bb, BUF_BYTES);
        tma_load_4d(base + B_QG, &map_qg, bb, 0, h, tg, b);
        tma_load_4d(base + B_QG + 8192, &map_qg, bb, 64, h, tg, b);
        tma_load_4d(base + B_DZ, &map_dzr, bb, 0, h, tg, b);
        tma_load_4d(base + B_DZ + 8192, &map_dzr, bb, 64, h, tg, b);
        tma_load_4d(base + B_DO, &map_do, bb, 64 * ch, h, tg, b);
        tma_load_4d(base + B_Q, &map_q, bb, 64 * ch, h, tg, b);
    };
    auto issue_sx = [&](int r) {
        mbar_arrive_expect_tx(&bar[BAR_SX], 16384);
        bulk_load(sm + OFF_SX, ck + static_cast<size_t>(r) * kCkptChunkBytes + 32768 + 16384 * ch, 16384, &bar[BAR_SX]);
    };
    if (tid == 0 && NC > 0) {
        issue(NC - 1, 0);
        if (NC > 1) issue(NC - 2, 1);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();

    float em_next = 1.f;  // e^{Gmid_{r+1}} (1 past the last chunk)
    for (int it = 0; it < NC; ++it) {
        const int r = NC - 1 - it, buf = it & 1;
        const uint32_t bpar = (it >> 1) & 1;
        const size_t ci = chunk0 + r;
        const float *cvec = a.chunk_vec + ci * 3 * kD;
        const float f = cvec[row], em = cvec[kD + row], ddm = cvec[2 * kD + row];
        if (it > 0) {
            // the update of chunk r+1 and Sx_{r+1} have landed; the previous images are out
            mbar_wait(&bar[BAR_MMA], (it - 1) & 1, abort_flag, status);
            mbar_wait(&bar[BAR_SX], (it - 1) & 1, abort_flag, status);
            if (tid == 0) tma_store_wait_read();
            __syncthreads();
            tc_fence_after();
            if (tid == 0 && !*abort_flag && r + 1 >= 2) issue(r - 1, buf ^ 1);  // chunk r+1's buffer is free
        }
        // X holds e^{-Gmid_{r+1}} dS_{r+1}: its gate carry rowsum(X * Sx_{r+1}) (chunk r's), then
        // Diag(e^{Gc_r - Gmid_r}) dS_{r+1} = (f_r e^{Gmid_{r+1}}) X as the image and in place
        const float hs = f * em_next;
        float cs = 0.f;
        {
            float x[32];
            tmem_ld32(tq + TM_X + 32 * th, x);
            if (it > 0) {
                uint64_t cs2 = 0;  // fp32 pairs: two chains
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) {
                    const uint4 sr = *reinterpret_cast<const uint4 *>(sm + OFF_SX + t64_chunk(row, 4 * th + q4));
                    const uint32_t sw[4] = {sr.x, sr.y, sr.z, sr.w};
#pragma unroll
                    for (int w = 0; w < 4; ++w)
                        cs2 = f2_fma(f2_make(x[8 * q4 + 2 * w], x[8 * q4 + 2 * w + 1]), f2_from_bf16x2(sw[w]), cs2);
                }
                const float2 cv = f2_split(cs2);
                cs = cv.x + cv.y;
            }
            const uint64_t hs2 = f2_make(hs, hs);
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                const float2 y = f2_split(f2_mul(f2_make(x[2 * e], x[2 * e + 1]), hs2));
                x[2 * e] = y.x;
                x[2 * e + 1] = y.y;
            }
#pragma unroll
            for (int q4 = 0; q4 < 4; ++q4) store_row_chunk(sm + OFF_IMG, row, 4 * th + q4, x + 8 * q4);
            tmem_st32(tq + TM_X + 32 * th, x);
            float y[32];
            tmem_ld32(tq + TM_DC + 32 * th, y);
#pragma unroll
            for (int q4 = 0; q4 < 4; ++q4) store_row_chunk(sm + OFF_IMG + 16384, row, 4 * th + q4, y + 8 * q4);
        }
        if (it > 0) carry[th * kD + row] = cs;
        em_next = em;
        tmem_wait_st();
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        if (th == 0) {
            if (ch == 0) a.state_vec[ci * 3 * kD + row] = Dm[row];
            a.state_vec[ci * 3 * kD + (1 + ch) * kD + row] = carry[row] + carry[kD + row];
            Dm[row] += ddm;  // Dm_r
        }
        if (tid == 0 && !*abort_flag && r >= 1) issue_sx(r);  // Sx_{r+1} has been read
        mbar_wait(&bar[BAR_IN0 + buf], bpar, abort_flag, status);
        if (tid == 0 && !*abort_flag) {
            bulk_store(a.state_img + ci * 65536 + 16384 * ch, sm + OFF_IMG, 16384);
            bulk_store(a.state_img + ci * 65536 + 32768 + 16384 * ch, sm + OFF_IMG + 16384, 16384);
            tma_store_commit();
            tc_fence_after();
            const uint32_t base = sb + buf * BUF_BYTES;
            const uint64_t dQGm = make_desc(base + B_QG, 8192, 1024), dDOm = make_desc(base + B_DO, 8192, 1024);
            const uint64_t dDZm = make_desc(base + B_DZ, 8192, 1024), dQm = make_desc(base + B_Q, 8192, 1024);
            for (int k = 0; k < 4; ++k)  // X += QG^T dO  (-> e^{-Gmid_r} dS_r), this CTA's columns
                mma_bf16(tbase + TM_X, dQGm + k * 128, dDOm + k * 128, ID_128x64_MM, 1);
            for (int k = 0; k < 4; ++k)  // DC += (DZ / |q|)^T q  (= DZ^T Qbar), this CTA's columns
                mma_bf16(tbase + TM_DC, dDZm + k * 128, dQm + k * 128, ID_128x64_MM, 1);
            mma_commit(&bar[BAR_MMA]);
        }
    }

    if (NC > 0) mbar_wait(&bar[BAR_MMA], (NC - 1) & 1, abort_flag, status);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    {
        const size_t grow = static_cast<size_t>(bh) * kD + row;
        const float e0 = em_next;  // e^{Gmid_0}: dS_0 = e^{Gmid_0} X
        {
            float x[32];
            tmem_ld32(tq + TM_X + 32 * th, x);
            if (a.dS0)
#pragma unroll
                for (int e = 0; e < 8; ++e)
                    reinterpret_cast<float4 *>(a.dS0 + grow * kD + 32 * c)[e] =
                        make_float4(e0 * x[4 * e], e0 * x[4 * e + 1], e0 * x[4 * e + 2], e0 * x[4 * e + 3]);
            tmem_ld32(tq + TM_DC + 32 * th, x);
            if (a.dC0)
#pragma unroll
                for (int e = 0; e < 8; ++e)
                    reinterpret_cast<float4 *>(a.dC0 + grow * kD + 32 * c)[e] =
                        make_float4(x[4 * e], x[4 * e + 1], x[4 * e + 2], x[4 * e + 3]);
        }
        if (a.dm0 && ch == 0 && th == 0) a.dm0[grow] = Dm[row];
    }
    if (tid == 0) tma_store_wait_all();
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tbase, 128);
    }
}

// =====================================================================================
// gla_bwd_kv_kernel: one CTA per (sequence, head, chunk)
// =====================================================================================
namespace kv {
constexpr uint32_t OFF_K = 0;        // kbar; then dk (staged)
constexpr uint32_t OFF_V = 16384;    // v; then dv (staged)
constexpr uint32_t OFF_DO = 32768;   // do
constexpr uint32_t OFF_KD = 49152;   // raw gates (fp32: KD + EG); then Kd
constexpr uint32_t OFF_EG = 65536;   // EG
constexpr uint32_t OFF_QG = 81920;   // QG               (from gla_bwd_q_kernel)
constexpr uint32_t OFF_DKC = 98304;  // local CCQ part of dkbar (from gla_bwd_q_kernel)
constexpr uint32_t OFF_GQ = 114688;  // qc * dqc         (from gla_bwd_q_kernel)
constexpr uint32_t OFF_DS = 131072;  // Diag(e^{Gc-Gmid}) dS_{r+1} } one image record of the state
constexpr uint32_t OFF_DC = 163840;  // DC_{r+1}                   } pass, one bulk copy
constexpr uint32_t OFF_P1 = 196608;  // P1
constexpr uint32_t OFF_SA = 204800;  // SA
constexpr uint32_t OFF_DG = 131072;  // fp32 dG [64][kDgStride], over the two images once they are dead
constexpr int kDgStride = 129;
constexpr uint32_t OFF_MISC = 212992;
constexpr uint32_t M_VEC = 0,        // [3][128] Dm_{r+1}, the gate carry's two column-half sums (state pass)
                   M_RK = 1536, M_GQ4 = 1792, M_RED = 3840, M_BAR = 4864, M_TMEM = 4896, M_ABORT = 4900;
constexpr uint32_t kMisc = 4992;
constexpr uint32_t kSmem = OFF_MISC + kMisc + 1024;
static_assert(OFF_DG + 64 * kDgStride * 4 <= OFF_P1, "dG scratch reaches P1");
static_assert(OFF_DC == OFF_DS + 32768, "a state image record lands as one block");
static_assert(kSmem <= 232448, "exceeds the 227 KB per-CTA limit");
enum { BAR_IN = 0, BAR_INB, BAR_R1, BAR_R2, kBars };
static_assert(M_BAR + 8 * kBars <= M_TMEM, "barriers reach the TMEM slot");
constexpr uint32_t TM_KC = 0, TM_T1 = 128, TM_SA = 192, TM_DK = 256, TM_DV = 384;
}  // namespace kv

__global__ void __launch_bounds__(kThreadsLoad, 1)
gla_bwd_kv_kernel(const __grid_constant__ CUtensorMap map_k, const __grid_constant__ CUtensorMap map_v,
                  const __grid_constant__ CUtensorMap map_do, const __grid_constant__ CUtensorMap map_g,
                  const __grid_constant__ CUtensorMap map_qg, const __grid_constant__ CUtensorMap map_dkc,
                  const __grid_constant__ CUtensorMap map_gq, const __grid_constant__ CUtensorMap map_dk,
                  const __grid_constant__ CUtensorMap map_dv, const BwdArgs a) {
    using namespace kv;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = smem_align1024(smem_raw);
    const uint32_t sb = smem_addr(sm);
    uint8_t *misc = sm + OFF_MISC;
    float *vec = reinterpret_cast<float *>(misc + M_VEC);
    float *rkv = reinterpret_cast<float *>(misc + M_RK);
    float *gq4 = reinterpret_cast<float *>(misc + M_GQ4);
    float *red = reinterpret_cast<float *>(misc + M_RED);  // [2 groups][128] partial sums
    float *dG = reinterpret_cast<float *>(sm + OFF_DG);
    uint64_t *bar = reinterpret_cast<uint64_t *>(misc + M_BAR);
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(misc + M_TMEM);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(misc + M_ABORT);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int qd = warp & 3, grp = warp >> 2;  // TMEM lane quadrant, warp group
    const int T = a.T, H = a.H, NC = (T + kC - 1) / kC;
    const int bh = blockIdx.x / NC, r = blockIdx.x % NC, b = bh / H, h = bh % H;
    const int c0 = r * kC;
    const bool gate_f32 = a.gate_dtype != 0;
    const uint32_t g_bytes = gate_f32 ? kC * kD * 4 : kC * kD * 2;
    int *status = a.status;

    // The load warp issues k and the gates (the row norms and the gate prefix) first, then,
    // once the compute threads are released, the rest.
    if (warp == kLoadWarp && lane == 0) {
        for (int i = 0; i < kBars; ++i) mbar_init(&bar[i], 1);
        *abort_flag = 0;
        fence_barrier_init();
        uint64_t *ba = &bar[BAR_IN], *bb = &bar[BAR_INB];
        mbar_arrive_expect_tx(ba, 16384 + g_bytes);
        mbar_arrive_expect_tx(bb, 5 * 16384 + 65536 + 1536);
        tma_load_4d(sm + OFF_K, &map_k, ba, 0, h, c0, b);
        tma_load_4d(sm + OFF_K + 8192, &map_k, ba, 64, h, c0, b);
        tma_load_4d(sm + OFF_KD, &map_g, ba, 0, h, c0, b);
    }
    if (warp == 0) tmem_alloc(tmem_slot, 512);
    __syncthreads();
    if (warp == kLoadWarp) {
        if (lane == 0) {
            uint64_t *bb = &bar[BAR_INB];
            tma_load_4d(sm + OFF_V, &map_v, bb, 0, h, c0, b);
            tma_load_4d(sm + OFF_V + 8192, &map_v, bb, 64, h, c0, b);
            tma_load_4d(sm + OFF_DO, &map_do, bb, 0, h, c0, b);
            tma_load_4d(sm + OFF_DO + 8192, &map_do, bb, 64, h, c0, b);
            tma_load_4d(sm + OFF_QG, &map_qg, bb, 0, h, c0, b);
            tma_load_4d(sm + OFF_QG + 8192, &map_qg, bb, 64, h, c0, b);
            tma_load_4d(sm + OFF_DKC, &map_dkc, bb, 0, h, c0, b);
            tma_load_4d(sm + OFF_DKC + 8192, &map_dkc, bb, 64, h, c0, b);
            tma_load_4d(sm + OFF_GQ, &map_gq, bb, 0, h, c0, b);
            tma_load_4d(sm + OFF_GQ + 8192, &map_gq, bb, 64, h, c0, b);
            bulk_load(sm + OFF_DS, a.state_img + static_cast<size_t>(blockIdx.x) * 65536, 65536, bb);
            bulk_load(misc + M_VEC, a.state_vec + static_cast<size_t>(blockIdx.x) * 3 * kD, 1536, bb);
            // the chunk one wave later finds its inputs in L2
            const int nx = blockIdx.x + a.wave;
            if (a.wave > 0 && nx < static_cast<int>(gridDim.x)) {
                const int bh2 = nx / NC, r2 = nx % NC, b2 = bh2 / H, h2 = bh2 % H, c2 = r2 * kC;
                const CUtensorMap *maps[6] = {&map_k, &map_v, &map_do, &map_qg, &map_dkc, &map_gq};
#pragma unroll
                for (int u = 0; u < 6; ++u) {
                    tma_prefetch_l2_4d(maps[u], 0, h2, c2, b2);
                    tma_prefetch_l2_4d(maps[u], 64, h2, c2, b2);
                }
                tma_prefetch_l2_4d(&map_g, 0, h2, c2, b2);
                bulk_prefetch_l2(a.state_img + static_cast<size_t>(nx) * 65536, 65536);
                bulk_prefetch_l2(a.state_vec + static_cast<size_t>(nx) * 3 * kD, 1536);
            }
        }
        return;
    }
    tc_fence_after();
    const uint32_t tbase = *tmem_slot;
    const uint32_t tq = tbase + (static_cast<uint32_t>(32 * qd) << 16);

    const int i = 16 * qd + (lane & 15), hf = lane >> 4;
    const uint64_t dK = make_desc(sb + OFF_K, 16, 1024);
    const uint64_t dV = make_desc(sb + OFF_V, 16, 1024);
    const uint64_t dDO = make_desc(sb + OFF_DO, 16, 1024), dDOm = make_desc(sb + OFF_DO, 8192, 1024);
    const uint64_t dKD = make_desc(sb + OFF_KD, 16, 1024);
    const uint64_t dQG = make_desc(sb + OFF_QG, 16, 1024), dQGm = make_desc(sb + OFF_QG, 8192, 1024);
    const uint64_t dDS = make_desc(sb + OFF_DS, 16, 1024), dDSm = make_desc(sb + OFF_DS, 16384, 1024);
    const uint64_t dDC = make_desc(sb + OFF_DC, 16, 1024), dDCm = make_desc(sb + OFF_DC, 16384, 1024);
    const uint64_t dP1m = make_desc(sb + OFF_P1, 8192, 1024);
    const uint64_t dSA = make_desc(sb + OFF_SA, 16, 1024);

    mbar_wait(&bar[BAR_IN], 0, abort_flag, status);
    prep_chunk(nullptr, sm + OFF_K, sm + OFF_KD, sm + OFF_EG, gate_f32, a.l2norm, nullptr, nullptr, nullptr,
               rkv, gq4, nullptr, nullptr, tid);
    mbar_wait(&bar[BAR_INB], 0, abort_flag, status);
    if (tid == 0 && !*abort_flag) {
        tc_fence_after();
        for (int k = 0; k < 8; ++k) {  // T1 = dO V^T, SA = Kd QG^T
            const uint64_t ko = (k >> 2) * 512 + (k & 3) * 2;
            mma_bf16(tbase + TM_T1, dDO + ko, dV + ko, ID_64x64_KK, k != 0);
        }
        for (int k = 0; k < 8; ++k) {
            const uint64_t ko = (k >> 2) * 512 + (k & 3) * 2;
            mma_bf16(tbase + TM_SA, dKD + ko, dQG + ko, ID_64x64_KK, k != 0);
        }
        for (int k = 0; k < 8; ++k) {  // dkw = V dSs^T, dv = Kd dSs, dkc inter = Kbar DC + Kbar DC^T
            const uint64_t ka = (k >> 2) * 512 + (k & 3) * 2, kb = (k >> 2) * 1024 + (k & 3) * 2;
            mma_bf16(tbase + TM_DK, dV + ka, dDS + kb, ID_64x128_KK, k != 0);
            mma_bf16(tbase + TM_DV, dKD + ka, dDSm + k * 128, ID_64x128_KM, k != 0);
            mma_bf16(tbase + TM_KC, dK + ka, dDCm + k * 128, ID_64x128_KM, k != 0);
            mma_bf16(tbase + TM_KC, dK + ka, dDC + kb, ID_64x128_KK, 1);
        }
        mma_commit(&bar[BAR_R1]);
    }
    mbar_wait(&bar[BAR_R1], 0, abort_flag, status);
    tc_fence_after();
    if (grp == 0) {
        float t1[32];
        tmem_ld16x2_32<32>(tq + TM_T1, t1);
        masked_row(sm + OFF_P1, i, hf, t1, 0.f);  // P1[t][j] = [j <= t] do_t . v_j
    } else {
        float sa[32];
        tmem_ld16x2_32<32>(tq + TM_SA, sa);
        // SA[j][t] = [t >= j] Kd_j . QG_t (row i is key j)
#pragma unroll
        for (int q4 = 0; q4 < 4; ++q4) {
            float w[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                const int t = 32 * hf + 8 * q4 + e;
                w[e] = (t >= i) ? sa[8 * q4 + e] : 0.f;
            }
            store_row_chunk(sm + OFF_SA, i, 4 * hf + q4, w);
        }
    }
    fence_proxy_async_smem();
    tc_fence_before();
    compute_sync();
    if (tid == 0 && !*abort_flag) {
        tc_fence_after();
        for (int k = 0; k < 4; ++k)  // dkw += P1^T QG, dv += SA dO
            mma_bf16(tbase + TM_DK, dP1m + k * 128, dQGm + k * 128, ID_64x128_MM, 1);
        for (int k = 0; k < 4; ++k)
            mma_bf16(tbase + TM_DV, dSA + k * 2, dDOm + k * 128, ID_64x128_KM, 1);
        mma_commit(&bar[BAR_R2]);
    }
    mbar_wait(&bar[BAR_R2], 0, abort_flag, status);
    tc_fence_after();
    {
        // dk: dkbar = e^{Gmid-G} dkw + (local CCQ part) + Kbar (DC + DC^T) + Dm_{r+1};
        // normalisation backward; dG
        const float rk = rkv[i];
        const float *Dh = vec + 64 * hf;  // Dm_{r+1}
        uint8_t *kt = sm + OFF_K + hf * 8192;
        const uint8_t *egt = sm + OFF_EG + hf * 8192;
        const uint8_t *dkct = sm + OFF_DKC + hf * 8192;
        const uint8_t *gqt = sm + OFF_GQ + hf * 8192;
        float *dgrow = dG + i * kDgStride + 64 * hf;
        const int h2 = grp;  // this group's 32-column slice of each 128-column product
        uint64_t dkb[16];    // fp32 pairs over consecutive columns
        float dot;
        {
            float x[32], y[32];
            tmem_ld16x2_32<64>(tq + TM_DK + 32 * h2, x);
            tmem_ld16x2_32<64>(tq + TM_KC + 32 * h2, y);
            uint64_t dot2 = 0;
#pragma unroll
            for (int q4 = 0; q4 < 4; ++q4) {
                const int cc = 4 * h2 + q4;
                const uint32_t off = t64_chunk(i, cc);
                const uint4 er = *reinterpret_cast<const uint4 *>(egt + off);
                const uint4 kr = *reinterpret_cast<const uint4 *>(kt + off);
                const uint4 cr = *reinterpret_cast<const uint4 *>(dkct + off);
                const uint4 gr = *reinterpret_cast<const uint4 *>(gqt + off);
                const ulonglong2 dlo = *reinterpret_cast<const ulonglong2 *>(Dh + 8 * cc);
                const ulonglong2 dhi = *reinterpret_cast<const ulonglong2 *>(Dh + 8 * cc + 4);
                const uint32_t ew[4] = {er.x, er.y, er.z, er.w}, kw[4] = {kr.x, kr.y, kr.z, kr.w};
                const uint32_t cw[4] = {cr.x, cr.y, cr.z, cr.w}, gw[4] = {gr.x, gr.y, gr.z, gr.w};
                const uint64_t dm[4] = {dlo.x, dlo.y, dhi.x, dhi.y};
#pragma unroll
                for (int w = 0; w < 4; ++w) {
                    const int e = 8 * q4 + 2 * w;
                    const float2 eg = f2_split(f2_from_bf16x2(ew[w]));
                    const uint64_t kb2 = f2_from_bf16x2(kw[w]);
                    const uint64_t dkw = f2_mul(f2_make(x[e], x[e + 1]), f2_make(__frcp_rn(eg.x), __frcp_rn(eg.y)));
                    const uint64_t v = f2_add(f2_add(f2_add(dkw, f2_from_bf16x2(cw[w])), f2_make(y[e], y[e + 1])), dm[w]);
                    dkb[4 * q4 + w] = v;
                    dot2 = f2_fma(kb2, v, dot2);
                    const float2 g = f2_split(f2_fma(f2_mul(kb2, f2_make(-1.f, -1.f)), dkw, f2_from_bf16x2(gw[w])));
                    dgrow[8 * cc + 2 * w] = g.x;
                    dgrow[8 * cc + 2 * w + 1] = g.y;
                }
            }
            const float2 dv = f2_split(dot2);
            dot = dv.x + dv.y;
        }
        dot += __shfl_xor_sync(0xffffffffu, dot, 16);
        if (hf == 0) red[grp * 128 + i] = dot;
        uint8_t *vt = sm + OFF_V + hf * 8192;
        {
            float x[32];
            tmem_ld16x2_32<64>(tq + TM_DV + 32 * h2, x);
#pragma unroll
            for (int q4 = 0; q4 < 4; ++q4) store_row_chunk(vt, i, 4 * h2 + q4, x + 8 * q4);
        }
        compute_sync();
        dot = red[i] + red[128 + i];
        const uint64_t ndot = f2_make(-dot, -dot), rk2 = f2_make(rk, rk);
#pragma unroll
        for (int q4 = 0; q4 < 4; ++q4) {
            const int cc = 4 * h2 + q4;
            const uint4 kr = *reinterpret_cast<const uint4 *>(kt + t64_chunk(i, cc));
            const uint32_t kw[4] = {kr.x, kr.y, kr.z, kr.w};
            uint32_t ow[4];
#pragma unroll
            for (int w = 0; w < 4; ++w) {
                const uint64_t v = dkb[4 * q4 + w];
                ow[w] = bf16x2_from_f2(a.l2norm ? f2_mul(rk2, f2_fma(ndot, f2_from_bf16x2(kw[w]), v)) : v);
            }
            *reinterpret_cast<uint4 *>(kt + t64_chunk(i, cc)) = make_uint4(ow[0], ow[1], ow[2], ow[3]);
        }
    }
    fence_proxy_async_smem();
    tc_fence_before();
    compute_sync();
    if (tid == 0 && !*abort_flag) {
        tma_store_4d(&map_dk, sm + OFF_K, 0, h, c0, b);
        tma_store_4d(&map_dk, sm + OFF_K + 8192, 64, h, c0, b);
        tma_store_4d(&map_dv, sm + OFF_V, 0, h, c0, b);
        tma_store_4d(&map_dv, sm + OFF_V + 8192, 64, h, c0, b);
        tma_store_commit();
    }
    {
        // dgk_t = sum_{s >= t in the chunk} dG_s + rowsum(dS_{r+1} * S_{r+1}): column
        // d, tokens in reverse, in two 32-row halves (half hh = rows [32 hh, 32 hh + 32))
        const int d = tid & 127, hh = tid >> 7;
        float x[32], tot = 0.f;
#pragma unroll
        for (int u = 0; u < 32; ++u) {
            x[u] = dG[(32 * hh + u) * kDgStride + d];
            tot += x[u];
        }
        red[hh * 128 + d] = tot;
        compute_sync();
        float acc = vec[kD + d] + vec[2 * kD + d] + (hh == 0 ? red[128 + d] : 0.f);
        const int nvalid = min(kC, T - c0);
#pragma unroll
        for (int u = 31; u >= 0; --u) {
            acc += x[u];
            const int t = 32 * hh + u;
            if (t < nvalid) {
                const size_t o = ((static_cast<size_t>(b) * T + c0 + t) * H + h) * kD + d;
                if (gate_f32) static_cast<float *>(a.dgk)[o] = acc;
                else static_cast<__nv_bfloat16 *>(a.dgk)[o] = __float2bfloat16_rn(acc);
            }
        }
    }
    if (tid == 0) tma_store_wait_read();  // shared memory outlives the stores' reads
    tc_fence_before();
    compute_sync();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tbase, 512);
    }
}

}  // namespace

cudaError_t launch_gla_bwd(const BwdArgs &a, const BwdMaps &m, cudaStream_t s) {
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(gla_bwd_q_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(qk::kSmem));
        if (e != cudaSuccess) return e;
        e = cudaFuncSetAttribute(gla_bwd_state_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 static_cast<int>(st::kSmem));
        if (e != cudaSuccess) return e;
        e = cudaFuncSetAttribute(gla_bwd_kv_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 static_cast<int>(kv::kSmem));
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    const int nc = (a.T + kC - 1) / kC;
    const int chunks = a.B * a.H * nc;
    gla_bwd_q_kernel<<<chunks, kThreadsLoad, qk::kSmem, s>>>(m.q, m.k, m.v, m.dO, m.g, m.dq, m.qg, m.dkc, m.gq,
                                                          m.dzr, a);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    gla_bwd_state_kernel<<<a.B * a.H * 2, kThreads, st::kSmem, s>>>(m.qg, m.dO, m.dzr, m.q, a);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    gla_bwd_kv_kernel<<<chunks, kThreadsLoad, kv::kSmem, s>>>(m.k, m.v, m.dO, m.g, m.qg, m.dkc, m.gq, m.dk, m.dv, a);
    return cudaGetLastError();
}

}  // namespace ccq
