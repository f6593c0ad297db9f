// ccq_gdn_segment.cu -- sequence-segment parallelism for long CCQ-Gated-DeltaNet sequences.
//
// With few (batch, head) sequences, each sequence is cut into `nseg` segments of whole
// chunks, as for CCQ-GLA (ccq_gla_segment.cu).  The gated delta state is affine in the
// state entering a chunk: with H = S^T [Dk][Dv], Tb = Tt diag(beta) and the chunk factors
// of ccq_gdn_chunk.cu,
//   H_{r+1} = A_r H_r + B_r,   A_r = e^{gC} I - Kd^T Tb Ke,   Ke = Diag(e^{gc}) Kbar,
//   Kd = Diag(e^{gC - gc}) Kbar,   B_r = Kd^T Tb V,
// every factor an exponential of a non-positive argument, so a segment maps its entering
// state H to P H + Q, with P the product of its A_r and Q the state it reaches from zero.
// The covariance C and key sum m are plain sums.  Three launches replace the long walk:
//   1. gdn_segment_state_kernel: per (sequence, segment), from a zero state, Q, P, dC, dm.
//      P is updated exactly like the state without its V term, so one set of products
//      serves both: with Z = [Q | P] (Dk x 2Dv),
//        Y^T = Z^T Ke^T,  R^T = [V^T - Y_Q^T | -Y_P^T],  U^T = R^T Tb^T,
//        [Q | P] = e^{gC} [Q | P] + Kd^T U
//      (M = 128 products over the transposed operands, so everything fits 512 TMEM columns).
//   2. gdn_segment_combine_kernel: per (sequence, 16 state columns), H_{s+1} = P_s H_s + Q_s,
//      C and m by prefix sums, in fp32; each slot then holds its segment's entering states.
//   3. gdn_chunk_kernel with one CTA per (sequence, segment) (ccq_gdn_chunk.cu).
// Workspace per (sequence, segment): kGdnSegFloats floats -- S (Q, then the entering H),
// P, C (dC, then the entering C), m (dm, then the entering m), and 128 spare.
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
constexpr int kThreads = 256;
constexpr float kLog2e = 1.4426950408889634f;
constexpr int kSS = kD * kD;

// shared memory: two slots of {k 16K, v 16K, Tb 8K}, then Ke, Kd, Z, R/U and scratch
constexpr uint32_t SL_BYTES = 40960;
constexpr uint32_t SL_K = 0, SL_V = 16384, SL_TB = 32768;
constexpr uint32_t OFF_KE = 81920;    // 16K  e^{gc} kbar (K-major B of Y^T)
constexpr uint32_t OFF_KD = 98304;    // 16K  e^{gC - gc} kbar (MN-major A of the state update)
constexpr uint32_t OFF_Z = 114688;    // 64K  bf16 [Q | P], [128 rows][256 cols] as four T64 tiles
constexpr uint32_t OFF_RU = 180224;   // 32K  bf16 R^T, then U^T: [256 rows][64 cols] as two T64 tiles
constexpr uint32_t OFF_MISC = 212992;
constexpr uint32_t M_GC = 0;      // [64] cumulative log decay
constexpr uint32_t M_EP = 256;    // [64] e^{gc}
constexpr uint32_t M_EN = 512;    // [64] e^{gC - gc}
constexpr uint32_t M_RK = 768;    // [64] 1/|k|
constexpr uint32_t M_DMP = 1024;  // [4][128] key-sum quarters
constexpr uint32_t M_BAR = 3072;  // in[2], mma
constexpr uint32_t M_TMEM = 3104, M_ABORT = 3108;
constexpr uint32_t kSmem = OFF_MISC + 4096 + 1024;
static_assert(kSmem <= 232448, "smem");

// TMEM columns
constexpr uint32_t TM_X = 0, TM_PT = 128, TM_DC = 256, TM_YU = 384;  // Q, P, dC, Y^T / U^T

constexpr uint32_t ID_Y = make_idesc(128, 64, 1, 0);     // Y^T = Z^T Ke^T
constexpr uint32_t ID_U = make_idesc(128, 64, 0, 0);     // U^T = R^T Tb^T
constexpr uint32_t ID_ST = make_idesc(128, 256, 1, 0);   // [Q | P] += Kd^T U
constexpr uint32_t ID_DC = make_idesc(128, 128, 1, 1);   // dC += Kbar^T Kbar

__device__ __forceinline__ void store_row_chunk(uint8_t *tile, int row, int chunk, const float *w) {
    uint4 u;
    u.x = pack_bf16(w[0], w[1]);
    u.y = pack_bf16(w[2], w[3]);
    u.z = pack_bf16(w[4], w[5]);
    u.w = pack_bf16(w[6], w[7]);
    *reinterpret_cast<uint4 *>(tile + t64_chunk(row, chunk)) = u;
}

__global__ void __launch_bounds__(kThreads, 1)
gdn_segment_state_kernel(const __grid_constant__ CUtensorMap map_k, const __grid_constant__ CUtensorMap map_v,
                         const __grid_constant__ CUtensorMap map_tb, const ChunkArgs a) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = smem_align1024(smem_raw);
    const uint32_t sb = smem_addr(sm);
    uint8_t *misc = sm + OFF_MISC;
    float *gc = reinterpret_cast<float *>(misc + M_GC);
    float *epv = reinterpret_cast<float *>(misc + M_EP);
    float *env = reinterpret_cast<float *>(misc + M_EN);
    float *rkv = reinterpret_cast<float *>(misc + M_RK);
    float *dmp = reinterpret_cast<float *>(misc + M_DMP);
    uint64_t *bar = reinterpret_cast<uint64_t *>(misc + M_BAR);
    uint32_t *tslot = reinterpret_cast<uint32_t *>(misc + M_TMEM);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(misc + M_ABORT);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int seq = blockIdx.x / a.nseg, seg = blockIdx.x % a.nseg;
    const int b = seq / a.H, h = seq % a.H;
    const int T = a.T, H = a.H;
    const int NCt = (T + kC - 1) / kC;
    const int cb = seg * a.seg_chunks;
    const int n = min(NCt, cb + a.seg_chunks) - cb;  // chunks of this segment (>= 1)
    const int wrow0 = seq * NCt * kC;                 // first Tb row of this sequence
    int *status = a.status;

    if (tid == 0) {
        for (int i = 0; i < 3; ++i) mbar_init(&bar[i], 1);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 0) tmem_alloc(tslot, 512);
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *tslot;
    const uint32_t tq = tbase + (static_cast<uint32_t>(32 * (warp & 3)) << 16);
    const int hz = warp >> 2;                  // column half of the state pair / of R^T, U^T
    const int row = 32 * (warp & 3) + lane;    // TMEM lane: state row a, or R^T / U^T row d

    auto issue_in = [&](int r) {  // k, v, Tb of local chunk r into slot r & 1
        const int s = r & 1, tg = (cb + r) * kC;
        uint8_t *base = sm + s * SL_BYTES;
        mbar_arrive_expect_tx(&bar[s], 5 * 8192);
        tma_load_4d(base + SL_K, &map_k, &bar[s], 0, h, tg, b);
        tma_load_4d(base + SL_K + 8192, &map_k, &bar[s], 64, h, tg, b);
        tma_load_4d(base + SL_V, &map_v, &bar[s], 0, h, tg, b);
        tma_load_4d(base + SL_V + 8192, &map_v, &bar[s], 64, h, tg, b);
        tma_load_2d(base + SL_TB, &map_tb, &bar[s], 0, wrow0 + (cb + r) * kC);
    };
    if (tid == 0) {
        tma_prefetch_desc(&map_k);
        tma_prefetch_desc(&map_v);
        tma_prefetch_desc(&map_tb);
        issue_in(0);
    }
    // Q = 0, P = I, dC = 0 (this thread: row `row`, the 128 columns of half hz)
    {
        float x[32];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
#pragma unroll
            for (int e = 0; e < 32; ++e) x[e] = (hz == 1 && 32 * c + e == row) ? 1.f : 0.f;
            tmem_st32(tq + (hz ? TM_PT : TM_X) + 32 * c, x);
#pragma unroll
            for (int e = 0; e < 32; ++e) x[e] = 0.f;
            if (hz == 0) tmem_st32(tq + TM_DC + 32 * c, x);
        }
        tmem_wait_st();
    }
    float g_reg = 0.f;
    if (tid < 64) {
        const int t = cb * kC + tid;
        g_reg = t < T ? a.g[(static_cast<size_t>(b) * T + t) * H + h] : 0.f;
    }
    float dm_acc = 0.f;      // key sum of dim tid (tid < 128)
    tc_fence_before();
    __syncthreads();

    for (int r = 0; r < n; ++r) {
        const int s = r & 1;
        uint8_t *slot = sm + s * SL_BYTES;
        // the previous chunk's state update has run: Ke, Kd, the other slot and Z are free
        if (r > 0) mbar_wait(&bar[2], (3 * (r - 1) + 2) & 1, abort_flag, status);
        if (tid == 0 && r + 1 < n && !*abort_flag) issue_in(r + 1);
        // ---- prep: cumulative decay, factors, norms, kbar, Ke, Kd, key sum
        if (tid < 64) gc[tid] = g_reg;
        if (tid < 64) {
            const int t = (cb + r + 1) * kC + tid;
            g_reg = t < T ? a.g[(static_cast<size_t>(b) * T + t) * H + h] : 0.f;
        }
        mbar_wait(&bar[s], (r >> 1) & 1, abort_flag, status);
        __syncthreads();
        if (warp == 0) {
            const float x0 = gc[2 * lane], x1 = gc[2 * lane + 1];
            float pv = x0 + x1;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const float y = __shfl_up_sync(0xffffffffu, pv, o);
                if (lane >= o) pv += y;
            }
            gc[2 * lane] = pv - x1;
            gc[2 * lane + 1] = pv;
        }
        // row norms: thread = (row j, column quarter)
        const int j = tid >> 2, qq = tid & 3;
        uint8_t *kq = slot + SL_K + (qq >> 1) * 8192;
        uint4 kv[4];
#pragma unroll
        for (int c = 0; c < 4; ++c) kv[c] = *reinterpret_cast<const uint4 *>(kq + t64_chunk(j, 4 * (qq & 1) + c));
        {
            uint64_t s0 = 0, s1 = 0;
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                const uint64_t p0 = f2_from_bf16x2(kv[c].x), p1 = f2_from_bf16x2(kv[c].y),
                               p2 = f2_from_bf16x2(kv[c].z), p3 = f2_from_bf16x2(kv[c].w);
                s0 = f2_fma(p0, p0, s0); s1 = f2_fma(p1, p1, s1);
                s0 = f2_fma(p2, p2, s0); s1 = f2_fma(p3, p3, s1);
            }
            const float2 sv = f2_split(f2_add(s0, s1));
            float ss = sv.x + sv.y;
            ss += __shfl_xor_sync(0xffffffffu, ss, 1);
            ss += __shfl_xor_sync(0xffffffffu, ss, 2);
            if (qq == 0) rkv[j] = a.l2norm ? rsqrtf(fmaxf(ss, 1e-12f)) : 1.f;
        }
        __syncthreads();  // gc, rk visible
        const float gC = gc[63];
        if (tid < 64) {
            epv[tid] = fast_exp2(gc[tid] * kLog2e);         // e^{gc} <= 1
            env[tid] = fast_exp2((gC - gc[tid]) * kLog2e);  // e^{gC - gc} <= 1
        }
        __syncthreads();  // factors visible
        {
            const float rk = rkv[j];
            const uint64_t rk2 = f2_make(rk, rk), ep2 = f2_make(epv[j], epv[j]), en2 = f2_make(env[j], env[j]);
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                const uint32_t w[4] = {kv[c].x, kv[c].y, kv[c].z, kv[c].w};
                uint32_t ob[4], oe[4], od[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const uint64_t kb = f2_mul(f2_from_bf16x2(w[u]), rk2);
                    ob[u] = bf16x2_from_f2(kb);
                    oe[u] = bf16x2_from_f2(f2_mul(kb, ep2));
                    od[u] = bf16x2_from_f2(f2_mul(kb, en2));
                }
                const uint32_t off = (qq >> 1) * 8192 + t64_chunk(j, 4 * (qq & 1) + c);
                *reinterpret_cast<uint4 *>(slot + SL_K + off) = make_uint4(ob[0], ob[1], ob[2], ob[3]);
                *reinterpret_cast<uint4 *>(sm + OFF_KE + off) = make_uint4(oe[0], oe[1], oe[2], oe[3]);
                *reinterpret_cast<uint4 *>(sm + OFF_KD + off) = make_uint4(od[0], od[1], od[2], od[3]);
            }
        }
        fence_proxy_async_smem();
        __syncthreads();  // kbar, Ke, Kd written
        // key sum: thread = (dim pair, token quarter)
        {
            const int p = tid & 63, tq4 = tid >> 6, d0 = 2 * p;
            const uint8_t *kt = slot + SL_K + (d0 >> 6) * 8192;
            uint64_t acc = 0;
#pragma unroll
            for (int u = 0; u < 16; ++u)
                acc = f2_add(acc, f2_from_bf16x2(*reinterpret_cast<const uint32_t *>(kt + t64_offset(16 * tq4 + u, d0 & 63))));
            const float2 sv = f2_split(acc);
            dmp[tq4 * kD + d0] = sv.x;
            dmp[tq4 * kD + d0 + 1] = sv.y;
        }
        // dC += Kbar^T Kbar
        if (tid == 0 && !*abort_flag) {
            tc_fence_after();
            const uint64_t dKm = make_desc(sb + s * SL_BYTES + SL_K, 8192, 1024);
            for (int k = 0; k < 4; ++k) mma_bf16(tbase + TM_DC, dKm + k * 128, dKm + k * 128, ID_DC, 1);
        }
        // ---- Z = [Q | P] as bf16; the TMEM copies scaled by e^{gC}, onto which the state
        // update of this chunk accumulates
        tc_fence_after();
        {
            const float hs = fast_exp2(gC * kLog2e);
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                float x[32];
                tmem_ld32(tq + (hz ? TM_PT : TM_X) + 32 * c, x);
                uint8_t *tile = sm + OFF_Z + (2 * hz + (c >> 1)) * 16384;
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) store_row_chunk(tile, row, 4 * (c & 1) + q4, x + 8 * q4);
#pragma unroll
                for (int e = 0; e < 32; ++e) x[e] *= hs;
                tmem_st32(tq + (hz ? TM_PT : TM_X) + 32 * c, x);
            }
            tmem_wait_st();
        }
        __syncthreads();
        if (tid < kD) dm_acc += (dmp[tid] + dmp[kD + tid]) + (dmp[2 * kD + tid] + dmp[3 * kD + tid]);
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();  // Z written
        // ---- Y^T = Z^T Ke^T (two M = 128 halves, N = 64 tokens, K = 128)
        if (tid == 0 && !*abort_flag) {
            tc_fence_after();
            const uint64_t dKe = make_desc(sb + OFF_KE, 16, 1024);
            for (int half = 0; half < 2; ++half) {
                const uint64_t dZ = make_desc(sb + OFF_Z + half * 32768, 16384, 1024);
                for (int k = 0; k < 8; ++k)
                    mma_bf16(tbase + TM_YU + 64 * half, dZ + k * 128, dKe + (k >> 2) * 512 + (k & 3) * 2, ID_Y,
                             k != 0);
            }
            mma_commit(&bar[2]);
        }
        mbar_wait(&bar[2], (3 * r) & 1, abort_flag, status);
        tc_fence_after();
        // ---- R^T: [V^T - Y_Q^T | -Y_P^T], this thread row d = `row` of half hz
        {
            const uint8_t *vt = slot + SL_V + (row >> 6) * 8192;
#pragma unroll
            for (int c = 0; c < 2; ++c) {
                float y[32];
                tmem_ld32(tq + TM_YU + 64 * hz + 32 * c, y);
                if (hz == 0) {
#pragma unroll
                    for (int e = 0; e < 32; ++e) {
                        const float vv = __bfloat162float(
                            *reinterpret_cast<const __nv_bfloat16 *>(vt + t64_offset(32 * c + e, row & 63)));
                        y[e] = vv - y[e];
                    }
                } else {
#pragma unroll
                    for (int e = 0; e < 32; ++e) y[e] = -y[e];
                }
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) store_row_chunk(sm + OFF_RU + hz * 16384, row, 4 * c + q4, y + 8 * q4);
            }
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        // ---- U^T = R^T Tb^T (two halves, N = 64 tokens, K = 64 tokens)
        if (tid == 0 && !*abort_flag) {
            tc_fence_after();
            const uint64_t dTb = make_desc(sb + s * SL_BYTES + SL_TB, 16, 1024);
            for (int half = 0; half < 2; ++half) {
                const uint64_t dR = make_desc(sb + OFF_RU + half * 16384, 16, 1024);
                for (int k = 0; k < 4; ++k) mma_bf16(tbase + TM_YU + 64 * half, dR + k * 2, dTb + k * 2, ID_U, k != 0);
            }
            mma_commit(&bar[2]);
        }
        mbar_wait(&bar[2], (3 * r + 1) & 1, abort_flag, status);
        tc_fence_after();
        {
#pragma unroll
            for (int c = 0; c < 2; ++c) {
                float y[32];
                tmem_ld32(tq + TM_YU + 64 * hz + 32 * c, y);
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) store_row_chunk(sm + OFF_RU + hz * 16384, row, 4 * c + q4, y + 8 * q4);
            }
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        // ---- [Q | P] += Kd^T U (N = 256: U^T rows 0..255 across both tiles)
        if (tid == 0 && !*abort_flag) {
            tc_fence_after();
            const uint64_t dKDm = make_desc(sb + OFF_KD, 8192, 1024);
            const uint64_t dU = make_desc(sb + OFF_RU, 16, 1024);
            for (int k = 0; k < 4; ++k) mma_bf16(tbase + TM_X, dKDm + k * 128, dU + k * 2, ID_ST, 1);
            mma_commit(&bar[2]);
        }
    }
    // ---- outputs: Q, P, dC, dm
    if (n > 0) mbar_wait(&bar[2], (3 * (n - 1) + 2) & 1, abort_flag, status);
    tc_fence_after();
    float *out = a.seg_ws + static_cast<size_t>(blockIdx.x) * kGdnSegFloats;
    {
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            float x[32];
            tmem_ld32(tq + (hz ? TM_PT : TM_X) + 32 * c, x);
            float4 *dst = reinterpret_cast<float4 *>(out + hz * kSS + row * kD + 32 * c);
#pragma unroll
            for (int e = 0; e < 8; ++e) dst[e] = make_float4(x[4 * e], x[4 * e + 1], x[4 * e + 2], x[4 * e + 3]);
            if (hz == 0) {
                tmem_ld32(tq + TM_DC + 32 * c, x);
                float4 *dc = reinterpret_cast<float4 *>(out + 2 * kSS + row * kD + 32 * c);
#pragma unroll
                for (int e = 0; e < 8; ++e) dc[e] = make_float4(x[4 * e], x[4 * e + 1], x[4 * e + 2], x[4 * e + 3]);
            }
        }
    }
    if (tid < kD) out[3 * kSS + tid] = dm_acc;
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tbase, 512);
    }
}

// Per (sequence, block of 16 state columns): walks the segments, replacing each slot's
// S (Q), C (dC) and m (dm) with the states entering that segment:
//   H_{s+1} = P_s H_s + Q_s,  C_{s+1} = C_s + dC_s,  m_{s+1} = m_s + dm_s.
// P_s is staged in shared memory with coalesced loads into rows padded to kPS floats (the
// row-per-lane reads of the product then spread over the banks); the loads of segment s+1
// (P, Q, dC) are in flight while segment s computes.
constexpr int kCols = 16;
constexpr int kPS = kD + 4;
constexpr int kCombineSmem = (kD * kPS + kD * kCols) * 4;

__global__ void __launch_bounds__(256)
gdn_segment_combine_kernel(const ChunkArgs a) {
    extern __shared__ float csm[];
    float *Ps = csm;               // [128][kPS]
    float *hcur = csm + kD * kPS;  // [128][16]
    const int nblk = kD / kCols;
    const int seq = blockIdx.x / nblk, cblk = blockIdx.x % nblk;
    const size_t sq = static_cast<size_t>(seq);
    const int tid = threadIdx.x;
    const int arow = tid >> 1, cl = 8 * (tid & 1), c0 = kCols * cblk + cl;  // row arow, 8 columns
    float hreg[8], creg[8];
    {
        const float4 *h4 = a.S0 ? reinterpret_cast<const float4 *>(a.S0 + sq * kSS + arow * kD + c0) : nullptr;
        const float4 *c4 = a.C0 ? reinterpret_cast<const float4 *>(a.C0 + sq * kSS + arow * kD + c0) : nullptr;
#pragma unroll
        for (int u = 0; u < 2; ++u) {
            const float4 hv = h4 ? h4[u] : make_float4(0.f, 0.f, 0.f, 0.f);
            const float4 cv = c4 ? c4[u] : make_float4(0.f, 0.f, 0.f, 0.f);
            hreg[4 * u] = hv.x; hreg[4 * u + 1] = hv.y; hreg[4 * u + 2] = hv.z; hreg[4 * u + 3] = hv.w;
            creg[4 * u] = cv.x; creg[4 * u + 1] = cv.y; creg[4 * u + 2] = cv.z; creg[4 * u + 3] = cv.w;
        }
    }
    float mreg = (cblk == 0 && tid < kD) ? (a.m0 ? a.m0[sq * kD + tid] : 0.f) : 0.f;
    // segment s+1's operands in registers while segment s computes
    float4 pv[16], qv[2], dv[2];
    auto load_next = [&](int s) {
        const float *slot = a.seg_ws + (sq * a.nseg + s) * kGdnSegFloats;
        const float4 *src = reinterpret_cast<const float4 *>(slot + kSS);
#pragma unroll
        for (int u = 0; u < 16; ++u) pv[u] = src[u * 256 + tid];
        const float4 *q4 = reinterpret_cast<const float4 *>(slot + arow * kD + c0);
        const float4 *d4 = reinterpret_cast<const float4 *>(slot + 2 * kSS + arow * kD + c0);
        qv[0] = q4[0]; qv[1] = q4[1];
        dv[0] = d4[0]; dv[1] = d4[1];
    };
    if (a.nseg > 0) load_next(0);
    for (int s = 0; s < a.nseg; ++s) {
        float *slot = a.seg_ws + (sq * a.nseg + s) * kGdnSegFloats;
        // stage P_s (element e = 4 (256 u + tid): row e / 128, column e % 128) and H_s
#pragma unroll
        for (int u = 0; u < 16; ++u) {
            const int e = 4 * (u * 256 + tid);
            *reinterpret_cast<float4 *>(Ps + (e >> 7) * kPS + (e & 127)) = pv[u];
        }
#pragma unroll
        for (int u = 0; u < 2; ++u)
            *reinterpret_cast<float4 *>(hcur + arow * kCols + cl + 4 * u) =
                make_float4(hreg[4 * u], hreg[4 * u + 1], hreg[4 * u + 2], hreg[4 * u + 3]);
        float acc[8] = {qv[0].x, qv[0].y, qv[0].z, qv[0].w, qv[1].x, qv[1].y, qv[1].z, qv[1].w};  // Q_s
        const float dcv[8] = {dv[0].x, dv[0].y, dv[0].z, dv[0].w, dv[1].x, dv[1].y, dv[1].z, dv[1].w};
        __syncthreads();
        if (s + 1 < a.nseg) load_next(s + 1);
        const float *P = Ps + arow * kPS;
#pragma unroll 4
        for (int bb = 0; bb < kD; bb += 4) {
            const float4 p4 = *reinterpret_cast<const float4 *>(P + bb);
            const float pw[4] = {p4.x, p4.y, p4.z, p4.w};
#pragma unroll
            for (int t = 0; t < 4; ++t) {
                const float4 h0 = *reinterpret_cast<const float4 *>(hcur + (bb + t) * kCols + cl);
                const float4 h1 = *reinterpret_cast<const float4 *>(hcur + (bb + t) * kCols + cl + 4);
                const float hv[8] = {h0.x, h0.y, h0.z, h0.w, h1.x, h1.y, h1.z, h1.w};
#pragma unroll
                for (int u = 0; u < 8; ++u) acc[u] = fmaf(pw[t], hv[u], acc[u]);
            }
        }
        // this slot now holds the states entering segment s
#pragma unroll
        for (int u = 0; u < 2; ++u) {
            *reinterpret_cast<float4 *>(slot + arow * kD + c0 + 4 * u) =
                make_float4(hreg[4 * u], hreg[4 * u + 1], hreg[4 * u + 2], hreg[4 * u + 3]);
            *reinterpret_cast<float4 *>(slot + 2 * kSS + arow * kD + c0 + 4 * u) =
                make_float4(creg[4 * u], creg[4 * u + 1], creg[4 * u + 2], creg[4 * u + 3]);
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            hreg[u] = acc[u];
            creg[u] += dcv[u];
        }
        if (cblk == 0 && tid < kD) {
            const float dm = slot[3 * kSS + tid];
            slot[3 * kSS + tid] = mreg;
            mreg += dm;
        }
        __syncthreads();  // Ps and hcur are rewritten by the next segment
    }
}

}  // namespace

cudaError_t launch_gdn_segments(const ChunkArgs &a, const GdnMaps &m, cudaStream_t s) {
    cudaError_t e = launch_gdn_wy(a, m, s);
    if (e != cudaSuccess) return e;
    static bool attr_set = false;
    if (!attr_set) {
        e = cudaFuncSetAttribute(gdn_segment_state_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 static_cast<int>(kSmem));
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    gdn_segment_state_kernel<<<a.B * a.H * a.nseg, kThreads, kSmem, s>>>(m.k, m.v, m.tb, a);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    static bool attr_combine = false;
    if (!attr_combine) {
        e = cudaFuncSetAttribute(gdn_segment_combine_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 kCombineSmem);
        if (e != cudaSuccess) return e;
        attr_combine = true;
    }
    gdn_segment_combine_kernel<<<a.B * a.H * (kD / kCols), 256, kCombineSmem, s>>>(a);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    return launch_gdn_chunk_only(a, m, s);
}

}  // namespace ccq
