// ccq_gdn_chunk.cu -- chunkwise CCQ-Gated-DeltaNet forward on sm_103a tensor cores.
//
// The gated delta rule S_t = alpha_t S_{t-1}(I - beta_t kbar_t kbar_t^T) + beta_t v_t kbar_t^T
// (the Gated DeltaNet write, Sec. 2.2) is kept as H = S^T [Dk][Dv].  Inside a 64-token
// chunk with start state H0, gc_i the in-chunk cumulative log-decay and gC its value at the
// chunk's end, unrolling the recurrence gives (chunkwise form):
//   A_ij = beta_i e^{gc_i - gc_j} kbar_i . kbar_j   (j < i),   Tt = (I + A)^{-1}
//   U    = Tb (V - Diag(e^{gc}) Kbar H0),   Tb = Tt diag(beta)
//   o_i  = scale [ e^{gc_i} q_clean_i H0 + sum_{j<=i} e^{gc_i - gc_j}(q_clean_i . kbar_j) U_j ]
//   H_C  = e^{gC} H0 + sum_j e^{gC - gc_j} kbar_j U_j^T
// Every decay factor is e^{x} with x <= 0 (gc_i, gC - gc_j and, per score entry, gc_i - gc_j
// for j <= i), so no factor overflows however strong the forgetting, and a decay that
// underflows contributes an exact zero.  Tb depends only on the chunk's own keys, gates and
// betas, so it is computed for every chunk in parallel by gdn_wy_kernel (64 x 64 bf16 per
// chunk, into a caller workspace); gdn_chunk_kernel then walks the chunks of each (batch,
// head) sequentially with the same warp-specialised structure as the GLA kernel and the same
// CCQ read (App. B):
//
//   G2  Sc  = Q Kbar^T           D2  KH = Kbar H0
//   (epilogue: W' of the CCQ mean fold;  R = V - Diag(e^{gc}) KH -> bf16 R tile)
//   G1  P   = Q S^K              DU  U = Tb R            G3  P += W' Kbar
//   (epilogue: U -> bf16 U tile; q_clean into the Q tile)
//   D6  X  += Kd^T U             G8  S^K += Kbar^T Kbar      (Kd = kbar e^{gC - gc})
//   D4  QK  = Qc Kbar^T          D3  O1^T = H0^T Qc^T
//   (epilogue: Pm_ij = [j<=i] QK_ij e^{gc_i - gc_j})
//   D5  O2^T = U^T Pm^T
//   (epilogue: o_i = scale (e^{gc_i} O1_i + O2_i), TMA store)
// The two output products are transposed (M = 128 = Dv, N = 64 rows) into their own TMEM
// accumulators, so the row factor e^{gc_i} of the inter-chunk read is applied in the output
// epilogue.  X = H stays in TMEM; the snapshot that copies H0 to bf16 for D2 and D3 also
// scales the TMEM copy by e^{gC}, so that D6 accumulates H_C onto it.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "ccq_internal.h"
#include "sm100_ptx.cuh"

namespace ccq {

namespace {

__device__ __forceinline__ void st_shared_b32(uint32_t addr, uint32_t v) {
    asm volatile("st.shared.b32 [%0], %1;" ::"r"(addr), "r"(v));
}

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
// One CTA (128 threads, five per SM) per (batch, head, chunk).  Writes Tb = Tt diag(beta)
// as the bf16 rows [((b*H + h)*NC + r)*64 + i][0..63] of the workspace.

constexpr uint32_t WY_K = 0;        // 16K  raw k (dead once the KK product and the norms have read it)
constexpr uint32_t WY_A = 0;        // 64 x 68 fp32 A over k; after the inversion the bf16 Tb tile
constexpr uint32_t WY_T = 17408;    // 64 x 68 fp32: Tt
constexpr uint32_t WY_Y = 34816;    // 3 x 256 fp32 block products of the inversion
constexpr uint32_t WY_MISC = 37888; // gc, beta, factors, rk, barriers
constexpr uint32_t WY_SMEM = WY_MISC + 2048 + 1024;  // 40 KB: five CTAs per SM
constexpr int kAS = 68;             // padded fp32 row stride of A and Tt

__global__ void __launch_bounds__(128, 5)
gdn_wy_kernel(const __grid_constant__ CUtensorMap map_k, const __grid_constant__ CUtensorMap map_tb,
              const ChunkArgs a, int NC) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = smem_align1024(smem_raw);
    const uint32_t sb = smem_addr(sm);
    float *A = reinterpret_cast<float *>(sm + WY_A);
    float *Tt = reinterpret_cast<float *>(sm + WY_T);
    float *Y = reinterpret_cast<float *>(sm + WY_Y);
    float *gcs = reinterpret_cast<float *>(sm + WY_MISC);        // [64] cumulative log decay
    float *bet = gcs + 64;                                        // [64] beta
    float *epos = gcs + 128;                                      // [64] beta / |k|
    float *eneg = gcs + 192;                                      // [64] gc log2(e)
    float *rk = gcs + 256;                                        // [64] 1/|k|
    uint64_t *bar = reinterpret_cast<uint64_t *>(sm + WY_MISC + 1536);
    uint32_t *tslot = reinterpret_cast<uint32_t *>(sm + WY_MISC + 1560);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(sm + WY_MISC + 1564);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int item = blockIdx.x;
    const int H = a.H;
    // packed sequences: item = (packed chunk) * H + head; otherwise item = (b H + h) NC + r
    const bool vl = a.cu != nullptr;
    int b, h, r, nc_b;
    if (vl) {
        const int gci = item / H;
        h = item % H;
        b = a.chunk_seq[gci];
        r = gci - a.cbase[b];
        nc_b = a.cbase[b + 1] - a.cbase[b];
    } else {
        r = item % NC;
        b = item / NC / H;
        h = item / NC % H;
        nc_b = NC;
    }
    const int tok0 = vl ? static_cast<int>(a.cu[b]) : 0;
    const int T = vl ? static_cast<int>(a.cu[b + 1] - a.cu[b]) : a.T;
    const int bt = vl ? 0 : b;
    const size_t rowbase = vl ? static_cast<size_t>(tok0) : static_cast<size_t>(b) * a.T;
    const int tbrow = ((vl ? a.cbase[b] : b * NC) * H + h * nc_b + r) * kC;  // first Tb row of the chunk
    const int c0 = r * kC;
    int *status = a.status;

    if (tid == 0) {
        for (int i = 0; i < 2; ++i) mbar_init(&bar[i], 1);
        *abort_flag = 0;
        fence_barrier_init();
        mbar_arrive_expect_tx(&bar[0], 2 * 8192);
        tma_load_4d(sm + WY_K, &map_k, &bar[0], 0, h, tok0 + c0, bt);
        tma_load_4d(sm + WY_K + 8192, &map_k, &bar[0], 64, h, tok0 + c0, bt);
    }
    if (warp == 0) tmem_alloc(tslot, 64);
    if (tid < 64) {
        // past the end of a packed sequence: beta = 0 and no decay, so the rows of the next
        // sequence's keys in the tile add nothing
        const int t = c0 + tid;
        const size_t row = (rowbase + t) * H + h;
        gcs[tid] = t < T ? a.g[row] : 0.f;
        bet[tid] = t < T ? a.beta[row] : 0.f;
    }
    __syncthreads();
    tc_fence_after();
    const uint32_t tb = *tslot;
    const uint32_t tq = tb + (static_cast<uint32_t>(32 * warp) << 16);

    // ---- cumulative decay (warp 2: two values per lane, shuffle scan)
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
    // ---- KK = K K^T on the raw keys (M = 64: rows 16w..16w+15 in lanes 32w..32w+15); the
    // key norms are its diagonal, and they scale A instead of the keys
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
    const int i = 16 * warp + (lane & 15), hf = lane >> 4;  // row i, columns 32 hf .. 32 hf + 31
    float kk[32];
    tmem_ld16x2_32<32>(tq, kk);
    if ((i >> 5) == hf) {  // this thread holds KK_ii = |k_i|^2
        // column i & 31 = 16 (warp & 1) + (lane & 15): a select tree on those bits, which keeps
        // kk in registers
        const int e = i & 31;
        float v[16];
#pragma unroll
        for (int u = 0; u < 16; ++u) v[u] = (e & 16) ? kk[16 + u] : kk[u];
#pragma unroll
        for (int w = 8; w >= 1; w >>= 1)
#pragma unroll
            for (int u = 0; u < w; ++u) v[u] = (e & w) ? v[w + u] : v[u];
        const float d = v[0];
        rk[i] = a.l2norm ? rsqrtf(fmaxf(d, 1e-12f)) : 1.f;
    }
    __syncthreads();
    // row and column factors of A: A_ij = (beta_i rk_i) (rk_j) KK_ij e^{gc_i - gc_j}; the decay
    // is one exponential of gc_i - gc_j <= 0 per entry (j < i), so no factor can overflow
    // however strong the forgetting, and a decay that underflows gives an exact zero
    if (tid < 64) {
        epos[tid] = bet[tid] * rk[tid];
        eneg[tid] = gcs[tid] * kLog2e;  // log2 of the cumulative decay
    }
    __syncthreads();
    {
        // A_ij for j < i, written over the k tile (the product has read it)
        const float ri = epos[i], li = eneg[i];
#pragma unroll
        for (int q4 = 0; q4 < 8; ++q4) {
            const float4 rkj = *reinterpret_cast<const float4 *>(rk + 32 * hf + 4 * q4);
            const float4 lj = *reinterpret_cast<const float4 *>(eneg + 32 * hf + 4 * q4);
            const float rkv[4] = {rkj.x, rkj.y, rkj.z, rkj.w}, lv[4] = {lj.x, lj.y, lj.z, lj.w};
            float w[4];
#pragma unroll
            for (int e = 0; e < 4; ++e)
                w[e] = (32 * hf + 4 * q4 + e < i) ? ri * rkv[e] * kk[4 * q4 + e] * fast_exp2(li - lv[e]) : 0.f;
            *reinterpret_cast<float4 *>(A + i * kAS + 32 * hf + 4 * q4) = make_float4(w[0], w[1], w[2], w[3]);
        }
    }
    __syncthreads();
    // ---- Tt = (I + A)^{-1}: the four 16 x 16 diagonal blocks by forward substitution
    // (thread = one column c of block bb; the row's A entries as float4 loads)
    if (tid < 64) {
        const int bb = tid >> 4, c = tid & 15, o = 16 * bb;
        float x[16];
#pragma unroll
        for (int rr = 0; rr < 16; ++rr) {
            float s = 0.f;
#pragma unroll
            for (int j4 = 0; j4 < 4; ++j4) {
                if (4 * j4 < rr) {
                    const float4 av = *reinterpret_cast<const float4 *>(A + (o + rr) * kAS + o + 4 * j4);
                    s = fmaf(av.x, x[4 * j4], s);
                    if (4 * j4 + 1 < rr) s = fmaf(av.y, x[4 * j4 + 1], s);
                    if (4 * j4 + 2 < rr) s = fmaf(av.z, x[4 * j4 + 2], s);
                    if (4 * j4 + 3 < rr) s = fmaf(av.w, x[4 * j4 + 3], s);
                }
            }
            x[rr] = (rr < c) ? 0.f : ((rr == c) ? 1.f : -s);
        }
#pragma unroll
        for (int rr = 0; rr < 16; ++rr) Tt[(o + rr) * kAS + o + c] = x[rr];
    }
    __syncthreads();
    // off-diagonal blocks, by distance from the diagonal:
    //   Tt_IJ = -Tt_II sum_{K=J}^{I-1} A_IK Tt_KJ
    // one warp per 16 x 16 block, each thread a 4-row x 2-column sub-tile in fp32 pairs
    for (int dist = 1; dist < 4; ++dist) {
        const int nblk = 4 - dist;
        const int blk = warp, r0 = 4 * (lane >> 3), cq = 2 * (lane & 7);
        const int J = blk, I = blk + dist;
        if (blk < nblk) {
            uint64_t acc[4] = {0, 0, 0, 0};
            for (int K = J; K < I; ++K) {
#pragma unroll
                for (int m = 0; m < 16; m += 4) {
                    float4 av[4];
                    uint64_t tv[4];
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        av[u] = *reinterpret_cast<const float4 *>(A + (16 * I + r0 + u) * kAS + 16 * K + m);
                        tv[u] = *reinterpret_cast<const uint64_t *>(Tt + (16 * K + m + u) * kAS + 16 * J + cq);
                    }
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        acc[u] = f2_fma(f2_make(av[u].x, av[u].x), tv[0], acc[u]);
                        acc[u] = f2_fma(f2_make(av[u].y, av[u].y), tv[1], acc[u]);
                        acc[u] = f2_fma(f2_make(av[u].z, av[u].z), tv[2], acc[u]);
                        acc[u] = f2_fma(f2_make(av[u].w, av[u].w), tv[3], acc[u]);
                    }
                }
            }
#pragma unroll
            for (int u = 0; u < 4; ++u)
                *reinterpret_cast<uint64_t *>(Y + blk * 256 + (r0 + u) * 16 + cq) = acc[u];
        }
        __syncthreads();
        if (blk < nblk) {
            uint64_t acc[4] = {0, 0, 0, 0};
#pragma unroll
            for (int m = 0; m < 16; m += 4) {
                float4 av[4];
                uint64_t yv[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    av[u] = *reinterpret_cast<const float4 *>(Tt + (16 * I + r0 + u) * kAS + 16 * I + m);
                    yv[u] = *reinterpret_cast<const uint64_t *>(Y + blk * 256 + (m + u) * 16 + cq);
                }
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    acc[u] = f2_fma(f2_make(av[u].x, av[u].x), yv[0], acc[u]);
                    acc[u] = f2_fma(f2_make(av[u].y, av[u].y), yv[1], acc[u]);
                    acc[u] = f2_fma(f2_make(av[u].z, av[u].z), yv[2], acc[u]);
                    acc[u] = f2_fma(f2_make(av[u].w, av[u].w), yv[3], acc[u]);
                }
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const float2 v = f2_split(acc[u]);
                *reinterpret_cast<float2 *>(Tt + (16 * I + r0 + u) * kAS + 16 * J + cq) = make_float2(-v.x, -v.y);
            }
        }
        __syncthreads();
    }
    // ---- the fp32 Tt itself for the backward (one row half per thread, as float4 stores;
    // the blocks above the diagonal were never written: zeros)
    if (a.tt_out) {
        const int i2 = tid >> 1, hf2 = tid & 1;
        float4 *dst = reinterpret_cast<float4 *>(a.tt_out + (static_cast<size_t>(item) * kC + i2) * kC + 32 * hf2);
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            const int j0 = 32 * hf2 + 4 * q;
            const float4 t = *reinterpret_cast<const float4 *>(Tt + i2 * kAS + j0);
            dst[q] = make_float4(j0 <= i2 ? t.x : 0.f, j0 + 1 <= i2 ? t.y : 0.f, j0 + 2 <= i2 ? t.z : 0.f,
                                 j0 + 3 <= i2 ? t.w : 0.f);
        }
    }
    // ---- Tb = Tt diag(beta) (zero above the diagonal) as the bf16 T64 tile in A's place
    {
        const int i = tid >> 1, hf = tid & 1;
#pragma unroll
        for (int q4 = 0; q4 < 4; ++q4) {
            float wb[8];
            const float4 t0 = *reinterpret_cast<const float4 *>(Tt + i * kAS + 32 * hf + 8 * q4);
            const float4 t1 = *reinterpret_cast<const float4 *>(Tt + i * kAS + 32 * hf + 8 * q4 + 4);
            const float4 b0 = *reinterpret_cast<const float4 *>(bet + 32 * hf + 8 * q4);
            const float4 b1 = *reinterpret_cast<const float4 *>(bet + 32 * hf + 8 * q4 + 4);
            const float tr[8] = {t0.x, t0.y, t0.z, t0.w, t1.x, t1.y, t1.z, t1.w};
            const float br[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                const int j = 32 * hf + 8 * q4 + e;
                wb[e] = (j <= i) ? tr[e] * br[e] : 0.f;
            }
            store_row_chunk(sm + WY_A, i, 4 * hf + q4, wb);
        }
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    if (tid == 0 && !*abort_flag) {
        asm volatile(
            "cp.async.bulk.tensor.2d.global.shared::cta.tile.bulk_group [%0, {%2, %3}], [%1];" ::"l"(
                reinterpret_cast<uint64_t>(&map_tb)),
            "r"(smem_addr(sm + WY_A)), "r"(0), "r"(tbrow)
            : "memory");
        tma_store_commit();
        tma_store_wait_read();  // shared memory must outlive the store's read
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tb, 64);
    }
}


// ============================================================================ main kernel
//
// Warp specialisation (14 warps), as in the GLA kernel:
//   EPI   (warps 0-7)   the epilogues of chunk r -- W', R and U, q_clean, Pm,
//                       output -- and the bf16 copies of S^K_{r+1} (while D4 runs) and
//                       H_{r+1} (while G2 of chunk r+1 runs).  Warps w and w+4 share
//                       TMEM lane quadrant w % 4 and split its columns.
//   PREP  (warps 8-11)  prep of chunk r+1: row norms, cumulative decay, kbar, Kd.
//   COPY  (warp 13)     every per-chunk TMA copy and the L2 prefetch of chunk r + 2; the
//                       output is staged in the slot's Kd tile, so R and U never wait on it.
//   ISSUE (warp 12)     every tcgen05.mma, in the order
//                       G2 D2 | G1 | DU G3 G8 | D4 D6 D3 | D5.  D2 (Kbar H0) lands in the
//                       P/O accumulator, so EPI reads it out first and frees the accumulator
//                       for G1 before it builds R; U = Tb R lands in TMEM columns 384-511
//                       (Sc has been read, QK comes later).
// R, then U share one 16 KB tile; the output is staged in the Kd tile of the chunk's slot.

constexpr int kThreads = 448;
constexpr int kEpiThreads = 256;
constexpr int kPrepWarp0 = 8, kIssueWarp = 12, kCopyWarp = 13;
constexpr int kSyncCount = kEpiThreads + 32;
constexpr uint32_t SLOT_BYTES = 49152;
constexpr uint32_t SO_Q = 0;        // raw q, then q_clean
constexpr uint32_t SO_K = 16384;    // raw k, then kbar
constexpr uint32_t SO_KD = 32768;   // kbar e^{gC - gc}
constexpr uint32_t OFF_V = 98304;   // 16K  v of the chunk
constexpr uint32_t OFF_TB = 114688; // 8K   Tb of the chunk (workspace), [64][64]
constexpr uint32_t OFF_UB = 122880; // 16K  R, then U (bf16, rows j)
constexpr uint32_t OFF_WM = 139264; // 8K   W' of the CCQ fold, then Pm
constexpr uint32_t OFF_SK = 147456; // 32K  bf16 S^K
constexpr uint32_t OFF_HB = 180224; // 32K  bf16 H0, the state entering the chunk
constexpr uint32_t OFF_MISC = 212992;
constexpr uint32_t MS_BYTES = 3072;
constexpr uint32_t MS_RQ = 0, MS_MQ = 256, MS_LT = 512, MS_RK = 768, MS_EP = 1024, MS_EN = 1280,
                   MS_SCAL = 1536, MS_MST = 2048, MS_ITI = 2560, MS_QN = 2816;
// EP: e^{gc}, EN: e^{gC - gc}, SCAL: [1] e^{gC}, [2..65] gc;  LT = lambda / t, ITI = 1 / t, QN = |q|
constexpr uint32_t M_DMP = 6144;     // [2][128] key-sum halves of the chunk
constexpr uint32_t M_DMPREV = 7168;  // [128]
constexpr uint32_t M_BAR = 7680;     // mbarriers
constexpr uint32_t M_TMEM = 7824;
constexpr uint32_t M_ABORT = 7828;
constexpr uint32_t M_EPO = 7936;     // [2][64] e^{gc} of the chunk whose output is being written
constexpr uint32_t kMiscBytes = 8448;
constexpr uint32_t kSmemBytes = OFF_MISC + kMiscBytes + 1024;
static_assert(kSmemBytes <= 232448, "exceeds the 227 KB per-CTA limit");
static_assert(MS_SCAL + 66 * 4 <= MS_MST, "scalar area overlaps");

enum {
    BAR_IN0 = 0, BAR_IN1 = 1, BAR_WU = 2, BAR_GA1 = 3, BAR_GA2 = 4, BAR_GB = 5, BAR_GK = 6, BAR_GC = 7,
    BAR_GC2 = 8, BAR_GD = 9, BAR_PREP0 = 10, BAR_PREP1 = 11, BAR_SNAPK = 12, BAR_SNAPS = 13,
    BAR_OST0 = 14, BAR_OST1 = 15, BAR_GP = 16, kNumBars = 17
};
static_assert(M_BAR + 8 * kNumBars <= M_TMEM, "barrier area");
enum { NB_PO = 1, NB_W = 2, NB_QC = 3, NB_MASK = 4, NB_OUT = 5, NB_PREP = 6, NB_EPI = 7 };

constexpr uint32_t TM_S = 0, TM_SK = 128, TM_PO = 256, TM_SA = 384, TM_U = 384, kTmemCols = 512;
// the transposed output accumulators (M = 128 layout) inside the P/O region
constexpr uint32_t TM_O1 = 256, TM_O2 = 320;
constexpr uint32_t ID_64x64_KK = make_idesc(64, 64, 0, 0);
constexpr uint32_t ID_64x128_KK = make_idesc(64, 128, 0, 0);
constexpr uint32_t ID_64x128_KM = make_idesc(64, 128, 0, 1);
constexpr uint32_t ID_128x128_MM = make_idesc(128, 128, 1, 1);
constexpr uint32_t ID_128x64_MK = make_idesc(128, 64, 1, 0);

__global__ void __launch_bounds__(kThreads, 1)
gdn_chunk_kernel(const __grid_constant__ CUtensorMap map_q, const __grid_constant__ CUtensorMap map_k,
                 const __grid_constant__ CUtensorMap map_v, const __grid_constant__ CUtensorMap map_tb,
                 const __grid_constant__ CUtensorMap map_o, const ChunkArgs a) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = smem_align1024(smem_raw);
    const uint32_t sb = smem_addr(sm);
    uint8_t *misc = sm + OFF_MISC;
    float *dmp = reinterpret_cast<float *>(misc + M_DMP);
    float *dmprev = reinterpret_cast<float *>(misc + M_DMPREV);
    uint64_t *bar = reinterpret_cast<uint64_t *>(misc + M_BAR);
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(misc + M_TMEM);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(misc + M_ABORT);
    auto slot_f = [&](int s, uint32_t off) {
        return reinterpret_cast<float *>(misc + s * MS_BYTES + off);
    };

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int bh = blockIdx.x / a.nseg, seg = blockIdx.x % a.nseg, b = bh / a.H, h = bh % a.H;
    const int H = a.H;
    // packed sequences: sequence b is rows tok0 .. tok0 + T of a [1][a.T][H][D] tensor
    const bool vl = a.cu != nullptr;
    const int tok0 = vl ? static_cast<int>(a.cu[b]) : 0;
    const int T = vl ? static_cast<int>(a.cu[b + 1] - a.cu[b]) : a.T;
    const int bt = vl ? 0 : b;
    const size_t rowbase = vl ? static_cast<size_t>(tok0) : static_cast<size_t>(b) * a.T;
    const int NCt = (T + kC - 1) / kC;
    const int cb = a.nseg > 1 ? seg * a.seg_chunks : 0;  // first chunk of this CTA
    const int NC = a.nseg > 1 ? min(NCt, cb + a.seg_chunks) - cb : NCt;
    const bool last_seg = seg == a.nseg - 1;
    // a segment starts from the states its slot of the workspace holds (ccq_gdn_segment.cu)
    const float *segst = a.nseg > 1 ? a.seg_ws + static_cast<size_t>(blockIdx.x) * kGdnSegFloats : nullptr;
    const float *S0 = segst ? segst : a.S0;
    const float *C0 = segst ? segst + 2 * kD * kD : a.C0;
    const float *m0 = segst ? segst + 3 * kD * kD : a.m0;
    const int64_t t0 = (a.t0 ? a.t0[b] : 0) + static_cast<int64_t>(cb) * kC;  // position before the CTA's first token
    int *status = a.status;
    const int wrow0 = ((vl ? a.cbase[b] * H + h * NCt : bh * NCt) + cb) * kC;  // first Tb row of this CTA's chunks

    if (tid == 0) {
        for (int i = 0; i < kNumBars; ++i) mbar_init(&bar[i], 1);
        *abort_flag = 0;
        fence_barrier_init();
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
        const int tg = (cb + r) * kC;
        tma_load_4d(base + SO_Q, &map_q, bb, 0, h, tok0 + tg, bt);
        tma_load_4d(base + SO_Q + 8192, &map_q, bb, 64, h, tok0 + tg, bt);
        tma_load_4d(base + SO_K, &map_k, bb, 0, h, tok0 + tg, bt);
        tma_load_4d(base + SO_K + 8192, &map_k, bb, 64, h, tok0 + tg, bt);
        if (r + 2 < NC) {  // chunk r + 2 into L2, so that its loads hit there
            tma_prefetch_l2_4d(&map_q, 0, h, tok0 + tg + 2 * kC, bt);
            tma_prefetch_l2_4d(&map_q, 64, h, tok0 + tg + 2 * kC, bt);
            tma_prefetch_l2_4d(&map_k, 0, h, tok0 + tg + 2 * kC, bt);
            tma_prefetch_l2_4d(&map_k, 64, h, tok0 + tg + 2 * kC, bt);
        }
    };
    auto issue_wu = [&](int r) {  // v and Tb of chunk r
        uint64_t *bb = &bar[BAR_WU];
        mbar_arrive_expect_tx(bb, 3 * 8192);
        tma_load_4d(sm + OFF_V, &map_v, bb, 0, h, tok0 + (cb + r) * kC, bt);
        tma_load_4d(sm + OFF_V + 8192, &map_v, bb, 64, h, tok0 + (cb + r) * kC, bt);
        tma_load_2d(sm + OFF_TB, &map_tb, bb, 0, wrow0 + r * kC);
        if (r + 2 < NC) {
            tma_prefetch_l2_4d(&map_v, 0, h, tok0 + (cb + r + 2) * kC, bt);
            tma_prefetch_l2_4d(&map_v, 64, h, tok0 + (cb + r + 2) * kC, bt);
            asm volatile("cp.async.bulk.prefetch.tensor.2d.L2.global.tile [%0, {%1, %2}];" ::"l"(
                             reinterpret_cast<uint64_t>(&map_tb)),
                         "r"(0), "r"(wrow0 + (r + 2) * kC)
                         : "memory");
        }
    };

    // the last chunk of a packed sequence ends inside the tile: its rows past the end belong to
    // the next sequence, so its output is written row by row (not by a TMA store of the tile)
    auto partial = [&](int r) { return vl && T - (cb + r) * kC < kC; };

    // ---- set-up: initial states into TMEM (EPI), key sum (PREP), first loads (ISSUE)
    if (warp < kPrepWarp0) {
        const size_t bhs = static_cast<size_t>(bh);
        const int row = 32 * (warp & 3) + lane, grp = warp >> 2;
        for (int m = 0; m < 2; ++m) {
            const float *src = m == 0 ? S0 : C0;
            const uint32_t col0 = m == 0 ? TM_S : TM_SK;
#pragma unroll
            for (int cc = 0; cc < 2; ++cc) {
                const int c = 2 * grp + cc;
                float x[32];
                if (src) {
                    const float4 *p4 = reinterpret_cast<const float4 *>(
                        src + (segst ? static_cast<size_t>(row) * kD : (bhs * kD + row) * kD) + 32 * c);
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
    } else if (warp < kIssueWarp) {
        const int wt = tid - 32 * kPrepWarp0;
        slot_f(0, MS_MST)[wt] = m0 ? m0[(segst ? 0 : static_cast<size_t>(bh) * kD) + wt] : 0.f;
        dmprev[wt] = 0.f;
    } else if (warp == kIssueWarp && lane == 0) {
        tma_prefetch_desc(&map_q);
        tma_prefetch_desc(&map_k);
        tma_prefetch_desc(&map_v);
        tma_prefetch_desc(&map_tb);
        tma_prefetch_desc(&map_o);
        if (NC > 0) {
            issue_in(0);
            issue_wu(0);
        }
        if (NC > 1) issue_in(1);
    }
    tc_fence_before();
    __syncthreads();

    if (warp < kPrepWarp0) {
        // =============================================================== EPI
        const int grp = warp >> 2;
        const int i = 16 * (warp & 3) + (lane & 15);
        const int hf = lane >> 4;
        const int row = 32 * (warp & 3) + lane;  // state row of the M = 128 layout
        // (with a.sk_out / a.hs_out the snapshots of chunk ch of this sequence also write the
        // fp32 states to the backward's arrays)
        auto snap_sk = [&](int ch) {
            tc_fence_after();
#pragma unroll
            for (int cc = 0; cc < 2; ++cc) {
                float x[32];
                tmem_ld32(tq + TM_SK + 64 * grp + 32 * cc, x);
                if (a.sk_out) {
                    float4 *dst = reinterpret_cast<float4 *>(
                        a.sk_out + ((static_cast<size_t>(bh) * NCt + ch) * kD + row) * kD + 64 * grp + 32 * cc);
#pragma unroll
                    for (int e = 0; e < 8; ++e) dst[e] = make_float4(x[4 * e], x[4 * e + 1], x[4 * e + 2], x[4 * e + 3]);
                }
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4)
                    store_row_chunk(sm + OFF_SK + grp * 16384, row, 4 * cc + q4, x + 8 * q4);
            }
            fence_proxy_async_smem();
            tc_fence_before();
            named_bar(NB_EPI, kEpiThreads);
            if (tid == 0) mbar_arrive(&bar[BAR_SNAPK]);
        };
        // bf16 copy of the state H entering the next chunk; the TMEM copy is scaled by that
        // chunk's e^{gC} (hs), onto which D6 accumulates the chunk's write
        auto snap_s = [&](float hs, int ch) {
            tc_fence_after();
#pragma unroll
            for (int cc = 0; cc < 2; ++cc) {
                float x[32];
                tmem_ld32(tq + TM_S + 64 * grp + 32 * cc, x);
                if (a.hs_out) {
                    float4 *dst = reinterpret_cast<float4 *>(
                        a.hs_out + ((static_cast<size_t>(bh) * NCt + ch) * kD + row) * kD + 64 * grp + 32 * cc);
#pragma unroll
                    for (int e = 0; e < 8; ++e) dst[e] = make_float4(x[4 * e], x[4 * e + 1], x[4 * e + 2], x[4 * e + 3]);
                }
                const uint64_t hs2 = f2_make(hs, hs);
                uint32_t w[16];
#pragma unroll
                for (int e = 0; e < 16; ++e) {
                    w[e] = pack_bf16(x[2 * e], x[2 * e + 1]);
                    const float2 y = f2_split(f2_mul(f2_make(x[2 * e], x[2 * e + 1]), hs2));
                    x[2 * e] = y.x;
                    x[2 * e + 1] = y.y;
                }
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4)
                    *reinterpret_cast<uint4 *>(sm + OFF_HB + grp * 16384 + t64_chunk(row, 4 * cc + q4)) =
                        make_uint4(w[4 * q4], w[4 * q4 + 1], w[4 * q4 + 2], w[4 * q4 + 3]);
                tmem_st32(tq + TM_S + 64 * grp + 32 * cc, x);
            }
            tmem_wait_st();
            fence_proxy_async_smem();
            tc_fence_before();
            named_bar(NB_EPI, kEpiThreads);
            if (tid == 0) mbar_arrive(&bar[BAR_SNAPS]);
        };
        float *epo = reinterpret_cast<float *>(misc + M_EPO);
        if (NC > 0) {
            mbar_wait(&bar[BAR_PREP0], 0, abort_flag, status);
            snap_sk(cb);
            snap_s(slot_f(0, MS_SCAL)[1], cb);
        }
        for (int r = 0; r < NC; ++r) {
            const int s = r & 1;
            const uint32_t sp = (r >> 1) & 1, par = r & 1;
            uint8_t *slot = sm + s * SLOT_BYTES;
            mbar_wait(&bar[BAR_PREP0 + s], sp, abort_flag, status);
            const float rqi = slot_f(s, MS_RQ)[i];
            const float mqi = slot_f(s, MS_MQ)[i];
            const float iti = slot_f(s, MS_ITI)[i];
            const float qni = slot_f(s, MS_QN)[i];
            const float lt = slot_f(s, MS_LT)[i];
            const float ep = slot_f(s, MS_EP)[i];
            // ---- W' of the CCQ mean fold
            mbar_wait(&bar[BAR_GA1], par, abort_flag, status);
            tc_fence_after();
            float c = 0.f;
            {
                float sc[32];
                tmem_ld16x2_32<32>(tq + TM_SA, sc);
                float pa[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                for (int jj = 0; jj < 32; ++jj)
                    if (32 * hf + jj <= i) pa[jj & 3] += sc[jj];
                float part = (pa[0] + pa[1]) + (pa[2] + pa[3]);
                part += __shfl_xor_sync(0xffffffffu, part, 16);
                const float cq = mqi + rqi * part;
                c = a.centered ? cq * iti : 0.f;
                const float cn = c * qni;
#pragma unroll
                for (int q2 = 0; q2 < 2; ++q2) {
                    float w[8];
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        const int jj = 8 * q2 + e;
                        const float v = grp ? sc[16 + jj] : sc[jj];
                        w[e] = (32 * hf + 16 * grp + jj <= i) ? v - cn : 0.f;
                    }
                    store_row_chunk(sm + OFF_WM, i, 4 * hf + 2 * grp + q2, w);
                }
            }
            fence_proxy_async_smem();  // W' is read by G3, issued with G1 after NB_PO
            // ---- R = V - e^{gc} Kbar H0: read Kbar H0 out of the P/O accumulator
            // first, freeing it for G1
            mbar_wait(&bar[BAR_GA2], par, abort_flag, status);
            tc_fence_after();
            {
                float x[32];
                tmem_ld16x2_32<32>(tq + TM_PO + 64 * grp, x);  // columns 64 grp + 32 hf ..
                tc_fence_before();
                named_bar_arrive(NB_PO, kSyncCount);
                mbar_wait(&bar[BAR_WU], par, abort_flag, status);  // v of the chunk
                const uint8_t *vt = sm + OFF_V + grp * 8192;
                uint8_t *rt = sm + OFF_UB + grp * 8192;
                const uint64_t nep = f2_make(-ep, -ep);
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) {
                    const uint4 v4 = *reinterpret_cast<const uint4 *>(vt + t64_chunk(i, 4 * hf + q4));
                    const uint32_t vw[4] = {v4.x, v4.y, v4.z, v4.w};
                    uint32_t ow[4];
#pragma unroll
                    for (int w = 0; w < 4; ++w)
                        ow[w] = bf16x2_from_f2(f2_fma(nep, f2_make(x[8 * q4 + 2 * w], x[8 * q4 + 2 * w + 1]),
                                                      f2_from_bf16x2(vw[w])));
                    *reinterpret_cast<uint4 *>(rt + t64_chunk(i, 4 * hf + q4)) = make_uint4(ow[0], ow[1], ow[2], ow[3]);
                }
            }
            fence_proxy_async_smem();
            tc_fence_before();
            named_bar_arrive(NB_W, kSyncCount);
            // ---- q_clean (Eq. clean) into the Q tile
            {
                uint8_t *qt = slot + SO_Q + grp * 8192;
                const float *Mst = slot_f(s, MS_MST) + 64 * grp + 32 * hf;
                uint4 qraw[4];
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) qraw[q4] = *reinterpret_cast<const uint4 *>(qt + t64_chunk(i, 4 * hf + q4));
                mbar_wait(&bar[BAR_GP], par, abort_flag, status);
                tc_fence_after();
                const float cm = lt * c;
                float p[32];
                tmem_ld16x2_32<32>(tq + TM_PO + 64 * grp, p);
                // the read scale is applied here: both output products are linear in q_clean
                const float rqs = rqi * a.scale, cms = cm * a.scale;
                const uint64_t nlt = f2_make(-lt, -lt), rq2 = f2_make(rqs, rqs), cm2 = f2_make(cms, cms);
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) {
                    const ulonglong2 m01 = *reinterpret_cast<const ulonglong2 *>(Mst + 8 * q4);
                    const ulonglong2 m23 = *reinterpret_cast<const ulonglong2 *>(Mst + 8 * q4 + 4);
                    const uint64_t mp[4] = {m01.x, m01.y, m23.x, m23.y};
                    const uint32_t qw[4] = {qraw[q4].x, qraw[q4].y, qraw[q4].z, qraw[q4].w};
                    uint32_t ow[4];
#pragma unroll
                    for (int w = 0; w < 4; ++w) {
                        const uint64_t p2 = f2_make(p[8 * q4 + 2 * w], p[8 * q4 + 2 * w + 1]);
                        const uint64_t t = f2_fma(nlt, p2, f2_from_bf16x2(qw[w]));
                        ow[w] = bf16x2_from_f2(f2_fma(rq2, t, f2_mul(cm2, mp[w])));
                    }
                    *reinterpret_cast<uint4 *>(qt + t64_chunk(i, 4 * hf + q4)) = make_uint4(ow[0], ow[1], ow[2], ow[3]);
                }
            }
            // U = Tb R (the MMA has read R; it ran while q_clean was formed) -> bf16 U tile in
            // R's place
            mbar_wait(&bar[BAR_GB], par, abort_flag, status);
            tc_fence_after();
            {
                float u[32];
                tmem_ld16x2_32<32>(tq + TM_U + 64 * grp, u);
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4)
                    store_row_chunk(sm + OFF_UB + grp * 8192, i, 4 * hf + q4, u + 8 * q4);
            }
            // gc_i - gc_j (log2 units) of this thread's 16 key columns, and e^{gc} of the rows for
            // the output epilogue, read before the slot is released
            float ev[16];
            {
                const float *gcv = slot_f(s, MS_SCAL) + 2;
                const float gi = gcv[i];
#pragma unroll
                for (int q = 0; q < 16; ++q) ev[q] = (gi - gcv[32 * hf + 16 * grp + q]) * kLog2e;
                if (tid < 64) epo[(r & 1) * 64 + tid] = slot_f(s, MS_EP)[tid];
            }
            fence_proxy_async_smem();
            tc_fence_before();
            named_bar_arrive(NB_QC, kSyncCount);
            // ---- S^K_{r+1} while D4 runs
            if (r + 1 < NC) {
                mbar_wait(&bar[BAR_GK], par, abort_flag, status);
                snap_sk(cb + r + 1);
            }
            // ---- Pm_ij = [j<=i] QK_ij e^{gc_i - gc_j} (one exponential of a non-positive argument)
            mbar_wait(&bar[BAR_GC], par, abort_flag, status);
            tc_fence_after();
            {
                float sc[32];
                tmem_ld16x2_32<32>(tq + TM_SA, sc);
#pragma unroll
                for (int q2 = 0; q2 < 2; ++q2) {
                    float w[8];
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        const int jj = 8 * q2 + e;
                        const float v = grp ? sc[16 + jj] : sc[jj];
                        w[e] = (32 * hf + 16 * grp + jj <= i) ? v * fast_exp2(ev[jj]) : 0.f;
                    }
                    store_row_chunk(sm + OFF_WM, i, 4 * hf + 2 * grp + q2, w);
                }
            }
            fence_proxy_async_smem();
            tc_fence_before();
            named_bar_arrive(NB_MASK, kSyncCount);
            // ---- output o_i = e^{gc_i} O1_i + O2_i (q_clean carries the read scale), staged for
            // the copy warp's TMA store in the slot's Kd tile (its last reader, D6, completed
            // before GD).  O1^T, O2^T are M = 128 accumulators: this thread holds value column
            // `row` for the chunk rows 32 grp .. 32 grp + 31.  A lane pair swaps one value per two
            // rows so that each lane writes a bf16 pair of adjacent columns: the even lane row e,
            // the odd lane row e + 1 (half the shared-memory stores of one column per thread).
            named_bar(NB_EPI, kEpiThreads);  // epo of this chunk visible
            mbar_wait(&bar[BAR_GD], par, abort_flag, status);
            tc_fence_after();
            {
                const bool direct = partial(r), odd = lane & 1;
                const int c2 = row & ~1;  // first column of this lane's pair
                // Shared addresses of the pair in tile row 0 + odd for the four swizzle classes of
                // the even rows (row & 7 = 0, 2, 4, 6); a row adds 128 bytes.
                const uint32_t ob = smem_addr(slot + SO_KD + (row >> 6) * 8192) + (odd ? 128u : 0u) +
                                    (static_cast<uint32_t>(c2 & 7) << 1);
                const uint32_t cx = (static_cast<uint32_t>(c2 & 63) >> 3) ^ (odd ? 1u : 0u);
                uint32_t bk[4];
#pragma unroll
                for (int k = 0; k < 4; ++k) bk[k] = ob + ((cx ^ (2u * k)) << 4);
#pragma unroll 1
                for (int hh = 0; hh < 2; ++hh) {
                    const int i0 = 32 * grp + 16 * hh;
                    float o1[16], o2[16];
                    tmem_ld16(tq + TM_O1 + i0, o1);
                    tmem_ld16(tq + TM_O2 + i0, o2);
                    const float *ep_r = epo + (r & 1) * 64 + i0;
                    const uint32_t rb = static_cast<uint32_t>(i0) * 128u;
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        const float4 e4 = *reinterpret_cast<const float4 *>(ep_r + 4 * q);
                        const float ev4[4] = {e4.x, e4.y, e4.z, e4.w};
                        float ov[4];
#pragma unroll
                        for (int u = 0; u < 4; ++u) ov[u] = fmaf(ev4[u], o1[4 * q + u], o2[4 * q + u]);
#pragma unroll
                        for (int u = 0; u < 4; u += 2) {
                            const float y = __shfl_xor_sync(0xffffffffu, odd ? ov[u] : ov[u + 1], 1);
                            const uint32_t pr = odd ? pack_bf16(y, ov[u + 1]) : pack_bf16(ov[u], y);
                            if (!direct) {
                                st_shared_b32(bk[(2 * q + u / 2) & 3] + rb + (4 * q + u) * 128, pr);
                            } else {
                                const int tpos = (cb + r) * kC + i0 + 4 * q + u + (odd ? 1 : 0);
                                if (tpos < T && !a.skip_o)
                                    *reinterpret_cast<uint32_t *>(a.o + ((rowbase + tpos) * H + h) * kD + c2) = pr;
                            }
                        }
                    }
                }
                fence_proxy_async_smem();
            }
            tc_fence_before();
            named_bar_arrive(NB_OUT, kSyncCount);
            // ---- H_{r+1} while G2 of chunk r+1 runs (D3, D6 of chunk r have run: GD follows them)
            if (r + 1 < NC) {
                mbar_wait(&bar[BAR_PREP0 + (s ^ 1)], ((r + 1) >> 1) & 1, abort_flag, status);
                snap_s(slot_f(s ^ 1, MS_SCAL)[1], cb + r + 1);
            }
        }
        // final states: H_T (the TMEM state after the last chunk), S^K
        if ((NC > 0 || vl) && last_seg) {  // (an empty packed sequence: the initial states)
            tc_fence_after();
            const size_t bhs = static_cast<size_t>(bh);
#pragma unroll
            for (int cc = 0; cc < 2; ++cc) {
                const int cl = 2 * grp + cc;
                float x[32];
                tmem_ld32(tq + TM_S + 32 * cl, x);
                if (a.ST) {
                    float4 *dst = reinterpret_cast<float4 *>(a.ST + (bhs * kD + row) * kD + 32 * cl);
#pragma unroll
                    for (int e = 0; e < 8; ++e)
                        dst[e] = make_float4(x[4 * e], x[4 * e + 1], x[4 * e + 2], x[4 * e + 3]);
                }
                tmem_ld32(tq + TM_SK + 32 * cl, x);
                if (a.CT) {
                    float4 *dst = reinterpret_cast<float4 *>(a.CT + (bhs * kD + row) * kD + 32 * cl);
#pragma unroll
                    for (int e = 0; e < 8; ++e) dst[e] = make_float4(x[4 * e], x[4 * e + 1], x[4 * e + 2], x[4 * e + 3]);
                }
            }
        }
    } else if (warp < kIssueWarp) {
        // =============================================================== PREP
        const int wt = tid - 32 * kPrepWarp0;
        float lam_reg, g_reg;
        {
            const int tn = cb * kC + (wt >> 1), tg = cb * kC + wt;
            lam_reg = (tn < T) ? a.lambda[(rowbase + tn) * H + h] : 0.f;
            g_reg = (wt < 64 && tg < T) ? a.g[(rowbase + tg) * H + h] : 0.f;
        }
        for (int r = 0; r < NC; ++r) {
            const int s = r & 1;
            const uint32_t sp = (r >> 1) & 1;
            uint8_t *slot = sm + s * SLOT_BYTES;
            float *Mst = slot_f(s, MS_MST);
            float *scal = slot_f(s, MS_SCAL);
            mbar_wait(&bar[BAR_IN0 + s], sp, abort_flag, status);
            if (r > 0) Mst[wt] = slot_f(s ^ 1, MS_MST)[wt] + dmprev[wt];
            if (a.mk_out) a.mk_out[(static_cast<size_t>(bh) * NCt + cb + r) * kD + wt] = Mst[wt];
            const float lam_cur = lam_reg;
            if (wt < 64) scal[2 + wt] = g_reg;
            {
                const int tn = (cb + r + 1) * kC + (wt >> 1);
                lam_reg = (tn < T) ? a.lambda[(rowbase + tn) * H + h] : 0.f;
                const int tg = (cb + r + 1) * kC + wt;
                g_reg = (wt < 64 && tg < T) ? a.g[(rowbase + tg) * H + h] : 0.f;
            }
            named_bar(NB_PREP, 128);  // key sum and raw decays visible
            // in-chunk cumulative log decay gc: one warp, a shuffle scan over two tokens a lane
            if (wt < 32) {
                const float x0 = scal[2 + 2 * lane], x1 = scal[2 + 2 * lane + 1];
                float pv = x0 + x1;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const float y = __shfl_up_sync(0xffffffffu, pv, o);
                    if (lane >= o) pv += y;
                }
                scal[2 + 2 * lane] = pv - x1;
                scal[2 + 2 * lane + 1] = pv;
            }
            // row norms of q and k and M . q (thread pair per row, one T64 tile each)
            {
                const int j = wt >> 1, hh = wt & 1;
                uint4 qv[8], kv[8];
#pragma unroll
                for (int cc = 0; cc < 8; ++cc) {
                    qv[cc] = *reinterpret_cast<const uint4 *>(slot + SO_Q + hh * 8192 + t64_chunk(j, cc));
                    kv[cc] = *reinterpret_cast<const uint4 *>(slot + SO_K + hh * 8192 + t64_chunk(j, cc));
                }
                const float *Mh = Mst + 64 * hh;
                uint64_t sq0 = 0, sq1 = 0, sk0 = 0, sk1 = 0, md0 = 0, md1 = 0;
#pragma unroll
                for (int cc = 0; cc < 8; ++cc) {
                    const ulonglong2 m01 = *reinterpret_cast<const ulonglong2 *>(Mh + 8 * cc);
                    const ulonglong2 m23 = *reinterpret_cast<const ulonglong2 *>(Mh + 8 * cc + 4);
                    const uint32_t qw[4] = {qv[cc].x, qv[cc].y, qv[cc].z, qv[cc].w};
                    const uint32_t kw[4] = {kv[cc].x, kv[cc].y, kv[cc].z, kv[cc].w};
                    const uint64_t mp[4] = {m01.x, m01.y, m23.x, m23.y};
#pragma unroll
                    for (int w = 0; w < 4; ++w) {
                        const uint64_t q2 = f2_from_bf16x2(qw[w]), k2 = f2_from_bf16x2(kw[w]);
                        if (w & 1) {
                            sq1 = f2_fma(q2, q2, sq1); sk1 = f2_fma(k2, k2, sk1); md1 = f2_fma(q2, mp[w], md1);
                        } else {
                            sq0 = f2_fma(q2, q2, sq0); sk0 = f2_fma(k2, k2, sk0); md0 = f2_fma(q2, mp[w], md0);
                        }
                    }
                }
                const float2 a0 = f2_split(f2_add(sq0, sq1)), b0 = f2_split(f2_add(sk0, sk1)),
                             c0v = f2_split(f2_add(md0, md1));
                float ssq = a0.x + a0.y, ssk = b0.x + b0.y, mdt = c0v.x + c0v.y;
                ssq += __shfl_xor_sync(0xffffffffu, ssq, 1);
                ssk += __shfl_xor_sync(0xffffffffu, ssk, 1);
                mdt += __shfl_xor_sync(0xffffffffu, mdt, 1);
                if (hh == 0) {
                    const float rq = a.l2norm ? rsqrtf(fmaxf(ssq, 1e-12f)) : 1.f;
                    const float iti = 1.f / static_cast<float>(t0 + r * kC + j + 1);
                    slot_f(s, MS_RQ)[j] = rq;
                    slot_f(s, MS_MQ)[j] = mdt * rq;
                    slot_f(s, MS_ITI)[j] = iti;
                    slot_f(s, MS_QN)[j] = a.l2norm ? fmaxf(ssq, 1e-12f) * rq : 1.f;
                    slot_f(s, MS_LT)[j] = lam_cur * iti;
                } else {
                    // rows past the end of a packed sequence hold the next one's keys: zero them
                    const bool in_seq = (cb + r) * kC + j < T;
                    slot_f(s, MS_RK)[j] = !in_seq ? 0.f : a.l2norm ? rsqrtf(fmaxf(ssk, 1e-12f)) : 1.f;
                }
            }
            named_bar(NB_PREP, 128);  // gc, rk visible
            if (wt < 64) {
                const float gC = scal[2 + 63];
                slot_f(s, MS_EP)[wt] = fast_exp2(scal[2 + wt] * kLog2e);           // e^{gc} <= 1
                slot_f(s, MS_EN)[wt] = fast_exp2((gC - scal[2 + wt]) * kLog2e);    // e^{gC - gc} <= 1
                if (wt == 0) scal[1] = fast_exp2(gC * kLog2e);
            }
            named_bar(NB_PREP, 128);  // e^{gC - gc} visible
            // kbar (in place) and Kd = kbar e^{gC - gc}: thread = (row, T64 tile); the Kd tile
            // held the output of chunk r - 2 until the copy warp's store read it
            if (r >= 2) mbar_wait(&bar[BAR_OST0 + s], ((r >> 1) - 1) & 1, abort_flag, status);
            {
                const int j = wt >> 1, hh = wt & 1;
                const float rkj = slot_f(s, MS_RK)[j], enj = slot_f(s, MS_EN)[j];
                const uint64_t rk2 = f2_make(rkj, rkj), en2 = f2_make(enj, enj);
                uint8_t *kt = slot + SO_K + hh * 8192;
                uint8_t *kd = slot + SO_KD + hh * 8192;
                uint4 kv[8];
#pragma unroll
                for (int cc = 0; cc < 8; ++cc) kv[cc] = *reinterpret_cast<const uint4 *>(kt + t64_chunk(j, cc));
#pragma unroll
                for (int cc = 0; cc < 8; ++cc) {
                    const uint32_t kw[4] = {kv[cc].x, kv[cc].y, kv[cc].z, kv[cc].w};
                    uint32_t ob[4], od[4];
#pragma unroll
                    for (int w = 0; w < 4; ++w) {
                        const uint64_t kb2 = f2_mul(f2_from_bf16x2(kw[w]), rk2);
                        ob[w] = bf16x2_from_f2(kb2);
                        od[w] = bf16x2_from_f2(f2_mul(kb2, en2));
                    }
                    *reinterpret_cast<uint4 *>(kt + t64_chunk(j, cc)) = make_uint4(ob[0], ob[1], ob[2], ob[3]);
                    *reinterpret_cast<uint4 *>(kd + t64_chunk(j, cc)) = make_uint4(od[0], od[1], od[2], od[3]);
                }
            }
            fence_proxy_async_smem();
            named_bar(NB_PREP, 128);
            // key sum of the chunk (from the bf16 kbar tile): thread = (dim pair, token half)
            {
                const int p = wt & 63, th = wt >> 6, d0 = 2 * p;
                const uint8_t *kt = slot + SO_K + (d0 >> 6) * 8192;
                uint64_t acc0 = 0, acc1 = 0;
#pragma unroll
                for (int jj = 0; jj < 32; jj += 2) {
                    const int j = 32 * th + jj;
                    acc0 = f2_add(acc0, f2_from_bf16x2(*reinterpret_cast<const uint32_t *>(kt + t64_offset(j, d0 & 63))));
                    acc1 = f2_add(acc1, f2_from_bf16x2(*reinterpret_cast<const uint32_t *>(kt + t64_offset(j + 1, d0 & 63))));
                }
                const float2 sv = f2_split(f2_add(acc0, acc1));
                dmp[th * kD + d0] = sv.x;
                dmp[th * kD + d0 + 1] = sv.y;
            }
            named_bar(NB_PREP, 128);
            dmprev[wt] = dmp[wt] + dmp[kD + wt];
            if (wt == 0) mbar_arrive(&bar[BAR_PREP0 + s]);
        }
        if ((NC > 0 || vl) && a.mT && last_seg) {
            const int sl = NC > 0 ? (NC - 1) & 1 : 0;
            a.mT[static_cast<size_t>(bh) * kD + wt] = slot_f(sl, MS_MST)[wt] + dmprev[wt];
        }
    } else if (warp == kIssueWarp) {
        // =============================================================== ISSUE
        const bool lead = lane == 0;
        const uint64_t dWm = make_desc(sb + OFF_WM, 16, 1024);
        const uint64_t dSK = make_desc(sb + OFF_SK, 16, 1024);
        const uint64_t dHB = make_desc(sb + OFF_HB, 16384, 1024);
        const uint64_t dTB = make_desc(sb + OFF_TB, 16, 1024);
        const uint64_t dUBm = make_desc(sb + OFF_UB, 8192, 1024);
        for (int r = 0; r < NC; ++r) {
            const int s = r & 1;
            const uint32_t sp = (r >> 1) & 1, par = r & 1;
            const uint32_t ss = sb + s * SLOT_BYTES;
            const uint64_t dQ = make_desc(ss + SO_Q, 16, 1024);
            const uint64_t dK = make_desc(ss + SO_K, 16, 1024);
            const uint64_t dKm = make_desc(ss + SO_K, 8192, 1024);
            const uint64_t dKDm = make_desc(ss + SO_KD, 8192, 1024);
            mbar_wait(&bar[BAR_PREP0 + s], sp, abort_flag, status);
            tc_fence_after();
            // G2 Sc = Q Kbar^T (SA is free: the Pm epilogue of chunk r-1 has read it)
            if (lead && !*abort_flag) {
                for (int k = 0; k < 8; ++k) {
                    const uint64_t ko = (k >> 2) * 512 + (k & 3) * 2;
                    mma_bf16(tbase + TM_SA, dQ + ko, dK + ko, ID_64x64_KK, k != 0);
                }
                mma_commit(&bar[BAR_GA1]);
            }
            __syncwarp();
            // D2 KH = Kbar H0 (needs the H0 copy)
            mbar_wait(&bar[BAR_SNAPS], par, abort_flag, status);
            tc_fence_after();
            if (lead && !*abort_flag)
                for (int k = 0; k < 8; ++k)
                    mma_bf16(tbase + TM_PO, dK + (k >> 2) * 512 + (k & 3) * 2, dHB + k * 128, ID_64x128_KM, k != 0);
            if (lead && !*abort_flag) mma_commit(&bar[BAR_GA2]);
            __syncwarp();
            // G1 P = Q S^K once Kbar H0 is out of the accumulator, G3 P += W' Kbar (W' is
            // written before NB_PO)
            named_bar(NB_PO, kSyncCount);
            mbar_wait(&bar[BAR_SNAPK], par, abort_flag, status);
            tc_fence_after();
            if (lead && !*abort_flag) {
                for (int k = 0; k < 8; ++k)
                    mma_bf16(tbase + TM_PO, dQ + (k >> 2) * 512 + (k & 3) * 2,
                             dSK + (k >> 2) * 1024 + (k & 3) * 2, ID_64x128_KK, k != 0);
                for (int k = 0; k < 4; ++k) mma_bf16(tbase + TM_PO, dWm + k * 2, dKm + k * 128, ID_64x128_KM, 1);
                mma_commit(&bar[BAR_GP]);
            }
            __syncwarp();
            // DU U = Tb R, G8 S^K += Kbar^T Kbar
            mbar_wait(&bar[BAR_WU], par, abort_flag, status);  // Tb of the chunk
            named_bar(NB_W, kSyncCount);
            tc_fence_after();
            if (lead && !*abort_flag) {
                for (int k = 0; k < 4; ++k) mma_bf16(tbase + TM_U, dTB + k * 2, dUBm + k * 128, ID_64x128_KM, k != 0);
                mma_commit(&bar[BAR_GB]);
                for (int k = 0; k < 4; ++k) mma_bf16(tbase + TM_SK, dKm + k * 128, dKm + k * 128, ID_128x128_MM, 1);
                mma_commit(&bar[BAR_GK]);
            }
            __syncwarp();
            // D4 QK = Qc Kbar^T, D6 X += Kd^T U, D3 O1^T = H0^T Qc^T
            named_bar(NB_QC, kSyncCount);
            tc_fence_after();
            if (lead && !*abort_flag) {
                for (int k = 0; k < 8; ++k) {
                    const uint64_t ko = (k >> 2) * 512 + (k & 3) * 2;
                    mma_bf16(tbase + TM_SA, dQ + ko, dK + ko, ID_64x64_KK, k != 0);
                }
                mma_commit(&bar[BAR_GC]);
                for (int k = 0; k < 4; ++k) mma_bf16(tbase + TM_S, dKDm + k * 128, dUBm + k * 128, ID_128x128_MM, 1);
                // D3 O1^T = H0^T Qc^T (A = the H0 copy, MN-major; B = Qc, K-major)
                for (int k = 0; k < 8; ++k)
                    mma_bf16(tbase + TM_O1, dHB + k * 128, dQ + (k >> 2) * 512 + (k & 3) * 2, ID_128x64_MK, k != 0);
                mma_commit(&bar[BAR_GC2]);
            }
            __syncwarp();
            // D5 O2^T = U^T Pm^T (A = U, MN-major; B = Pm, K-major)
            named_bar(NB_MASK, kSyncCount);
            tc_fence_after();
            if (lead && !*abort_flag) {
                for (int k = 0; k < 4; ++k) mma_bf16(tbase + TM_O2, dUBm + k * 128, dWm + k * 2, ID_128x64_MK, k != 0);
                mma_commit(&bar[BAR_GD]);
            }
            __syncwarp();
        }
    } else {
        // =============================================================== COPY
        // Every per-chunk copy, off the issuing thread (a copy can hold its thread while the
        // copy engine is busy): v and Tb of chunk r + 1 once DU of chunk r has read them (GB);
        // q and k of chunk r + 2 into the slot once D3 and D4 of chunk r have read it (GC2);
        // the store of O (staged in the slot's Kd tile), whose read releases that tile to the
        // prep of chunk r + 2 (OST).
        const bool lead = lane == 0;
        for (int r = 0; r < NC; ++r) {
            const int s = r & 1;
            if (r + 1 < NC) {
                mbar_wait(&bar[BAR_GB], r & 1, abort_flag, status);
                if (lead && !*abort_flag) issue_wu(r + 1);
                __syncwarp();
            }
            if (r + 2 < NC) {
                mbar_wait(&bar[BAR_GC2], r & 1, abort_flag, status);
                if (lead && !*abort_flag) issue_in(r + 2);
                __syncwarp();
            }
            named_bar(NB_OUT, kSyncCount);  // O of chunk r staged
            if (lead) {
                uint8_t *st = sm + s * SLOT_BYTES + SO_KD;
                if (!partial(r) && !a.skip_o) {
                    tma_store_4d(&map_o, st, 0, h, tok0 + (cb + r) * kC, bt);
                    tma_store_4d(&map_o, st + 8192, 64, h, tok0 + (cb + r) * kC, bt);
                    tma_store_commit();
                }
                tma_store_wait_read();
                mbar_arrive(&bar[BAR_OST0 + s]);
            }
            __syncwarp();
        }
        if (lead) {
            tma_store_wait_all();
            if (NC > 0 && *abort_flag) {
                // after a give-up, wait (bounded) for the copies still in flight
                mbar_drain(&bar[BAR_WU], (NC - 1) & 1);
                for (int r = (NC > 2 ? NC - 2 : 0); r < NC; ++r) mbar_drain(&bar[BAR_IN0 + (r & 1)], (r >> 1) & 1);
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
    const int items = a.cu ? a.vl_chunks * a.H : a.B * a.H * NC;
    if (items == 0) return cudaSuccess;
    gdn_wy_kernel<<<items, 128, WY_SMEM, s>>>(m.k, m.tb, a, NC);
    return cudaGetLastError();
}

}  // namespace ccq

namespace ccq {

cudaError_t launch_gdn_chunk_only(const ChunkArgs &a, const GdnMaps &m, cudaStream_t s) {
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(gdn_chunk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(kSmemBytes));
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    gdn_chunk_kernel<<<a.B * a.H * a.nseg, kThreads, kSmemBytes, s>>>(m.q, m.k, m.v, m.tb, m.o, a);
    return cudaGetLastError();
}

cudaError_t launch_gdn_chunk(const ChunkArgs &a, const GdnMaps &m, cudaStream_t s) {
    cudaError_t e = launch_gdn_wy(a, m, s);
    if (e != cudaSuccess) return e;
    return launch_gdn_chunk_only(a, m, s);
}

size_t gdn_workspace_bytes(int B, int T, int H) {
    const size_t nc = static_cast<size_t>((T + kC - 1) / kC);
    return static_cast<size_t>(B) * H * nc * kC * kC * sizeof(__nv_bfloat16);
}

}  // namespace ccq
