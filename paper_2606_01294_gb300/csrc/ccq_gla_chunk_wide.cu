// ccq_gla_chunk_wide.cu -- chunkwise CCQ-GLA forward on sm_103a tensor cores for strongly
// forgetting gates (algo CCQ_ALGO_CHUNKWISE_WIDE).
//
// The default kernel (ccq_gla_chunk.cu) measures every gate factor of a chunk from one
// reference, the chunk midpoint, which is exact while each 32-token half of a chunk sums its
// log gates to more than about -82 per key dimension.  This kernel gives each half of the
// chunk its own reference, so that no factor spans more than 16 tokens of decay, at the price
// of a 96-row key tile, a second query tile and two more warps (about twice the time of the
// default kernel on the 4K workload).
//
// One CTA per (batch, head) walks the 64-token chunks of Algorithm 1
// (Dk = Dv = 128).  The two recurrent states stay in tensor memory as fp32
// accumulators for the whole sequence:
//   S   [Dk lanes][Dv cols]   the GLA state, transposed (S[a][e]), kept as
//                             X = Diag(e^{G47}) S_r + ... between chunks (below)
//   SK  [Dk lanes][Dk cols]   the undecayed key second-moment sum S^K (App. B)
// and every product of a chunk is a tcgen05.mma with bf16 operands in
// 128-byte-swizzled shared-memory tiles (q, k, v loaded by TMA):
//
//   group A  G2  Sc  = Q Kbar^T                   (CCQ intra scores, raw q)
//            G1  P   = Q S^K                      (CCQ inter read, App. B P^prev)
//   group B  G3  P  += W Kbar                     (CCQ intra read with the mean fold)
//   group C  G4  A'  = Qg K'^T                    (gated GLA scores, two references)
//            G6  O   = Qe S_r                     (GLA inter read)
//   group S  G7  X  += K47^T V                    (GLA state update)
//            G8  S^K += Kbar^T Kbar               (second-moment update)
//   group D  G5  O  += [j<=i] A V                 (GLA intra read)
//
// Notation (chunk r, positions t_i = t_r + i + 1, rq_i = 1/|q_i|):
//   cq_i = CumK_i . qbar_i = M . qbar_i + rq_i sum_{j<=i} Sc_ij,   c_i = cq_i / t_i,
//   W_ij = [j<=i] (Sc_ij - c_i |q_i|), so that rq_i P_i = S^K qbar_i
//   + sum_{j<=i} (qbar_i . kbar_j - c_i) kbar_j and
//   D (P^prev + P^intra) - MeanCorr = (rq_i P_i - c_i M) / t_i     (App. B, re-associated)
//   q_clean_i = qbar_i - lambda_i (rq_i P_i - c_i M) / t_i          (Eq. clean)
//
// Gate factors.  G_i is the in-chunk cumulative log gate (per key dimension, non-increasing).
// The GLA terms need e^{G_i - G_j} (j <= i, intra), e^{G_i} (inter read) and e^{G63 - G_j}
// (state write), all at most 1, but the intra scores must factor into a query side and a key
// side.  Each half of the chunk has its own reference, token 15 for rows 0-31 and token 47
// for rows 32-63:
//   Qg_i = q_clean_i e^{G_i - G_ref(i)}             (|G_i - G_ref| spans at most 16 tokens)
//   K'   = [ kbar_j e^{G15 - G_j}, j < 32  ;  kbar_j e^{G47 - G_j}, j < 64 ]   (96 rows)
//   A_ij = Qg_i . K'_(row of j for ref(i))           (G4: N = 96, each half reads its block)
// so no factor spans more than 16 tokens of decay: the kernel is exact (up to rounding) while
// every 16 consecutive log gates of a chunk sum to more than about -87 per key dimension
// (about -5.4 per token), and records CCQ_ERR_RANGE in the status word otherwise.  The inter
// read uses Qe_i = q_clean_i e^{G_i} (at most 1) against the unscaled S_r, and the state
// carries X = e^{G47} S_r + K47^T V (K47 the rows of K' with reference 47) with
// S_{r+1} = e^{G63 - G47} X applied when the next chunk's snapshot is taken.
//
// Warp specialisation (14 warps):
//   EPI   (warps 0-7)   the epilogues of chunk r -- W, q_clean, mask of A, output --
//                       and the bf16 operand copies of the states, placed where EPI
//                       would otherwise wait on an MMA: S^K_{r+1} while G4 runs,
//                       S_{r+1} (rescaling X in TMEM) while G2 of chunk r+1 runs.  The
//                       64-row products are M = 64 MMAs (rows 16q..16q+15 in TMEM lanes
//                       32q..32q+15); warps w and w+4 share lane quadrant q = w % 4 and
//                       split its columns.
//   PREP  (warps 8-11)  chunk r+1 while the chain runs chunk r: the gates (read from
//                       global memory), row norms, kbar, e^{G - G_ref}, M . qbar, lambda;
//                       then, once G4 of chunk r has read it, the key tile K' of chunk r+1.
//   ISSUE (warp 12)     one thread issues every tcgen05.mma (and, unless COPY does,
//                       the per-chunk TMA copies), in the order G2 | G1 | G3 G8 | G7 |
//                       G4 G6 | G5, so that G1, G7 and G6 run under the epilogues.  An MMA
//                       instruction holds its issuing thread for its whole execution,
//                       which is why no epilogue thread issues.  EPI signals the issuer
//                       with named-barrier arrives; the issuer signals EPI with commits.
//   COPY  (warp 13)     in the COPY instance: the loads of chunk r+2, the store of O and the
//                       next v, plus an L2 prefetch of chunk r+2 (q, k, gates, v).
// q, k and the factor tile are double-buffered (two slots); the loads of chunk r+2 start as
// soon as chunk r's last MMA reader of the slot (G6) completes.  v and K' are
// single-buffered: v is reloaded once G5 of the previous chunk completes, K' rewritten once
// G4 of the previous chunk (the later of its two readers) completes.
// Rows past T load as zeros: zero keys add nothing to any sum, zero gates keep the
// cumulative gate, so the ragged tail needs no special arithmetic.
// With a.ckpt set, EPI also writes each chunk's checkpoint record for the backward
// (ccq_gla_bwd.cu): the S^K tile (one bulk copy), the image of the tile e^{G31} S_r (from
// registers) and the key sum; the last segment writes S_T there.
// With a.nseg > 1 every CTA walks one segment (a range of whole chunks) of one
// sequence, starting from the segment's initial states in a.seg_ws
// (ccq_gla_segment.cu); only the last segment writes the final states.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <type_traits>

#include "ccq_internal.h"
#include "sm100_ptx.cuh"

namespace ccq {

namespace {

constexpr int kC = 64;         // chunk length
constexpr int kD = 128;        // Dk = Dv
constexpr int kEpiThreads = 256;
constexpr int kPrepWarp0 = 8, kKpWarp0 = 12, kIssueWarp = 14, kCopyWarp = 15;
constexpr int kThreadsNoCopy = 32 * kCopyWarp;       // 480
constexpr int kThreadsCopy = 32 * (kCopyWarp + 1);    // 512
constexpr int kKpThreads = 32 * (kIssueWarp - kKpWarp0);  // 64
constexpr int kSyncCount = kEpiThreads + 32;          // EPI + the issuing warp
constexpr float kLog2e = 1.4426950408889634f;
// largest exponent (log2 units) a gate factor may have: a state accumulated over a chunk
// from keys scaled by up to 2^118 stays inside the fp32 range
constexpr float kMaxExp2 = 118.f;

// ---- shared memory map (bytes from the 1024-aligned base)
// two slots of per-chunk tiles, each [64 rows][128 cols] bf16 as two T64 tiles of 8 KB:
constexpr uint32_t SLOT_BYTES = 49152;
constexpr uint32_t SO_Q = 0;       // raw q, then Qg = q_clean e^{G - G_ref}
constexpr uint32_t SO_K = 16384;   // raw k, then kbar
constexpr uint32_t SO_EG = 32768;  // e^{G - G_ref}, then Qe = q_clean e^{G}
constexpr uint32_t OFF_KP = 98304;   // 24K  K' [96 rows][128 cols] as two T64 tiles of 12 KB
constexpr uint32_t KP_TILE = 12288;
constexpr uint32_t OFF_V = 122880;   // 16K  v; after G5 the output staging of the TMA store
constexpr uint32_t OFF_W = 139264;   // 8K   W, then the masked A ([64][64], one T64 tile)
constexpr uint32_t OFF_SK = 147456;  // 32K  bf16 S^K ([128][128], two T64 tiles of 16 KB)
constexpr uint32_t OFF_S = 180224;   // 32K  bf16 S_r ([128][128], two T64 tiles of 16 KB)
constexpr uint32_t OFF_MISC = 212992;
// misc: per-slot arrays (4096 B per slot)
constexpr uint32_t MS_BYTES = 5632;
constexpr uint32_t MS_RQ = 0;      // [64] 1/|q_i|
constexpr uint32_t MS_MQ = 256;    // [64] M . qbar_i
constexpr uint32_t MS_LT = 512;    // [64] lambda_i / t_i
constexpr uint32_t MS_RK = 768;    // [64] 1/|k_j|
constexpr uint32_t MS_ER0 = 1024;  // [128] e^{G15}
constexpr uint32_t MS_F = 1536;    // [128] e^{G63 - G47}
constexpr uint32_t MS_MST = 2048;  // [128] key sum M at the chunk start
constexpr uint32_t MS_ITI = 2560;  // [64] 1 / t_i
constexpr uint32_t MS_QN = 2816;   // [64] |q_i| (1 without the l2 norm)
constexpr uint32_t MS_ER1 = 3072;  // [128] e^{G47}
constexpr uint32_t MS_EMID = 3584; // [128] e^{G31} (checkpoint tiles)
constexpr uint32_t MS_G15 = 4096;  // [128] G15  (the reference gate sums, for the K' warps)
constexpr uint32_t MS_G31 = 4608;  // [128] G31
constexpr uint32_t MS_G47 = 5120;  // [128] G47
constexpr uint32_t M_DMP = 11264;  // [2][128] partial key sums of the chunk (prep)
constexpr uint32_t M_DMPREV = 12288; // [128] key sum of the previous chunk
constexpr uint32_t M_GT0 = 12800;  // [128] G31 (gate sum over tokens 0..31), prep scratch
constexpr uint32_t M_G47 = 13312;  // [128] G47 - G31, prep scratch
constexpr uint32_t M_BAR = 13824;  // mbarriers
constexpr uint32_t M_TMEM = 13952;
constexpr uint32_t M_ABORT = 13956;
constexpr uint32_t kMiscBytes = 14016;
constexpr uint32_t kSmemBytes = OFF_MISC + kMiscBytes + 1024;  // + alignment slack
static_assert(kSmemBytes <= 232448, "exceeds the 227 KB per-CTA limit");
static_assert(2 * SLOT_BYTES == OFF_KP && OFF_KP + 2 * KP_TILE == OFF_V, "tile map");
static_assert(2 * MS_BYTES == M_DMP, "misc map");

enum {
    BAR_IN0 = 0, BAR_IN1 = 1, BAR_V = 2, BAR_GA = 3, BAR_GB = 4, BAR_GK = 5, BAR_GC = 6,
    BAR_GC2 = 7, BAR_GD = 8, BAR_PREP0 = 9, BAR_PREP1 = 10, BAR_SNAPK = 11, BAR_SNAPS = 12,
    BAR_KP = 13, kNumBars = 14
};
static_assert(M_BAR + 8 * kNumBars <= M_TMEM, "barrier area");
// named barriers (0 is __syncthreads)
enum { NB_W = 1, NB_QC = 2, NB_MASK = 3, NB_OUT = 4, NB_PREP = 5, NB_EPI = 6, NB_KP = 7 };

// ---- tensor memory columns
constexpr uint32_t TM_S = 0;     // 128 cols
constexpr uint32_t TM_SK = 128;  // 128 cols
constexpr uint32_t TM_PO = 256;  // 128 cols: P, then O (M = 64 layout)
constexpr uint32_t TM_SA = 384;  // 96 cols: Sc (64), then A' (96) (M = 64 layout)
constexpr uint32_t kTmemCols = 512;

constexpr uint32_t ID_64x64_KK = make_idesc(64, 64, 0, 0);
constexpr uint32_t ID_64x96_KK = make_idesc(64, 96, 0, 0);
constexpr uint32_t ID_64x128_KK = make_idesc(64, 128, 0, 0);
constexpr uint32_t ID_64x128_KM = make_idesc(64, 128, 0, 1);
constexpr uint32_t ID_128x128_MM = make_idesc(128, 128, 1, 1);

__device__ __forceinline__ void store_row_chunk(uint8_t *tile, int row, int chunk, const float *w) {
    uint4 u;
    u.x = pack_bf16(w[0], w[1]);
    u.y = pack_bf16(w[2], w[3]);
    u.z = pack_bf16(w[4], w[5]);
    u.w = pack_bf16(w[6], w[7]);
    *reinterpret_cast<uint4 *>(tile + t64_chunk(row, chunk)) = u;
}

// The gate words of N tokens starting at t0 (dims d0, d0 + 1) of one thread: a bf16 pair or an
// fp32 pair; zero past the end of the sequence.  The loads are volatile
// so that they issue where they are written -- a chunk ahead of their use -- and are all in
// flight at once (plain read-only loads were scheduled next to their first use, in small
// batches, which exposed their latency on every chunk).
template <bool F32>
using GateWord = typename std::conditional<F32, uint64_t, uint32_t>::type;

template <bool F32, int N>
__device__ __forceinline__ void load_gate_words(GateWord<F32> (&g)[N], const void *gk, int b, int h, int T,
                                                int H, int t0, int d0) {
#pragma unroll
    for (int jj = 0; jj < N; ++jj) {
        const int t = t0 + jj;
        const int tt = t < T ? t : 0;  // an in-bounds address; the value is replaced below
        const size_t e = ((static_cast<size_t>(b) * T + tt) * H + h) * kD + d0;
        if constexpr (F32) {
            uint32_t lo, hi;
            asm volatile("ld.global.nc.v2.u32 {%0, %1}, [%2];" : "=r"(lo), "=r"(hi)
                         : "l"(static_cast<const float *>(gk) + e));
            g[jj] = t < T ? ((static_cast<uint64_t>(hi) << 32) | lo) : 0;
        } else {
            uint32_t lo;
            asm volatile("ld.global.nc.u32 %0, [%1];" : "=r"(lo) : "l"(static_cast<const __nv_bfloat16 *>(gk) + e));
            g[jj] = t < T ? lo : 0u;
        }
    }
}

// A gate word as an fp32 pair.
template <bool F32>
__device__ __forceinline__ uint64_t gate_pair(GateWord<F32> w) {
    if constexpr (F32) return w;
    else return f2_from_bf16x2(w);
}

template <bool COPY, bool GF32>
__global__ void __launch_bounds__(COPY ? kThreadsCopy : kThreadsNoCopy, 1)
gla_chunk_wide_kernel(const __grid_constant__ CUtensorMap map_q, const __grid_constant__ CUtensorMap map_k,
                 const __grid_constant__ CUtensorMap map_v, const __grid_constant__ CUtensorMap map_g,
                 const __grid_constant__ CUtensorMap map_o, const ChunkArgs a) {
    // the output barrier: EPI and the issuing warp, and the copy warp when there is one
    constexpr int kOutCount = kEpiThreads + (COPY ? 64 : 32);
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = smem_align1024(smem_raw);
    const uint32_t sb = smem_addr(sm);
    uint8_t *misc = sm + OFF_MISC;
    float *dmp = reinterpret_cast<float *>(misc + M_DMP);
    float *dmprev = reinterpret_cast<float *>(misc + M_DMPREV);
    float *gt0 = reinterpret_cast<float *>(misc + M_GT0);
    float *g47 = reinterpret_cast<float *>(misc + M_G47);
    uint64_t *bar = reinterpret_cast<uint64_t *>(misc + M_BAR);
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(misc + M_TMEM);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(misc + M_ABORT);
    auto slot_f = [&](int s, uint32_t off) {
        return reinterpret_cast<float *>(misc + s * MS_BYTES + off);
    };

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int bh = blockIdx.x / a.nseg, seg = blockIdx.x % a.nseg, b = bh / a.H, h = bh % a.H;
    const int T = a.T, H = a.H;
    const int NCt = (T + kC - 1) / kC;
    const int cb = a.nseg > 1 ? seg * a.seg_chunks : 0;  // first chunk of this CTA
    const int NC = a.nseg > 1 ? min(NCt, cb + a.seg_chunks) - cb : NCt;
    const bool last_seg = seg == a.nseg - 1;
    const float *segst = a.nseg > 1 ? a.seg_ws + static_cast<size_t>(blockIdx.x) * kSegFloats : nullptr;
    const float *S0 = segst ? segst : a.S0;
    const float *C0 = segst ? segst + kD * kD : a.C0;
    const float *m0 = segst ? segst + 2 * kD * kD : a.m0;
    const int64_t tseq0 = a.t0 ? a.t0[b] : 0;  // position before the sequence
    int *status = a.status;

    if (tid == 0) {
        for (int i = 0; i < kNumBars; ++i) mbar_init(&bar[i], 1);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 0) tmem_alloc(tmem_slot, kTmemCols);
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *tmem_slot;
    const uint32_t tq = tbase + (static_cast<uint32_t>(32 * (warp & 3)) << 16);  // warp's lane quadrant

    auto issue_in = [&](int r) {  // q and k of local chunk r into slot r & 1
        const int s = r & 1, tg = (cb + r) * kC;
        uint8_t *base = sm + s * SLOT_BYTES;
        uint64_t *bb = &bar[BAR_IN0 + s];
        mbar_arrive_expect_tx(bb, 4 * 8192);
        tma_load_4d(base + SO_Q, &map_q, bb, 0, h, tg, b);
        tma_load_4d(base + SO_Q + 8192, &map_q, bb, 64, h, tg, b);
        tma_load_4d(base + SO_K, &map_k, bb, 0, h, tg, b);
        tma_load_4d(base + SO_K + 8192, &map_k, bb, 64, h, tg, b);
        if (COPY && r + 2 < NC) {  // chunk r + 2 into L2, so that its loads hit there
            const int tp = tg + 2 * kC;
            tma_prefetch_l2_4d(&map_q, 0, h, tp, b);
            tma_prefetch_l2_4d(&map_q, 64, h, tp, b);
            tma_prefetch_l2_4d(&map_k, 0, h, tp, b);
            tma_prefetch_l2_4d(&map_k, 64, h, tp, b);
            tma_prefetch_l2_4d(&map_g, 0, h, tg + kC, b);  // read by the prep and K' warps a chunk later
        }
    };
    auto issue_v = [&](int r) {
        const int tg = (cb + r) * kC;
        mbar_arrive_expect_tx(&bar[BAR_V], 2 * 8192);
        tma_load_4d(sm + OFF_V, &map_v, &bar[BAR_V], 0, h, tg, b);
        tma_load_4d(sm + OFF_V + 8192, &map_v, &bar[BAR_V], 64, h, tg, b);
        if (COPY && r + 2 < NC) {
            tma_prefetch_l2_4d(&map_v, 0, h, tg + 2 * kC, b);
            tma_prefetch_l2_4d(&map_v, 64, h, tg + 2 * kC, b);
        }
    };

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
    } else if (warp < kKpWarp0) {
        const int wt = tid - 32 * kPrepWarp0;
        slot_f(0, MS_MST)[wt] = m0 ? m0[(segst ? 0 : static_cast<size_t>(bh) * kD) + wt] : 0.f;
        dmprev[wt] = 0.f;
    } else if (warp == kIssueWarp && lane == 0) {
        tma_prefetch_desc(&map_q);
        tma_prefetch_desc(&map_k);
        tma_prefetch_desc(&map_v);
        tma_prefetch_desc(&map_g);
        tma_prefetch_desc(&map_o);
        if (NC > 0) {
            issue_in(0);
            issue_v(0);
        }
        if (NC > 1) issue_in(1);
    }
    tc_fence_before();
    __syncthreads();

    if (warp < kPrepWarp0) {
        // =============================================================== EPI
        const int grp = warp >> 2;              // column group
        const int i = 16 * (warp & 3) + (lane & 15);  // chunk row owned by this thread
        const int hf = lane >> 4;               // column half
        const int row = 32 * (warp & 3) + lane;  // state row a (key dim) of the M = 128 layout
        const bool upper = (warp & 3) >= 2;     // rows 32-63: reference token 47
        uint8_t *ck_head = a.ckpt ? a.ckpt + static_cast<size_t>(bh) * ckpt_head_bytes(T) : nullptr;
        // bf16 copy of S^K (this thread: row a, columns 64 grp .. 64 grp + 63)
        auto snap_sk = [&]() {
            if (ck_head) {
                // the previous checkpoint copy must have read the tile before it changes
                if (tid == 0) tma_store_wait_read();
                named_bar(NB_EPI, kEpiThreads);
            }
            tc_fence_after();
#pragma unroll
            for (int cc = 0; cc < 2; ++cc) {
                float x[32];
                tmem_ld32(tq + TM_SK + 64 * grp + 32 * cc, x);
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4)
                    store_row_chunk(sm + OFF_SK + grp * 16384, row, 4 * cc + q4, x + 8 * q4);
            }
            fence_proxy_async_smem();
            tc_fence_before();
            named_bar(NB_EPI, kEpiThreads);
            if (tid == 0) mbar_arrive(&bar[BAR_SNAPK]);
        };
        // S_r = fs X (state row `row`): its bf16 copy for G6, e^{G47_r} S_r back into TMEM for
        // G7, and for a checkpoint the image of e^{G31_r} S_r plus the S^K tile and M_r
        auto snap_s = [&](int r, float fs, float er, float em) {
            uint8_t *rec = ck_head ? ck_head + static_cast<size_t>(cb + r) * kCkptChunkBytes : nullptr;
            const uint64_t fs2 = f2_make(fs, fs), er2 = f2_make(er, er), em2 = f2_make(em, em);
            tc_fence_after();
#pragma unroll
            for (int cc = 0; cc < 2; ++cc) {
                float x[32];
                tmem_ld32(tq + TM_S + 64 * grp + 32 * cc, x);
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) {
                    uint32_t w[4], wc[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const int k2 = 8 * q4 + 2 * e;
                        const uint64_t y2 = f2_mul(f2_make(x[k2], x[k2 + 1]), fs2);
                        w[e] = bf16x2_from_f2(y2);
                        wc[e] = bf16x2_from_f2(f2_mul(y2, em2));
                        const float2 t2 = f2_split(f2_mul(y2, er2));
                        x[k2] = t2.x;
                        x[k2 + 1] = t2.y;
                    }
                    const uint32_t off = grp * 16384 + t64_chunk(row, 4 * cc + q4);
                    *reinterpret_cast<uint4 *>(sm + OFF_S + off) = make_uint4(w[0], w[1], w[2], w[3]);
                    if (rec) *reinterpret_cast<uint4 *>(rec + 32768 + off) = make_uint4(wc[0], wc[1], wc[2], wc[3]);
                }
                tmem_st32(tq + TM_S + 64 * grp + 32 * cc, x);
            }
            tmem_wait_st();
            fence_proxy_async_smem();
            tc_fence_before();
            named_bar(NB_EPI, kEpiThreads);
            if (tid == 0) mbar_arrive(&bar[BAR_SNAPS]);
            if (rec) {
                if (grp == 0) reinterpret_cast<float *>(rec + 65536)[row] = slot_f(r & 1, MS_MST)[row];
                if (tid == 0) {
                    bulk_store(rec, sm + OFF_SK, 32768);
                    tma_store_commit();
                }
            }
        };
        float f_cur = 1.f;  // e^{G63 - G47} of the chunk in flight, state row `row`
        if (NC > 0) {
            mbar_wait(&bar[BAR_PREP0], 0, abort_flag, status);
            snap_sk();
            snap_s(0, 1.f, slot_f(0, MS_ER1)[row], slot_f(0, MS_EMID)[row]);
        }
        for (int r = 0; r < NC; ++r) {
            const int s = r & 1;
            const uint32_t sp = (r >> 1) & 1, par = r & 1;
            uint8_t *slot = sm + s * SLOT_BYTES;
            mbar_wait(&bar[BAR_PREP0 + s], sp, abort_flag, status);
            f_cur = slot_f(s, MS_F)[row];
            const float rqi = slot_f(s, MS_RQ)[i];
            const float mqi = slot_f(s, MS_MQ)[i];
            const float iti = slot_f(s, MS_ITI)[i];  // 1 / t_i
            const float qni = slot_f(s, MS_QN)[i];   // |q_i|
            const float lt = slot_f(s, MS_LT)[i];    // lambda_i / t_i
            // ---- W epilogue: c_i and W_ij = [j<=i](Sc_ij - c_i |q_i|)
            mbar_wait(&bar[BAR_GA], par, abort_flag, status);
            tc_fence_after();
            float c;
            {
                float sc[32];
                tmem_ld16x2_32<32>(tq + TM_SA, sc);  // row i, columns 32 hf .. 32 hf + 31
                float pa[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                for (int jj = 0; jj < 32; ++jj)
                    if (32 * hf + jj <= i) pa[jj & 3] += sc[jj];
                float part = (pa[0] + pa[1]) + (pa[2] + pa[3]);
                part += __shfl_xor_sync(0xffffffffu, part, 16);
                const float cq = mqi + rqi * part;
                c = a.centered ? cq * iti : 0.f;
                const float cn = c * qni;  // c_i |q_i|
#pragma unroll
                for (int q2 = 0; q2 < 2; ++q2) {
                    float w[8];
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        const int jj = 8 * q2 + e;
                        const float v = grp ? sc[16 + jj] : sc[jj];
                        w[e] = (32 * hf + 16 * grp + jj <= i) ? v - cn : 0.f;
                    }
                    store_row_chunk(sm + OFF_W, i, 4 * hf + 2 * grp + q2, w);
                }
            }
            fence_proxy_async_smem();
            tc_fence_before();
            named_bar_arrive(NB_W, kSyncCount);
            // ---- q_clean epilogue (Eq. clean): u = rq (q - (lambda/t) P) + (lambda c / t) M;
            // Qg = u e^{G - G_ref} into the Q tile, Qe = Qg e^{G_ref} = u e^{G} into the factor tile.
            // This thread: row i, columns 64 grp + 32 hf .. +31 (T64 tile grp, chunks 4 hf ..)
            {
                uint8_t *qt = slot + SO_Q + grp * 8192;
                uint8_t *et = slot + SO_EG + grp * 8192;
                const float *Mst = slot_f(s, MS_MST) + 64 * grp + 32 * hf;
                const float *Er = slot_f(s, upper ? MS_ER1 : MS_ER0) + 64 * grp + 32 * hf;
                uint4 qraw[4], eraw[4];
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) {
                    qraw[q4] = *reinterpret_cast<const uint4 *>(qt + t64_chunk(i, 4 * hf + q4));
                    eraw[q4] = *reinterpret_cast<const uint4 *>(et + t64_chunk(i, 4 * hf + q4));
                }
                mbar_wait(&bar[BAR_GB], par, abort_flag, status);
                tc_fence_after();
                const float cm = lt * c;  // lambda_i c_i / t_i
                float p[32];
                tmem_ld16x2_32<32>(tq + TM_PO + 64 * grp, p);
                const uint64_t nlt = f2_make(-lt, -lt), rq2 = f2_make(rqi, rqi), cm2 = f2_make(cm, cm);
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) {
                    const ulonglong2 m01 = *reinterpret_cast<const ulonglong2 *>(Mst + 8 * q4);
                    const ulonglong2 m23 = *reinterpret_cast<const ulonglong2 *>(Mst + 8 * q4 + 4);
                    const ulonglong2 e01 = *reinterpret_cast<const ulonglong2 *>(Er + 8 * q4);
                    const ulonglong2 e23 = *reinterpret_cast<const ulonglong2 *>(Er + 8 * q4 + 4);
                    const uint64_t mp[4] = {m01.x, m01.y, m23.x, m23.y};
                    const uint64_t rp[4] = {e01.x, e01.y, e23.x, e23.y};
                    const uint32_t qw[4] = {qraw[q4].x, qraw[q4].y, qraw[q4].z, qraw[q4].w};
                    const uint32_t ew[4] = {eraw[q4].x, eraw[q4].y, eraw[q4].z, eraw[q4].w};
                    uint32_t ow[4], xw[4];
#pragma unroll
                    for (int w = 0; w < 4; ++w) {
                        const uint64_t p2 = f2_make(p[8 * q4 + 2 * w], p[8 * q4 + 2 * w + 1]);
                        const uint64_t t = f2_fma(nlt, p2, f2_from_bf16x2(qw[w]));     // q - (lambda/t) P
                        const uint64_t u = f2_fma(rq2, t, f2_mul(cm2, mp[w]));          // rq (.) + (lambda c/t) M
                        const uint64_t g = f2_mul(f2_from_bf16x2(ew[w]), u);            // * e^{G - G_ref}
                        ow[w] = bf16x2_from_f2(g);
                        xw[w] = bf16x2_from_f2(f2_mul(g, rp[w]));                     // * e^{G_ref}
                    }
                    *reinterpret_cast<uint4 *>(qt + t64_chunk(i, 4 * hf + q4)) = make_uint4(ow[0], ow[1], ow[2], ow[3]);
                    *reinterpret_cast<uint4 *>(et + t64_chunk(i, 4 * hf + q4)) = make_uint4(xw[0], xw[1], xw[2], xw[3]);
                }
            }
            fence_proxy_async_smem();
            tc_fence_before();
            named_bar_arrive(NB_QC, kSyncCount);
            // ---- S^K_{r+1} while G4 runs (G8 of chunk r has run, after its G1 read)
            if (r + 1 < NC) {
                mbar_wait(&bar[BAR_GK], par, abort_flag, status);
                snap_sk();
            }
            // ---- causal mask of A: rows 0-31 read the reference-15 block (columns 0-31 of A'),
            // rows 32-63 the reference-47 block (columns 32-95)
            mbar_wait(&bar[BAR_GC], par, abort_flag, status);
            tc_fence_after();
            {
                float sc[32];
                tmem_ld16x2_32<32>(tq + TM_SA + (upper ? 32 : 0), sc);
#pragma unroll
                for (int q2 = 0; q2 < 2; ++q2) {
                    float w[8];
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        const int jj = 8 * q2 + e;
                        const float v = grp ? sc[16 + jj] : sc[jj];
                        w[e] = (32 * hf + 16 * grp + jj <= i) ? v : 0.f;
                    }
                    store_row_chunk(sm + OFF_W, i, 4 * hf + 2 * grp + q2, w);
                }
            }
            fence_proxy_async_smem();
            tc_fence_before();
            named_bar_arrive(NB_MASK, kSyncCount);
            // ---- output: o = scale O staged (bf16, swizzled) in the v tile, which G5 has
            // finished reading; the issuing thread stores it with one TMA copy (rows past T
            // fall outside the tensor and are not written)
            mbar_wait(&bar[BAR_GD], par, abort_flag, status);
            tc_fence_after();
            if (!a.skip_o) {
                float x[32];
                tmem_ld16x2_32<32>(tq + TM_PO + 64 * grp, x);
                const uint64_t sc2 = f2_make(a.scale, a.scale);
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) {
                    uint32_t w[4];
#pragma unroll
                    for (int u = 0; u < 4; ++u)
                        w[u] = bf16x2_from_f2(f2_mul(f2_make(x[8 * q4 + 2 * u], x[8 * q4 + 2 * u + 1]), sc2));
                    *reinterpret_cast<uint4 *>(sm + OFF_V + grp * 8192 + t64_chunk(i, 4 * hf + q4)) = make_uint4(w[0], w[1], w[2], w[3]);
                }
                fence_proxy_async_smem();
            }
            tc_fence_before();
            named_bar_arrive(NB_OUT, kOutCount);
            // ---- S_{r+1} while G2 of chunk r+1 runs (G6 and G7 of chunk r have run: GD
            // follows them)
            if (r + 1 < NC) {
                mbar_wait(&bar[BAR_PREP0 + (s ^ 1)], ((r + 1) >> 1) & 1, abort_flag, status);
                snap_s(r + 1, f_cur, slot_f(s ^ 1, MS_ER1)[row], slot_f(s ^ 1, MS_EMID)[row]);
            }
        }
        if (ck_head && tid == 0) tma_store_wait_all();
        // final states: S_T = e^{G63 - G47} X (last chunk), S^K
        if (NC > 0 && last_seg) {
            tc_fence_after();
            const float fs = f_cur;
            const size_t bhs = static_cast<size_t>(bh);
#pragma unroll
            for (int cc = 0; cc < 2; ++cc) {
                const int c = 2 * grp + cc;
                float x[32];
                tmem_ld32(tq + TM_S + 32 * c, x);
                if (a.ST) {
                    float4 *dst = reinterpret_cast<float4 *>(a.ST + (bhs * kD + row) * kD + 32 * c);
#pragma unroll
                    for (int e = 0; e < 8; ++e)
                        dst[e] = make_float4(fs * x[4 * e], fs * x[4 * e + 1], fs * x[4 * e + 2],
                                             fs * x[4 * e + 3]);
                }
                if (ck_head) {
                    float4 *dst = reinterpret_cast<float4 *>(
                        ck_head + static_cast<size_t>(NCt) * kCkptChunkBytes + (static_cast<size_t>(row) * kD + 32 * c) * 4);
#pragma unroll
                    for (int e = 0; e < 8; ++e)
                        dst[e] = make_float4(fs * x[4 * e], fs * x[4 * e + 1], fs * x[4 * e + 2],
                                             fs * x[4 * e + 3]);
                }
                tmem_ld32(tq + TM_SK + 32 * c, x);
                if (a.CT) {
                    float4 *dst = reinterpret_cast<float4 *>(a.CT + (bhs * kD + row) * kD + 32 * c);
#pragma unroll
                    for (int e = 0; e < 8; ++e) dst[e] = make_float4(x[4 * e], x[4 * e + 1], x[4 * e + 2], x[4 * e + 3]);
                }
            }
        }
    } else if (warp < kKpWarp0) {
        // =============================================================== PREP
        const int wt = tid - 32 * kPrepWarp0;
        const int p = wt & 63, th = wt >> 6;  // key-dim pair (2p, 2p+1), token half
        const int d0 = 2 * p;
        const uint32_t tcol = (d0 >> 6) * 8192;     // T64 tile of dims d0, d0+1 (q, k, factors)
        float lam_reg = 0.f;  // lambda of row wt >> 1
        {
            const int tn = cb * kC + (wt >> 1);
            lam_reg = (tn < T) ? a.lambda[(static_cast<size_t>(b) * T + tn) * H + h] : 0.f;
        }
        // gate words of the chunk being prepared (loaded one chunk ahead), then its cumulative
        // gates within this thread's token half, as fp32 pairs
        GateWord<GF32> gw[32];
        uint64_t g2[32];
        if (NC > 0) load_gate_words<GF32>(gw, a.gk, b, h, T, H, cb * kC + 32 * th, d0);
        float emax = 0.f;  // largest |exponent| (log2 units) of a factor met
        const uint64_t l2e = f2_make(kLog2e, kLog2e);
        for (int r = 0; r < NC; ++r) {
            const int s = r & 1;
            const uint32_t sp = (r >> 1) & 1;
            uint8_t *slot = sm + s * SLOT_BYTES;
            float *Mst = slot_f(s, MS_MST);
            mbar_wait(&bar[BAR_IN0 + s], sp, abort_flag, status);
            // key sum at the chunk start and lambda of the chunk
            if (r > 0) Mst[wt] = slot_f(s ^ 1, MS_MST)[wt] + dmprev[wt];
            const float lam_cur = lam_reg;
            {
                const int tn = (cb + r + 1) * kC + (wt >> 1);
                lam_reg = (tn < T) ? a.lambda[(static_cast<size_t>(b) * T + tn) * H + h] : 0.f;
            }
            named_bar(NB_PREP, 128);
            // row norms of q and k and M . q: thread pair (2j, 2j+1) takes row j, each
            // thread one 64-column half (one T64 tile) of both q and k, in fp32 pairs
            {
                // (q and k in turn, which keeps half as many registers live beside the gate words
                // of the next chunk)
                const int j = wt >> 1, hh = wt & 1;
                const float *Mh = Mst + 64 * hh;
                uint64_t sq0 = 0, sq1 = 0, sk0 = 0, sk1 = 0, md0 = 0, md1 = 0;
                {
                    uint4 qv[8];
#pragma unroll
                    for (int cc = 0; cc < 8; ++cc)
                        qv[cc] = *reinterpret_cast<const uint4 *>(slot + SO_Q + hh * 8192 + t64_chunk(j, cc));
#pragma unroll
                    for (int cc = 0; cc < 8; ++cc) {
                        const ulonglong2 m01 = *reinterpret_cast<const ulonglong2 *>(Mh + 8 * cc);
                        const ulonglong2 m23 = *reinterpret_cast<const ulonglong2 *>(Mh + 8 * cc + 4);
                        const uint32_t qw[4] = {qv[cc].x, qv[cc].y, qv[cc].z, qv[cc].w};
                        const uint64_t mp[4] = {m01.x, m01.y, m23.x, m23.y};
#pragma unroll
                        for (int w = 0; w < 4; ++w) {
                            const uint64_t q2 = f2_from_bf16x2(qw[w]);
                            if (w & 1) {
                                sq1 = f2_fma(q2, q2, sq1); md1 = f2_fma(q2, mp[w], md1);
                            } else {
                                sq0 = f2_fma(q2, q2, sq0); md0 = f2_fma(q2, mp[w], md0);
                            }
                        }
                    }
                }
                {
                    uint4 kv[8];
#pragma unroll
                    for (int cc = 0; cc < 8; ++cc)
                        kv[cc] = *reinterpret_cast<const uint4 *>(slot + SO_K + hh * 8192 + t64_chunk(j, cc));
#pragma unroll
                    for (int cc = 0; cc < 8; ++cc) {
                        const uint32_t kw[4] = {kv[cc].x, kv[cc].y, kv[cc].z, kv[cc].w};
#pragma unroll
                        for (int w = 0; w < 4; ++w) {
                            const uint64_t k2 = f2_from_bf16x2(kw[w]);
                            if (w & 1) sk1 = f2_fma(k2, k2, sk1);
                            else sk0 = f2_fma(k2, k2, sk0);
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
                    const float iti = 1.f / static_cast<float>(tseq0 + (cb + r) * kC + j + 1);
                    slot_f(s, MS_RQ)[j] = rq;
                    slot_f(s, MS_MQ)[j] = mdt * rq;
                    slot_f(s, MS_ITI)[j] = iti;
                    slot_f(s, MS_QN)[j] = a.l2norm ? fmaxf(ssq, 1e-12f) * rq : 1.f;
                    slot_f(s, MS_LT)[j] = lam_cur * iti;
                } else {
                    slot_f(s, MS_RK)[j] = a.l2norm ? rsqrtf(fmaxf(ssk, 1e-12f)) : 1.f;
                }
            }
            // cumulative gates of this thread's 32 tokens: G_j (th 0) or G_j - G31 (th 1)
            {
                uint64_t r2 = 0;  // (0.f, 0.f)
#pragma unroll
                for (int jj = 0; jj < 32; ++jj) {
                    r2 = f2_add(r2, gate_pair<GF32>(gw[jj]));
                    g2[jj] = r2;
                }
                const float2 rv = th ? f2_split(g2[15]) : f2_split(r2);
                float *dst = th ? g47 : gt0;  // G47 - G31, or G31
                dst[d0] = rv.x;
                dst[d0 + 1] = rv.y;
                if (th == 0) {
                    const float2 l15 = f2_split(g2[15]);
                    slot_f(s, MS_G15)[d0] = l15.x;
                    slot_f(s, MS_G15)[d0 + 1] = l15.y;
                    slot_f(s, MS_G31)[d0] = rv.x;
                    slot_f(s, MS_G31)[d0 + 1] = rv.y;
                }
            }
            named_bar(NB_PREP, 128);  // norms, G31 and G47 visible
            const float2 l15 = f2_split(g2[15]);  // G15 (th 0) or G47 - G31 (th 1)
            {
                const float2 l31 = f2_split(g2[31]);
                if (th == 0) {
                    slot_f(s, MS_ER0)[d0] = fast_exp2(l15.x * kLog2e);
                    slot_f(s, MS_ER0)[d0 + 1] = fast_exp2(l15.y * kLog2e);
                    slot_f(s, MS_EMID)[d0] = fast_exp2(l31.x * kLog2e);
                    slot_f(s, MS_EMID)[d0 + 1] = fast_exp2(l31.y * kLog2e);
                } else {
                    slot_f(s, MS_ER1)[d0] = fast_exp2((gt0[d0] + l15.x) * kLog2e);
                    slot_f(s, MS_ER1)[d0 + 1] = fast_exp2((gt0[d0 + 1] + l15.y) * kLog2e);
                    slot_f(s, MS_G47)[d0] = gt0[d0] + l15.x;
                    slot_f(s, MS_G47)[d0 + 1] = gt0[d0 + 1] + l15.y;
                    slot_f(s, MS_F)[d0] = fast_exp2((l31.x - l15.x) * kLog2e);
                    slot_f(s, MS_F)[d0 + 1] = fast_exp2((l31.y - l15.y) * kLog2e);
                }
            }
            {
                // kbar (in place), e^{G - G_ref} and the chunk's key sum: four batches of eight
                // tokens, every load of a batch issued before its stores (the in-place kbar
                // store may alias a later load)
                const uint64_t ref2 = f2_make(-l15.x * kLog2e, -l15.y * kLog2e);
                const float *rk = slot_f(s, MS_RK);
                uint64_t dm2 = 0;
#pragma unroll
                for (int bt = 0; bt < 4; ++bt) {
                    uint32_t kraw[8];
#pragma unroll
                    for (int u = 0; u < 8; ++u) {
                        const int j = 32 * th + 8 * bt + u;
                        kraw[u] = *reinterpret_cast<const uint32_t *>(slot + SO_K + tcol + t64_offset(j, d0 & 63));
                    }
                    const float4 rka = *reinterpret_cast<const float4 *>(rk + 32 * th + 8 * bt);
                    const float4 rkb = *reinterpret_cast<const float4 *>(rk + 32 * th + 8 * bt + 4);
                    const float rkv[8] = {rka.x, rka.y, rka.z, rka.w, rkb.x, rkb.y, rkb.z, rkb.w};
#pragma unroll
                    for (int u = 0; u < 8; ++u) {
                        const int jj = 8 * bt + u, j = 32 * th + jj;
                        const uint32_t off = tcol + t64_offset(j, d0 & 63);
                        const uint64_t k2 = f2_mul(f2_from_bf16x2(kraw[u]), f2_make(rkv[u], rkv[u]));
                        const float2 x = f2_split(f2_fma(g2[jj], l2e, ref2));  // (G_j - G_ref) log2(e)
                        emax = fmaxf(emax, fmaxf(fabsf(x.x), fabsf(x.y)));
                        *reinterpret_cast<uint32_t *>(slot + SO_K + off) = bf16x2_from_f2(k2);
                        *reinterpret_cast<uint32_t *>(slot + SO_EG + off) = pack_bf16(fast_exp2(x.x), fast_exp2(x.y));
                        dm2 = f2_add(dm2, k2);
                    }
                }
                const float2 dmv = f2_split(dm2);
                dmp[th * kD + d0] = dmv.x;
                dmp[th * kD + d0 + 1] = dmv.y;
            }
            fence_proxy_async_smem();
            named_bar(NB_PREP, 128);
            dmprev[wt] = dmp[wt] + dmp[kD + wt];
            if (wt == 0) mbar_arrive(&bar[BAR_PREP0 + s]);
            // the gate words of the next chunk, in flight while this warp waits for its q and k
            if (r + 1 < NC) load_gate_words<GF32>(gw, a.gk, b, h, T, H, (cb + r + 1) * kC + 32 * th, d0);
        }
        // a factor beyond 2^kMaxExp2 (16 tokens of decay stronger than about e^-82) cannot be
        // represented: report it rather than return silently wrong values
        if (emax > kMaxExp2) atomicExch(status, kStatusRange);
        // final key sum
        if (NC > 0 && a.mT && last_seg) {
            const int sl = (NC - 1) & 1;
            a.mT[static_cast<size_t>(bh) * kD + wt] = slot_f(sl, MS_MST)[wt] + dmprev[wt];
        }
    } else if (warp < kIssueWarp) {
        // =============================================================== K'
        // The key tile K' of chunk r, once the prep has normalised its keys (and published the
        // reference gate sums G15, G31, G47) and G4 of chunk r-1, the later of K's two readers,
        // has run.  Thread: dims d0, d0 + 1 over all 64 tokens, the cumulative gates G_j
        // recomputed from the gate words in fp32 as the prep computes them.
        const int kt = tid - 32 * kKpWarp0;
        const int d0 = 2 * kt;
        const uint32_t tcol = (d0 >> 6) * 8192, kcol = (d0 >> 6) * KP_TILE;
        const uint64_t nl2e = f2_make(-kLog2e, -kLog2e);
        float emax = 0.f;
        GateWord<GF32> gw[32];  // gate words of one half of the chunk
        if (NC > 0) load_gate_words<GF32>(gw, a.gk, b, h, T, H, cb * kC, d0);
        for (int r = 0; r < NC; ++r) {
            const int s = r & 1;
            const uint32_t sp = (r >> 1) & 1;
            const uint8_t *slot = sm + s * SLOT_BYTES;
            mbar_wait(&bar[BAR_PREP0 + s], sp, abort_flag, status);
            if (r > 0) mbar_wait(&bar[BAR_GC], (r - 1) & 1, abort_flag, status);
            const uint64_t r15 = f2_make(slot_f(s, MS_G15)[d0] * kLog2e, slot_f(s, MS_G15)[d0 + 1] * kLog2e);
            const uint64_t r47 = f2_make(slot_f(s, MS_G47)[d0] * kLog2e, slot_f(s, MS_G47)[d0 + 1] * kLog2e);
            uint64_t run = 0;  // G_j (fp32 pair)
#pragma unroll 1
            for (int half = 0; half < 2; ++half) {
                if (half == 1) load_gate_words<GF32>(gw, a.gk, b, h, T, H, (cb + r) * kC + 32, d0);
#pragma unroll
                for (int jj = 0; jj < 32; ++jj) {
                    const int j = 32 * half + jj;
                    run = f2_add(run, gate_pair<GF32>(gw[jj]));
                    const uint64_t kb =
                        f2_from_bf16x2(*reinterpret_cast<const uint32_t *>(slot + SO_K + tcol + t64_offset(j, d0 & 63)));
                    // (G_ref - G_j) log2(e): reference 15 for keys 0-31 (row j), 47 for all keys
                    // (row 32 + j)
                    const float2 x4 = f2_split(f2_fma(run, nl2e, r47));
                    *reinterpret_cast<uint32_t *>(sm + OFF_KP + kcol + t64_offset(32 + j, d0 & 63)) =
                        bf16x2_from_f2(f2_mul(kb, f2_make(fast_exp2(x4.x), fast_exp2(x4.y))));
                    if (half == 0) {
                        const float2 x = f2_split(f2_fma(run, nl2e, r15));
                        emax = fmaxf(emax, fmaxf(fabsf(x.x), fabsf(x.y)));
                        *reinterpret_cast<uint32_t *>(sm + OFF_KP + kcol + t64_offset(j, d0 & 63)) =
                            bf16x2_from_f2(f2_mul(kb, f2_make(fast_exp2(x.x), fast_exp2(x.y))));
                    } else {
                        emax = fmaxf(emax, fmaxf(fabsf(x4.x), fabsf(x4.y)));
                    }
                }
            }
            fence_proxy_async_smem();
            named_bar(NB_KP, kKpThreads);
            if (kt == 0) mbar_arrive(&bar[BAR_KP]);
            if (r + 1 < NC) load_gate_words<GF32>(gw, a.gk, b, h, T, H, (cb + r + 1) * kC, d0);
        }
        if (emax > kMaxExp2) atomicExch(status, kStatusRange);
    } else if (warp == kIssueWarp) {
        // =============================================================== ISSUE
        const bool lead = lane == 0;
        // descriptor bases (start-address field advanced per K slice: +2 per 32 B)
        const uint64_t dW = make_desc(sb + OFF_W, 16, 1024);
        const uint64_t dSK = make_desc(sb + OFF_SK, 16, 1024);
        const uint64_t dS = make_desc(sb + OFF_S, 16384, 1024);
        const uint64_t dV = make_desc(sb + OFF_V, 8192, 1024);
        const uint64_t dKP = make_desc(sb + OFF_KP, 16, 1024);                 // K', K-major (N = 96)
        const uint64_t dK47m = make_desc(sb + OFF_KP + 32 * 128, KP_TILE, 1024);  // rows 32-95, MN-major
        for (int r = 0; r < NC; ++r) {
            const int s = r & 1;
            const uint32_t sp = (r >> 1) & 1, par = r & 1;
            const uint32_t ss = sb + s * SLOT_BYTES;
            const uint64_t dQ = make_desc(ss + SO_Q, 16, 1024);
            const uint64_t dK = make_desc(ss + SO_K, 16, 1024);
            const uint64_t dKm = make_desc(ss + SO_K, 8192, 1024);
            const uint64_t dE = make_desc(ss + SO_EG, 16, 1024);
            mbar_wait(&bar[BAR_PREP0 + s], sp, abort_flag, status);
            tc_fence_after();
            // G2 Sc = Q Kbar^T (SA is free: the mask epilogue of chunk r-1 has read A)
            if (lead && !*abort_flag) {
                for (int k = 0; k < 8; ++k) {
                    const uint64_t ko = (k >> 2) * 512 + (k & 3) * 2;
                    mma_bf16(tbase + TM_SA, dQ + ko, dK + ko, ID_64x64_KK, k != 0);
                }
                mma_commit(&bar[BAR_GA]);
            }
            __syncwarp();
            if (r > 0) {
                // O of chunk r-1 has left PO (staged in the v tile): store it (unless the copy
                // warp does)
                mbar_wait(&bar[BAR_GD], (r - 1) & 1, abort_flag, status);
                named_bar(NB_OUT, kOutCount);
                if (lead && !COPY && !a.skip_o) {
                    const int cp = (cb + r - 1) * kC;
                    tma_store_4d(&map_o, sm + OFF_V, 0, h, cp, b);
                    tma_store_4d(&map_o, sm + OFF_V + 8192, 64, h, cp, b);
                    tma_store_commit();
                }
                __syncwarp();
            }
            // G1 P = Q S^K
            mbar_wait(&bar[BAR_SNAPK], par, abort_flag, status);
            tc_fence_after();
            if (lead && !*abort_flag)
                for (int k = 0; k < 8; ++k)
                    mma_bf16(tbase + TM_PO, dQ + (k >> 2) * 512 + (k & 3) * 2,
                             dSK + (k >> 2) * 1024 + (k & 3) * 2, ID_64x128_KK, k != 0);
            // v of chunk r replaces the staged output once the store has read it
            if (r > 0 && lead && !COPY) {
                tma_store_wait_read();
                if (!*abort_flag) issue_v(r);
            }
            __syncwarp();
            // G3 P += W Kbar, then G8 S^K += Kbar^T Kbar
            named_bar(NB_W, kSyncCount);
            tc_fence_after();
            if (lead && !*abort_flag) {
                for (int k = 0; k < 4; ++k)
                    mma_bf16(tbase + TM_PO, dW + k * 2, dKm + k * 128, ID_64x128_KM, 1);
                mma_commit(&bar[BAR_GB]);
                for (int k = 0; k < 4; ++k)
                    mma_bf16(tbase + TM_SK, dKm + k * 128, dKm + k * 128, ID_128x128_MM, 1);
                mma_commit(&bar[BAR_GK]);
            }
            __syncwarp();
            // G7 X += K47^T V (X rescaled by the snapshot of chunk r; v and K' landed)
            mbar_wait(&bar[BAR_SNAPS], par, abort_flag, status);
            mbar_wait(&bar[BAR_V], par, abort_flag, status);
            mbar_wait(&bar[BAR_KP], par, abort_flag, status);
            tc_fence_after();
            if (lead && !*abort_flag)
                for (int k = 0; k < 4; ++k)
                    mma_bf16(tbase + TM_S, dK47m + k * 128, dV + k * 128, ID_128x128_MM, 1);
            __syncwarp();
            // G4 A' = Qg K'^T (N = 96), G6 O = Qe S_r
            named_bar(NB_QC, kSyncCount);
            tc_fence_after();
            if (lead && !*abort_flag) {
                for (int k = 0; k < 8; ++k) {
                    const uint64_t ko = (k >> 2) * 512 + (k & 3) * 2;
                    const uint64_t kp = (k >> 2) * (KP_TILE >> 4) + (k & 3) * 2;
                    mma_bf16(tbase + TM_SA, dQ + ko, dKP + kp, ID_64x96_KK, k != 0);
                }
                mma_commit(&bar[BAR_GC]);
                for (int k = 0; k < 8; ++k)
                    mma_bf16(tbase + TM_PO, dE + (k >> 2) * 512 + (k & 3) * 2, dS + k * 128, ID_64x128_KM,
                             k != 0);
                mma_commit(&bar[BAR_GC2]);
            }
            __syncwarp();
            // G5 O += A V
            named_bar(NB_MASK, kSyncCount);
            tc_fence_after();
            if (lead && !*abort_flag) {
                for (int k = 0; k < 4; ++k)
                    mma_bf16(tbase + TM_PO, dW + k * 2, dV + k * 128, ID_64x128_KM, 1);
                mma_commit(&bar[BAR_GD]);
            }
            __syncwarp();
            // the slot's last MMA reader (G6) is done: load chunk r + 2 into it
            if (!COPY && r + 2 < NC) {
                mbar_wait(&bar[BAR_GC2], par, abort_flag, status);
                if (lead && !*abort_flag) issue_in(r + 2);
                __syncwarp();
            }
        }
        if (NC > 0) {
            mbar_wait(&bar[BAR_GD], (NC - 1) & 1, abort_flag, status);
            named_bar(NB_OUT, kOutCount);
            if (lead && !COPY && !a.skip_o) {
                const int cp = (cb + NC - 1) * kC;
                tma_store_4d(&map_o, sm + OFF_V, 0, h, cp, b);
                tma_store_4d(&map_o, sm + OFF_V + 8192, 64, h, cp, b);
                tma_store_commit();
            }
            if (lead) tma_store_wait_all();
            // after a give-up, wait (bounded) for the copies still in flight
            if (lead && *abort_flag) {
                mbar_drain(&bar[BAR_V], (NC - 1) & 1);
                for (int r = (NC > 2 ? NC - 2 : 0); r < NC; ++r) mbar_drain(&bar[BAR_IN0 + (r & 1)], (r >> 1) & 1);
            }
        }
    } else {
        // =============================================================== COPY
        // The per-chunk copies, which can hold a thread for a thousand
        // cycles while the copy engine is busy -- the loads of chunk r + 2 once G6 of chunk r
        // has read the slot, the store of O (staged in the v tile), the next v once that
        // store has read it (the instance without this warp has the issuer make them).
        const bool lead = lane == 0;
        for (int r = 0; r < NC; ++r) {
            if (COPY && r + 2 < NC) {
                mbar_wait(&bar[BAR_GC2], r & 1, abort_flag, status);
                if (lead && !*abort_flag) issue_in(r + 2);
                __syncwarp();
            }
            named_bar(NB_OUT, kOutCount);  // O of chunk r staged in the v tile
            if (lead && COPY) {
                if (!a.skip_o) {
                    const int cp = (cb + r) * kC;
                    tma_store_4d(&map_o, sm + OFF_V, 0, h, cp, b);
                    tma_store_4d(&map_o, sm + OFF_V + 8192, 64, h, cp, b);
                    tma_store_commit();
                }
                if (r + 1 < NC) {
                    tma_store_wait_read();
                    if (!*abort_flag) issue_v(r + 1);
                }
            }
            __syncwarp();
        }
        if (lead) tma_store_wait_all();
        if (lead && COPY && NC > 0 && *abort_flag) {
            mbar_drain(&bar[BAR_V], (NC - 1) & 1);
            for (int r = (NC > 2 ? NC - 2 : 0); r < NC; ++r) mbar_drain(&bar[BAR_IN0 + (r & 1)], (r >> 1) & 1);
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

template <bool COPY, bool GF32>
static cudaError_t launch_one(const ChunkArgs &a, const ChunkMaps &m, cudaStream_t s) {
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(gla_chunk_wide_kernel<COPY, GF32>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(kSmemBytes));
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    const int grid = COPY ? a.B * a.H : a.B * a.H * a.nseg;
    gla_chunk_wide_kernel<COPY, GF32><<<grid, COPY ? kThreadsCopy : kThreadsNoCopy, kSmemBytes, s>>>(m.q, m.k, m.v, m.g,
                                                                                               m.o, a);
    return cudaGetLastError();
}

cudaError_t launch_gla_chunk_wide(const ChunkArgs &a, const ChunkMaps &m, cudaStream_t s) {
    if (!a.gk) return cudaErrorInvalidValue;
    // The copy warp (with the L2 prefetch of chunk r + 2) measured faster for whole sequences
    // without checkpoints and slower with segments or checkpoint copies.
    const bool copy = a.nseg == 1 && a.ckpt == nullptr;
    if (a.gate_dtype != 0) return copy ? launch_one<true, true>(a, m, s) : launch_one<false, true>(a, m, s);
    return copy ? launch_one<true, false>(a, m, s) : launch_one<false, false>(a, m, s);
}

}  // namespace ccq
