// ccq_gla_chunk.cu -- chunkwise CCQ-GLA forward on sm_103a tensor cores.
//
// One CTA per (batch, head) walks the 64-token chunks of Algorithm 1
// (Dk = Dv = 128).  The two recurrent states stay in tensor memory as fp32
// accumulators for the whole sequence:
//   S   [Dk lanes][Dv cols]   the GLA state, transposed (S[a][e]), kept as
//                             X = Diag(e^{Gmid - Gtot}) S between chunks
//   SK  [Dk lanes][Dk cols]   the undecayed key second-moment sum S^K (App. B)
// and every product of a chunk is a tcgen05.mma with bf16 operands in
// 128-byte-swizzled shared-memory tiles (q, k, v, gates loaded by TMA):
//
//   group A  G2  Sc  = Q Kbar^T                   (CCQ intra scores, raw q)
//            G1  P   = Q S^K                      (CCQ inter read, App. B P^prev)
//   group B  G3  P  += W Kbar                     (CCQ intra read with the mean fold)
//   group C  G4  A   = Qg Kg^T                    (gated GLA scores)
//            G6  O   = Qg Ssnap                   (GLA inter read)
//   group S  G7  X  += Kg^T V                     (GLA state update)
//            G8  S^K += Kbar^T Kbar               (second-moment update)
//   group D  G5  O  += [j<=i] A V                 (GLA intra read)
// Group S is issued right after group C: it runs under the mask epilogue and
// releases the next chunk's state snapshot early.
//
// Notation (chunk r, positions t_i = t_r + i + 1, rq_i = 1/|q_i|):
//   cq_i = CumK_i . qbar_i = M . qbar_i + rq_i sum_{j<=i} Sc_ij,   c_i = cq_i / t_i,
//   W_ij = [j<=i] (Sc_ij - c_i |q_i|), so that rq_i P_i = S^K qbar_i
//   + sum_{j<=i} (qbar_i . kbar_j - c_i) kbar_j and
//   D (P^prev + P^intra) - MeanCorr = (rq_i P_i - c_i M) / t_i     (App. B, re-associated)
//   q_clean_i = qbar_i - lambda_i (rq_i P_i - c_i M) / t_i          (Eq. clean)
// GLA gates are measured from the chunk midpoint Gmid: Qg = scale q_clean e^{G - Gmid},
// Kg = kbar * e^{Gmid - G}, Ssnap = e^{Gmid} S_r, and S_{r+1} = e^{Gtot - Gmid} X_{r+1}
// (that factor is applied at the next snapshot).  A factor e^{G - Gmid} of a row before the
// midpoint grows with the decay between that row and the midpoint, so the factoring is exact
// (up to rounding) only while each 32-token half of a chunk sums its log gates to more than
// about -82 per key dimension (2^118, where the state update from keys scaled that much still
// fits fp32).  The prep warps check every factor's exponent and record CCQ_ERR_RANGE in the
// status word when a chunk goes beyond that; the two-reference kernel (ccq_gla_chunk_wide.cu,
// algo CCQ_ALGO_CHUNKWISE_WIDE) halves the span of every factor.
//
// Warp specialisation (18 warps, 96 registers a thread):
//   EPI   (warps 0-7)   the epilogues of chunk r -- W, q_clean, mask of A, output --
//                       and the bf16 operand copies of the states, placed where EPI
//                       would otherwise wait on an MMA: e^{Gmid} S_r (rescaling X in
//                       TMEM) while G3 runs, S^K_{r+1} while G4 runs.  The 64-row
//                       products are M = 64 MMAs (rows 16q..16q+15 in TMEM lanes
//                       32q..32q+15); warps w and w+4 share lane quadrant q = w % 4
//                       and split its columns.
//   PREP  (warps 8-15)  prep of chunk r+1 while the chain runs chunk r: row norms
//                       (q and M . qbar on warps 8-11, k on 12-15), gate cumsum in
//                       four token quarters, kbar, Kg, e^{G-Gmid}, lambda.
//   ISSUE (warp 16)     one thread issues every tcgen05.mma (and, unless COPY does,
//                       the per-chunk TMA copies), in the order G2 | G1 | G3 G8 | G7 |
//                       G4 G6 | G5, so that G1, G7 and G6 run under the epilogues.  An MMA
//                       instruction holds its issuing thread for its whole execution,
//                       which is why no epilogue thread issues.  EPI signals the issuer
//                       with named-barrier arrives; the issuer signals EPI with commits.
//   COPY  (warp 17)     in the COPY instance: the loads of chunk r+2, the store of O and the
//                       next v, plus an L2 prefetch of chunk r+2 beyond each load.
// Per-chunk tiles are double-buffered (two slots); the loads of chunk r+2 start as
// soon as chunk r's last MMA reader of the slot (G6) completes.  v is single-buffered
// and reloaded once G5 of the previous chunk completes.
// Rows past T load as zeros: zero keys add nothing to any sum, zero gates keep
// the cumulative gate, so the ragged tail needs no special arithmetic.
// With a.ckpt set, EPI also copies each chunk's two state tiles and key sum to
// the checkpoint buffer (bulk copies) and the last segment writes
// S_T there; the backward (ccq_gla_bwd.cu) reads them.
// With a.nseg > 1 every CTA walks one segment (a range of whole chunks) of one
// sequence, starting from the segment's initial states in a.seg_ws
// (ccq_gla_segment.cu); only the last segment writes the final states.
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
constexpr int kEpiThreads = 256;
constexpr int kPrepWarp0 = 8, kIssueWarp = 16, kCopyWarp = 17;
constexpr int kPrepThreads = 32 * (kIssueWarp - kPrepWarp0);  // 256
constexpr int kThreadsNoCopy = 32 * kCopyWarp;       // 544
constexpr int kThreadsCopy = 32 * (kCopyWarp + 1);    // 576
constexpr int kSyncCount = kEpiThreads + 32;          // EPI + the issuing warp
// largest exponent (log2 units) a gate factor may have: a state accumulated over a chunk
// from keys scaled by up to 2^118 stays inside the fp32 range
constexpr float kMaxExp2 = 118.f;

// ---- shared memory map (bytes from the 1024-aligned base)
// two slots of per-chunk tiles, each [64 rows][128 cols] bf16 as two T64 tiles of 8 KB:
constexpr uint32_t SLOT_BYTES = 49152;
constexpr uint32_t SO_Q = 0;       // raw q, then q_clean * e^{G - Gmid}
constexpr uint32_t SO_KG = 16384;  // raw gates land here (bf16: 16 KB, fp32: KG+EG 32 KB); then Kg
constexpr uint32_t SO_EG = 32768;  // e^{G - Gmid}
// The keys of both slots and the bf16 S^K share one region per 64-column half h of the
// key dimension: [kbar of slot 0 (64 rows)][S^K (128 rows)][kbar of slot 1 (64 rows)],
// 128 B per row (T64 tiles, K-major for G2 and G1, MN-major for G3 and G8).
constexpr uint32_t OFF_KS = 98304;   // 2 x 32K
constexpr uint32_t KS_HALF = 32768;  // distance between the two halves
constexpr uint32_t KS_SK = 8192;     // S^K rows within a half
constexpr uint32_t KS_K1 = 24576;    // kbar of slot 1 within a half
constexpr uint32_t OFF_V = 163840;   // 16K  v; after G5 the output staging of the TMA store
constexpr uint32_t OFF_W = 180224;   // 8K   W, then the masked A ([64][64], one T64 tile)
constexpr uint32_t OFF_S = 188416;   // 32K  bf16 e^{Gmid} S ([128][128], two T64 tiles of 16 KB)
constexpr uint32_t OFF_MISC = 221184;
static_assert(2 * SLOT_BYTES == OFF_KS && OFF_KS + 2 * KS_HALF == OFF_V, "shared memory map");
// the kbar tile of slot s, key columns 64 h .. 64 h + 63
__host__ __device__ constexpr uint32_t kbar_off(int s, int h) {
    return OFF_KS + static_cast<uint32_t>(h) * KS_HALF + (s ? KS_K1 : 0u);
}
// misc: per-slot arrays (3072 B per slot)
constexpr uint32_t MS_BYTES = 3072;
constexpr uint32_t MS_RQ = 0;      // [64] 1/|q_i|
constexpr uint32_t MS_MQ = 256;    // [64] M . qbar_i
constexpr uint32_t MS_LT = 512;    // [64] lambda_i / t_i
constexpr uint32_t MS_RK = 768;    // [64] 1/|k_j|
constexpr uint32_t MS_EGM = 1024;  // [128] e^{Gmid}
constexpr uint32_t MS_F = 1536;    // [128] e^{Gtot - Gmid}
constexpr uint32_t MS_MST = 2048;  // [128] key sum M at the chunk start
constexpr uint32_t MS_ITI = 2560;  // [64] 1 / t_i
constexpr uint32_t MS_QN = 2816;   // [64] |q_i| (1 without the l2 norm)
constexpr uint32_t M_DMP = 6144;   // [4][128] per token quarter: gate sums, then key sums (prep)
constexpr uint32_t M_DMPREV = 8192;  // [128] key sum of the previous chunk
constexpr uint32_t M_BAR = 8704;   // mbarriers
constexpr uint32_t M_TMEM = 8816;
constexpr uint32_t M_ABORT = 8820;
constexpr uint32_t kMiscBytes = 8832;
constexpr uint32_t kSmemBytes = OFF_MISC + kMiscBytes + 1024;  // + alignment slack
static_assert(kSmemBytes <= 232448, "exceeds the 227 KB per-CTA limit");

enum {
    BAR_IN0 = 0, BAR_IN1 = 1, BAR_V = 2, BAR_GA = 3, BAR_GB = 4, BAR_GK = 5, BAR_GC = 6,
    BAR_GC2 = 7, BAR_GD = 8, BAR_PREP0 = 9, BAR_PREP1 = 10, BAR_SNAPK = 11, BAR_SNAPS = 12,
    kNumBars = 13
};
static_assert(M_BAR + 8 * kNumBars <= M_TMEM, "barrier area");
// named barriers (0 is __syncthreads)
enum { NB_W = 1, NB_QC = 2, NB_MASK = 3, NB_OUT = 4, NB_PREP = 5, NB_EPI = 6 };

// ---- tensor memory columns
constexpr uint32_t TM_S = 0;     // 128 cols
constexpr uint32_t TM_SK = 128;  // 128 cols
constexpr uint32_t TM_PO = 256;  // 128 cols: P, then O (M = 64 layout)
constexpr uint32_t TM_SA = 384;  // 64 cols: Sc, then A (M = 64 layout)
constexpr uint32_t kTmemCols = 512;

constexpr uint32_t ID_64x64_KK = make_idesc(64, 64, 0, 0);
constexpr uint32_t ID_64x128_KM = make_idesc(64, 128, 0, 1);
constexpr uint32_t ID_64x128_KK = make_idesc(64, 128, 0, 0);
constexpr uint32_t ID_128x128_MM = make_idesc(128, 128, 1, 1);

__device__ __forceinline__ void store_row_chunk(uint8_t *tile, int row, int chunk, const float *w) {
    uint4 u;
    u.x = pack_bf16(w[0], w[1]);
    u.y = pack_bf16(w[2], w[3]);
    u.z = pack_bf16(w[4], w[5]);
    u.w = pack_bf16(w[6], w[7]);
    *reinterpret_cast<uint4 *>(tile + t64_chunk(row, chunk)) = u;
}

template <bool COPY>
__global__ void __maxnreg__(96)
gla_chunk_kernel(const __grid_constant__ CUtensorMap map_q, const __grid_constant__ CUtensorMap map_k,
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
    const int tok0 = vl ? static_cast<int>(a.cu[b]) : 0;                  // token coordinate offset
    const int T = vl ? static_cast<int>(a.cu[b + 1] - a.cu[b]) : a.T;     // this sequence's length
    const int bt = vl ? 0 : b;                                            // batch coordinate
    const size_t rowbase = vl ? static_cast<size_t>(tok0) : static_cast<size_t>(b) * a.T;  // its first [., H] row
    const int NCt = (T + kC - 1) / kC;
    const int cb = a.nseg > 1 ? seg * a.seg_chunks : 0;  // first chunk of this CTA
    const int NC = a.nseg > 1 ? min(NCt, cb + a.seg_chunks) - cb : NCt;
    const bool last_seg = seg == a.nseg - 1;
    const float *segst = a.nseg > 1 ? a.seg_ws + static_cast<size_t>(blockIdx.x) * kSegFloats : nullptr;
    const float *S0 = segst ? segst : a.S0;
    const float *C0 = segst ? segst + kD * kD : a.C0;
    const float *m0 = segst ? segst + 2 * kD * kD : a.m0;
    const bool gate_f32 = a.gate_dtype != 0;
    const uint32_t g_bytes = gate_f32 ? kC * kD * 4 : kC * kD * 2;
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

    auto issue_in = [&](int r) {  // q, k, gates of local chunk r into slot r & 1
        const int s = r & 1, tg = (cb + r) * kC;
        uint8_t *base = sm + s * SLOT_BYTES;
        uint64_t *bb = &bar[BAR_IN0 + s];
        mbar_arrive_expect_tx(bb, 4 * 8192 + g_bytes);
        tma_load_4d(base + SO_Q, &map_q, bb, 0, h, tok0 + tg, bt);
        tma_load_4d(base + SO_Q + 8192, &map_q, bb, 64, h, tok0 + tg, bt);
        tma_load_4d(sm + kbar_off(s, 0), &map_k, bb, 0, h, tok0 + tg, bt);
        tma_load_4d(sm + kbar_off(s, 1), &map_k, bb, 64, h, tok0 + tg, bt);
        tma_load_4d(base + SO_KG, &map_g, bb, 0, h, tok0 + tg, bt);
        if (COPY && r + 2 < NC) {  // chunk r + 2 into L2, so that its loads hit there
            const int tp = tok0 + tg + 2 * kC;
            tma_prefetch_l2_4d(&map_q, 0, h, tp, bt);
            tma_prefetch_l2_4d(&map_q, 64, h, tp, bt);
            tma_prefetch_l2_4d(&map_k, 0, h, tp, bt);
            tma_prefetch_l2_4d(&map_k, 64, h, tp, bt);
            tma_prefetch_l2_4d(&map_g, 0, h, tp, bt);
        }
    };
    auto issue_v = [&](int r) {
        const int tg = (cb + r) * kC;
        mbar_arrive_expect_tx(&bar[BAR_V], 2 * 8192);
        tma_load_4d(sm + OFF_V, &map_v, &bar[BAR_V], 0, h, tok0 + tg, bt);
        tma_load_4d(sm + OFF_V + 8192, &map_v, &bar[BAR_V], 64, h, tok0 + tg, bt);
        if (COPY && r + 2 < NC) {
            tma_prefetch_l2_4d(&map_v, 0, h, tok0 + tg + 2 * kC, bt);
            tma_prefetch_l2_4d(&map_v, 64, h, tok0 + tg + 2 * kC, bt);
        }
    };
    // the last chunk of a packed sequence ends inside the tile: its rows past the end belong to
    // the next sequence, so its output is written row by row (not by a TMA store of the tile)
    auto partial = [&](int r) { return vl && T - (cb + r) * kC < kC; };
    auto store_o = [&](int r) {  // TMA store of the output of local chunk r staged in the v tile
        if (a.skip_o || partial(r)) return;
        const int cp = (cb + r) * kC;
        tma_store_4d(&map_o, sm + OFF_V, 0, h, tok0 + cp, bt);
        tma_store_4d(&map_o, sm + OFF_V + 8192, 64, h, tok0 + cp, bt);
        tma_store_commit();
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
    } else if (warp < kIssueWarp) {
        const int wt = tid - 32 * kPrepWarp0;
        if (wt < kD) {
            slot_f(0, MS_MST)[wt] = m0 ? m0[(segst ? 0 : static_cast<size_t>(bh) * kD) + wt] : 0.f;
            dmprev[wt] = 0.f;
        }
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
        uint8_t *ck_head = a.ckpt ? a.ckpt + static_cast<size_t>(bh) * ckpt_head_bytes(T) : nullptr;
        // bf16 copy of S^K (this thread: row a, columns 64 grp .. 64 grp + 63)
        auto snap_sk = [&]() {
            if (ck_head) {
                // the previous checkpoint copy must have read the tiles before they change
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
                    store_row_chunk(sm + OFF_KS + grp * KS_HALF + KS_SK, row, 4 * cc + q4, x + 8 * q4);
            }
            fence_proxy_async_smem();
            tc_fence_before();
            named_bar(NB_EPI, kEpiThreads);
            if (tid == 0) mbar_arrive(&bar[BAR_SNAPK]);
        };
        // bf16 copy of e^{Gmid_r} S_r = hs X, with X rescaled in TMEM; then the checkpoint record
        auto snap_s = [&](int r, float hs) {
            tc_fence_after();
#pragma unroll
            for (int cc = 0; cc < 2; ++cc) {
                float x[32];
                tmem_ld32(tq + TM_S + 64 * grp + 32 * cc, x);
                const uint64_t hs2 = f2_make(hs, hs);
                uint32_t w[16];
#pragma unroll
                for (int e = 0; e < 16; ++e) {
                    const float2 y = f2_split(f2_mul(f2_make(x[2 * e], x[2 * e + 1]), hs2));
                    x[2 * e] = y.x;
                    x[2 * e + 1] = y.y;
                    w[e] = pack_bf16(y.x, y.y);
                }
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4)
                    *reinterpret_cast<uint4 *>(sm + OFF_S + grp * 16384 + t64_chunk(row, 4 * cc + q4)) =
                        make_uint4(w[4 * q4], w[4 * q4 + 1], w[4 * q4 + 2], w[4 * q4 + 3]);
                tmem_st32(tq + TM_S + 64 * grp + 32 * cc, x);
            }
            tmem_wait_st();
            fence_proxy_async_smem();
            tc_fence_before();
            named_bar(NB_EPI, kEpiThreads);
            if (tid == 0) mbar_arrive(&bar[BAR_SNAPS]);
            if (ck_head) {
                // checkpoint of chunk cb + r: the S^K and e^{Gmid} S tiles, then M_r
                uint8_t *rec = ck_head + static_cast<size_t>(cb + r) * kCkptChunkBytes;
                if (grp == 0) reinterpret_cast<float *>(rec + 65536)[row] = slot_f(r & 1, MS_MST)[row];
                if (tid == 0) {
                    bulk_store(rec, sm + OFF_KS + KS_SK, 16384);
                    bulk_store(rec + 16384, sm + OFF_KS + KS_HALF + KS_SK, 16384);
                    bulk_store(rec + 32768, sm + OFF_S, 32768);
                    tma_store_commit();
                }
            }
        };
        float f_cur = 1.f;  // e^{Gtot - Gmid} of the chunk in flight, state row `row`
        if (NC > 0) {
            mbar_wait(&bar[BAR_PREP0], 0, abort_flag, status);
            snap_sk();
            snap_s(0, slot_f(0, MS_EGM)[row]);
        }
        for (int r = 0; r < NC; ++r) {
            const int s = r & 1;
            const uint32_t sp = (r >> 1) & 1, par = r & 1;
            uint8_t *slot = sm + s * SLOT_BYTES;
            mbar_wait(&bar[BAR_PREP0 + s], sp, abort_flag, status);
            const float f_prev = f_cur;  // e^{Gtot - Gmid} of chunk r - 1
            const float egm = slot_f(s, MS_EGM)[row];
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
            // ---- e^{Gmid_r} S_r while G3 runs (G6 and G7 of chunk r-1 have run: the output
            // epilogue of chunk r-1 waited for GD, which follows them).  The instance without
            // the copy warp (segments, checkpoints) writes it at the end of chunk r-1 instead, so
            // that the checkpoint copy issued with it has read the tiles before S^K_{r+1} is
            // written over them.
            if (COPY && r > 0) snap_s(r, f_prev * egm);
            // ---- q_clean epilogue (Eq. clean), scaled by e^{G - Gmid}, into the Q tile.
            // q_clean e^{G-Gmid} = e^{G-Gmid} (rq (q - (lambda/t) P) + (lambda c / t) M);
            // this thread: row i, columns 64 grp + 32 hf .. +31 (T64 tile grp, chunks 4 hf ..)
            {
                uint8_t *qt = slot + SO_Q + grp * 8192;
                const uint8_t *et = slot + SO_EG + grp * 8192;
                const float *Mst = slot_f(s, MS_MST) + 64 * grp + 32 * hf;
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
                // the read scale is applied here: O is linear in the scaled q_clean
                const float rqs = rqi * a.scale, cms = cm * a.scale;
                const uint64_t nlt = f2_make(-lt, -lt), rq2 = f2_make(rqs, rqs), cm2 = f2_make(cms, cms);
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) {
                    const ulonglong2 m01 = *reinterpret_cast<const ulonglong2 *>(Mst + 8 * q4);
                    const ulonglong2 m23 = *reinterpret_cast<const ulonglong2 *>(Mst + 8 * q4 + 4);
                    const uint64_t mp[4] = {m01.x, m01.y, m23.x, m23.y};
                    const uint32_t qw[4] = {qraw[q4].x, qraw[q4].y, qraw[q4].z, qraw[q4].w};
                    const uint32_t ew[4] = {eraw[q4].x, eraw[q4].y, eraw[q4].z, eraw[q4].w};
                    uint32_t ow[4];
#pragma unroll
                    for (int w = 0; w < 4; ++w) {
                        const uint64_t p2 = f2_make(p[8 * q4 + 2 * w], p[8 * q4 + 2 * w + 1]);
                        const uint64_t t = f2_fma(nlt, p2, f2_from_bf16x2(qw[w]));     // q - (lambda/t) P
                        const uint64_t u = f2_fma(rq2, t, f2_mul(cm2, mp[w]));          // rq (.) + (lambda c/t) M
                        ow[w] = bf16x2_from_f2(f2_mul(f2_from_bf16x2(ew[w]), u));      // * e^{G - Gmid}
                    }
                    *reinterpret_cast<uint4 *>(qt + t64_chunk(i, 4 * hf + q4)) = make_uint4(ow[0], ow[1], ow[2], ow[3]);
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
            // ---- causal mask of A
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
                        w[e] = (32 * hf + 16 * grp + jj <= i) ? v : 0.f;
                    }
                    store_row_chunk(sm + OFF_W, i, 4 * hf + 2 * grp + q2, w);
                }
            }
            fence_proxy_async_smem();
            tc_fence_before();
            named_bar_arrive(NB_MASK, kSyncCount);
            // ---- output: o = O (q_clean carries the read scale) staged (bf16, swizzled) in the
            // v tile, which G5 has finished reading; the copy warp stores it with one TMA copy
            // (rows past T fall outside the tensor and are not written)
            mbar_wait(&bar[BAR_GD], par, abort_flag, status);
            tc_fence_after();
            if (!a.skip_o) {
                float x[32];
                tmem_ld16x2_32<32>(tq + TM_PO + 64 * grp, x);
                const int tpos = (cb + r) * kC + i;  // position of row i in the sequence
                const bool direct = partial(r);
                uint4 *dst = reinterpret_cast<uint4 *>(a.o + ((rowbase + tpos) * H + h) * kD + 64 * grp + 32 * hf);
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) {
                    uint32_t w[4];
#pragma unroll
                    for (int u = 0; u < 4; ++u)
                        w[u] = pack_bf16(x[8 * q4 + 2 * u], x[8 * q4 + 2 * u + 1]);
                    if (!direct)
                        *reinterpret_cast<uint4 *>(sm + OFF_V + grp * 8192 + t64_chunk(i, 4 * hf + q4)) = make_uint4(w[0], w[1], w[2], w[3]);
                    else if (tpos < T)
                        dst[q4] = make_uint4(w[0], w[1], w[2], w[3]);
                }
                fence_proxy_async_smem();
            }
            tc_fence_before();
            named_bar_arrive(NB_OUT, kOutCount);
            if (!COPY && r + 1 < NC) {
                mbar_wait(&bar[BAR_PREP0 + (s ^ 1)], ((r + 1) >> 1) & 1, abort_flag, status);
                snap_s(r + 1, f_cur * slot_f(s ^ 1, MS_EGM)[row]);
            }
        }
        if (ck_head && tid == 0) tma_store_wait_all();
        // final states: S_T = e^{Gtot - Gmid} X (last chunk), S^K (an empty packed sequence:
        // the initial states, still in TMEM as set up)
        if ((NC > 0 || vl) && last_seg) {
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
    } else if (warp < kIssueWarp) {
        // =============================================================== PREP
        // Eight warps.  Row norms: warps 0-3 take the rows of q (and M . q), warps 4-7 those
        // of k; lanes l and l + 16 of a warp share row j, each one 64-column half (one T64
        // tile), so eight consecutive lanes read eight different rows (no bank conflicts).
        // Gates: thread (p, tq) takes key dims 2p, 2p+1 over the sixteen tokens of quarter tq.
        const int wt = tid - 32 * kPrepWarp0;
        const int pw = wt >> 5;
        const bool nq = pw < 4;
        const int j = 16 * (pw & 3) + (lane & 15), hh = lane >> 4;
        const int p = wt & 63, tq = wt >> 6;
        const int d0 = 2 * p;
        constexpr float kLog2e = 1.4426950408889634f;
        float lam_reg = 0.f;  // lambda of row j of the next chunk (q warps)
        if (nq) {
            const int tn = cb * kC + j;
            lam_reg = (tn < T) ? a.lambda[(rowbase + tn) * H + h] : 0.f;
        }
        float emax = 0.f;  // largest |exponent| (log2 units) of a gate factor met
        for (int r = 0; r < NC; ++r) {
            const int s = r & 1;
            const uint32_t sp = (r >> 1) & 1;
            uint8_t *slot = sm + s * SLOT_BYTES;
            float *Mst = slot_f(s, MS_MST);
            mbar_wait(&bar[BAR_IN0 + s], sp, abort_flag, status);
            // key sum at the chunk start and lambda of the chunk
            if (r > 0 && wt < kD) Mst[wt] = slot_f(s ^ 1, MS_MST)[wt] + dmprev[wt];
            const float lam_cur = lam_reg;
            if (nq) {
                const int tn = (cb + r + 1) * kC + j;
                lam_reg = (tn < T) ? a.lambda[(rowbase + tn) * H + h] : 0.f;
            }
            named_bar(NB_PREP, kPrepThreads);
            if (nq) {
                // |q_j|^2 and M . q_j in fp32 pairs
                uint4 qv[8];
#pragma unroll
                for (int cc = 0; cc < 8; ++cc)
                    qv[cc] = *reinterpret_cast<const uint4 *>(slot + SO_Q + hh * 8192 + t64_chunk(j, cc));
                const float *Mh = Mst + 64 * hh;
                uint64_t sq0 = 0, sq1 = 0, md0 = 0, md1 = 0;
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
                const float2 a0 = f2_split(f2_add(sq0, sq1)), c0v = f2_split(f2_add(md0, md1));
                float ssq = a0.x + a0.y, mdt = c0v.x + c0v.y;
                ssq += __shfl_xor_sync(0xffffffffu, ssq, 16);
                mdt += __shfl_xor_sync(0xffffffffu, mdt, 16);
                if (hh == 0) {
                    const float rq = a.l2norm ? rsqrtf(fmaxf(ssq, 1e-12f)) : 1.f;
                    const float iti = 1.f / static_cast<float>(tseq0 + (cb + r) * kC + j + 1);
                    slot_f(s, MS_RQ)[j] = rq;
                    slot_f(s, MS_MQ)[j] = mdt * rq;
                    slot_f(s, MS_ITI)[j] = iti;
                    slot_f(s, MS_QN)[j] = a.l2norm ? fmaxf(ssq, 1e-12f) * rq : 1.f;
                    slot_f(s, MS_LT)[j] = lam_cur * iti;
                }
            } else {
                // |k_j|^2
                uint4 kv[8];
#pragma unroll
                for (int cc = 0; cc < 8; ++cc)
                    kv[cc] = *reinterpret_cast<const uint4 *>(sm + kbar_off(s, hh) + t64_chunk(j, cc));
                uint64_t sk0 = 0, sk1 = 0;
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
                const float2 b0 = f2_split(f2_add(sk0, sk1));
                float ssk = b0.x + b0.y;
                ssk += __shfl_xor_sync(0xffffffffu, ssk, 16);
                if (hh == 0) {
                    // rows past the end of a packed sequence hold the next one's keys: zero them
                    const bool in_seq = (cb + r) * kC + j < T;
                    slot_f(s, MS_RK)[j] = !in_seq ? 0.f : a.l2norm ? rsqrtf(fmaxf(ssk, 1e-12f)) : 1.f;
                }
            }
            // gate cumsum over this thread's sixteen tokens for dims d0, d0+1, as fp32 pairs
            uint64_t g2[16];
            {
                uint64_t r2 = 0;  // (0.f, 0.f)
                const int rem = T - (cb + r) * kC;  // tokens of the sequence in this chunk
#pragma unroll
                for (int u = 0; u < 16; ++u) {
                    const int jt = 16 * tq + u;
                    const uint64_t x2 =
                        jt >= rem ? 0
                        : gate_f32 ? *reinterpret_cast<const uint64_t *>(slot + SO_KG + (jt * kD + d0) * 4)
                                   : f2_from_bf16x2(*reinterpret_cast<const uint32_t *>(slot + SO_KG + (jt * kD + d0) * 2));
                    r2 = f2_add(r2, x2);
                    g2[u] = r2;
                }
                *reinterpret_cast<uint64_t *>(dmp + tq * kD + d0) = r2;  // the quarter's gate sums
            }
            named_bar(NB_PREP, kPrepThreads);  // raw gates all read, norms and quarter sums visible
            uint64_t dm2 = 0;
            {
                // G at this quarter's start (sum of the earlier quarters) and Gmid = G at token 31
                uint64_t q2[4];
#pragma unroll
                for (int qq = 0; qq < 4; ++qq) q2[qq] = *reinterpret_cast<const uint64_t *>(dmp + qq * kD + d0);
                uint64_t gs = 0;
#pragma unroll
                for (int qq = 0; qq < 3; ++qq)
                    if (qq < tq) gs = f2_add(gs, q2[qq]);
                const float2 gm = f2_split(f2_add(q2[0], q2[1]));
                const float2 gsv = f2_split(gs);
                // exponents in log2 units relative to Gmid: x = (G - Gmid) log2(e)
                const uint64_t o2 = f2_make((gsv.x - gm.x) * kLog2e, (gsv.y - gm.y) * kLog2e);
                const uint64_t l2e = f2_make(kLog2e, kLog2e);
                if (tq == 3) {
                    // f = e^{Gtot - Gmid} (the last token's factor), e^{Gmid}
                    const float2 xl = f2_split(f2_fma(g2[15], l2e, o2));
                    slot_f(s, MS_F)[d0] = fast_exp2(xl.x);
                    slot_f(s, MS_F)[d0 + 1] = fast_exp2(xl.y);
                    slot_f(s, MS_EGM)[d0] = fast_exp2(gm.x * kLog2e);
                    slot_f(s, MS_EGM)[d0 + 1] = fast_exp2(gm.y * kLog2e);
                }
                if (tq == 0 || tq == 3) {
                    // log gates are <= 0, so G falls monotonically and the factors' exponents are
                    // largest in magnitude at the chunk's first and last tokens
                    const float2 xe = f2_split(f2_fma(tq ? g2[15] : g2[0], l2e, o2));
                    emax = fmaxf(emax, fmaxf(fabsf(xe.x), fabsf(xe.y)));
                }
                const float *rk = slot_f(s, MS_RK);
                uint8_t *kt = sm + kbar_off(s, d0 >> 6);  // kbar tile of these key columns
                // two batches of eight tokens: every load of a batch is issued before its
                // stores (the in-place kbar store may alias a later load)
#pragma unroll
                for (int bt = 0; bt < 2; ++bt) {
                    uint32_t kraw[8];
#pragma unroll
                    for (int u = 0; u < 8; ++u) {
                        const int jt = 16 * tq + 8 * bt + u;
                        kraw[u] = *reinterpret_cast<const uint32_t *>(kt + t64_offset(jt, d0 & 63));
                    }
                    const float4 rka = *reinterpret_cast<const float4 *>(rk + 16 * tq + 8 * bt);
                    const float4 rkb = *reinterpret_cast<const float4 *>(rk + 16 * tq + 8 * bt + 4);
                    const float rkv[8] = {rka.x, rka.y, rka.z, rka.w, rkb.x, rkb.y, rkb.z, rkb.w};
#pragma unroll
                    for (int u = 0; u < 8; ++u) {
                        const int ju = 8 * bt + u, jt = 16 * tq + ju;
                        const uint32_t off = t64_offset(jt, d0 & 63);
                        const uint32_t toff = (d0 >> 6) * 8192 + off;  // in the slot's Kg / EG tiles
                        const uint64_t k2 = f2_mul(f2_from_bf16x2(kraw[u]), f2_make(rkv[u], rkv[u]));
                        const float2 x = f2_split(f2_fma(g2[ju], l2e, o2));
                        *reinterpret_cast<uint32_t *>(kt + off) = bf16x2_from_f2(k2);
                        *reinterpret_cast<uint32_t *>(slot + SO_KG + toff) =
                            bf16x2_from_f2(f2_mul(k2, f2_make(fast_exp2(-x.x), fast_exp2(-x.y))));
                        *reinterpret_cast<uint32_t *>(slot + SO_EG + toff) = pack_bf16(fast_exp2(x.x), fast_exp2(x.y));
                        dm2 = f2_add(dm2, k2);
                    }
                }
            }
            fence_proxy_async_smem();
            named_bar(NB_PREP, kPrepThreads);  // tiles and scalars written, quarter sums read
            if (wt == 0) mbar_arrive(&bar[BAR_PREP0 + s]);
            *reinterpret_cast<uint64_t *>(dmp + tq * kD + d0) = dm2;  // the quarter's key sums
            named_bar(NB_PREP, kPrepThreads);
            if (wt < kD) dmprev[wt] = (dmp[wt] + dmp[kD + wt]) + (dmp[2 * kD + wt] + dmp[3 * kD + wt]);
        }
        // a factor beyond 2^kMaxExp2 cannot be represented: report it rather than return
        // silently wrong values
        if (emax > kMaxExp2) atomicExch(status, kStatusRange);
        // final key sum
        if ((NC > 0 || vl) && a.mT && last_seg && wt < kD) {
            const int sl = NC > 0 ? (NC - 1) & 1 : 0;
            a.mT[static_cast<size_t>(bh) * kD + wt] = slot_f(sl, MS_MST)[wt] + dmprev[wt];
        }
    } else if (warp == kIssueWarp) {
        // =============================================================== ISSUE
        const bool lead = lane == 0;
        // descriptor bases (start-address field advanced per K slice: +2 per 32 B)
        const uint64_t dW = make_desc(sb + OFF_W, 16, 1024);
        const uint64_t dSK = make_desc(sb + OFF_KS + KS_SK, 16, 1024);
        const uint64_t dS = make_desc(sb + OFF_S, 16384, 1024);
        const uint64_t dV = make_desc(sb + OFF_V, 8192, 1024);
        for (int r = 0; r < NC; ++r) {
            const int s = r & 1;
            const uint32_t sp = (r >> 1) & 1, par = r & 1;
            const uint32_t ss = sb + s * SLOT_BYTES;
            const uint64_t dQ = make_desc(ss + SO_Q, 16, 1024);
            const uint64_t dK = make_desc(sb + kbar_off(s, 0), 16, 1024);
            const uint64_t dKm = make_desc(sb + kbar_off(s, 0), KS_HALF, 1024);
            const uint64_t dKG = make_desc(ss + SO_KG, 16, 1024);
            const uint64_t dKGm = make_desc(ss + SO_KG, 8192, 1024);
            const uint32_t tp = tbase + TM_PO, tsa = tbase + TM_SA;
            mbar_wait(&bar[BAR_PREP0 + s], sp, abort_flag, status);
            tc_fence_after();
            // G2 Sc = Q Kbar^T (SA is free: the mask epilogue of chunk r-1 has read A)
            if (lead && !*abort_flag) {
                for (int k = 0; k < 8; ++k)
                    mma_bf16(tsa, dQ + (k >> 2) * 512 + (k & 3) * 2, dK + (k >> 2) * (KS_HALF >> 4) + (k & 3) * 2,
                             ID_64x64_KK, k != 0);
                mma_commit(&bar[BAR_GA]);
            }
            __syncwarp();
            if (r > 0) {
                // O of chunk r-1 has left PO (staged in the v tile): store it (unless the copy
                // warp does)
                mbar_wait(&bar[BAR_GD], (r - 1) & 1, abort_flag, status);
                named_bar(NB_OUT, kOutCount);
                if (lead && !COPY) store_o(r - 1);
                __syncwarp();
            }
            // G1 P = Q S^K
            mbar_wait(&bar[BAR_SNAPK], par, abort_flag, status);
            tc_fence_after();
            if (lead && !*abort_flag)
                for (int k = 0; k < 8; ++k)
                    mma_bf16(tp, dQ + (k >> 2) * 512 + (k & 3) * 2, dSK + (k >> 2) * (KS_HALF >> 4) + (k & 3) * 2,
                             ID_64x128_KK, k != 0);
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
                    mma_bf16(tp, dW + k * 2, dKm + k * 128, ID_64x128_KM, 1);
                mma_commit(&bar[BAR_GB]);
                for (int k = 0; k < 4; ++k)
                    mma_bf16(tbase + TM_SK, dKm + k * 128, dKm + k * 128, ID_128x128_MM, 1);
                mma_commit(&bar[BAR_GK]);
            }
            __syncwarp();
            // G7 X += Kg^T V (X rescaled by the snapshot of chunk r; v landed)
            mbar_wait(&bar[BAR_SNAPS], par, abort_flag, status);
            mbar_wait(&bar[BAR_V], par, abort_flag, status);
            tc_fence_after();
            if (lead && !*abort_flag)
                for (int k = 0; k < 4; ++k)
                    mma_bf16(tbase + TM_S, dKGm + k * 128, dV + k * 128, ID_128x128_MM, 1);
            __syncwarp();
            // G4 A = Qg Kg^T, G6 O = Qg Ssnap
            named_bar(NB_QC, kSyncCount);
            tc_fence_after();
            if (lead && !*abort_flag) {
                for (int k = 0; k < 8; ++k) {
                    const uint64_t ko = (k >> 2) * 512 + (k & 3) * 2;
                    mma_bf16(tsa, dQ + ko, dKG + ko, ID_64x64_KK, k != 0);
                }
                mma_commit(&bar[BAR_GC]);
                for (int k = 0; k < 8; ++k)
                    mma_bf16(tp, dQ + (k >> 2) * 512 + (k & 3) * 2, dS + k * 128, ID_64x128_KM, k != 0);
                mma_commit(&bar[BAR_GC2]);
            }
            __syncwarp();
            // G5 O += A V
            named_bar(NB_MASK, kSyncCount);
            tc_fence_after();
            if (lead && !*abort_flag) {
                for (int k = 0; k < 4; ++k)
                    mma_bf16(tp, dW + k * 2, dV + k * 128, ID_64x128_KM, 1);
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
            if (lead && !COPY) store_o(NC - 1);
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
                store_o(r);
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

cudaError_t launch_gla_chunk(const ChunkArgs &a, const ChunkMaps &m, cudaStream_t s) {
    if (a.wide) return launch_gla_chunk_wide(a, m, s);
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(gla_chunk_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(kSmemBytes));
        if (e != cudaSuccess) return e;
        e = cudaFuncSetAttribute(gla_chunk_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 static_cast<int>(kSmemBytes));
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    // The copy warp (with the L2 prefetch of chunk r + 2) measured faster for whole sequences
    // without checkpoints (4K: 268 -> 253 us) and slower with segments or checkpoint copies.
    if (a.nseg == 1 && a.ckpt == nullptr)
        gla_chunk_kernel<true><<<a.B * a.H, kThreadsCopy, kSmemBytes, s>>>(m.q, m.k, m.v, m.g, m.o, a);
    else
        gla_chunk_kernel<false><<<a.B * a.H * a.nseg, kThreadsNoCopy, kSmemBytes, s>>>(m.q, m.k, m.v, m.g, m.o, a);
    return cudaGetLastError();
}

}  // namespace ccq
