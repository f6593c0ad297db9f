// ccq_internal.h -- launch descriptors shared by the C ABI and the kernels.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace ccq {

// Arguments of the token-by-token kernel (ccq_recurrent.cu).  dtype codes
// follow ccq_dtype (0 = bf16, 1 = fp32).
struct RecurrentArgs {
    int backbone;  // 0 GLA, 1 Gated DeltaNet
    int B, T, H, Dk, Dv;
    int in_dtype, gate_dtype;
    int l2norm, centered;
    float scale;
    const void *q, *k, *v, *gate;
    const float *beta, *lambda;
    const float *S0, *C0, *m0;
    const int64_t *t0;
    void *o;
    float *ST, *CT, *mT;
};

cudaError_t launch_recurrent(const RecurrentArgs &a, cudaStream_t s);

// tT[b] = t0[b] + T (t0 NULL: T), one thread per batch row.  The kernels leave
// the final count to this launch, enqueued after them: tT may alias t0, and
// every (batch, head) CTA reads t0[b] while it runs.
cudaError_t launch_t_update(const int64_t *t0, int64_t *tT, int B, int T, cudaStream_t s);
// tT[s] = t0[s] + (cu[s+1] - cu[s]) (t0 NULL: 0 +) for packed sequences (device cu).
cudaError_t launch_t_update_varlen(const int64_t *t0, int64_t *tT, const int64_t *cu, int num_seqs,
                                   cudaStream_t s);

// Arguments of the chunkwise tensor-core kernels (Dk = Dv = 128, chunk 64,
// bf16 q/k/v/o).
struct ChunkArgs {
    int B, T, H;
    int gate_dtype;  // GLA gate: 0 bf16, 1 fp32
    int l2norm, centered;
    float scale;
    const float *lambda;
    const float *g, *beta;  // Gated DeltaNet scalar log-decay and beta
    const void *gk = nullptr;  // GLA log-forget gate [B][T][H][128] (gate_dtype), read by the wide kernel's prep warps
    int wide = 0;              // GLA: the two-reference kernel (ccq_gla_chunk_wide.cu)
    const float *S0, *C0, *m0;
    const int64_t *t0;
    __nv_bfloat16 *o;
    float *ST, *CT, *mT;
    int *status;  // device status word (bounded-wait give-ups)
    // sequence segments (long sequences): nseg segments of seg_chunks chunks each
    // (the last one shorter); seg_ws holds kSegFloats (GLA) or kGdnSegFloats (Gated
    // DeltaNet) floats per (sequence, segment).
    int nseg = 1;
    int seg_chunks = 0;
    float *seg_ws = nullptr;
    // GLA only: when set, the chunk-start states of every chunk are saved for the
    // backward (layout below).  skip_o suppresses the output write (both backbones).
    uint8_t *ckpt = nullptr;
    int skip_o = 0;
    // Packed variable-length sequences (cu != NULL): the batch index b is the sequence, B the
    // number of sequences, T the packed length; rows cu[b] .. cu[b+1] of the [1][T][H][D]
    // token tensors (and of lambda, the gates, beta) are sequence b, its states are row b.
    // Gated DeltaNet: cbase[b] is the first chunk of sequence b in the packed chunk order
    // (cbase[B] the total), chunk_seq[c] the sequence of packed chunk c; the UT factor of
    // chunk r of (b, h) is at rows (cbase[b] * H + h * NC_b + r) * 64 of the workspace.
    // Device arrays; only with nseg = 1 and no checkpoints.
    const int64_t *cu = nullptr;
    const int *cbase = nullptr;
    const int *chunk_seq = nullptr;
    int vl_chunks = 0;  // cbase[B]: the packed chunk count
    // Gated DeltaNet, for the backward (no packed sequences): when set, the forward writes per
    // chunk ch = (b H + h) NC + r of every (sequence, head), in fp32, what the backward reads:
    // tt_out[ch][64][64] = Tt = (I + A)^{-1} (the WY kernel), and the states entering the chunk
    // hs_out[ch][Dk][Dv] = H_r, sk_out[ch][Dk][Dk] = S^K_r, mk_out[ch][Dk] = M_r (the chunk kernel).
    float *tt_out = nullptr, *hs_out = nullptr, *sk_out = nullptr, *mk_out = nullptr;
};

// Per (sequence, segment) workspace: S [128][128], C [128][128], m [128], D [128].
constexpr int kSegFloats = 2 * 128 * 128 + 2 * 128;

// GLA checkpoints, per (sequence, head): one record per chunk r, then the final
// state.  A chunk record is the byte image of the forward kernel's bf16 operand
// tiles -- S^K_r ([128][128] as two T64 tiles) then e^{Gmid_r} S_r (same) --
// followed by the key sum M_r (128 fp32).  The final record is S_T (fp32
// [128][128], row-major, key dim first).
constexpr size_t kCkptChunkBytes = 65536 + 512;
constexpr size_t kCkptFinalBytes = 65536;
__host__ __device__ inline size_t ckpt_head_bytes(int T) {
    return static_cast<size_t>((T + 63) / 64) * kCkptChunkBytes + kCkptFinalBytes;
}


// Device address of the library's status word on the current device.
int *device_status_word();

// Store `msg` as this host thread's ccq_last_error() text and return `st`.
// (ccq_status is an int-valued enum of include/ccq.h.)
int record_error_code(int st, const char *msg);

// Tensor maps of q, k, v (and the GLA gate) viewed as 4-D [B][T][H][D]
// tensors, so that rows past T load as zeros.
struct ChunkMaps {
    CUtensorMap q, k, v, g, o;
};

cudaError_t launch_gla_chunk(const ChunkArgs &a, const ChunkMaps &m, cudaStream_t s);
// The two-reference CCQ-GLA forward (ccq_gla_chunk_wide.cu); launch_gla_chunk dispatches to it
// when a.wide is set.
cudaError_t launch_gla_chunk_wide(const ChunkArgs &a, const ChunkMaps &m, cudaStream_t s);

// Segment-parallel CCQ-GLA (ccq_gla_segment.cu): state deltas per segment, an
// exclusive combine, then gla_chunk_kernel on every (sequence, segment).
cudaError_t launch_gla_segments(const ChunkArgs &a, const ChunkMaps &m, cudaStream_t s);

// Chunkwise Gated DeltaNet: tensor maps of q, k, v, o ([B][T][H][128], 64 x 64
// boxes) and of the workspace matrix Tb = Tt diag(beta) of every chunk
// ([B*H*NC*64][64] bf16).
struct GdnMaps {
    CUtensorMap q, k, v, o, tb;
};

// Launches the per-chunk WY kernel then the sequential chunk kernel (launch_gdn_chunk),
// either one alone, or -- for a.nseg > 1 -- WY, the segment states, their combine and
// the chunk kernel on every (sequence, segment) (launch_gdn_segments).
cudaError_t launch_gdn_chunk(const ChunkArgs &a, const GdnMaps &m, cudaStream_t s);
cudaError_t launch_gdn_wy(const ChunkArgs &a, const GdnMaps &m, cudaStream_t s);
cudaError_t launch_gdn_chunk_only(const ChunkArgs &a, const GdnMaps &m, cudaStream_t s);
cudaError_t launch_gdn_segments(const ChunkArgs &a, const GdnMaps &m, cudaStream_t s);

// Per (sequence, segment) workspace of the segmented Gated DeltaNet forward:
// S [128][128] (the segment's state from zero, then its entering state), P [128][128]
// (the segment's transition), C [128][128] (its covariance sum, then the entering C),
// m [128] (its key sum, then the entering m), 128 spare.
constexpr int kGdnSegFloats = 3 * 128 * 128 + 2 * 128;

// Workspace bytes of the chunkwise Gated DeltaNet path (Tb of every chunk).
size_t gdn_workspace_bytes(int B, int T, int H);

// Arguments of the chunkwise CCQ-GLA backward (ccq_gla_bwd.cu).  ckpt holds
// the forward checkpoints (layout above); dgk is written in the gate dtype.
struct BwdArgs {
    int B, T, H;
    int gate_dtype;
    int l2norm, centered;
    float scale;
    const float *lambda;
    const int64_t *t0;
    const uint8_t *ckpt;
    const float *dST, *dCT, *dmT;
    float *dlambda;
    void *dgk;
    float *dS0, *dC0, *dm0;
    int *status;
    // per chunk (flat index (b*H + h)*NC + r), in the workspace:
    float *chunk_vec;    // [3][128] written by the q kernel: e^{Gc-Gmid}, e^{Gmid}, Dm increment
    uint8_t *state_img;  // 64 KB written by the state pass: the bf16 tile images of
                         // Diag(e^{Gc-Gmid}) dS_{r+1} and DC_{r+1} (two T64 tiles each)
    float *state_vec;    // [3][128] written by the state pass: Dm_{r+1}, rowsum(dS_{r+1} S_{r+1}) as
                         // the sums over the two column halves
    int wave = 0;        // chunk CTAs resident at once (one per SM): each prefetches into L2 the
                         // inputs of the chunk one wave after its own
};

// Tensor maps ([B][T][H][128], 64 x 64 swizzled boxes; g as in ChunkMaps) of
// the inputs, the outputs dq, dk, dv and the four bf16 tensors the backward
// kernels exchange (QG, the chunk-local CCQ part of dkbar, qc * dqc, DZ / |q|).
struct BwdMaps {
    CUtensorMap q, k, v, dO, g, dq, dk, dv, qg, dkc, gq, dzr;
};

// Launches the backward: gla_bwd_q_kernel (one CTA per chunk), the sequential
// gla_bwd_state_kernel (one CTA per sequence and head), gla_bwd_kv_kernel (one
// CTA per chunk).
cudaError_t launch_gla_bwd(const BwdArgs &a, const BwdMaps &m, cudaStream_t s);

// Encode the tensor map of a row-major [rows][128] bf16 matrix with 64 x 64 boxes
// (128-byte swizzle).
bool make_rows_map(CUtensorMap *map, const void *base, long long rows, int cols = 128);

// Encode the tensor map of a [B][T][H][D] tensor with a (box_inner x 1 x 64 x 1)
// box.  swizzle128 selects the 128-byte swizzle (bf16 MMA operands, box_inner
// 64); otherwise the box lands as a plain row-major [64][box_inner] array.
// Returns false when the driver entry point is missing or rejects the map.
bool make_token_map(CUtensorMap *map, const void *base, int elem_bytes, int B, int T, int H,
                    int D, int box_inner, bool swizzle128);

}  // namespace ccq
