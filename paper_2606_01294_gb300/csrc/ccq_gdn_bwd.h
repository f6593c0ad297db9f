// ccq_gdn_bwd.h -- launch interfaces of the CUDA-core CCQ-Gated-DeltaNet kernels (the backward,
// ccq_gdn_bwd.cu, and the decay-aligned-covariance forward, ccq_gdn_decayed.cu), used by the C ABI.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace ccq {

namespace gbwd {
struct GdnBwdArgs;
}

// Arguments of the CUDA-core CCQ-Gated-DeltaNet backward (ccq_gdn_bwd.cu): the C ABI's
// pointers as given (token tensors [B][T][H][D] in bf16 or fp32, D = Dk = Dv) and a
// caller workspace of gdn_bwd_workspace_bytes() bytes.
struct GdnBwdCall {
    int B, T, H, D, bf16, l2norm, centered;
    float scale;
    const void *q, *k, *v, *dout;
    const float *g, *beta, *lambda, *S0, *C0, *m0;
    const int64_t *t0;
    const float *dST, *dCT, *dmT;
    void *dq, *dk, *dv;
    float *dg, *dbeta, *dlambda, *dS0, *dC0, *dm0;
    void *workspace;
    // 1: the forward's per-chunk quantities (Tt, S^K_r, M_r, H_r) are already in the workspace
    // arrays that gdn_bwd_state_arrays() names (written by the tensor-core forward); the three
    // launches that would compute them are skipped.
    int states_ready = 0;
};
size_t gdn_bwd_workspace_bytes(int B, int T, int H, int D);
// The workspace arrays of the forward's per-chunk quantities (layout: ChunkArgs::tt_out etc.).
void gdn_bwd_state_arrays(const GdnBwdCall &c, float **tt, float **sk, float **mk, float **hs);
cudaError_t launch_gdn_bwd(const GdnBwdCall &c, cudaStream_t s);
// The reverse state pass on tensor cores (ccq_gdn_bwd_state_tc.cu): Dk = Dv = 128, bf16 keys k.
cudaError_t launch_gdn_dstate_tc(const gbwd::GdnBwdArgs &a, const void *k, cudaStream_t s);
// A 2-D tensor map over an fp32 [rows][cols] array with (box_cols x box_rows) boxes, 128-byte
// swizzled (box_cols * 4 = 128).
bool make_f32_rows_map(CUtensorMap *map, const void *base, long long rows, int cols, int box_cols, int box_rows);

// Arguments of the CUDA-core CCQ-Gated-DeltaNet forward with the decay-aligned covariance
// (ccq_gdn_decayed.cu); n0/nT are the decayed counts [B][H].
struct GdecCall {
    int B, T, H, D, bf16, l2norm, centered;
    float scale;
    const void *q, *k, *v;
    const float *g, *beta, *lambda, *S0, *C0, *m0, *n0;
    void *o;
    float *ST, *CT, *mT, *nT;
    void *workspace;
    int cov_decay = 1;    // 1: decay-aligned statistics; 0: the paper's undecayed ones (n = t)
    int contraction = 0;  // 0: I - lambda Sigma; 1: (I + lambda Sigma)^{-1}; 2: exp(-lambda Sigma)
};
size_t gdn_decayed_workspace_bytes(int B, int T, int H, int D);
cudaError_t launch_gdn_decayed(const GdecCall &c, cudaStream_t s);

}  // namespace ccq
