// ccq_gdn_decayed.cu -- launches of the CUDA-core CCQ-Gated-DeltaNet forward with the
// decay-aligned covariance (kernels: ccq_gdn_decayed_kernels.cuh).
#include <cuda_runtime.h>
#include <stdint.h>

#include "ccq_gdn_bwd.h"
#include "ccq_gdn_decayed_kernels.cuh"

namespace ccq {

namespace {

// Workspace floats per chunk: Tt, the undecayed key statistics of the shared prep kernel,
// H_r, the decayed increments / entering statistics of C, m, and n with the chunk's decay.
size_t per_chunk_floats(int D) {
    const size_t d = static_cast<size_t>(D);
    return 64 * 64 + 3 * d * d + 2 * d + 4;
}

template <typename K>
cudaError_t allow_smem(K kernel, size_t bytes) {
    return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(bytes));
}

// The forward state pass, instantiated per count of value-column blocks.
template <int D, typename Tin, int NS>
cudaError_t launch_fstate_ns(const gbwd::GdnBwdArgs &a, unsigned bh, cudaStream_t s) {
    using namespace gbwd;
    cudaError_t e = allow_smem(gdn_bwd_fstate_kernel<D, Tin, NS>, fstate_smem<D, NS>());
    if (e != cudaSuccess) return e;
    gdn_bwd_fstate_kernel<D, Tin, NS><<<bh * NS, 512, fstate_smem<D, NS>(), s>>>(a);
    return cudaSuccess;
}
template <int D, typename Tin>
cudaError_t launch_fstate(const gbwd::GdnBwdArgs &a, unsigned bh, cudaStream_t s) {
    return a.nsplit == 4 ? launch_fstate_ns<D, Tin, 4>(a, bh, s)
         : a.nsplit == 2 ? launch_fstate_ns<D, Tin, 2>(a, bh, s) : launch_fstate_ns<D, Tin, 1>(a, bh, s);
}

template <int D, typename Tin>
cudaError_t run(const gbwd::GdecArgs &g, cudaStream_t s) {
    using namespace gbwd;
    const GdnBwdArgs &a = g.base;
    cudaError_t e;
    if ((e = allow_smem(gdn_bwd_prep_kernel<D, Tin>, prep_smem<D>())) != cudaSuccess) return e;
    if ((e = allow_smem(gdec_stats_kernel<D, Tin>, gdec_stats_smem<D>())) != cudaSuccess) return e;
    if ((e = allow_smem(gdec_out_kernel<D, Tin>, gdec_out_smem<D>())) != cudaSuccess) return e;
    const unsigned nch = static_cast<unsigned>(a.B * a.H * a.NC), bh = static_cast<unsigned>(a.B * a.H);
    const long long elems = (static_cast<long long>(D) * D + D + 1) * a.B * a.H;
    const unsigned eblocks = static_cast<unsigned>((elems + 255) / 256);
    gdn_bwd_prep_kernel<D, Tin><<<nch, 256, prep_smem<D>(), s>>>(a);
    if ((e = launch_fstate<D, Tin>(a, bh, s)) != cudaSuccess) return e;
    gdec_stats_kernel<D, Tin><<<nch, 256, gdec_stats_smem<D>(), s>>>(g);
    gdec_scan_kernel<D><<<eblocks, 256, 0, s>>>(g);
    gdec_out_kernel<D, Tin><<<nch, 256, gdec_out_smem<D>(), s>>>(g);
    return cudaGetLastError();
}

}  // namespace

size_t gdn_decayed_workspace_bytes(int B, int T, int H, int D) {
    const size_t chunks = static_cast<size_t>(B) * H * ((T + 63) / 64);
    return chunks * per_chunk_floats(D) * sizeof(float);
}

cudaError_t launch_gdn_decayed(const GdecCall &c, cudaStream_t s) {
    gbwd::GdecArgs g{};
    gbwd::GdnBwdArgs &a = g.base;
    a.B = c.B; a.T = c.T; a.H = c.H; a.NC = (c.T + 63) / 64;
    a.nsplit = gbwd::seq_split(c.B, c.H);
    a.l2norm = c.l2norm; a.centered = c.centered; a.scale = c.scale;
    a.q = c.q; a.k = c.k; a.v = c.v;
    a.g = c.g; a.beta = c.beta; a.lambda = c.lambda;
    a.S0 = c.S0; a.C0 = c.C0; a.m0 = c.m0;
    a.hT = c.ST;
    g.n0 = c.n0; g.o = c.o; g.CT = c.CT; g.mT = c.mT; g.nT = c.nT;
    g.cov_decay = c.cov_decay; g.contraction = c.contraction;
    const size_t chunks = static_cast<size_t>(c.B) * c.H * a.NC;
    const size_t d = static_cast<size_t>(c.D);
    float *p = static_cast<float *>(c.workspace);
    auto take = [&](size_t per) { float *r = p; p += chunks * per; return r; };
    a.tt = take(64 * 64); a.sk = take(d * d); a.mk = take(d); a.hs = take(d * d);
    g.dC = take(d * d); g.dmv = take(d); g.dn = take(4);
    if (c.D == 128) return c.bf16 ? run<128, __nv_bfloat16>(g, s) : run<128, float>(g, s);
    if (c.D == 64) return c.bf16 ? run<64, __nv_bfloat16>(g, s) : run<64, float>(g, s);
    return cudaErrorInvalidValue;
}

}  // namespace ccq
