// ccq_gdn_bwd.cu -- launches of the CUDA-core CCQ-Gated-DeltaNet backward
// (kernels and the adjoint they evaluate: ccq_gdn_bwd_kernels.cuh).
#include <cuda_runtime.h>
#include <stdint.h>

#include <type_traits>

#include "ccq_gdn_bwd_kernels.cuh"
#include "ccq_gdn_bwd.h"
#include "ccq_internal.h"

namespace ccq {

namespace {

// Workspace floats per chunk (layout of gbwd::GdnBwdArgs): Tt, S^K_r, M_r, H_r, dH, DC, Dm,
// P^T D, (diag(E) Qc)^T D, qbar, qc, U, R, W and the row vectors.
size_t per_chunk_floats(int D) {
    const size_t d = static_cast<size_t>(D);
    return 64 * 64 + 5 * d * d + 2 * d + 6 * 64 * d + 4 * 64;
}

template <typename K>
cudaError_t allow_smem(K kernel, size_t bytes) {
    return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(bytes));
}

// The sequential passes, instantiated per count of value-column blocks.
template <int D, typename Tin, int NS>
cudaError_t launch_fstate_ns(const gbwd::GdnBwdArgs &a, unsigned bh, cudaStream_t s) {
    using namespace gbwd;
    cudaError_t e = allow_smem(gdn_bwd_fstate_kernel<D, Tin, NS>, fstate_smem<D, NS>());
    if (e != cudaSuccess) return e;
    gdn_bwd_fstate_kernel<D, Tin, NS><<<bh * NS, 512, fstate_smem<D, NS>(), s>>>(a);
    return cudaSuccess;
}
template <int D, typename Tin, int NS>
cudaError_t launch_dstate_ns(const gbwd::GdnBwdArgs &a, unsigned bh, cudaStream_t s) {
    using namespace gbwd;
    cudaError_t e = allow_smem(gdn_bwd_dstate_kernel<D, Tin, NS>, dstate_smem<D, NS>());
    if (e != cudaSuccess) return e;
    gdn_bwd_dstate_kernel<D, Tin, NS><<<bh * NS, 512, dstate_smem<D, NS>(), s>>>(a);
    return cudaSuccess;
}
template <int D, typename Tin>
cudaError_t launch_fstate(const gbwd::GdnBwdArgs &a, unsigned bh, cudaStream_t s) {
    return a.nsplit == 4 ? launch_fstate_ns<D, Tin, 4>(a, bh, s)
         : a.nsplit == 2 ? launch_fstate_ns<D, Tin, 2>(a, bh, s) : launch_fstate_ns<D, Tin, 1>(a, bh, s);
}
template <int D, typename Tin>
cudaError_t launch_dstate(const gbwd::GdnBwdArgs &a, unsigned bh, cudaStream_t s) {
    return a.nsplit == 4 ? launch_dstate_ns<D, Tin, 4>(a, bh, s)
         : a.nsplit == 2 ? launch_dstate_ns<D, Tin, 2>(a, bh, s) : launch_dstate_ns<D, Tin, 1>(a, bh, s);
}

template <int D, typename Tin>
cudaError_t run(gbwd::GdnBwdArgs a, cudaStream_t s) {
    using namespace gbwd;
    // bf16 inputs: the per-chunk kernels' products on the tensor cores (bf16 operands, the
    // forward's precision); fp32 inputs keep fp32 products on the CUDA cores
    constexpr bool kTc = std::is_same<Tin, __nv_bfloat16>::value;
    cudaError_t e;
    if (kTc && !(a.status = device_status_word())) return cudaErrorInvalidValue;
    if ((e = allow_smem(gdn_bwd_prep_kernel<D, Tin>, prep_smem<D>())) != cudaSuccess) return e;
    if ((e = allow_smem(gdn_bwd_local_kernel<D, Tin, kTc>, local_smem<D, kTc>())) != cudaSuccess) return e;
    if ((e = allow_smem(gdn_bwd_kv_kernel<D, Tin, kTc>, kv_smem<D, kTc>())) != cudaSuccess) return e;
    const unsigned nch = static_cast<unsigned>(a.B * a.H * a.NC), bh = static_cast<unsigned>(a.B * a.H);
    const long long elems = (static_cast<long long>(D) * D + D) * a.B * a.H;
    const unsigned eblocks = static_cast<unsigned>((elems + 255) / 256);
    if (!a.states_ready) {
        gdn_bwd_prep_kernel<D, Tin><<<nch, 256, prep_smem<D>(), s>>>(a);
        gdn_bwd_prefix_kernel<D><<<eblocks, 256, 0, s>>>(a);
        if ((e = launch_fstate<D, Tin>(a, bh, s)) != cudaSuccess) return e;
    }
    gdn_bwd_local_kernel<D, Tin, kTc><<<nch, kBwdThreads, local_smem<D, kTc>(), s>>>(a);
    if (D == 128 && std::is_same<Tin, __nv_bfloat16>::value && a.states_ready) {
        // bf16, Dk = 128: the reverse state pass on tensor cores
        if ((e = launch_gdn_dstate_tc(a, a.k, s)) != cudaSuccess) return e;
    } else if ((e = launch_dstate<D, Tin>(a, bh, s)) != cudaSuccess) {
        return e;
    }
    gdn_bwd_suffix_kernel<D><<<eblocks, 256, 0, s>>>(a);
    gdn_bwd_kv_kernel<D, Tin, kTc><<<nch, kBwdThreads, kv_smem<D, kTc>(), s>>>(a);
    return cudaGetLastError();
}

}  // namespace

void gdn_bwd_state_arrays(const GdnBwdCall &c, float **tt, float **sk, float **mk, float **hs) {
    const size_t chunks = static_cast<size_t>(c.B) * c.H * ((c.T + 63) / 64);
    const size_t d = static_cast<size_t>(c.D);
    float *p = static_cast<float *>(c.workspace);
    *tt = p;
    *sk = p + chunks * 64 * 64;
    *mk = *sk + chunks * d * d;
    *hs = *mk + chunks * d;
}

size_t gdn_bwd_workspace_bytes(int B, int T, int H, int D) {
    const size_t chunks = static_cast<size_t>(B) * H * ((T + 63) / 64);
    return chunks * per_chunk_floats(D) * sizeof(float);
}

cudaError_t launch_gdn_bwd(const GdnBwdCall &c, cudaStream_t s) {
    gbwd::GdnBwdArgs a{};
    a.B = c.B; a.T = c.T; a.H = c.H; a.NC = (c.T + 63) / 64;
    a.nsplit = gbwd::seq_split(c.B, c.H);
    a.states_ready = c.states_ready;
    a.l2norm = c.l2norm; a.centered = c.centered; a.scale = c.scale;
    a.q = c.q; a.k = c.k; a.v = c.v; a.dout = c.dout;
    a.g = c.g; a.beta = c.beta; a.lambda = c.lambda;
    a.S0 = c.S0; a.C0 = c.C0; a.m0 = c.m0; a.t0 = c.t0;
    a.dST = c.dST; a.dCT = c.dCT; a.dmT = c.dmT;
    a.dq = c.dq; a.dk = c.dk; a.dv = c.dv;
    a.dg = c.dg; a.dbeta = c.dbeta; a.dlambda = c.dlambda;
    a.dS0 = c.dS0; a.dC0 = c.dC0; a.dm0 = c.dm0;
    const size_t chunks = static_cast<size_t>(c.B) * c.H * a.NC;
    const size_t d = static_cast<size_t>(c.D);
    float *p = static_cast<float *>(c.workspace);
    auto take = [&](size_t per) { float *r = p; p += chunks * per; return r; };
    a.tt = take(64 * 64); a.sk = take(d * d); a.mk = take(d); a.hs = take(d * d); a.dh = take(d * d);
    a.dc = take(d * d); a.dm = take(d); a.x1 = take(64 * d); a.y1 = take(d * d);
    a.qb = take(64 * d); a.qc = take(64 * d); a.u = take(64 * d); a.r = take(64 * d); a.w = take(64 * d);
    a.vec = take(4 * 64);
    if (c.D == 128) return c.bf16 ? run<128, __nv_bfloat16>(a, s) : run<128, float>(a, s);
    if (c.D == 64) return c.bf16 ? run<64, __nv_bfloat16>(a, s) : run<64, float>(a, s);
    return cudaErrorInvalidValue;
}

}  // namespace ccq
