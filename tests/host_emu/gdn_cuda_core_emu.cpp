// Host build of the CUDA-core CCQ-Gated-DeltaNet kernels (the backward and the forward with
// the decay-aligned covariance), for a CPU test of their arithmetic and indexing against the
// fp64 oracle (tests/test_gdn_bwd_host.py, tests/test_gdn_decayed_host.py).  Test
// infrastructure only: the library never builds or loads this file.
//
// The kernels are written as phases separated by __syncthreads(), in each of which every
// thread strides over the elements it owns and reads only what earlier phases wrote.  Run
// with one thread per CTA, each phase therefore computes exactly what the whole CTA computes
// on the GPU, so the CTAs are executed one after another, phase by phase.  Each CTA gets a
// fresh heap block of exactly the kernel's dynamic shared-memory size, filled with NaN, so
// that a read of shared memory no phase wrote shows up in the results and an access past the
// end is visible to an address sanitizer.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstdlib>
#include <cstring>
#include <type_traits>
#include <vector>

static uint3 threadIdx, blockIdx;
static dim3 blockDim, gridDim;
#define __syncthreads() ((void)0)
#undef __launch_bounds__
#define __launch_bounds__(...)
static inline float atomicAdd(float *p, float v) {
    const float o = *p;
    *p += v;
    return o;
}
using std::min;
// The kernels' `extern __shared__ float4 gbwd_smem4[]` becomes a block-scope declaration of
// this pointer (to the current CTA's block) in their namespace.
namespace ccq {
namespace gbwd {
float4 (*g_smem)[];
}  // namespace gbwd
}  // namespace ccq
#define gbwd_smem4 (*g_smem)
#include "../../paper_2606_01294_gb300/csrc/ccq_gdn_decayed_kernels.cuh"
#undef gbwd_smem4
using namespace ccq::gbwd;

template <typename F>
static void run_blocks(F f, long long grid, size_t smem_bytes) {
    blockDim = dim3(1);
    threadIdx = make_uint3(0, 0, 0);
    for (long long bx = 0; bx < grid; ++bx) {
        blockIdx = make_uint3(static_cast<unsigned>(bx), 0, 0);
        void *blk = nullptr;
        if (smem_bytes) {
            blk = std::malloc(smem_bytes);
            std::memset(blk, 0xff, smem_bytes);  // NaN
        }
        ccq::gbwd::g_smem = reinterpret_cast<float4 (*)[]>(blk);
        f();
        std::free(blk);
    }
}

// The sequential passes are instantiated per count of value-column blocks (1, 2 or 4).
template <int D, typename Tin>
static void run_fstate(const GdnBwdArgs &a, long long bh) {
    if (a.nsplit == 4) run_blocks([&] { gdn_bwd_fstate_kernel<D, Tin, 4>(a); }, bh * 4, fstate_smem<D, 4>());
    else if (a.nsplit == 2) run_blocks([&] { gdn_bwd_fstate_kernel<D, Tin, 2>(a); }, bh * 2, fstate_smem<D, 2>());
    else run_blocks([&] { gdn_bwd_fstate_kernel<D, Tin, 1>(a); }, bh, fstate_smem<D, 1>());
}
template <int D, typename Tin>
static void run_dstate(const GdnBwdArgs &a, long long bh) {
    if (a.nsplit == 4) run_blocks([&] { gdn_bwd_dstate_kernel<D, Tin, 4>(a); }, bh * 4, dstate_smem<D, 4>());
    else if (a.nsplit == 2) run_blocks([&] { gdn_bwd_dstate_kernel<D, Tin, 2>(a); }, bh * 2, dstate_smem<D, 2>());
    else run_blocks([&] { gdn_bwd_dstate_kernel<D, Tin, 1>(a); }, bh, dstate_smem<D, 1>());
}

template <int D, typename Tin>
static void run(const GdnBwdArgs &a) {
    const long long nch = static_cast<long long>(a.B) * a.H * a.NC, bh = static_cast<long long>(a.B) * a.H;
    const long long elems = (static_cast<long long>(D) * D + D) * bh;
    run_blocks([&] { gdn_bwd_prep_kernel<D, Tin>(a); }, nch, prep_smem<D>());
    run_blocks([&] { gdn_bwd_prefix_kernel<D>(a); }, elems, 0);
    run_fstate<D, Tin>(a, bh);
    // bf16 inputs with D >= 64 take the kernels' tensor-core instantiation, as the library does; on
    // the host its products are computed in place on bf16-rounded operands (ccq_gdn_bwd_tc.cuh)
    constexpr bool kTc = std::is_same<Tin, __nv_bfloat16>::value && D >= 64;
    run_blocks([&] { gdn_bwd_local_kernel<D, Tin, kTc>(a); }, nch, local_smem<D, kTc>());
    run_dstate<D, Tin>(a, bh);
    run_blocks([&] { gdn_bwd_suffix_kernel<D>(a); }, elems, 0);
    run_blocks([&] { gdn_bwd_kv_kernel<D, Tin, kTc>(a); }, nch, kv_smem<D, kTc>());
}

template <typename Tin>
static std::vector<Tin> to_in(const float *x, size_t n) {
    std::vector<Tin> y(n);
    for (size_t i = 0; i < n; ++i) y[i] = from_f<Tin>(x[i]);
    return y;
}

template <typename Tin>
static void to_out(const std::vector<Tin> &y, float *x) {
    for (size_t i = 0; i < y.size(); ++i) x[i] = to_f(y[i]);
}

template <int D, typename Tin>
static int go(int B, int T, int H, int l2norm, int centered, float scale, const float *const *in,
              const int64_t *t0, float *const *out) {
    // in: q, k, v, dout, g, beta, lambda, S0, C0, m0, dST, dCT, dmT
    // out: dq, dk, dv, dg, dbeta, dlambda, dS0, dC0, dm0
    const size_t ntok = static_cast<size_t>(B) * T * H * D;
    auto q = to_in<Tin>(in[0], ntok), k = to_in<Tin>(in[1], ntok), v = to_in<Tin>(in[2], ntok),
         dout = to_in<Tin>(in[3], ntok);
    std::vector<Tin> dq(ntok), dk(ntok), dv(ntok);
    GdnBwdArgs a{};
    a.B = B; a.T = T; a.H = H; a.NC = (T + 63) / 64;
    a.nsplit = 1 << (T % 3);  // 1, 2 or 4 value-column blocks in the sequential passes, by T
    a.l2norm = l2norm; a.centered = centered; a.scale = scale;
    a.q = q.data(); a.k = k.data(); a.v = v.data(); a.dout = dout.data();
    a.g = in[4]; a.beta = in[5]; a.lambda = in[6]; a.S0 = in[7]; a.C0 = in[8]; a.m0 = in[9]; a.t0 = t0;
    a.dST = in[10]; a.dCT = in[11]; a.dmT = in[12];
    a.dq = dq.data(); a.dk = dk.data(); a.dv = dv.data();
    a.dg = out[3]; a.dbeta = out[4]; a.dlambda = out[5]; a.dS0 = out[6]; a.dC0 = out[7]; a.dm0 = out[8];
    const size_t chunks = static_cast<size_t>(B) * H * a.NC, d = D;
    std::vector<float> ws(chunks * (64 * 64 + 5 * d * d + 2 * d + 6 * 64 * d + 4 * 64), NAN);
    float *p = ws.data();
    auto take = [&](size_t per) { float *r = p; p += chunks * per; return r; };
    a.tt = take(64 * 64); a.sk = take(d * d); a.mk = take(d); a.hs = take(d * d); a.dh = take(d * d);
    a.dc = take(d * d); a.dm = take(d); a.x1 = take(64 * d); a.y1 = take(d * d);
    a.qb = take(64 * d); a.qc = take(64 * d); a.u = take(64 * d); a.r = take(64 * d); a.w = take(64 * d);
    a.vec = take(4 * 64);
    run<D, Tin>(a);
    to_out(dq, out[0]);
    to_out(dk, out[1]);
    to_out(dv, out[2]);
    return 0;
}

extern "C" int gdn_bwd_emu(int D, int bf16, int B, int T, int H, int l2norm, int centered, float scale,
                           const float *const *in, const int64_t *t0, float *const *out) {
    if (D == 16) return bf16 ? go<16, __nv_bfloat16>(B, T, H, l2norm, centered, scale, in, t0, out)
                             : go<16, float>(B, T, H, l2norm, centered, scale, in, t0, out);
    if (D == 64) return bf16 ? go<64, __nv_bfloat16>(B, T, H, l2norm, centered, scale, in, t0, out)
                             : go<64, float>(B, T, H, l2norm, centered, scale, in, t0, out);
    if (D == 128 && bf16) return go<128, __nv_bfloat16>(B, T, H, l2norm, centered, scale, in, t0, out);
    return -1;
}

template <int D, typename Tin>
static int go_dec(int B, int T, int H, int l2norm, int centered, float scale, int contraction, int decayed,
                  const float *const *in, float *const *out) {
    // in: q, k, v, g, beta, lambda, S0, C0, m0, n0;  out: o, ST, CT, mT, nT
    const size_t ntok = static_cast<size_t>(B) * T * H * D;
    auto q = to_in<Tin>(in[0], ntok), k = to_in<Tin>(in[1], ntok), v = to_in<Tin>(in[2], ntok);
    std::vector<Tin> o(ntok);
    GdecArgs g{};
    GdnBwdArgs &a = g.base;
    a.B = B; a.T = T; a.H = H; a.NC = (T + 63) / 64;
    a.nsplit = 1 << (T % 3);  // 1, 2 or 4 value-column blocks in the sequential passes, by T
    a.l2norm = l2norm; a.centered = centered; a.scale = scale;
    a.q = q.data(); a.k = k.data(); a.v = v.data();
    a.g = in[3]; a.beta = in[4]; a.lambda = in[5]; a.S0 = in[6]; a.C0 = in[7]; a.m0 = in[8];
    g.n0 = in[9];
    g.o = o.data();
    g.contraction = contraction;
    g.cov_decay = decayed;
    a.hT = out[1]; g.CT = out[2]; g.mT = out[3]; g.nT = out[4];
    const size_t chunks = static_cast<size_t>(B) * H * a.NC, d = D;
    std::vector<float> ws(chunks * (64 * 64 + 3 * d * d + 2 * d + 4), NAN);
    float *p = ws.data();
    auto take = [&](size_t per) { float *r = p; p += chunks * per; return r; };
    a.tt = take(64 * 64); a.sk = take(d * d); a.mk = take(d); a.hs = take(d * d);
    g.dC = take(d * d); g.dmv = take(d); g.dn = take(4);
    const long long nch = static_cast<long long>(chunks), bh = static_cast<long long>(B) * H;
    run_blocks([&] { gdn_bwd_prep_kernel<D, Tin>(a); }, nch, prep_smem<D>());
    run_fstate<D, Tin>(a, bh);
    run_blocks([&] { gdec_stats_kernel<D, Tin>(g); }, nch, gdec_stats_smem<D>());
    run_blocks([&] { gdec_scan_kernel<D>(g); }, (static_cast<long long>(D) * D + D + 1) * bh, 0);
    run_blocks([&] { gdec_out_kernel<D, Tin>(g); }, nch, gdec_out_smem<D>());
    to_out(o, out[0]);
    return 0;
}

extern "C" int gdn_spectral_emu(int D, int bf16, int B, int T, int H, int l2norm, int centered, float scale,
                                int contraction, int decayed, const float *const *in, float *const *out) {
    if (D == 16)
        return bf16 ? go_dec<16, __nv_bfloat16>(B, T, H, l2norm, centered, scale, contraction, decayed, in, out)
                    : go_dec<16, float>(B, T, H, l2norm, centered, scale, contraction, decayed, in, out);
    if (D == 64 && !bf16) return go_dec<64, float>(B, T, H, l2norm, centered, scale, contraction, decayed, in, out);
    return -1;
}
