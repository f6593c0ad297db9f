// ccq_gdn_decayed_kernels.cuh -- CCQ-Gated-DeltaNet forward with a decay-aligned covariance,
// CUDA-core kernels (fp32 arithmetic).
//
// The paper names a covariance built from gamma-weighted running statistics as the variant
// that matches a forgetting backbone, without fixing the weights or the normaliser.  Here
// gamma_{j,t} is the product of the backbone's own scalar decays over j < s <= t and the
// normaliser is the decayed count, so the statistics follow
//   C_t = alpha_t C_{t-1} + kbar_t kbar_t^T,  m_t = alpha_t m_{t-1} + kbar_t,  n_t = alpha_t n_{t-1} + 1,
//   Sigma^gamma_t = C_t / n_t - (m_t / n_t)(m_t / n_t)^T,   q_clean = qbar - lambda Sigma^gamma_t qbar
// (the gamma-weighted sample covariance; every alpha = 1 gives the undecayed statistics with
// n = t).  Inside a chunk entered with (C_r, m_r, n_r), row i sees
//   C_i qbar_i = E_i C_r qbar_i + sum_{j<=i} Gamma_ij (kbar_j . qbar_i) kbar_j,
//   m_i = E_i m_r + sum_{j<=i} Gamma_ij kbar_j,  n_i = E_i n_r + sum_{j<=i} Gamma_ij,
// (E_i = e^{gc_i}, Gamma_ij = e^{gc_i - gc_j}, gc the in-chunk cumulative log decay), and the
// output is the Gated DeltaNet chunk form O = scale (diag(E) Qc H_r + P U).  Launches: the
// backward's gdn_bwd_prep_kernel (Tt) and gdn_bwd_fstate_kernel (H_r, S_T), then
//   gdec_stats_kernel  per chunk: the chunk's decayed increments of C, m, n and its decay
//   gdec_scan_kernel   the statistics entering every chunk, and the final ones
//   gdec_out_kernel    per chunk: q_clean with Sigma^gamma, U, o
#pragma once

#include "ccq_gdn_bwd_kernels.cuh"

namespace ccq {
namespace gbwd {

// Extra arguments of the decayed-covariance forward; the GdnBwdArgs part carries the inputs,
// S0, the workspace arrays tt, sk, mk (prep), hs (entering states) and hT (final state).
struct GdecArgs {
    GdnBwdArgs base;
    const float *n0;           // [B][H] decayed count entering (NULL: zero, with C0, m0)
    void *o;                   // [B][T][H][D] in the input dtype
    float *CT, *mT, *nT;       // final statistics (each may be NULL)
    // workspace, per chunk: the chunk's increments, then the statistics entering it
    float *dC;                 // [D][D]
    float *dmv;                // [D]
    float *dn;                 // [4]: increment of n, the chunk's total decay e^{gc_last}, spare
};

// Per chunk: dC = sum_j e^{gc_last - gc_j} kbar_j kbar_j^T, dm likewise, dn = sum over the
// chunk's tokens of e^{gc_last - gc_j}, and the chunk's decay e^{gc_last}.
template <int D, typename Tin>
__global__ void __launch_bounds__(256) gdec_stats_kernel(const GdecArgs g) {
    extern __shared__ float4 gbwd_smem4[];
    const GdnBwdArgs &a = g.base;
    float *sm = reinterpret_cast<float *>(gbwd_smem4);
    float *Kb = sm;               // [64][D]
    float *graw = Kb + kC * D;    // [64]
    float *gc = graw + kC, *rk = gc + kC, *w = rk + kC;

    const int ch = blockIdx.x, r = ch % a.NC, bh = ch / a.NC, b = bh / a.H, h = bh % a.H;
    const int n = min(kC, a.T - r * kC);
    load_tile<D, Tin>(Kb, a.k, a, b, h, r);
    GBWD_FOR(i, kC) {
        const int t = r * kC + i;
        graw[i] = i < n ? a.g[tok_row(a, b, t < a.T ? t : 0, h)] : 0.f;
    }
    __syncthreads();
    row_rnorm<D>(Kb, rk, a.l2norm);
    gate_prefix(graw, gc);
    __syncthreads();
    GBWD_FOR(idx, kC * D) Kb[idx] *= rk[idx / D];
    GBWD_FOR(i, kC) w[i] = i < n ? expf(gc[kC - 1] - gc[i]) : 0.f;
    __syncthreads();
    float *dC = g.dC + static_cast<size_t>(ch) * D * D;
    GBWD_FOR(idx, D * D) {
        const int p = idx / D, c = idx % D;
        float acc = 0.f;
        for (int i = 0; i < kC; ++i) acc += w[i] * Kb[i * D + p] * Kb[i * D + c];
        dC[idx] = acc;
    }
    float *dm = g.dmv + static_cast<size_t>(ch) * D;
    GBWD_FOR(c, D) {
        float acc = 0.f;
        for (int i = 0; i < kC; ++i) acc += w[i] * Kb[i * D + c];
        dm[c] = acc;
    }
    if (threadIdx.x == 0) {
        float acc = 0.f;
        for (int i = 0; i < kC; ++i) acc += w[i];
        float *dn = g.dn + static_cast<size_t>(ch) * 4;
        dn[0] = acc;
        dn[1] = expf(gc[kC - 1]);
        dn[2] = dn[3] = 0.f;
    }
}

// Decayed scan over the chunks of each sequence and head, one thread per element of
// (C, m, n): x_{r+1} = e^{gc_last,r} x_r + dx_r.  Replaces every increment by the value
// entering its chunk and writes the final values.
template <int D>
__global__ void __launch_bounds__(256) gdec_scan_kernel(const GdecArgs g) {
    const GdnBwdArgs &a = g.base;
    const long long per = static_cast<long long>(D) * D + D + 1;
    const long long gid = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (gid >= per * a.B * a.H) return;
    const int bh = static_cast<int>(gid / per);
    const int e = static_cast<int>(gid % per);
    const size_t nc = static_cast<size_t>(a.NC);
    float *base;
    size_t stride;
    float acc = 0.f;
    if (e < D * D) {
        base = g.dC + static_cast<size_t>(bh) * nc * D * D + e;
        stride = static_cast<size_t>(D) * D;
        if (a.C0) acc = a.C0[static_cast<size_t>(bh) * D * D + e];
    } else if (e < D * D + D) {
        const int em = e - D * D;
        base = g.dmv + static_cast<size_t>(bh) * nc * D + em;
        stride = D;
        if (a.m0) acc = a.m0[static_cast<size_t>(bh) * D + em];
    } else {
        base = g.dn + static_cast<size_t>(bh) * nc * 4;
        stride = 4;
        if (g.n0) acc = g.n0[bh];
    }
    const float *decay = g.dn + static_cast<size_t>(bh) * nc * 4 + 1;
    for (size_t r = 0; r < nc; ++r) {
        const float x = base[r * stride];
        base[r * stride] = acc;
        acc = decay[r * 4] * acc + x;
    }
    if (e < D * D) {
        if (g.CT) g.CT[static_cast<size_t>(bh) * D * D + e] = acc;
    } else if (e < D * D + D) {
        if (g.mT) g.mT[static_cast<size_t>(bh) * D + (e - D * D)] = acc;
    } else if (g.nT) {
        g.nT[bh] = acc;
    }
}

// Per chunk: q_clean with the decayed statistics, U = Tt diag(beta)(V - diag(E) Kbar H_r),
// o = scale (diag(E) Qc H_r + P U).
template <int D, typename Tin>
__global__ void __launch_bounds__(256) gdec_out_kernel(const GdecArgs g) {
    extern __shared__ float4 gbwd_smem4[];
    const GdnBwdArgs &a = g.base;
    float *sm = reinterpret_cast<float *>(gbwd_smem4);
    float *Qb = sm;                // [64][D] qbar, then qc
    float *Kb = Qb + kC * D;       // [64][D]
    float *Rv = Kb + kC * D;       // [64][D] V, then R
    float *Uu = Rv + kC * D;       // [64][D] U
    float *Zz = Uu + kC * D;       // [64][D] Sigma^gamma qbar
    float *sA = Zz + kC * D;       // [64][64] (Qbar Kbar^T) o Gamma o causal, then P
    float *graw = sA + kC * kC;
    float *gc = graw + kC, *E = gc + kC, *be = E + kC, *lam = be + kC, *rq = lam + kC, *rk = rq + kC;
    float *nn = rk + kC, *mq = nn + kC;

    const int ch = blockIdx.x, r = ch % a.NC, bh = ch / a.NC, b = bh / a.H, h = bh % a.H;
    const int n = min(kC, a.T - r * kC);
    const float c = a.centered ? 1.f : 0.f;
    const float *H = a.hs + static_cast<size_t>(ch) * D * D;
    const float *Cr = g.dC + static_cast<size_t>(ch) * D * D;
    const float *mr = g.dmv + static_cast<size_t>(ch) * D;
    const float nr = g.dn[static_cast<size_t>(ch) * 4];
    const float *Tt = a.tt + static_cast<size_t>(ch) * kC * kC;

    load_tile<D, Tin>(Qb, a.q, a, b, h, r);
    load_tile<D, Tin>(Kb, a.k, a, b, h, r);
    load_tile<D, Tin>(Rv, a.v, a, b, h, r);
    GBWD_FOR(i, kC) {
        const int t = r * kC + i;
        const size_t row = tok_row(a, b, t < a.T ? t : 0, h);
        graw[i] = i < n ? a.g[row] : 0.f;
        be[i] = i < n ? a.beta[row] : 0.f;
        lam[i] = i < n ? a.lambda[row] : 0.f;
    }
    __syncthreads();
    row_rnorm<D>(Qb, rq, a.l2norm);
    row_rnorm<D>(Kb, rk, a.l2norm);
    gate_prefix(graw, gc);
    __syncthreads();
    GBWD_FOR(idx, kC * D) {
        Qb[idx] *= rq[idx / D];
        Kb[idx] *= rk[idx / D];
    }
    GBWD_FOR(i, kC) E[i] = expf(gc[i]);
    __syncthreads();
    // decayed causal scores (diagonal included);  R = V - diag(E) Kbar H_r
    GBWD_FOR(idx, kC * kC) {
        const int i = idx / kC, j = idx % kC;
        float acc = 0.f;
        if (j <= i) {
            for (int l = 0; l < D; ++l) acc += Qb[i * D + l] * Kb[j * D + l];
            acc *= expf(gc[i] - gc[j]);
        }
        sA[idx] = acc;
    }
    GBWD_FOR(idx, kC * D) {
        const int i = idx / D, j = idx % D;
        float acc = 0.f;
        for (int l = 0; l < D; ++l) acc += Kb[i * D + l] * H[l * D + j];
        Rv[idx] -= E[i] * acc;
    }
    __syncthreads();
    // n_i and m_i . qbar_i;  U = Tt diag(beta) R
    GBWD_FOR(i, kC) {
        float cnt = E[i] * nr, dot = 0.f;
        for (int j = 0; j <= i && j < n; ++j) cnt += expf(gc[i] - gc[j]);
        for (int l = 0; l < D; ++l) dot += mr[l] * Qb[i * D + l];
        dot *= E[i];
        for (int j = 0; j <= i; ++j) dot += sA[i * kC + j];
        nn[i] = cnt;
        mq[i] = dot;
    }
    GBWD_FOR(idx, kC * D) {
        const int i = idx / D, j = idx % D;
        float acc = 0.f;
        for (int l = 0; l <= i; ++l) acc += Tt[i * kC + l] * be[l] * Rv[l * D + j];
        Uu[idx] = acc;
    }
    __syncthreads();
    // Sigma^gamma qbar = C_i qbar_i / n_i - c m_i (m_i . qbar_i) / n_i^2
    GBWD_FOR(idx, kC * D) {
        const int i = idx / D, j = idx % D;
        float cq = 0.f, mi = 0.f;
        for (int l = 0; l < D; ++l) cq += Cr[j * D + l] * Qb[i * D + l];
        cq *= E[i];
        mi = E[i] * mr[j];
        for (int l = 0; l <= i; ++l) {
            cq += sA[i * kC + l] * Kb[l * D + j];
            mi += expf(gc[i] - gc[l]) * Kb[l * D + j];
        }
        const float ninv = i < n ? 1.f / nn[i] : 0.f;
        Zz[idx] = cq * ninv - c * mi * mq[i] * ninv * ninv;
    }
    __syncthreads();
    GBWD_FOR(idx, kC * D) Qb[idx] -= lam[idx / D] * Zz[idx];
    __syncthreads();
    // P = (Qc Kbar^T) o Gamma o causal
    GBWD_FOR(idx, kC * kC) {
        const int i = idx / kC, j = idx % kC;
        float acc = 0.f;
        if (j <= i) {
            for (int l = 0; l < D; ++l) acc += Qb[i * D + l] * Kb[j * D + l];
            acc *= expf(gc[i] - gc[j]);
        }
        sA[idx] = acc;
    }
    __syncthreads();
    {
        Tin *o = static_cast<Tin *>(g.o);
        GBWD_FOR(idx, kC * D) {
            const int i = idx / D, j = idx % D;
            if (i >= n) continue;
            float acc = 0.f;
            for (int l = 0; l < D; ++l) acc += Qb[i * D + l] * H[l * D + j];
            acc *= E[i];
            for (int l = 0; l <= i; ++l) acc += sA[i * kC + l] * Uu[l * D + j];
            o[tok_row(a, b, r * kC + i, h) * D + j] = from_f<Tin>(a.scale * acc);
        }
    }
}

template <int D> constexpr size_t gdec_stats_smem() { return sizeof(float) * (kC * D + 4 * kC); }
template <int D> constexpr size_t gdec_out_smem() { return sizeof(float) * (5 * kC * D + kC * kC + 9 * kC); }

}  // namespace gbwd
}  // namespace ccq
