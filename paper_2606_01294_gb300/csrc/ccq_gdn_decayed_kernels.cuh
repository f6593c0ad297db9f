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
// output is the Gated DeltaNet chunk form O = scale (diag(E) Qc H_r + P U).  With cov_decay = 0
// the statistics are the paper's undecayed sums (E and Gamma replaced by 1 in them, n = t).
// The contraction is the paper's q_clean = qbar - lambda Sigma qbar, or one of the two
// alternatives it names with that first-order form: (I + lambda Sigma)^{-1} qbar by conjugate
// gradients per row (I + lambda Sigma is symmetric with spectrum in [1, 1 + lambda], so ten
// iterations from the linear estimate leave an error below 1e-6 relative), or
// exp(-lambda Sigma) qbar by its Taylor series (|lambda Sigma| <= 1: twelve terms leave 1e-10).  Launches: the
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
    int cov_decay = 1;         // 1: decay-aligned statistics; 0: the paper's undecayed ones
    int contraction = 0;       // 0: I - lambda Sigma; 1: (I + lambda Sigma)^{-1}; 2: exp(-lambda Sigma)
};

constexpr int kCgIters = 10;   // conjugate-gradient iterations of the resolvent contraction
constexpr int kExpTerms = 12;  // Taylor terms of the exponential contraction

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
    GBWD_FOR(i, kC) w[i] = i < n ? (g.cov_decay ? expf(gc[kC - 1] - gc[i]) : 1.f) : 0.f;
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
        dn[1] = g.cov_decay ? expf(gc[kC - 1]) : 1.f;
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

// Row-wise Sigma_i p_i for the 64 rows of a chunk (three phases): with W the covariance
// weights (Gamma o causal, or the causal mask for undecayed statistics) and Ec_i the weight of
// the chunk-start statistics, Sigma_i p = (Ec_i C_r p + sum_{l<=i} W_il (kbar_l . p) kbar_l) / n_i
// - c m_i (m_i . p) / n_i^2,  m_i = Ec_i m_r + sum_{l<=i} W_il kbar_l.  Rows past n give 0.
template <int D>
__device__ __forceinline__ void apply_sigma(const float *P, float *out, const float *Kb, const float *Wc,
                                            const float *Ec, const float *ninv, const float *Cr,
                                            const float *mr, float c, float *sS, float *mp) {
    GBWD_FOR(idx, kC * kC) {
        const int i = idx / kC, l = idx % kC;
        float acc = 0.f;
        if (l <= i)
            for (int j = 0; j < D; ++j) acc += Kb[l * D + j] * P[i * D + j];
        sS[idx] = acc * Wc[idx];
    }
    __syncthreads();
    GBWD_FOR(i, kC) {
        float acc = 0.f;
        for (int j = 0; j < D; ++j) acc += mr[j] * P[i * D + j];
        acc *= Ec[i];
        for (int l = 0; l <= i; ++l) acc += sS[i * kC + l];
        mp[i] = acc;
    }
    __syncthreads();
    GBWD_FOR(idx, kC * D) {
        const int i = idx / D, j = idx % D;
        float cp = 0.f;
        for (int l = 0; l < D; ++l) cp += Cr[j * D + l] * P[i * D + l];
        cp *= Ec[i];
        float mi = Ec[i] * mr[j];
        for (int l = 0; l <= i; ++l) {
            cp += sS[i * kC + l] * Kb[l * D + j];
            mi += Wc[i * kC + l] * Kb[l * D + j];
        }
        out[idx] = cp * ninv[i] - c * mi * mp[i] * ninv[i] * ninv[i];
    }
    __syncthreads();
}

// Per chunk: q_clean with the chunk's statistics and contraction,
// U = Tt diag(beta)(V - diag(E) Kbar H_r), o = scale (diag(E) Qc H_r + P U).
template <int D, typename Tin>
__global__ void __launch_bounds__(256) gdec_out_kernel(const GdecArgs g) {
    extern __shared__ float4 gbwd_smem4[];
    const GdnBwdArgs &a = g.base;
    float *sm = reinterpret_cast<float *>(gbwd_smem4);
    float *Qb = sm;                // [64][D] qbar, then q_clean
    float *Kb = Qb + kC * D;       // [64][D]
    float *B1 = Kb + kC * D;       // [64][D] scratch, then R
    float *B2 = B1 + kC * D;       // [64][D] scratch, then U
    float *B3 = B2 + kC * D;       // [64][D] scratch
    float *sA = B3 + kC * D;       // [64][64] scores, then P
    float *Wc = sA + kC * kC;      // [64][64] covariance weights
    float *graw = Wc + kC * kC;
    float *gc = graw + kC, *E = gc + kC, *Ec = E + kC, *be = Ec + kC, *lam = be + kC, *rq = lam + kC;
    float *rk = rq + kC, *ninv = rk + kC, *mp = ninv + kC, *rr = mp + kC, *al = rr + kC, *bt = al + kC;

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
    GBWD_FOR(i, kC) {
        E[i] = expf(gc[i]);
        Ec[i] = g.cov_decay ? E[i] : 1.f;
    }
    GBWD_FOR(idx, kC * kC) {
        const int i = idx / kC, l = idx % kC;
        Wc[idx] = l <= i && l < n ? (g.cov_decay ? expf(gc[i] - gc[l]) : 1.f) : 0.f;
    }
    __syncthreads();
    GBWD_FOR(i, kC) {
        float cnt = Ec[i] * nr;
        for (int l = 0; l <= i; ++l) cnt += Wc[i * kC + l];
        ninv[i] = i < n ? 1.f / cnt : 0.f;
    }
    __syncthreads();
    // q_clean (into Qb)
    apply_sigma<D>(Qb, B3, Kb, Wc, Ec, ninv, Cr, mr, c, sA, mp);  // B3 = Sigma qbar
    if (g.contraction == 1) {
        // (I + lambda Sigma) x = qbar by conjugate gradients per row, from x0 = qbar - lambda Sigma qbar
        GBWD_FOR(idx, kC * D) B1[idx] = Qb[idx] - lam[idx / D] * B3[idx];
        __syncthreads();
        apply_sigma<D>(B1, B3, Kb, Wc, Ec, ninv, Cr, mr, c, sA, mp);
        GBWD_FOR(idx, kC * D) {
            const float res = Qb[idx] - B1[idx] - lam[idx / D] * B3[idx];
            Qb[idx] = res;  // r (qbar is no longer needed)
            B2[idx] = res;  // p
        }
        __syncthreads();
        GBWD_FOR(i, kC) {
            float acc = 0.f;
            for (int j = 0; j < D; ++j) acc += Qb[i * D + j] * Qb[i * D + j];
            rr[i] = acc;
        }
        __syncthreads();
        for (int it = 0; it < kCgIters; ++it) {
            apply_sigma<D>(B2, B3, Kb, Wc, Ec, ninv, Cr, mr, c, sA, mp);
            GBWD_FOR(idx, kC * D) B3[idx] = B2[idx] + lam[idx / D] * B3[idx];  // A p
            __syncthreads();
            GBWD_FOR(i, kC) {
                float pap = 0.f;
                for (int j = 0; j < D; ++j) pap += B2[i * D + j] * B3[i * D + j];
                al[i] = pap > 0.f ? rr[i] / pap : 0.f;
            }
            __syncthreads();
            GBWD_FOR(idx, kC * D) {
                const int i = idx / D;
                B1[idx] += al[i] * B2[idx];
                Qb[idx] -= al[i] * B3[idx];
            }
            __syncthreads();
            GBWD_FOR(i, kC) {
                float acc = 0.f;
                for (int j = 0; j < D; ++j) acc += Qb[i * D + j] * Qb[i * D + j];
                bt[i] = rr[i] > 0.f ? acc / rr[i] : 0.f;
                rr[i] = acc;
            }
            __syncthreads();
            GBWD_FOR(idx, kC * D) B2[idx] = Qb[idx] + bt[idx / D] * B2[idx];
            __syncthreads();
        }
        GBWD_FOR(idx, kC * D) Qb[idx] = B1[idx];
    } else if (g.contraction == 2) {
        // exp(-lambda Sigma) qbar = sum_k (-lambda Sigma)^k qbar / k!
        GBWD_FOR(idx, kC * D) {
            B1[idx] = Qb[idx] - lam[idx / D] * B3[idx];  // terms 0 and 1
            B2[idx] = -lam[idx / D] * B3[idx];           // term 1
        }
        __syncthreads();
        for (int k = 2; k <= kExpTerms; ++k) {
            apply_sigma<D>(B2, B3, Kb, Wc, Ec, ninv, Cr, mr, c, sA, mp);
            const float inv = 1.f / static_cast<float>(k);
            GBWD_FOR(idx, kC * D) {
                const float tv = -lam[idx / D] * inv * B3[idx];
                B2[idx] = tv;
                B1[idx] += tv;
            }
            __syncthreads();
        }
        GBWD_FOR(idx, kC * D) Qb[idx] = B1[idx];
    } else {
        GBWD_FOR(idx, kC * D) Qb[idx] -= lam[idx / D] * B3[idx];
    }
    __syncthreads();
    // the Gated DeltaNet chunk: R = V - diag(E) Kbar H_r (B1), U = Tt diag(beta) R (B2)
    load_tile<D, Tin>(B1, a.v, a, b, h, r);
    __syncthreads();
    GBWD_FOR(idx, kC * D) {
        const int i = idx / D, j = idx % D;
        float acc = 0.f;
        for (int l = 0; l < D; ++l) acc += Kb[i * D + l] * H[l * D + j];
        B1[idx] -= E[i] * acc;
    }
    __syncthreads();
    GBWD_FOR(idx, kC * D) {
        const int i = idx / D, j = idx % D;
        float acc = 0.f;
        for (int l = 0; l <= i; ++l) acc += Tt[i * kC + l] * be[l] * B1[l * D + j];
        B2[idx] = acc;
    }
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
            for (int l = 0; l <= i; ++l) acc += sA[i * kC + l] * B2[l * D + j];
            o[tok_row(a, b, r * kC + i, h) * D + j] = from_f<Tin>(a.scale * acc);
        }
    }
}

template <int D> constexpr size_t gdec_stats_smem() { return sizeof(float) * (kC * D + 4 * kC); }
template <int D> constexpr size_t gdec_out_smem() { return sizeof(float) * (5 * kC * D + 2 * kC * kC + 14 * kC); }

}  // namespace gbwd
}  // namespace ccq
