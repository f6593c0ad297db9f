/*
 * ccq_oracle.c -- fp64 CPU oracle for Curvature-Conditioned Query (CCQ).
 *
 * TEST INFRASTRUCTURE ONLY. This file is the plain, slow, obviously correct
 * statement of what the CCQ hot path computes. Only the test-suite, the smoke
 * check and the CPU-baseline leg of the benchmark may load it. The CUDA
 * library never links, includes or calls anything in this directory, and
 * this file includes nothing from the CUDA library.
 *
 * What it computes (arxiv 2606.01294):
 *   - running key statistics C_sum = sum_j kbar_j kbar_j^T and m_sum = sum_j kbar_j
 *     with the length normalisation 1/t (Sec. 3.2 "Idea 1"; App. A.2, Eq. hess);
 *   - Sigma_t = C_sum/t - (m_sum/t)(m_sum/t)^T, the centred sample covariance
 *     (App. A.2), or C_sum/t for the uncentred variant (App. D ablation);
 *   - the cleaned query q_clean = qbar - lambda_t Sigma_t qbar (Eq. clean,
 *     Algorithm 2), applied to the l2-normalised query (Algorithms 1 and 2);
 *   - the backbone write S_t = Update(S_{t-1}; kbar_t, v_t, ...) and the read
 *     o_t = scale * S_t q_clean (Eq. read).  The paper treats the backbone as a
 *     black box (Sec. 2.2); the two write rules are GLA's per-key-dimension
 *     forget gate and Gated DeltaNet's gated delta rule, as those methods
 *     define them and as Sec. 2.2 summarises them.
 *
 * State orientation: the paper's S is d_v x d_k.  Here every state is stored
 * as its transpose Hs[dk][dv] (row = key dimension), i.e. Hs = S^T.
 *
 * Readings of the paper that this file fixes (where the paper is silent):
 *   - zero-norm rows: l2-normalising an all-zero row yields the zero row
 *     (the paper gives no epsilon);
 *   - the position counter t is inclusive of the current token (sums over
 *     j <= t, Sec. 3.2) and continues from the caller's t0;
 *   - the read uses the state after token t has been written (Eq. read);
 *   - scale multiplies the read only.
 *
 * Every routine is fp64.  Work over (batch, head) pairs is spread over
 * POSIX threads; each pair is computed by exactly one thread in a fixed
 * order, so results do not depend on the thread count.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define CCQ_ORACLE_GLA 0
#define CCQ_ORACLE_GDN 1

typedef struct {
    int backbone, B, T, H, Dk, Dv, l2norm, centered, chunk;
    double scale;
    const double *q, *k, *v, *gate, *beta, *lam;
    const double *S0, *C0, *m0;
    const int64_t *t0;
    double *o, *ST, *CT, *mT, *qc_out;
    int64_t *tT;
    /* work queue over (b, h) pairs */
    int next;
    pthread_mutex_t mu;
} job_t;

/* l2-normalise x[0..n) into y; the zero row maps to the zero row. */
static void l2_normalise(const double *x, double *y, int n, int enabled) {
    if (!enabled) {
        memcpy(y, x, sizeof(double) * (size_t)n);
        return;
    }
    double s = 0.0;
    for (int i = 0; i < n; ++i) s += x[i] * x[i];
    double r = s > 0.0 ? 1.0 / sqrt(s) : 0.0;
    for (int i = 0; i < n; ++i) y[i] = x[i] * r;
}

static size_t row(const job_t *J, int b, int t, int h) {
    return ((size_t)b * J->T + t) * J->H + h;
}

/* Load the initial states of pair (b, h): zero when the pointer is NULL. */
static void load_states(const job_t *J, int b, int h, double *Hs, double *Cs,
                        double *ms, int64_t *t) {
    const int Dk = J->Dk, Dv = J->Dv;
    const size_t bh = (size_t)b * J->H + h;
    if (J->S0) memcpy(Hs, J->S0 + bh * Dk * Dv, sizeof(double) * Dk * Dv);
    else memset(Hs, 0, sizeof(double) * Dk * Dv);
    if (J->C0) memcpy(Cs, J->C0 + bh * Dk * Dk, sizeof(double) * Dk * Dk);
    else memset(Cs, 0, sizeof(double) * Dk * Dk);
    if (J->m0) memcpy(ms, J->m0 + bh * Dk, sizeof(double) * Dk);
    else memset(ms, 0, sizeof(double) * Dk);
    *t = J->t0 ? J->t0[b] : 0;
}

static void store_states(const job_t *J, int b, int h, const double *Hs,
                         const double *Cs, const double *ms, int64_t t) {
    const int Dk = J->Dk, Dv = J->Dv;
    const size_t bh = (size_t)b * J->H + h;
    if (J->ST) memcpy(J->ST + bh * Dk * Dv, Hs, sizeof(double) * Dk * Dv);
    if (J->CT) memcpy(J->CT + bh * Dk * Dk, Cs, sizeof(double) * Dk * Dk);
    if (J->mT) memcpy(J->mT + bh * Dk, ms, sizeof(double) * Dk);
    if (J->tT && h == 0) J->tT[b] = t;
}

/*
 * Sigma_t qbar from the running sums (App. A.2): C_sum qbar / t minus the
 * mean term m (m^T qbar) / t^2; the mean term is dropped when uncentred.
 */
static void sigma_times(const double *Cs, const double *ms, const double *qb,
                        int Dk, double t, int centered, double *out) {
    double mq = 0.0;
    for (int j = 0; j < Dk; ++j) mq += ms[j] * qb[j];
    for (int i = 0; i < Dk; ++i) {
        double acc = 0.0;
        for (int j = 0; j < Dk; ++j) acc += Cs[(size_t)i * Dk + j] * qb[j];
        out[i] = acc / t;
        if (centered) out[i] -= ms[i] * mq / (t * t);
    }
}

/*
 * One (b, h) pair, token by token: Algorithm 2 with the statistics kept as
 * unnormalised sums and divided by t on use (the same Sigma_t, App. A.2).
 */
static void recurrent_pair(const job_t *J, int b, int h) {
    const int Dk = J->Dk, Dv = J->Dv;
    double *Hs = malloc(sizeof(double) * Dk * Dv);
    double *Cs = malloc(sizeof(double) * Dk * Dk);
    double *ms = malloc(sizeof(double) * Dk);
    double *qb = malloc(sizeof(double) * Dk), *kb = malloc(sizeof(double) * Dk);
    double *sq = malloc(sizeof(double) * Dk), *qc = malloc(sizeof(double) * Dk);
    double *kS = malloc(sizeof(double) * Dv);
    int64_t t;
    load_states(J, b, h, Hs, Cs, ms, &t);

    for (int tl = 0; tl < J->T; ++tl) {
        const size_t r = row(J, b, tl, h);
        const double *qr = J->q + r * Dk, *kr = J->k + r * Dk, *vr = J->v + r * Dv;
        /* Algorithm 2: normalise query and key */
        l2_normalise(qr, qb, Dk, J->l2norm);
        l2_normalise(kr, kb, Dk, J->l2norm);
        /* key statistics include the current token (sums over j <= t) */
        t += 1;
        for (int i = 0; i < Dk; ++i) {
            for (int j = 0; j < Dk; ++j) Cs[(size_t)i * Dk + j] += kb[i] * kb[j];
            ms[i] += kb[i];
        }
        /* Eq. clean: q_clean = qbar - lambda Sigma_t qbar */
        const double lam = J->lam[r];
        sigma_times(Cs, ms, qb, Dk, (double)t, J->centered, sq);
        for (int i = 0; i < Dk; ++i) qc[i] = qb[i] - lam * sq[i];
        if (J->qc_out) memcpy(J->qc_out + r * Dk, qc, sizeof(double) * Dk);

        /* backbone write with the normalised key */
        if (J->backbone == CCQ_ORACLE_GLA) {
            /* GLA: S_t = S_{t-1} Diag(alpha_t) + v_t kbar_t^T, alpha = exp(gk) */
            const double *gr = J->gate + r * Dk;
            for (int i = 0; i < Dk; ++i) {
                const double a = exp(gr[i]);
                for (int j = 0; j < Dv; ++j)
                    Hs[(size_t)i * Dv + j] = a * Hs[(size_t)i * Dv + j] + kb[i] * vr[j];
            }
        } else {
            /* Gated DeltaNet: S_t = alpha_t S_{t-1} (I - beta_t k k^T) + beta_t v k^T */
            const double a = exp(J->gate[r]), be = J->beta[r];
            for (int j = 0; j < Dv; ++j) {
                double acc = 0.0;
                for (int i = 0; i < Dk; ++i) acc += kb[i] * Hs[(size_t)i * Dv + j];
                kS[j] = acc;
            }
            for (int i = 0; i < Dk; ++i)
                for (int j = 0; j < Dv; ++j)
                    Hs[(size_t)i * Dv + j] =
                        a * (Hs[(size_t)i * Dv + j] - be * kb[i] * kS[j]) + be * kb[i] * vr[j];
        }
        /* Eq. read: o_t = S_t q_clean (times the read scale) */
        double *orow = J->o + r * Dv;
        for (int j = 0; j < Dv; ++j) {
            double acc = 0.0;
            for (int i = 0; i < Dk; ++i) acc += Hs[(size_t)i * Dv + j] * qc[i];
            orow[j] = J->scale * acc;
        }
    }
    store_states(J, b, h, Hs, Cs, ms, t);
    free(Hs); free(Cs); free(ms); free(qb); free(kb); free(sq); free(qc); free(kS);
}

/*
 * One (b, h) pair in the chunkwise form of Algorithm 1 (App. B), with the
 * backbone's own chunk update.  This is a second statement of the same
 * computation used to check that the chunkwise re-association is exact; it
 * is not what the tests compare GPU results against.
 */
static void chunkwise_pair(const job_t *J, int b, int h) {
    const int Dk = J->Dk, Dv = J->Dv, C = J->chunk;
    double *Hs = malloc(sizeof(double) * Dk * Dv);
    double *SK = malloc(sizeof(double) * Dk * Dk);
    double *M = malloc(sizeof(double) * Dk);
    double *Qb = malloc(sizeof(double) * C * Dk), *Kb = malloc(sizeof(double) * C * Dk);
    double *P = malloc(sizeof(double) * C * Dk), *CumK = malloc(sizeof(double) * C * Dk);
    double *Qc = malloc(sizeof(double) * C * Dk);
    double *G = malloc(sizeof(double) * C * Dk); /* GLA: in-chunk cumulative log gate */
    double *gc = malloc(sizeof(double) * C);     /* GDN: in-chunk cumulative log decay */
    double *U = malloc(sizeof(double) * C * Dv); /* GDN: pseudo-values u_j */
    double *Hn = malloc(sizeof(double) * Dk * Dv);
    int64_t t;
    load_states(J, b, h, Hs, SK, M, &t);

    for (int c0 = 0; c0 < J->T; c0 += C) {
        const int n = (J->T - c0 < C) ? J->T - c0 : C;
        /* Algorithm 1: normalised queries and keys of the chunk */
        for (int i = 0; i < n; ++i) {
            const size_t r = row(J, b, c0 + i, h);
            l2_normalise(J->q + r * Dk, Qb + (size_t)i * Dk, Dk, J->l2norm);
            l2_normalise(J->k + r * Dk, Kb + (size_t)i * Dk, Dk, J->l2norm);
        }
        for (int i = 0; i < n; ++i) {
            const double *qi = Qb + (size_t)i * Dk;
            /* P_prev = S^K_r qbar_i (S^K symmetric) */
            for (int a = 0; a < Dk; ++a) {
                double acc = 0.0;
                for (int e = 0; e < Dk; ++e) acc += SK[(size_t)a * Dk + e] * qi[e];
                P[(size_t)i * Dk + a] = acc;
            }
            /* P_intra = sum_{j <= i} (qbar_i . kbar_j) kbar_j (mask includes the diagonal) */
            for (int j = 0; j <= i; ++j) {
                const double *kj = Kb + (size_t)j * Dk;
                double s = 0.0;
                for (int e = 0; e < Dk; ++e) s += qi[e] * kj[e];
                for (int a = 0; a < Dk; ++a) P[(size_t)i * Dk + a] += s * kj[a];
            }
            /* CumK = M_r + cumsum(kbar) */
            for (int a = 0; a < Dk; ++a)
                CumK[(size_t)i * Dk + a] =
                    (i == 0 ? M[a] : CumK[(size_t)(i - 1) * Dk + a]) + Kb[(size_t)i * Dk + a];
            /* D = 1/(t+i); MeanCorr_i = D^2 CumK_i (CumK_i . qbar_i), read row by row */
            const double tpos = (double)(t + i + 1);
            double cq = 0.0;
            for (int a = 0; a < Dk; ++a) cq += CumK[(size_t)i * Dk + a] * qi[a];
            const double lam = J->lam[row(J, b, c0 + i, h)];
            for (int a = 0; a < Dk; ++a) {
                double corr = P[(size_t)i * Dk + a] / tpos;
                if (J->centered) corr -= CumK[(size_t)i * Dk + a] * cq / (tpos * tpos);
                Qc[(size_t)i * Dk + a] = qi[a] - lam * corr;
            }
            if (J->qc_out)
                memcpy(J->qc_out + row(J, b, c0 + i, h) * Dk, Qc + (size_t)i * Dk,
                       sizeof(double) * Dk);
        }

        if (J->backbone == CCQ_ORACLE_GLA) {
            /* GLA chunk update: G_i = sum_{s <= i} gk_s within the chunk */
            for (int i = 0; i < n; ++i) {
                const double *gr = J->gate + row(J, b, c0 + i, h) * Dk;
                for (int a = 0; a < Dk; ++a)
                    G[(size_t)i * Dk + a] = (i ? G[(size_t)(i - 1) * Dk + a] : 0.0) + gr[a];
            }
            for (int i = 0; i < n; ++i) {
                double *orow = J->o + row(J, b, c0 + i, h) * Dv;
                const double *qi = Qc + (size_t)i * Dk, *Gi = G + (size_t)i * Dk;
                for (int e = 0; e < Dv; ++e) {
                    /* inter-chunk: (q_clean_i * exp(G_i)) S_r */
                    double acc = 0.0;
                    for (int a = 0; a < Dk; ++a)
                        acc += qi[a] * exp(Gi[a]) * Hs[(size_t)a * Dv + e];
                    orow[e] = acc;
                }
                /* intra-chunk: sum_{j <= i} (q_clean_i * exp(G_i - G_j) . kbar_j) v_j */
                for (int j = 0; j <= i; ++j) {
                    const double *Gj = G + (size_t)j * Dk, *kj = Kb + (size_t)j * Dk;
                    double s = 0.0;
                    for (int a = 0; a < Dk; ++a) s += qi[a] * exp(Gi[a] - Gj[a]) * kj[a];
                    const double *vj = J->v + row(J, b, c0 + j, h) * Dv;
                    for (int e = 0; e < Dv; ++e) orow[e] += s * vj[e];
                }
                for (int e = 0; e < Dv; ++e) orow[e] *= J->scale;
            }
            /* S_{r+1} = Diag(exp(G_n)) S_r + sum_j (kbar_j * exp(G_n - G_j)) v_j^T */
            const double *Gn = G + (size_t)(n - 1) * Dk;
            for (int a = 0; a < Dk; ++a)
                for (int e = 0; e < Dv; ++e) {
                    double acc = exp(Gn[a]) * Hs[(size_t)a * Dv + e];
                    for (int j = 0; j < n; ++j)
                        acc += Kb[(size_t)j * Dk + a] * exp(Gn[a] - G[(size_t)j * Dk + a]) *
                               J->v[row(J, b, c0 + j, h) * Dv + e];
                    Hn[(size_t)a * Dv + e] = acc;
                }
            memcpy(Hs, Hn, sizeof(double) * Dk * Dv);
        } else {
            /* Gated DeltaNet chunk update.  With H = S^T and gamma_i the in-chunk
             * decay product, the per-token write is H_i = alpha_i H_{i-1} + kbar_i u_i^T
             * with u_i = beta_i (v_i - alpha_i H_{i-1}^T kbar_i).  Unrolling gives the
             * unit lower-triangular system
             *   u_i + beta_i sum_{j<i} (gamma_i/gamma_j)(kbar_i . kbar_j) u_j
             *       = beta_i v_i - beta_i gamma_i H_0^T kbar_i,
             * solved here by forward substitution (the WY/UT form inverts the same
             * matrix). */
            for (int i = 0; i < n; ++i)
                gc[i] = (i ? gc[i - 1] : 0.0) + J->gate[row(J, b, c0 + i, h)];
            for (int i = 0; i < n; ++i) {
                const double be = J->beta[row(J, b, c0 + i, h)];
                const double *ki = Kb + (size_t)i * Dk;
                const double *vi = J->v + row(J, b, c0 + i, h) * Dv;
                double *ui = U + (size_t)i * Dv;
                for (int e = 0; e < Dv; ++e) {
                    double hk = 0.0;
                    for (int a = 0; a < Dk; ++a) hk += Hs[(size_t)a * Dv + e] * ki[a];
                    ui[e] = be * vi[e] - be * exp(gc[i]) * hk;
                }
                for (int j = 0; j < i; ++j) {
                    const double *kj = Kb + (size_t)j * Dk;
                    double s = 0.0;
                    for (int a = 0; a < Dk; ++a) s += ki[a] * kj[a];
                    const double Aij = be * exp(gc[i] - gc[j]) * s;
                    for (int e = 0; e < Dv; ++e) ui[e] -= Aij * U[(size_t)j * Dv + e];
                }
            }
            for (int i = 0; i < n; ++i) {
                double *orow = J->o + row(J, b, c0 + i, h) * Dv;
                const double *qi = Qc + (size_t)i * Dk;
                for (int e = 0; e < Dv; ++e) {
                    double acc = 0.0;
                    for (int a = 0; a < Dk; ++a) acc += qi[a] * Hs[(size_t)a * Dv + e];
                    orow[e] = exp(gc[i]) * acc;
                }
                for (int j = 0; j <= i; ++j) {
                    const double *kj = Kb + (size_t)j * Dk;
                    double s = 0.0;
                    for (int a = 0; a < Dk; ++a) s += qi[a] * kj[a];
                    s *= exp(gc[i] - gc[j]);
                    for (int e = 0; e < Dv; ++e) orow[e] += s * U[(size_t)j * Dv + e];
                }
                for (int e = 0; e < Dv; ++e) orow[e] *= J->scale;
            }
            for (int a = 0; a < Dk; ++a)
                for (int e = 0; e < Dv; ++e) {
                    double acc = exp(gc[n - 1]) * Hs[(size_t)a * Dv + e];
                    for (int j = 0; j < n; ++j)
                        acc += exp(gc[n - 1] - gc[j]) * Kb[(size_t)j * Dk + a] * U[(size_t)j * Dv + e];
                    Hn[(size_t)a * Dv + e] = acc;
                }
            memcpy(Hs, Hn, sizeof(double) * Dk * Dv);
        }
        /* S^K_{r+1} = S^K_r + Kbar^T Kbar ; M_{r+1} = M_r + sum_j kbar_j ; t += n */
        for (int j = 0; j < n; ++j) {
            const double *kj = Kb + (size_t)j * Dk;
            for (int a = 0; a < Dk; ++a) {
                for (int e = 0; e < Dk; ++e) SK[(size_t)a * Dk + e] += kj[a] * kj[e];
                M[a] += kj[a];
            }
        }
        t += n;
    }
    store_states(J, b, h, Hs, SK, M, t);
    free(Hs); free(SK); free(M); free(Qb); free(Kb); free(P); free(CumK); free(Qc);
    free(G); free(gc); free(U); free(Hn);
}

static void *worker(void *arg) {
    job_t *J = (job_t *)arg;
    for (;;) {
        pthread_mutex_lock(&J->mu);
        const int w = J->next++;
        pthread_mutex_unlock(&J->mu);
        if (w >= J->B * J->H) break;
        const int b = w / J->H, h = w % J->H;
        if (J->chunk > 0) chunkwise_pair(J, b, h);
        else recurrent_pair(J, b, h);
    }
    return NULL;
}

/*
 * Forward over a [B, T, H, D] sequence batch (D contiguous).
 *   backbone   0 = GLA (gate: log alpha [B,T,H,Dk]), 1 = Gated DeltaNet
 *              (gate: log alpha [B,T,H], beta [B,T,H]).
 *   lam        lambda_t [B,T,H].
 *   S0/C0/m0   initial S^T [B,H,Dk,Dv], C_sum [B,H,Dk,Dk], m_sum [B,H,Dk]; NULL = 0.
 *   t0         initial position per batch row [B]; NULL = 0.
 *   o          [B,T,H,Dv].  ST/CT/mT/tT final states (each may be NULL).
 *   qc_out     optional [B,T,H,Dk] cleaned queries (NULL = not written).
 *   chunk      0 = token-by-token recurrence; >0 = chunkwise form, chunk size.
 *   nthreads   worker threads (>= 1).
 * Returns 0, or -1 on a bad argument.
 */
int ccq_oracle_forward(int backbone, int B, int T, int H, int Dk, int Dv,
                       const double *q, const double *k, const double *v,
                       const double *gate, const double *beta, const double *lam,
                       const double *S0, const double *C0, const double *m0,
                       const int64_t *t0, double *o, double *ST, double *CT,
                       double *mT, int64_t *tT, double *qc_out, int l2norm,
                       int centered, double scale, int chunk, int nthreads) {
    if (B < 0 || T < 0 || H < 0 || Dk <= 0 || Dv <= 0 || chunk < 0 || nthreads < 1) return -1;
    if (!q || !k || !v || !gate || !lam || !o) return -1;
    if (backbone == CCQ_ORACLE_GDN && !beta) return -1;
    if (backbone != CCQ_ORACLE_GLA && backbone != CCQ_ORACLE_GDN) return -1;
    job_t J;
    memset(&J, 0, sizeof J);
    J.backbone = backbone; J.B = B; J.T = T; J.H = H; J.Dk = Dk; J.Dv = Dv;
    J.l2norm = l2norm; J.centered = centered; J.chunk = chunk; J.scale = scale;
    J.q = q; J.k = k; J.v = v; J.gate = gate; J.beta = beta; J.lam = lam;
    J.S0 = S0; J.C0 = C0; J.m0 = m0; J.t0 = t0;
    J.o = o; J.ST = ST; J.CT = CT; J.mT = mT; J.tT = tT; J.qc_out = qc_out;
    pthread_mutex_init(&J.mu, NULL);
    if (nthreads > B * H) nthreads = B * H > 0 ? B * H : 1;
    pthread_t *th = malloc(sizeof(pthread_t) * (size_t)nthreads);
    for (int i = 0; i < nthreads; ++i) pthread_create(&th[i], NULL, worker, &J);
    for (int i = 0; i < nthreads; ++i) pthread_join(th[i], NULL);
    free(th);
    pthread_mutex_destroy(&J.mu);
    /* T == 0: the per-pair loops still copy the initial states through */
    return 0;
}

/* ====================================================================== decay-aligned covariance
 *
 * The variant the paper names as future work for decayed backbones (Sec. 6 and the appendix
 * paragraph on decayed backbones): the covariance is computed from gamma-weighted running
 * statistics, gamma_{j,t} the factor by which the backbone has decayed key j's write by
 * token t.  The paper fixes neither gamma nor the normaliser; this oracle takes the reading
 *   gamma_{j,t} = prod_{s=j+1..t} alpha_s      (Gated DeltaNet's scalar decay),
 *   C_t = alpha_t C_{t-1} + kbar_t kbar_t^T,  m_t = alpha_t m_{t-1} + kbar_t,
 *   n_t = alpha_t n_{t-1} + 1                   (the decayed count, in place of t),
 *   Sigma_t = C_t / n_t - (m_t / n_t)(m_t / n_t)^T  (centred; C_t / n_t uncentred),
 * which is the undecayed definition when every alpha_t = 1.  Only a backbone with one decay
 * per key (Gated DeltaNet) has such a factor; GLA's per-dimension gates have none.
 */
typedef struct {
    int B, T, H, Dk, Dv, l2norm, centered;
    double scale;
    const double *q, *k, *v, *g, *beta, *lam, *S0, *C0, *m0, *n0;
    double *o, *ST, *CT, *mT, *nT, *qc_out;
    int next;
    pthread_mutex_t mu;
} djob_t;

static void decayed_pair(const djob_t *J, int b, int h) {
    const int Dk = J->Dk, Dv = J->Dv;
    const size_t bh = (size_t)b * J->H + h;
    double *Hs = calloc((size_t)Dk * Dv, sizeof(double));
    double *Cg = calloc((size_t)Dk * Dk, sizeof(double));
    double *mg = calloc((size_t)Dk, sizeof(double));
    double *qb = malloc(sizeof(double) * Dk), *kb = malloc(sizeof(double) * Dk);
    double *sg = malloc(sizeof(double) * Dk), *qcl = malloc(sizeof(double) * Dk);
    double *kS = malloc(sizeof(double) * Dv);
    if (J->S0) memcpy(Hs, J->S0 + bh * Dk * Dv, sizeof(double) * Dk * Dv);
    if (J->C0) memcpy(Cg, J->C0 + bh * Dk * Dk, sizeof(double) * Dk * Dk);
    if (J->m0) memcpy(mg, J->m0 + bh * Dk, sizeof(double) * Dk);
    double n = J->n0 ? J->n0[bh] : 0.0;
    for (int tl = 0; tl < J->T; ++tl) {
        const size_t r = ((size_t)b * J->T + tl) * J->H + h;
        const double *vr = J->v + r * Dv;
        l2_normalise(J->q + r * Dk, qb, Dk, J->l2norm);
        l2_normalise(J->k + r * Dk, kb, Dk, J->l2norm);
        const double a = exp(J->g[r]), be = J->beta[r], lam = J->lam[r];
        /* gamma-weighted statistics including token t */
        for (int i = 0; i < Dk; ++i) {
            for (int j = 0; j < Dk; ++j) Cg[(size_t)i * Dk + j] = a * Cg[(size_t)i * Dk + j] + kb[i] * kb[j];
            mg[i] = a * mg[i] + kb[i];
        }
        n = a * n + 1.0;
        /* Sigma^gamma_t qbar, then the cleaned query (Eq. clean with Sigma^gamma) */
        double mq = 0.0;
        for (int j = 0; j < Dk; ++j) mq += mg[j] * qb[j];
        for (int i = 0; i < Dk; ++i) {
            double acc = 0.0;
            for (int j = 0; j < Dk; ++j) acc += Cg[(size_t)i * Dk + j] * qb[j];
            sg[i] = acc / n - (J->centered ? mg[i] * mq / (n * n) : 0.0);
        }
        for (int i = 0; i < Dk; ++i) qcl[i] = qb[i] - lam * sg[i];
        if (J->qc_out) memcpy(J->qc_out + r * Dk, qcl, sizeof(double) * Dk);
        /* gated delta rule, written as S_t = a S_{t-1} + kbar u^T with u = beta (v - a S_{t-1}^T kbar) */
        for (int j = 0; j < Dv; ++j) {
            double acc = 0.0;
            for (int i = 0; i < Dk; ++i) acc += kb[i] * Hs[(size_t)i * Dv + j];
            kS[j] = be * (vr[j] - a * acc);
        }
        for (int i = 0; i < Dk; ++i)
            for (int j = 0; j < Dv; ++j) Hs[(size_t)i * Dv + j] = a * Hs[(size_t)i * Dv + j] + kb[i] * kS[j];
        double *orow = J->o + r * Dv;
        for (int j = 0; j < Dv; ++j) {
            double acc = 0.0;
            for (int i = 0; i < Dk; ++i) acc += Hs[(size_t)i * Dv + j] * qcl[i];
            orow[j] = J->scale * acc;
        }
    }
    if (J->ST) memcpy(J->ST + bh * Dk * Dv, Hs, sizeof(double) * Dk * Dv);
    if (J->CT) memcpy(J->CT + bh * Dk * Dk, Cg, sizeof(double) * Dk * Dk);
    if (J->mT) memcpy(J->mT + bh * Dk, mg, sizeof(double) * Dk);
    if (J->nT) J->nT[bh] = n;
    free(Hs); free(Cg); free(mg); free(qb); free(kb); free(sg); free(qcl); free(kS);
}

static void *dworker(void *arg) {
    djob_t *J = (djob_t *)arg;
    for (;;) {
        pthread_mutex_lock(&J->mu);
        const int w = J->next++;
        pthread_mutex_unlock(&J->mu);
        if (w >= J->B * J->H) break;
        decayed_pair(J, w / J->H, w % J->H);
    }
    return NULL;
}

/*
 * Gated DeltaNet forward with the decay-aligned covariance (reading above).  Arguments as
 * ccq_oracle_forward for the Gated DeltaNet backbone, except that the position count is
 * replaced by the decayed count: n0 [B,H] (NULL = 0) in, nT [B,H] out (may be NULL).
 * Returns 0, or -1 on a bad argument.
 */
int ccq_oracle_gdn_forward_decayed(int B, int T, int H, int Dk, int Dv, const double *q, const double *k,
                                   const double *v, const double *g, const double *beta,
                                   const double *lam, const double *S0, const double *C0,
                                   const double *m0, const double *n0, double *o, double *ST,
                                   double *CT, double *mT, double *nT, double *qc_out, int l2norm,
                                   int centered, double scale, int nthreads) {
    if (B < 0 || T < 0 || H < 0 || Dk <= 0 || Dv <= 0 || nthreads < 1) return -1;
    if (!q || !k || !v || !g || !beta || !lam || !o) return -1;
    djob_t J;
    memset(&J, 0, sizeof J);
    J.B = B; J.T = T; J.H = H; J.Dk = Dk; J.Dv = Dv; J.l2norm = l2norm; J.centered = centered;
    J.scale = scale;
    J.q = q; J.k = k; J.v = v; J.g = g; J.beta = beta; J.lam = lam;
    J.S0 = S0; J.C0 = C0; J.m0 = m0; J.n0 = n0;
    J.o = o; J.ST = ST; J.CT = CT; J.mT = mT; J.nT = nT; J.qc_out = qc_out;
    pthread_mutex_init(&J.mu, NULL);
    if (nthreads > B * H) nthreads = B * H > 0 ? B * H : 1;
    pthread_t *th = malloc(sizeof(pthread_t) * (size_t)nthreads);
    for (int i = 0; i < nthreads; ++i) pthread_create(&th[i], NULL, dworker, &J);
    for (int i = 0; i < nthreads; ++i) pthread_join(th[i], NULL);
    free(th);
    pthread_mutex_destroy(&J.mu);
    return 0;
}

/* ====================================================================== reverse mode
 *
 * Gradients of the CCQ-GLA forward (recurrent form above) with respect to every
 * input, by hand-written reverse mode.  Per (b, h): the forward states are
 * checkpointed at every 64-token boundary; the tokens of each block are
 * recomputed from its checkpoint (keeping every per-token state of the block),
 * then walked backwards.  For token t (all sums and products of Algorithm 2):
 *   o = scale S_t q_clean,  q_clean = qbar - lambda z,  z = Sigma_t qbar
 *   Sigma_t qbar = C_t qbar / t - m_t (m_t . qbar) / t^2,  C_t = C_{t-1} + kbar kbar^T,
 *   m_t = m_{t-1} + kbar,  S_t = Diag(e^{gk_t}) S_{t-1} + kbar v^T  (S stored [Dk][Dv]),
 * the adjoints are
 *   dq_clean = scale S_t do,  dS_t += scale q_clean do^T,  dz = -lambda dq_clean,
 *   dlambda = -z . dq_clean,  dqbar = dq_clean + Sigma_t dz,
 *   dC += dz qbar^T / t,  dm -= ((m . qbar) dz + (dz . m) qbar) / t^2,
 *   dkbar = dS v + (dC + dC^T) kbar + dm,  dv = dS^T kbar,
 *   dgk = e^{gk} * rowsum(dS * S_{t-1}),  dS <- Diag(e^{gk}) dS,
 *   dx = (dxbar - xbar (xbar . dxbar)) / |x| for x = q, k (l2 normalisation).
 */

typedef struct {
    int B, T, H, Dk, Dv, l2norm, centered;
    double scale;
    const double *q, *k, *v, *gk, *lam, *S0, *C0, *m0, *dout, *dST, *dCT, *dmT;
    const int64_t *t0;
    double *dq, *dk, *dv, *dgk, *dlam, *dS0, *dC0, *dm0;
    /* Gated DeltaNet only: gk is then the scalar log decay g [B,T,H], beta [B,T,H],
       and dgk receives dg [B,T,H] */
    const double *beta;
    double *dbeta;
    int next;
    pthread_mutex_t mu;
} bjob_t;

static size_t brow(const bjob_t *J, int b, int t, int h) { return ((size_t)b * J->T + t) * J->H + h; }

static void normalise_with_norm(const double *x, double *y, double *nrm, int n, int enabled) {
    if (!enabled) {
        memcpy(y, x, sizeof(double) * (size_t)n);
        *nrm = 1.0;
        return;
    }
    double s = 0.0;
    for (int i = 0; i < n; ++i) s += x[i] * x[i];
    *nrm = sqrt(s);
    const double r = s > 0.0 ? 1.0 / *nrm : 0.0;
    for (int i = 0; i < n; ++i) y[i] = x[i] * r;
}

/* dx = (dxbar - xbar (xbar . dxbar)) / |x|; the zero row maps to zero */
static void normalise_backward(const double *xbar, double nrm, const double *dxbar, double *dx, int n,
                               int enabled) {
    if (!enabled) {
        memcpy(dx, dxbar, sizeof(double) * (size_t)n);
        return;
    }
    if (nrm == 0.0) {
        for (int i = 0; i < n; ++i) dx[i] = 0.0;
        return;
    }
    double d = 0.0;
    for (int i = 0; i < n; ++i) d += xbar[i] * dxbar[i];
    for (int i = 0; i < n; ++i) dx[i] = (dxbar[i] - xbar[i] * d) / nrm;
}

static void backward_pair(const bjob_t *J, int b, int h) {
    const int Dk = J->Dk, Dv = J->Dv, T = J->T, BL = 64;
    const int NB = (T + BL - 1) / BL;
    const size_t bh = (size_t)b * J->H + h;
    const size_t SS = (size_t)Dk * Dv, CC = (size_t)Dk * Dk;
    /* checkpoints at block starts */
    double *ckS = malloc(sizeof(double) * SS * (NB + 1));
    double *ckC = malloc(sizeof(double) * CC * (NB + 1));
    double *ckm = malloc(sizeof(double) * Dk * (NB + 1));
    /* per-token states of one block: S after each token (BL + 1 incl. the block start), C, m */
    double *bS = malloc(sizeof(double) * SS * (BL + 1));
    double *bC = malloc(sizeof(double) * CC * (BL + 1));
    double *bm = malloc(sizeof(double) * Dk * (BL + 1));
    double *qb = malloc(sizeof(double) * Dk), *kb = malloc(sizeof(double) * Dk);
    double *z = malloc(sizeof(double) * Dk), *qc = malloc(sizeof(double) * Dk);
    double *dqc = malloc(sizeof(double) * Dk), *dz = malloc(sizeof(double) * Dk);
    double *dqb = malloc(sizeof(double) * Dk), *dkb = malloc(sizeof(double) * Dk);
    double *dS = malloc(sizeof(double) * SS), *dC = malloc(sizeof(double) * CC);
    double *dm = malloc(sizeof(double) * Dk);
    const int64_t tstart = J->t0 ? J->t0[b] : 0;

    if (J->S0) memcpy(ckS, J->S0 + bh * SS, sizeof(double) * SS); else memset(ckS, 0, sizeof(double) * SS);
    if (J->C0) memcpy(ckC, J->C0 + bh * CC, sizeof(double) * CC); else memset(ckC, 0, sizeof(double) * CC);
    if (J->m0) memcpy(ckm, J->m0 + bh * Dk, sizeof(double) * Dk); else memset(ckm, 0, sizeof(double) * Dk);

    /* forward over the blocks, keeping only the block-start checkpoints */
    for (int blk = 0; blk < NB; ++blk) {
        double *S = ckS + SS * (blk + 1), *C = ckC + CC * (blk + 1), *m = ckm + (size_t)Dk * (blk + 1);
        memcpy(S, ckS + SS * blk, sizeof(double) * SS);
        memcpy(C, ckC + CC * blk, sizeof(double) * CC);
        memcpy(m, ckm + (size_t)Dk * blk, sizeof(double) * Dk);
        for (int tl = blk * BL; tl < T && tl < (blk + 1) * BL; ++tl) {
            const size_t r = brow(J, b, tl, h);
            double nk;
            normalise_with_norm(J->k + r * Dk, kb, &nk, Dk, J->l2norm);
            for (int i = 0; i < Dk; ++i) {
                for (int j = 0; j < Dk; ++j) C[(size_t)i * Dk + j] += kb[i] * kb[j];
                m[i] += kb[i];
            }
            for (int i = 0; i < Dk; ++i) {
                const double a = exp(J->gk[r * Dk + i]);
                for (int e = 0; e < Dv; ++e)
                    S[(size_t)i * Dv + e] = a * S[(size_t)i * Dv + e] + kb[i] * J->v[r * Dv + e];
            }
        }
    }

    /* adjoints of the final states */
    if (J->dST) memcpy(dS, J->dST + bh * SS, sizeof(double) * SS); else memset(dS, 0, sizeof(double) * SS);
    if (J->dCT) memcpy(dC, J->dCT + bh * CC, sizeof(double) * CC); else memset(dC, 0, sizeof(double) * CC);
    if (J->dmT) memcpy(dm, J->dmT + bh * Dk, sizeof(double) * Dk); else memset(dm, 0, sizeof(double) * Dk);

    for (int blk = NB - 1; blk >= 0; --blk) {
        const int t_lo = blk * BL, t_hi = (T < (blk + 1) * BL) ? T : (blk + 1) * BL;
        /* recompute the block's per-token states: index 0 = block start, i + 1 = after token t_lo + i */
        memcpy(bS, ckS + SS * blk, sizeof(double) * SS);
        memcpy(bC, ckC + CC * blk, sizeof(double) * CC);
        memcpy(bm, ckm + (size_t)Dk * blk, sizeof(double) * Dk);
        for (int tl = t_lo; tl < t_hi; ++tl) {
            const int ix = tl - t_lo;
            const size_t r = brow(J, b, tl, h);
            double nk;
            normalise_with_norm(J->k + r * Dk, kb, &nk, Dk, J->l2norm);
            const double *Sp = bS + SS * ix, *Cp = bC + CC * ix, *mp = bm + (size_t)Dk * ix;
            double *Sn = bS + SS * (ix + 1), *Cn = bC + CC * (ix + 1), *mn = bm + (size_t)Dk * (ix + 1);
            for (int i = 0; i < Dk; ++i) {
                for (int j = 0; j < Dk; ++j) Cn[(size_t)i * Dk + j] = Cp[(size_t)i * Dk + j] + kb[i] * kb[j];
                mn[i] = mp[i] + kb[i];
                const double a = exp(J->gk[r * Dk + i]);
                for (int e = 0; e < Dv; ++e)
                    Sn[(size_t)i * Dv + e] = a * Sp[(size_t)i * Dv + e] + kb[i] * J->v[r * Dv + e];
            }
        }
        for (int tl = t_hi - 1; tl >= t_lo; --tl) {
            const int ix = tl - t_lo;
            const size_t r = brow(J, b, tl, h);
            const double tf = (double)(tstart + tl + 1);
            const double *St = bS + SS * (ix + 1), *Sp = bS + SS * ix;
            const double *Ct = bC + CC * (ix + 1), *mt = bm + (size_t)Dk * (ix + 1);
            const double lam = J->lam[r];
            const double *dor = J->dout + r * Dv, *vr = J->v + r * Dv, *gr = J->gk + r * Dk;
            double nq, nk;
            normalise_with_norm(J->q + r * Dk, qb, &nq, Dk, J->l2norm);
            normalise_with_norm(J->k + r * Dk, kb, &nk, Dk, J->l2norm);
            /* forward quantities of token t */
            double mq = 0.0;
            for (int j = 0; j < Dk; ++j) mq += mt[j] * qb[j];
            for (int i = 0; i < Dk; ++i) {
                double acc = 0.0;
                for (int j = 0; j < Dk; ++j) acc += Ct[(size_t)i * Dk + j] * qb[j];
                z[i] = acc / tf - (J->centered ? mt[i] * mq / (tf * tf) : 0.0);
                qc[i] = qb[i] - lam * z[i];
            }
            /* read: o = scale S_t q_clean */
            double dl = 0.0;
            for (int i = 0; i < Dk; ++i) {
                double acc = 0.0;
                for (int e = 0; e < Dv; ++e) {
                    acc += St[(size_t)i * Dv + e] * dor[e];
                    dS[(size_t)i * Dv + e] += J->scale * qc[i] * dor[e];
                }
                dqc[i] = J->scale * acc;
                dz[i] = -lam * dqc[i];
                dl -= z[i] * dqc[i];
            }
            J->dlam[r] = dl;
            /* clean: dqbar = dq_clean + Sigma_t dz; statistics adjoints */
            double mdz = 0.0;
            for (int j = 0; j < Dk; ++j) mdz += mt[j] * dz[j];
            for (int i = 0; i < Dk; ++i) {
                double acc = 0.0;
                for (int j = 0; j < Dk; ++j) acc += Ct[(size_t)i * Dk + j] * dz[j];
                dqb[i] = dqc[i] + acc / tf - (J->centered ? mt[i] * mdz / (tf * tf) : 0.0);
            }
            for (int i = 0; i < Dk; ++i) {
                for (int j = 0; j < Dk; ++j) dC[(size_t)i * Dk + j] += dz[i] * qb[j] / tf;
                if (J->centered) dm[i] -= (mq * dz[i] + mdz * qb[i]) / (tf * tf);
            }
            /* write: S_t = Diag(alpha) S_{t-1} + kbar v^T */
            for (int i = 0; i < Dk; ++i) {
                double acc = 0.0, gs = 0.0;
                for (int e = 0; e < Dv; ++e) {
                    acc += dS[(size_t)i * Dv + e] * vr[e];
                    gs += dS[(size_t)i * Dv + e] * Sp[(size_t)i * Dv + e];
                }
                dkb[i] = acc;
                const double a = exp(gr[i]);
                J->dgk[r * Dk + i] = a * gs;
            }
            for (int e = 0; e < Dv; ++e) {
                double acc = 0.0;
                for (int i = 0; i < Dk; ++i) acc += dS[(size_t)i * Dv + e] * kb[i];
                J->dv[r * Dv + e] = acc;
            }
            for (int i = 0; i < Dk; ++i) {
                const double a = exp(gr[i]);
                for (int e = 0; e < Dv; ++e) dS[(size_t)i * Dv + e] *= a;
            }
            /* statistics: C_t = C_{t-1} + kbar kbar^T, m_t = m_{t-1} + kbar */
            for (int i = 0; i < Dk; ++i) {
                double acc = 0.0;
                for (int j = 0; j < Dk; ++j) acc += (dC[(size_t)i * Dk + j] + dC[(size_t)j * Dk + i]) * kb[j];
                dkb[i] += acc + dm[i];
            }
            normalise_backward(qb, nq, dqb, J->dq + r * Dk, Dk, J->l2norm);
            normalise_backward(kb, nk, dkb, J->dk + r * Dk, Dk, J->l2norm);
        }
    }
    if (J->dS0) memcpy(J->dS0 + bh * SS, dS, sizeof(double) * SS);
    if (J->dC0) memcpy(J->dC0 + bh * CC, dC, sizeof(double) * CC);
    if (J->dm0) memcpy(J->dm0 + bh * Dk, dm, sizeof(double) * Dk);
    free(ckS); free(ckC); free(ckm); free(bS); free(bC); free(bm); free(qb); free(kb); free(z); free(qc);
    free(dqc); free(dz); free(dqb); free(dkb); free(dS); free(dC); free(dm);
}

static void *bworker(void *arg) {
    bjob_t *J = (bjob_t *)arg;
    for (;;) {
        pthread_mutex_lock(&J->mu);
        const int w = J->next++;
        pthread_mutex_unlock(&J->mu);
        if (w >= J->B * J->H) break;
        backward_pair(J, w / J->H, w % J->H);
    }
    return NULL;
}

/*
 * CCQ-GLA backward.  Inputs as ccq_oracle_forward (GLA) plus dout [B,T,H,Dv] and
 * optional adjoints of the final states dST [B,H,Dk,Dv], dCT [B,H,Dk,Dk],
 * dmT [B,H,Dk] (NULL = 0).  Outputs dq, dk [B,T,H,Dk], dv [B,T,H,Dv],
 * dgk [B,T,H,Dk], dlam [B,T,H], dS0, dC0, dm0 (each may be NULL only for the
 * initial-state gradients).  Returns 0, or -1 on a bad argument.
 */
int ccq_oracle_gla_backward(int B, int T, int H, int Dk, int Dv, const double *q, const double *k,
                            const double *v, const double *gk, const double *lam, const double *S0,
                            const double *C0, const double *m0, const int64_t *t0, const double *dout,
                            const double *dST, const double *dCT, const double *dmT, double *dq,
                            double *dk, double *dv, double *dgk, double *dlam, double *dS0, double *dC0,
                            double *dm0, int l2norm, int centered, double scale, int nthreads) {
    if (B < 0 || T < 0 || H < 0 || Dk <= 0 || Dv <= 0 || nthreads < 1) return -1;
    if (!q || !k || !v || !gk || !lam || !dout || !dq || !dk || !dv || !dgk || !dlam) return -1;
    bjob_t J;
    memset(&J, 0, sizeof J);
    J.B = B; J.T = T; J.H = H; J.Dk = Dk; J.Dv = Dv; J.l2norm = l2norm; J.centered = centered;
    J.scale = scale;
    J.q = q; J.k = k; J.v = v; J.gk = gk; J.lam = lam; J.S0 = S0; J.C0 = C0; J.m0 = m0; J.t0 = t0;
    J.dout = dout; J.dST = dST; J.dCT = dCT; J.dmT = dmT;
    J.dq = dq; J.dk = dk; J.dv = dv; J.dgk = dgk; J.dlam = dlam; J.dS0 = dS0; J.dC0 = dC0; J.dm0 = dm0;
    pthread_mutex_init(&J.mu, NULL);
    if (nthreads > B * H) nthreads = B * H > 0 ? B * H : 1;
    pthread_t *th = malloc(sizeof(pthread_t) * (size_t)nthreads);
    for (int i = 0; i < nthreads; ++i) pthread_create(&th[i], NULL, bworker, &J);
    for (int i = 0; i < nthreads; ++i) pthread_join(th[i], NULL);
    free(th);
    pthread_mutex_destroy(&J.mu);
    return 0;
}

/* ====================================================================== reverse mode, Gated DeltaNet
 *
 * Gradients of the CCQ-Gated-DeltaNet forward (recurrent form above), same scheme as the GLA
 * backward: block checkpoints every 64 tokens, each block recomputed and walked backwards.  The
 * write, with the state stored as Hs = S^T [Dk][Dv], a = e^{g_t}, u = Hs_{t-1}^T kbar, is
 *   Hs_t = a (Hs_{t-1} - beta kbar u^T) + beta kbar v^T,
 * and with G the adjoint of Hs_t its adjoints are
 *   dv = beta G^T kbar,  du = -a beta G^T kbar,
 *   dkbar (write) = G (beta v - a beta u) + Hs_{t-1} du,
 *   da = sum(G * (Hs_{t-1} - beta kbar u^T)),  dg = a da,
 *   dbeta = kbar^T G (v - a u),  dHs_{t-1} = a G + kbar du^T.
 * The read, the cleaned query and the key statistics are as in the GLA backward.
 */
static void backward_pair_gdn(const bjob_t *J, int b, int h) {
    const int Dk = J->Dk, Dv = J->Dv, T = J->T, BL = 64;
    const int NB = (T + BL - 1) / BL;
    const size_t bh = (size_t)b * J->H + h;
    const size_t SS = (size_t)Dk * Dv, CC = (size_t)Dk * Dk;
    double *ckS = malloc(sizeof(double) * SS * (NB + 1));
    double *ckC = malloc(sizeof(double) * CC * (NB + 1));
    double *ckm = malloc(sizeof(double) * Dk * (NB + 1));
    double *bS = malloc(sizeof(double) * SS * (BL + 1));
    double *bC = malloc(sizeof(double) * CC * (BL + 1));
    double *bm = malloc(sizeof(double) * Dk * (BL + 1));
    double *qb = malloc(sizeof(double) * Dk), *kb = malloc(sizeof(double) * Dk);
    double *z = malloc(sizeof(double) * Dk), *qc = malloc(sizeof(double) * Dk);
    double *dqc = malloc(sizeof(double) * Dk), *dz = malloc(sizeof(double) * Dk);
    double *dqb = malloc(sizeof(double) * Dk), *dkb = malloc(sizeof(double) * Dk);
    double *u = malloc(sizeof(double) * Dv), *gtk = malloc(sizeof(double) * Dv), *du = malloc(sizeof(double) * Dv);
    double *dS = malloc(sizeof(double) * SS), *dC = malloc(sizeof(double) * CC);
    double *dm = malloc(sizeof(double) * Dk);
    const int64_t tstart = J->t0 ? J->t0[b] : 0;

    if (J->S0) memcpy(ckS, J->S0 + bh * SS, sizeof(double) * SS); else memset(ckS, 0, sizeof(double) * SS);
    if (J->C0) memcpy(ckC, J->C0 + bh * CC, sizeof(double) * CC); else memset(ckC, 0, sizeof(double) * CC);
    if (J->m0) memcpy(ckm, J->m0 + bh * Dk, sizeof(double) * Dk); else memset(ckm, 0, sizeof(double) * Dk);

    /* one token's write: Sn = a (Sp - beta kb u^T) + beta kb v^T, u = Sp^T kb */
#define GDN_WRITE(Sp, Sn, r)                                                                  \
    do {                                                                                      \
        const double a_ = exp(J->gk[(r)]), be_ = J->beta[(r)];                                \
        const double *vr_ = J->v + (r) * Dv;                                                  \
        for (int e = 0; e < Dv; ++e) {                                                        \
            double acc = 0.0;                                                                 \
            for (int i = 0; i < Dk; ++i) acc += kb[i] * (Sp)[(size_t)i * Dv + e];             \
            u[e] = acc;                                                                       \
        }                                                                                     \
        for (int i = 0; i < Dk; ++i)                                                          \
            for (int e = 0; e < Dv; ++e)                                                      \
                (Sn)[(size_t)i * Dv + e] =                                                    \
                    a_ * ((Sp)[(size_t)i * Dv + e] - be_ * kb[i] * u[e]) + be_ * kb[i] * vr_[e]; \
    } while (0)

    for (int blk = 0; blk < NB; ++blk) {
        double *S = ckS + SS * (blk + 1), *C = ckC + CC * (blk + 1), *m = ckm + (size_t)Dk * (blk + 1);
        memcpy(bS, ckS + SS * blk, sizeof(double) * SS);
        memcpy(C, ckC + CC * blk, sizeof(double) * CC);
        memcpy(m, ckm + (size_t)Dk * blk, sizeof(double) * Dk);
        for (int tl = blk * BL; tl < T && tl < (blk + 1) * BL; ++tl) {
            const size_t r = brow(J, b, tl, h);
            double nk;
            normalise_with_norm(J->k + r * Dk, kb, &nk, Dk, J->l2norm);
            for (int i = 0; i < Dk; ++i) {
                for (int j = 0; j < Dk; ++j) C[(size_t)i * Dk + j] += kb[i] * kb[j];
                m[i] += kb[i];
            }
            GDN_WRITE(bS, bS + SS, r);
            memcpy(bS, bS + SS, sizeof(double) * SS);
        }
        memcpy(S, bS, sizeof(double) * SS);
    }

    if (J->dST) memcpy(dS, J->dST + bh * SS, sizeof(double) * SS); else memset(dS, 0, sizeof(double) * SS);
    if (J->dCT) memcpy(dC, J->dCT + bh * CC, sizeof(double) * CC); else memset(dC, 0, sizeof(double) * CC);
    if (J->dmT) memcpy(dm, J->dmT + bh * Dk, sizeof(double) * Dk); else memset(dm, 0, sizeof(double) * Dk);

    for (int blk = NB - 1; blk >= 0; --blk) {
        const int t_lo = blk * BL, t_hi = (T < (blk + 1) * BL) ? T : (blk + 1) * BL;
        /* recompute the block's per-token states: index 0 = block start, i + 1 = after token t_lo + i */
        memcpy(bS, ckS + SS * blk, sizeof(double) * SS);
        memcpy(bC, ckC + CC * blk, sizeof(double) * CC);
        memcpy(bm, ckm + (size_t)Dk * blk, sizeof(double) * Dk);
        for (int tl = t_lo; tl < t_hi; ++tl) {
            const int ix = tl - t_lo;
            const size_t r = brow(J, b, tl, h);
            double nk;
            normalise_with_norm(J->k + r * Dk, kb, &nk, Dk, J->l2norm);
            const double *Cp = bC + CC * ix, *mp = bm + (size_t)Dk * ix;
            double *Cn = bC + CC * (ix + 1), *mn = bm + (size_t)Dk * (ix + 1);
            for (int i = 0; i < Dk; ++i) {
                for (int j = 0; j < Dk; ++j) Cn[(size_t)i * Dk + j] = Cp[(size_t)i * Dk + j] + kb[i] * kb[j];
                mn[i] = mp[i] + kb[i];
            }
            GDN_WRITE(bS + SS * ix, bS + SS * (ix + 1), r);
        }
        for (int tl = t_hi - 1; tl >= t_lo; --tl) {
            const int ix = tl - t_lo;
            const size_t r = brow(J, b, tl, h);
            const double tf = (double)(tstart + tl + 1);
            const double *St = bS + SS * (ix + 1), *Sp = bS + SS * ix;
            const double *Ct = bC + CC * (ix + 1), *mt = bm + (size_t)Dk * (ix + 1);
            const double lam = J->lam[r], a = exp(J->gk[r]), be = J->beta[r];
            const double *dor = J->dout + r * Dv, *vr = J->v + r * Dv;
            double nq, nk;
            normalise_with_norm(J->q + r * Dk, qb, &nq, Dk, J->l2norm);
            normalise_with_norm(J->k + r * Dk, kb, &nk, Dk, J->l2norm);
            /* forward quantities of token t: z, q_clean, u = Hs_{t-1}^T kbar */
            double mq = 0.0;
            for (int j = 0; j < Dk; ++j) mq += mt[j] * qb[j];
            for (int i = 0; i < Dk; ++i) {
                double acc = 0.0;
                for (int j = 0; j < Dk; ++j) acc += Ct[(size_t)i * Dk + j] * qb[j];
                z[i] = acc / tf - (J->centered ? mt[i] * mq / (tf * tf) : 0.0);
                qc[i] = qb[i] - lam * z[i];
            }
            for (int e = 0; e < Dv; ++e) {
                double acc = 0.0;
                for (int i = 0; i < Dk; ++i) acc += kb[i] * Sp[(size_t)i * Dv + e];
                u[e] = acc;
            }
            /* read: o = scale Hs_t^T q_clean */
            double dl = 0.0;
            for (int i = 0; i < Dk; ++i) {
                double acc = 0.0;
                for (int e = 0; e < Dv; ++e) {
                    acc += St[(size_t)i * Dv + e] * dor[e];
                    dS[(size_t)i * Dv + e] += J->scale * qc[i] * dor[e];
                }
                dqc[i] = J->scale * acc;
                dz[i] = -lam * dqc[i];
                dl -= z[i] * dqc[i];
            }
            J->dlam[r] = dl;
            /* clean: dqbar = dq_clean + Sigma_t dz; statistics adjoints */
            double mdz = 0.0;
            for (int j = 0; j < Dk; ++j) mdz += mt[j] * dz[j];
            for (int i = 0; i < Dk; ++i) {
                double acc = 0.0;
                for (int j = 0; j < Dk; ++j) acc += Ct[(size_t)i * Dk + j] * dz[j];
                dqb[i] = dqc[i] + acc / tf - (J->centered ? mt[i] * mdz / (tf * tf) : 0.0);
            }
            for (int i = 0; i < Dk; ++i) {
                for (int j = 0; j < Dk; ++j) dC[(size_t)i * Dk + j] += dz[i] * qb[j] / tf;
                if (J->centered) dm[i] -= (mq * dz[i] + mdz * qb[i]) / (tf * tf);
            }
            /* write: G = dS is the adjoint of Hs_t */
            for (int e = 0; e < Dv; ++e) {
                double acc = 0.0;
                for (int i = 0; i < Dk; ++i) acc += dS[(size_t)i * Dv + e] * kb[i];
                gtk[e] = acc;                       /* G^T kbar */
                J->dv[r * Dv + e] = be * acc;
                du[e] = -a * be * acc;
            }
            double da = 0.0, dbe = 0.0;
            for (int i = 0; i < Dk; ++i) {
                double acc = 0.0, hs = 0.0, gsum = 0.0;
                for (int e = 0; e < Dv; ++e) {
                    const double G = dS[(size_t)i * Dv + e];
                    acc += G * (be * vr[e] - a * be * u[e]);
                    hs += Sp[(size_t)i * Dv + e] * du[e];
                    gsum += G * (Sp[(size_t)i * Dv + e] - be * kb[i] * u[e]);
                    dbe += kb[i] * G * (vr[e] - a * u[e]);
                }
                dkb[i] = acc + hs;
                da += gsum;
            }
            J->dgk[r] = a * da;
            J->dbeta[r] = dbe;
            for (int i = 0; i < Dk; ++i)
                for (int e = 0; e < Dv; ++e)
                    dS[(size_t)i * Dv + e] = a * dS[(size_t)i * Dv + e] + kb[i] * du[e];
            /* statistics: C_t = C_{t-1} + kbar kbar^T, m_t = m_{t-1} + kbar */
            for (int i = 0; i < Dk; ++i) {
                double acc = 0.0;
                for (int j = 0; j < Dk; ++j) acc += (dC[(size_t)i * Dk + j] + dC[(size_t)j * Dk + i]) * kb[j];
                dkb[i] += acc + dm[i];
            }
            normalise_backward(qb, nq, dqb, J->dq + r * Dk, Dk, J->l2norm);
            normalise_backward(kb, nk, dkb, J->dk + r * Dk, Dk, J->l2norm);
        }
    }
#undef GDN_WRITE
    if (J->dS0) memcpy(J->dS0 + bh * SS, dS, sizeof(double) * SS);
    if (J->dC0) memcpy(J->dC0 + bh * CC, dC, sizeof(double) * CC);
    if (J->dm0) memcpy(J->dm0 + bh * Dk, dm, sizeof(double) * Dk);
    free(ckS); free(ckC); free(ckm); free(bS); free(bC); free(bm); free(qb); free(kb); free(z); free(qc);
    free(dqc); free(dz); free(dqb); free(dkb); free(u); free(gtk); free(du); free(dS); free(dC); free(dm);
}

static void *bworker_gdn(void *arg) {
    bjob_t *J = (bjob_t *)arg;
    for (;;) {
        pthread_mutex_lock(&J->mu);
        const int w = J->next++;
        pthread_mutex_unlock(&J->mu);
        if (w >= J->B * J->H) break;
        backward_pair_gdn(J, w / J->H, w % J->H);
    }
    return NULL;
}

/*
 * CCQ-Gated-DeltaNet backward.  Inputs as ccq_oracle_forward (GDN: g the log decay and beta,
 * both [B,T,H]) plus dout [B,T,H,Dv] and optional adjoints of the final states (NULL = 0).
 * Outputs dq, dk [B,T,H,Dk], dv [B,T,H,Dv], dg and dbeta [B,T,H], dlam [B,T,H], dS0, dC0,
 * dm0 (each of the last three may be NULL).  Returns 0, or -1 on a bad argument.
 */
int ccq_oracle_gdn_backward(int B, int T, int H, int Dk, int Dv, const double *q, const double *k,
                            const double *v, const double *g, const double *beta, const double *lam,
                            const double *S0, const double *C0, const double *m0, const int64_t *t0,
                            const double *dout, const double *dST, const double *dCT, const double *dmT,
                            double *dq, double *dk, double *dv, double *dg, double *dbeta, double *dlam,
                            double *dS0, double *dC0, double *dm0, int l2norm, int centered, double scale,
                            int nthreads) {
    if (B < 0 || T < 0 || H < 0 || Dk <= 0 || Dv <= 0 || nthreads < 1) return -1;
    if (!q || !k || !v || !g || !beta || !lam || !dout || !dq || !dk || !dv || !dg || !dbeta || !dlam) return -1;
    bjob_t J;
    memset(&J, 0, sizeof J);
    J.B = B; J.T = T; J.H = H; J.Dk = Dk; J.Dv = Dv; J.l2norm = l2norm; J.centered = centered;
    J.scale = scale;
    J.q = q; J.k = k; J.v = v; J.gk = g; J.beta = beta; J.lam = lam; J.S0 = S0; J.C0 = C0; J.m0 = m0;
    J.t0 = t0; J.dout = dout; J.dST = dST; J.dCT = dCT; J.dmT = dmT;
    J.dq = dq; J.dk = dk; J.dv = dv; J.dgk = dg; J.dbeta = dbeta; J.dlam = dlam;
    J.dS0 = dS0; J.dC0 = dC0; J.dm0 = dm0;
    pthread_mutex_init(&J.mu, NULL);
    if (nthreads > B * H) nthreads = B * H > 0 ? B * H : 1;
    pthread_t *th = malloc(sizeof(pthread_t) * (size_t)nthreads);
    for (int i = 0; i < nthreads; ++i) pthread_create(&th[i], NULL, bworker_gdn, &J);
    for (int i = 0; i < nthreads; ++i) pthread_join(th[i], NULL);
    free(th);
    pthread_mutex_destroy(&J.mu);
    return 0;
}
