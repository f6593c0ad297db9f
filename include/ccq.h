/*
 * ccq.h -- C ABI of the GB300 (sm_103a) Curvature-Conditioned Query library.
 *
 * CCQ (arxiv 2606.01294) modifies only the read of a linear-attention layer:
 * before the query reads the fast-weight state S, it is contracted by
 * (I - lambda_t Sigma_t), where Sigma_t is the running, length-normalised key
 * covariance (Sec. 3.2, Eq. clean; App. A.2):
 *
 *   C_t = sum_{j<=t} kbar_j kbar_j^T,   m_t = sum_{j<=t} kbar_j,
 *   Sigma_t = C_t / t - (m_t / t)(m_t / t)^T            (centred, default)
 *   q_clean = qbar_t - lambda_t Sigma_t qbar_t           (Eq. clean, Algorithm 2)
 *   o_t     = scale * S_t q_clean                        (Eq. read)
 *
 * with qbar, kbar the per-head l2-normalised query and key (Algorithms 1, 2).
 * The backbone write S_t = Update(S_{t-1}; kbar_t, v_t, ...) is either
 *   GLA:            S_t = S_{t-1} Diag(alpha_t) + v_t kbar_t^T,   alpha_t = exp(gk_t) in R^{Dk}
 *   Gated DeltaNet: S_t = alpha_t S_{t-1} (I - beta_t kbar_t kbar_t^T) + beta_t v_t kbar_t^T,
 *                   alpha_t = exp(g_t) scalar
 * (Sec. 2.2; the paper treats the write rule as a black box).  The chunkwise
 * kernels follow Algorithm 1 (App. B): the key statistics are carried across
 * chunks as a d_k x d_k second-moment sum and a d_k key-sum vector.
 *
 * Conventions shared by every entry point
 *   - Pointers are DEVICE pointers owned by the caller and must be 16-byte
 *     aligned.  Nothing is allocated and nothing is freed by the library.
 *   - Token tensors are [B, T, H, D] with D contiguous (row-major).
 *   - States are fp32.  S is stored as its transpose: S[B, H, Dk, Dv], element
 *     [i][j] is the paper's S_{j,i}.  C is the second-moment SUM C_t
 *     [B, H, Dk, Dk] (not divided by t), m the key SUM m_t [B, H, Dk], and t the
 *     per-batch-row token count [B] (int64).  Algorithm 2's running means are
 *     C_t / t and m_t / t; keeping sums makes chunk, prefill and decode
 *     resumption exact.
 *   - Initial-state pointers may be NULL (zero state, t0 = 0).  Final-state
 *     pointers may be NULL (not written).  A final-state buffer may alias the
 *     corresponding initial-state buffer.
 *   - Calls are asynchronous on `stream` (a cudaStream_t; NULL = legacy default
 *     stream).  Argument errors are reported synchronously through the
 *     return value; the calls never abort the process.  Every in-kernel wait is
 *     bounded: a wait that runs out records CCQ_ERR_TIMEOUT in a device status
 *     word that ccq_device_status() reads back.
 */
#ifndef CCQ_H_
#define CCQ_H_

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define CCQ_API __attribute__((visibility("default")))
#else
#define CCQ_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    CCQ_OK = 0,
    CCQ_ERR_INVALID_ARG = 1, /* NULL or misaligned pointer, negative size, ...    */
    CCQ_ERR_UNSUPPORTED = 2, /* a valid request this build does not implement     */
    CCQ_ERR_CUDA = 3,        /* a CUDA runtime/driver call failed                 */
    CCQ_ERR_TIMEOUT = 4,     /* an in-kernel bounded wait ran out (device status) */
    CCQ_ERR_RANGE = 5        /* a chunk's gates left the range the kernel can factor (device status) */
} ccq_status;

typedef enum { CCQ_BF16 = 0, CCQ_FP32 = 1 } ccq_dtype;

/* Spectral contraction of the query (ccq_gdn_fwd_spectral): the paper's first-order operator
   and the two alternatives it names with that first-order form (Sec. 3.2, after Eq. clean). */
typedef enum {
    CCQ_CONTRACT_LINEAR = 0,     /* q_clean = (I - lambda Sigma) qbar (the paper's CCQ)      */
    CCQ_CONTRACT_RESOLVENT = 1,  /* q_clean = (I + lambda Sigma)^{-1} qbar                   */
    CCQ_CONTRACT_EXPONENTIAL = 2 /* q_clean = exp(-lambda Sigma) qbar                        */
} ccq_contraction;

typedef enum {
    CCQ_ALGO_AUTO = 0,      /* chunkwise tensor-core kernel when supported, else recurrent */
    CCQ_ALGO_RECURRENT = 1, /* token-by-token CUDA-core kernel (fp32 arithmetic)         */
    CCQ_ALGO_CHUNKWISE = 2, /* chunkwise tcgen05 kernel (bf16 operands, fp32 accumulate)  */
    CCQ_ALGO_CHUNKWISE_WIDE = 3 /* CCQ-GLA: the chunkwise kernel with two gate references per
                                   chunk, for strongly forgetting gates (see ccq_gla_fwd); about
                                   twice the time.  Gated DeltaNet: the same as CHUNKWISE.   */
} ccq_algo;

/* Contraction and read hyper-parameters. */
typedef struct {
    int l2norm_qk; /* 1: l2-normalise q and k per head row in the kernel (Algorithms 1, 2);
                      0: use q and k as given.  The norm uses rsqrt(max(|x|^2, 1e-12)),
                      so an all-zero row stays zero.                                     */
    float scale;   /* read scale multiplying o; <= 0 selects 1/sqrt(Dk) (paper silent)    */
    int centered;  /* 1: Sigma_t = C_t/t - mu_t mu_t^T (App. A.2); 0: uncentred C_t/t
                      (App. D ablation)                                                  */
    int chunk;     /* chunk length of the chunkwise kernels; 0 or 64 (Algorithm 1)        */
    int algo;      /* a ccq_algo value                                                   */
    int seq_split; /* chunkwise GLA only: segments each sequence is cut into so that few
                      long sequences still fill the GPU (states compose exactly across
                      segments); 0 = choose from B*H and the SM count, 1 = never split */
} ccq_params;

/* Fill *p with the defaults: l2norm_qk = 1, scale = 0 (1/sqrt(Dk)), centered = 1,
   chunk = 64, algo = CCQ_ALGO_AUTO, seq_split = 0. */
CCQ_API void ccq_default_params(ccq_params *p);

/*
 * CCQ-GLA chunkwise forward (Algorithm 1 with the GLA write rule).
 *   q, k      [B,T,H,Dk] in in_dtype;  v [B,T,H,Dv] in in_dtype.
 *   gk        log forget gate log(alpha) [B,T,H,Dk] in gate_dtype (<= 0).
 *   lambda    [B,T,H] fp32, the CCQ gate lambda_t in (0,1) (Eq. clean; the caller
 *             applies W_lambda and the sigmoid).
 *   S0/C0/m0/t0  initial states (see conventions); ST/CT/mT/tT final states.
 *   o         [B,T,H,Dv] in in_dtype.
 * Supported: Dk = Dv in {64, 128}; T >= 0; B, H >= 1.  in_dtype BF16 runs the
 * chunkwise tensor-core kernel for Dk = Dv = 128 and the recurrent kernel
 * otherwise; FP32 always runs the recurrent kernel (fp32 arithmetic).
 * Gate range of the chunkwise kernels.  A chunk's decays are applied as factors
 * measured from reference tokens inside the chunk.  The default kernel (AUTO,
 * CHUNKWISE) has one reference, the chunk midpoint; it is exact (up to rounding)
 * while, for every key dimension, the log gates of each 32-token half of a chunk
 * sum to more than about -82 (e.g. per-token log gates above -2.5).  CHUNKWISE_WIDE
 * has one reference per half, which doubles that range (each 16-token quarter
 * above about -82, e.g. per-token log gates above -5) at about twice the time.
 * Beyond its range a kernel records CCQ_ERR_RANGE in the device status word
 * (ccq_device_status) and its outputs are not valid; the recurrent path
 * (algo RECURRENT) has no range limit.  Within range, a decay that underflows
 * contributes an exact zero.  The backward (ccq_gla_bwd) has the default
 * kernel's range.
 *   workspace  caller-owned device scratch of at least ccq_gla_workspace_size()
 *              bytes (16-byte aligned) when that size is non-zero (long sequences
 *              split into segments); may be NULL otherwise.  Contents undefined on
 *              return.
 * Returns CCQ_OK or an error code; launches asynchronously on `stream`.
 */
CCQ_API ccq_status ccq_gla_fwd(const void *q, const void *k, const void *v, const void *gk,
                       const float *lambda, ccq_dtype in_dtype, ccq_dtype gate_dtype,
                       const float *S0, const float *C0, const float *m0, const int64_t *t0,
                       void *o, float *ST, float *CT, float *mT, int64_t *tT,
                       int B, int T, int H, int Dk, int Dv, void *workspace,
                       size_t workspace_bytes, const ccq_params *p, void *stream);

/*
 * Workspace bytes ccq_gla_fwd needs (the per-segment states of a split sequence;
 * 0 when sequences are not split).  The split depends on B*H, T and the current
 * device's SM count.  Queries the device but launches nothing.
 */
CCQ_API ccq_status ccq_gla_workspace_size(int B, int T, int H, int Dk, int Dv, ccq_dtype in_dtype,
                                          const ccq_params *p, size_t *bytes);

/*
 * CCQ-Gated-DeltaNet forward (the gated delta rule as the backbone).
 *   g         log decay log(alpha) [B,T,H] fp32 (<= 0);  beta [B,T,H] fp32 in [0,1].
 *   workspace caller-owned device scratch of at least the size ccq_gdn_workspace_size()
 *             reports (16-byte aligned), used by the chunkwise kernel to hold the
 *             per-chunk UT factor Tt diag(beta) (64 x 64 bf16 per chunk); may be NULL
 *             when that size is 0.  Its contents on entry do not matter and are
 *             undefined on return.
 * All other arguments as ccq_gla_fwd.  bf16 inputs with Dk = Dv = 128 run the chunkwise
 * tensor-core kernels (CCQ_ALGO_AUTO / CHUNKWISE / CHUNKWISE_WIDE, which are the same here;
 * CCQ_ERR_INVALID_ARG if the workspace is missing or too small); other inputs run the
 * recurrent kernel.  Every decay factor of the chunkwise kernels is an exponential of a
 * non-positive argument (e^{gc_i}, e^{gC - gc_j} and, per score entry, e^{gc_i - gc_j}), so
 * any g <= 0 is supported; a decay that underflows contributes an exact zero.
 */
CCQ_API ccq_status ccq_gdn_fwd(const void *q, const void *k, const void *v, const float *g,
                       const float *beta, const float *lambda, ccq_dtype in_dtype,
                       const float *S0, const float *C0, const float *m0, const int64_t *t0,
                       void *o, float *ST, float *CT, float *mT, int64_t *tT,
                       int B, int T, int H, int Dk, int Dv, void *workspace,
                       size_t workspace_bytes, const ccq_params *p, void *stream);

/*
 * Workspace bytes ccq_gdn_fwd needs for these sizes and parameters (0 when the
 * selected kernel needs none).  Host-only; launches nothing.
 */
CCQ_API ccq_status ccq_gdn_workspace_size(int B, int T, int H, int Dk, int Dv, ccq_dtype in_dtype,
                                          const ccq_params *p, size_t *bytes);

/*
 * One recurrent CCQ token for a batch of cached states (Algorithm 2), updating
 * the cache (S, C, m, t) IN PLACE and writing o.
 *   backbone  0 = GLA (gate: log alpha [B,H,Dk] in gate_dtype),
 *             1 = Gated DeltaNet (gate: log alpha [B,H] fp32; beta [B,H] fp32).
 *   q, k      [B,H,Dk]; v [B,H,Dv]; lambda [B,H] fp32; o [B,H,Dv] (in_dtype).
 *   S [B,H,Dk,Dv], C [B,H,Dk,Dk], m [B,H,Dk] fp32 and t [B] int64, read and written.
 */
CCQ_API ccq_status ccq_decode_step(int backbone, const void *q, const void *k, const void *v,
                           const void *gate, const float *beta, const float *lambda,
                           ccq_dtype in_dtype, ccq_dtype gate_dtype, float *S, float *C,
                           float *m, int64_t *t, void *o, int B, int H, int Dk, int Dv,
                           const ccq_params *p, void *stream);

/*
 * Bytes of the checkpoint buffer ccq_gla_fwd_save writes for these sizes: per
 * (sequence, head), 66048 bytes per 64-token chunk (the bf16 S^K and
 * e^{Gmid} S of the chunk start, the fp32 key sum) plus 65536 bytes (fp32 S_T).
 * Host-only.
 */
CCQ_API ccq_status ccq_gla_ckpt_size(int B, int T, int H, int Dk, int Dv, size_t *bytes);

/*
 * ccq_gla_fwd that also saves, into `ckpt` (device memory, at least
 * ccq_gla_ckpt_size() bytes, 16-byte aligned), the chunk-start states the
 * backward needs, so that ccq_gla_bwd does not recompute them (a training
 * step's forward).  Only the chunkwise tensor-core path saves checkpoints:
 * bf16 inputs, Dk = Dv = 128, T >= 1, algo AUTO, CHUNKWISE or CHUNKWISE_WIDE; anything else
 * returns CCQ_ERR_UNSUPPORTED.  All other arguments as ccq_gla_fwd.
 */
CCQ_API ccq_status ccq_gla_fwd_save(const void *q, const void *k, const void *v, const void *gk,
                                    const float *lambda, ccq_dtype in_dtype, ccq_dtype gate_dtype,
                                    const float *S0, const float *C0, const float *m0, const int64_t *t0,
                                    void *o, float *ST, float *CT, float *mT, int64_t *tT,
                                    int B, int T, int H, int Dk, int Dv, void *workspace,
                                    size_t workspace_bytes, void *ckpt, size_t ckpt_bytes,
                                    const ccq_params *p, void *stream);

/*
 * CCQ-GLA backward: the gradients of a scalar loss L through ccq_gla_fwd, given
 * dL/do and (optionally) dL/d(final states).  The paper times a backward pass
 * but does not write it out; it is the reverse mode of Eqs. clean/read, the
 * running sums of Sec. 3.2 and the GLA write, chunked like Algorithm 1.
 *   q, k, v, gk, lambda, in/gate dtypes, S0/C0/m0/t0   the forward's inputs.
 *   dout      dL/do [B,T,H,Dv] in in_dtype.
 *   dST [B,H,Dk,Dv], dCT [B,H,Dk,Dk], dmT [B,H,Dk] fp32: dL/d(ST, CT, mT); NULL = 0.
 *   ckpt      checkpoints written by ccq_gla_fwd_save on the same inputs, or
 *             NULL: the call then recomputes them (one forward pass without
 *             the output) into the workspace.
 *   dq, dk    [B,T,H,Dk], dv [B,T,H,Dv] in in_dtype; dgk [B,T,H,Dk] in
 *             gate_dtype: gradients of q, k, v and gk (the raw, un-normalised
 *             q and k when l2norm_qk = 1).
 *   dlambda   [B,T,H] fp32 (may be NULL);  dS0 [B,H,Dk,Dv], dC0 [B,H,Dk,Dk],
 *             dm0 [B,H,Dk] fp32 (each may be NULL): gradients of lambda and of
 *             the initial states.
 *   workspace at least ccq_gla_bwd_workspace_size() bytes (16-byte aligned):
 *             four bf16 [B,T,H,128] tensors and 67 KB per 64-token chunk that
 *             the backward kernels exchange, plus the checkpoints and forward
 *             scratch when ckpt is NULL.
 * Supported: bf16 inputs with Dk = Dv = 128 (the chunkwise tensor-core path),
 * algo AUTO or CHUNKWISE; otherwise CCQ_ERR_UNSUPPORTED.  T = 0 copies the
 * final-state gradients to the initial-state ones.
 */
CCQ_API ccq_status ccq_gla_bwd(const void *q, const void *k, const void *v, const void *gk,
                               const float *lambda, ccq_dtype in_dtype, ccq_dtype gate_dtype,
                               const float *S0, const float *C0, const float *m0, const int64_t *t0,
                               const void *dout, const float *dST, const float *dCT, const float *dmT,
                               const void *ckpt, void *dq, void *dk, void *dv, void *dgk,
                               float *dlambda, float *dS0, float *dC0, float *dm0,
                               int B, int T, int H, int Dk, int Dv, void *workspace,
                               size_t workspace_bytes, const ccq_params *p, void *stream);

/*
 * Workspace bytes ccq_gla_bwd needs; with_ckpt = 1 when the caller passes
 * checkpoints (then only the exchange tensors), 0 otherwise.  Queries the
 * device (the forward's segment split) but launches nothing.
 */
CCQ_API ccq_status ccq_gla_bwd_workspace_size(int B, int T, int H, int Dk, int Dv, ccq_dtype in_dtype,
                                              int with_ckpt, const ccq_params *p, size_t *bytes);

/*
 * CCQ-Gated-DeltaNet backward: the gradients of a scalar loss L through ccq_gdn_fwd,
 * given dL/do and (optionally) dL/d(final states).  The paper gives no backward; this is
 * the reverse mode of Eqs. clean/read, the running sums of Sec. 3.2 and the gated delta
 * rule, chunked like Algorithm 1 (only the state adjoint crosses chunks sequentially).
 *   q, k, v, g, beta, lambda, in_dtype, S0/C0/m0/t0   the forward's inputs.
 *   dout      dL/do [B,T,H,Dv] in in_dtype.
 *   dST [B,H,Dk,Dv], dCT [B,H,Dk,Dk], dmT [B,H,Dk] fp32: dL/d(ST, CT, mT); NULL = 0.
 *   dq, dk    [B,T,H,Dk], dv [B,T,H,Dv] in in_dtype: gradients of q, k, v (the raw,
 *             un-normalised q and k when l2norm_qk = 1).
 *   dg, dbeta [B,T,H] fp32: gradients of the log decay and of beta.
 *   dlambda   [B,T,H] fp32 (may be NULL);  dS0, dC0, dm0 fp32 (each may be NULL).
 *   workspace at least ccq_gdn_bwd_workspace_size() bytes (16-byte aligned): per
 *             64-token chunk of every (sequence, head), the chunk's forward states,
 *             state adjoints and intermediate tiles in fp32 (for bf16 inputs with
 *             Dk = 128, followed by the chunkwise forward's own workspace).
 * Supported: Dk = Dv in {64, 128}, bf16 or fp32 inputs.  The per-chunk forward quantities
 * the adjoint needs (the UT factor (I + A)^{-1}, the entering S^K, M and H of every chunk)
 * come, for bf16 inputs with Dk = 128, from the chunkwise tensor-core forward kernels of
 * ccq_gdn_fwd (which write them in fp32 and no output; their segment split follows
 * p->seq_split), and otherwise from three CUDA-core passes.  The products of the adjoint's
 * per-chunk kernels run, for bf16 inputs, on the tensor cores (bf16 operands, fp32 accumulation;
 * their element-wise parts stay fp32) and, for fp32 inputs, on the CUDA cores in fp32; its reverse
 * pass over the state adjoint runs, for bf16 inputs with Dk = 128, on the tensor cores, and
 * otherwise on the CUDA cores (the algo parameter is ignored).  A bounded wait of the tensor-core
 * kernels that gives up leaves the gradients invalid and CCQ_ERR_TIMEOUT for
 * ccq_device_status().  T = 0 copies the final-state gradients to the initial-state ones.
 */
CCQ_API ccq_status ccq_gdn_bwd(const void *q, const void *k, const void *v, const float *g,
                               const float *beta, const float *lambda, ccq_dtype in_dtype,
                               const float *S0, const float *C0, const float *m0, const int64_t *t0,
                               const void *dout, const float *dST, const float *dCT, const float *dmT,
                               void *dq, void *dk, void *dv, float *dg, float *dbeta, float *dlambda,
                               float *dS0, float *dC0, float *dm0, int B, int T, int H, int Dk, int Dv,
                               void *workspace, size_t workspace_bytes, const ccq_params *p, void *stream);

/* Workspace bytes ccq_gdn_bwd needs for these sizes (0 when T = 0).  Queries the device
 * (the forward's segment split, bf16 with Dk = 128) but launches nothing. */
CCQ_API ccq_status ccq_gdn_bwd_workspace_size(int B, int T, int H, int Dk, int Dv, ccq_dtype in_dtype,
                                              const ccq_params *p, size_t *bytes);

/*
 * CCQ-Gated-DeltaNet forward with a decay-aligned covariance.  The paper proposes a
 * covariance from gamma-weighted running statistics for backbones that forget
 * (Limitations; App. "Modelling choices and limitations", interaction with decayed
 * backbones) but fixes neither the weights nor the normaliser.  This entry point reads gamma_{j,t} as the product of the backbone's own
 * decays alpha_s = exp(g_s) over j < s <= t and normalises by the decayed count:
 *   C_t = alpha_t C_{t-1} + kbar_t kbar_t^T,  m_t = alpha_t m_{t-1} + kbar_t,
 *   n_t = alpha_t n_{t-1} + 1,  Sigma_t = C_t / n_t - (m_t / n_t)(m_t / n_t)^T
 * (uncentred with centered = 0), which is ccq_gdn_fwd's covariance when every alpha = 1.
 *   C0/CT [B,H,Dk,Dk], m0/mT [B,H,Dk]: the decayed sums;  n0/nT [B,H] fp32: the decayed
 *   count (replacing t0/tT).  NULL initial pointers mean zero; NULL final pointers are not
 *   written.
 *   workspace  at least ccq_gdn_decayed_workspace_size() bytes, 16-byte aligned (per 64-token
 *              chunk of every (sequence, head): the chunk's UT factor, entering state and
 *              entering statistics in fp32).
 * Other arguments as ccq_gdn_fwd.  Supported: Dk = Dv in {64, 128}, bf16 or fp32 inputs;
 * the kernels compute in fp32 on the CUDA cores (five launches; the algo parameter is
 * ignored).
 */
CCQ_API ccq_status ccq_gdn_fwd_decayed(const void *q, const void *k, const void *v, const float *g,
                                       const float *beta, const float *lambda, ccq_dtype in_dtype,
                                       const float *S0, const float *C0, const float *m0, const float *n0,
                                       void *o, float *ST, float *CT, float *mT, float *nT,
                                       int B, int T, int H, int Dk, int Dv, void *workspace,
                                       size_t workspace_bytes, const ccq_params *p, void *stream);

/*
 * CCQ-Gated-DeltaNet forward with a choice of spectral contraction and of covariance
 * statistics, on the same CUDA-core kernels as ccq_gdn_fwd_decayed.
 *   contraction  a ccq_contraction value.  RESOLVENT runs ten conjugate-gradient iterations
 *                per query from the linear estimate (I + lambda Sigma has spectrum in
 *                [1, 1 + lambda] for unit keys); EXPONENTIAL sums twelve Taylor terms
 *                (|lambda Sigma| <= 1).  Both rely on unit-norm keys for those bounds, so they
 *                need l2norm_qk = 1: with l2norm_qk = 0 they return CCQ_ERR_UNSUPPORTED
 *                (arbitrary key norms would leave the fixed iteration counts without an
 *                error bound).
 *   decayed      1: the decay-aligned statistics of ccq_gdn_fwd_decayed (n the decayed count);
 *                0: the paper's undecayed sums, C_t = sum kbar kbar^T, m_t = sum kbar, with n
 *                the token count t (n0/nT [B,H] fp32 carry it) -- with LINEAR this is the
 *                paper's CCQ-Gated-DeltaNet, computed in fp32 on the CUDA cores.
 * Other arguments, the workspace (ccq_gdn_decayed_workspace_size) and the supported sizes as
 * ccq_gdn_fwd_decayed, which equals this call with LINEAR and decayed = 1.
 */
CCQ_API ccq_status ccq_gdn_fwd_spectral(const void *q, const void *k, const void *v, const float *g,
                                        const float *beta, const float *lambda, ccq_dtype in_dtype,
                                        const float *S0, const float *C0, const float *m0, const float *n0,
                                        void *o, float *ST, float *CT, float *mT, float *nT,
                                        int B, int T, int H, int Dk, int Dv, int contraction, int decayed,
                                        void *workspace, size_t workspace_bytes, const ccq_params *p,
                                        void *stream);

/* Workspace bytes ccq_gdn_fwd_decayed and ccq_gdn_fwd_spectral need for these sizes (0 when
   T = 0).  Host-only. */
CCQ_API ccq_status ccq_gdn_decayed_workspace_size(int B, int T, int H, int Dk, int Dv, ccq_dtype in_dtype,
                                                  const ccq_params *p, size_t *bytes);

/*
 * Forward of packed variable-length sequences (GLA or Gated DeltaNet backbone): sequence s is
 * tokens [cu_seqlens[s], cu_seqlens[s+1]) of the packed tensors, and runs as one batch-1
 * ccq_gla_fwd / ccq_gdn_fwd call on them (the calls follow each other on `stream` and share
 * the workspace).  The paper trains on fixed-length sequences; this is for serving mixes.
 *   backbone     0 = GLA, 1 = Gated DeltaNet.
 *   q, k [total,H,Dk]; v, o [total,H,Dv] in in_dtype;  gate: GLA log forget gate
 *                [total,H,Dk] in gate_dtype, or Gated DeltaNet log decay [total,H] fp32;
 *                beta (GDN only) and lambda [total,H] fp32.
 *   cu_seqlens   HOST array of num_seqs + 1 offsets, cu_seqlens[0] = 0, non-decreasing
 *                (empty sequences allowed).  cu_seqlens[s] * H must be a multiple of 4 so that
 *                every sequence's fp32 rows start 16-byte aligned (any offsets when H % 4 = 0).
 *   S0, C0, m0, t0 / ST, CT, mT, tT  per-sequence states [num_seqs, H, ...] and [num_seqs], as
 *                in ccq_gla_fwd (NULL allowed as there).
 *   workspace    at least ccq_fwd_varlen_workspace_size() bytes (the largest per-sequence need).
 */
CCQ_API ccq_status ccq_fwd_varlen(int backbone, const void *q, const void *k, const void *v, const void *gate,
                                  const float *beta, const float *lambda, ccq_dtype in_dtype, ccq_dtype gate_dtype,
                                  const int64_t *cu_seqlens, int num_seqs, const float *S0, const float *C0,
                                  const float *m0, const int64_t *t0, void *o, float *ST, float *CT, float *mT,
                                  int64_t *tT, int H, int Dk, int Dv, void *workspace, size_t workspace_bytes,
                                  const ccq_params *p, void *stream);

/* Workspace bytes ccq_fwd_varlen needs for these sequences.  Queries the device (the segment
   split of long GLA sequences) but launches nothing. */
CCQ_API ccq_status ccq_fwd_varlen_workspace_size(int backbone, const int64_t *cu_seqlens, int num_seqs, int H,
                                                 int Dk, int Dv, ccq_dtype in_dtype, const ccq_params *p,
                                                 size_t *bytes);

/*
 * ccq_gla_fwd for callers that cannot supply any device memory of their own --
 * for instance an engine that gave all device memory to its own caches at
 * start-up, or code on a path where allocating is not allowed or would stall
 * the device.  The paper has no counterpart; this is a deployment convenience.
 * Same arguments as ccq_gla_fwd minus the workspace: the per-segment states of
 * split sequences live in a fixed 24 MiB array inside the library (190
 * (sequence, segment) states), which every GPU that loads the library keeps
 * until the process exits.  Nothing is allocated.
 *   - Requests needing more scratch than that (ccq_gla_workspace_size) fail with
 *     CCQ_ERR_INVALID_ARG and a message naming both sizes.
 *   - The first call on each device looks up the array's device address
 *     (cudaGetSymbolAddress); make that first call before any stream capture.
 *     The address is then kept for the life of the process, which assumes the
 *     device's primary context lives that long: after cudaDeviceReset (or any
 *     teardown and re-creation of that context) the kept address is stale, so
 *     do not reset a device while this library is in use on it.
 *   - All calls share the one array and it keeps the last call's contents: two
 *     calls whose work overlaps on the GPU (other streams, other host threads)
 *     race and corrupt each other's results; serialise them.
 */
CCQ_API ccq_status ccq_gla_fwd_fixed_scratch(const void *q, const void *k, const void *v, const void *gk,
                                             const float *lambda, ccq_dtype in_dtype, ccq_dtype gate_dtype,
                                             const float *S0, const float *C0, const float *m0,
                                             const int64_t *t0, void *o, float *ST, float *CT, float *mT,
                                             int64_t *tT, int B, int T, int H, int Dk, int Dv,
                                             const ccq_params *p, void *stream);

/*
 * Synchronise `stream`, then read and clear the device status word that the
 * kernels write.  Returns CCQ_OK, CCQ_ERR_RANGE (a chunkwise CCQ-GLA kernel met
 * gates stronger than its factored decays can represent: see ccq_gla_fwd), CCQ_ERR_TIMEOUT (a kernel gave
 * up waiting; its outputs are not valid) or CCQ_ERR_CUDA.
 */
CCQ_API ccq_status ccq_device_status(void *stream);

/* Static description of a status code. */
CCQ_API const char *ccq_status_string(ccq_status s);

/* Human-readable detail of the most recent error returned on this host thread. */
CCQ_API const char *ccq_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* CCQ_H_ */
