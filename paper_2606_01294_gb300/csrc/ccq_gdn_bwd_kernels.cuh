// ccq_gdn_bwd_kernels.cuh -- CCQ-Gated-DeltaNet backward kernels (fp32 tiles; the per-chunk kernels'
// products on the tensor cores for bf16 inputs).
//
// Reverse mode of the CCQ read (Eq. clean, Eq. read, the undecayed running sums of Sec. 3.2)
// with the Gated DeltaNet write as the backbone, chunked as Algorithm 1 chunks the forward.
// The paper gives no backward; the adjoint below is the reverse mode of the chunk map
//
//   A  = strict_lower(diag(beta) (Kbar Kbar^T) o Gamma),  Gamma_ij = e^{gc_i - gc_j},
//   Tt = (I + A)^{-1},  Tb = Tt diag(beta),  R = V - diag(E) Kbar H,  U = Tb R,  E_i = e^{gc_i}
//   O  = scale (diag(E) Qc H + P U),  P = (Qc Kbar^T) o Gamma o causal
//   H' = e^{gc_last} H + Kd^T U,  Kd = diag(e^{gc_last - gc}) Kbar
//
// (gc the in-chunk cumulative log decay, H the state entering the chunk with key dims as
// rows), with the CCQ contraction qc = qbar - lambda z, z = Sigma_t qbar.  Given the
// adjoint dH of H' and D = scale dO, per chunk:
//   dU  = P^T D + Kd dH,       dv = dR = Tb^T dU
//   dP  = (D U^T) o Gamma o causal,   dqc = diag(E) D H^T + dP Kbar
//   dH_enter = e^{gc_last} dH + (diag(E) Qc)^T D - (diag(E) Kbar)^T dR
//   dTb = dU R^T,  dbeta_j = sum_i dTb_ij Tt_ij + sum_l dA_jl Gamma_jl KK_jl,
//   dA  = strict_lower(-Tt^T (dTb diag(beta)) Tt^T),  dKK = diag(beta) (dA o Gamma)
//   dkbar = dP^T Qc + diag(e^{gc_last - gc}) U dH^T - diag(E) dR H^T + (dKK + dKK^T) Kbar
//           + the CCQ terms (as in the GLA backward)
//   dgc = rowsum - colsum of (dA o A) and (dP o S) + E o rowsum((Qc H) o D)
//         - rowsum(Kd o U dH^T) - E o rowsum((Kbar H) o dR),
//         plus e^{gc_last} <dH, H> + sum_i rowsum(Kd o U dH^T)_i at the last row;
//   dg  = the in-chunk reverse cumulative sum of dgc.
// Only dH crosses chunks sequentially: the CCQ adjoints DC, Dm are sums of chunk-local
// terms.  So the backward is seven launches:
//   gdn_bwd_prep_kernel    per chunk: Tt and the chunk's key statistics (Kbar^T Kbar, sum Kbar)
//   gdn_bwd_prefix_kernel  exclusive prefix of the key statistics over chunks (S^K_r, M_r)
//   gdn_bwd_fstate_kernel  per sequence and head, chunks in order: the entering states H_r
//   gdn_bwd_local_kernel   per chunk: z, qc, R, U, dqc, dq, dlambda, the CCQ increments of
//                          DC and Dm, and P^T D, (diag(E) Qc)^T D for the state pass
//   gdn_bwd_dstate_kernel  per sequence and head, chunks last to first: dH at every chunk end
//   gdn_bwd_suffix_kernel  exclusive suffix of the DC, Dm increments (DC_{r+1}, Dm_{r+1})
//   gdn_bwd_kv_kernel      per chunk: dv, dk, dbeta, dg
//
// Every kernel is a sequence of phases separated by __syncthreads(); inside a phase each
// thread strides over the elements it owns and reads only what earlier phases wrote (row
// reductions go through shared-memory atomics).  Arithmetic is fp32 on the CUDA cores, except
// that the local and kv kernels instantiated with TC = true (bf16 inputs) run their products on
// the tensor cores with bf16 operands and fp32 accumulation (tc_mm, ccq_gdn_bwd_tc.cuh).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stddef.h>
#include <stdint.h>
#include <string.h>

#include "ccq_gdn_bwd_tc.cuh"

namespace ccq {
namespace gbwd {

constexpr int kC = 64;  // chunk length
constexpr int kBwdThreads = 512;  // threads of the per-chunk local and kv kernels

#define GBWD_FOR(i, n) for (int i = static_cast<int>(threadIdx.x); i < (n); i += static_cast<int>(blockDim.x))

__device__ __forceinline__ float to_f(float x) { return x; }
__device__ __forceinline__ float to_f(__nv_bfloat16 x) { return __bfloat162float(x); }
template <typename T> __device__ __forceinline__ T from_f(float x);
template <> __device__ __forceinline__ float from_f<float>(float x) { return x; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f<__nv_bfloat16>(float x) { return __float2bfloat16_rn(x); }

// Kernel arguments.  Token tensors are [B][T][H][D]; g, beta, lambda [B][T][H] fp32.
// The workspace arrays are indexed by the chunk ch = (b*H + h)*NC + r.
struct GdnBwdArgs {
    int B, T, H, NC;
    int l2norm, centered;
    float scale;
    const void *q, *k, *v, *dout;
    const float *g, *beta, *lambda;
    const float *S0, *C0, *m0;  // may be NULL (zero)
    const int64_t *t0;          // may be NULL (zero)
    const float *dST, *dCT, *dmT;  // may be NULL (zero)
    void *dq, *dk, *dv;
    float *dg, *dbeta, *dlambda;   // dlambda may be NULL
    float *dS0, *dC0, *dm0;        // each may be NULL
    // workspace, per chunk
    float *tt;   // [64][64] Tt
    float *sk;   // [D][D]   chunk's Kbar^T Kbar, then S^K_r
    float *mk;   // [D]      chunk's sum Kbar, then M_r
    float *hs;   // [D][D]   H_r (the state entering the chunk)
    float *dh;   // [D][D]   adjoint of H_{r+1} (the state leaving the chunk)
    float *dc;   // [D][D]   chunk's increment of DC, then DC_{r+1}
    float *dm;   // [D]      chunk's increment of Dm, then Dm_{r+1}
    float *x1;   // [64][D]  P^T D
    float *y1;   // [D][D]   (diag(E) Qc)^T D
    float *qb, *qc, *u, *r, *w;  // [64][D] each: qbar, qc, U, R, W = dz / t
    float *vec;  // [4][64]  cq, cz, E o rowsum((Qc H) o D), spare
    float *hT = nullptr;  // [B][H][D][D]: when set, gdn_bwd_fstate_kernel writes the final state
    int nsplit = 1;       // value-column blocks of the sequential passes (a divisor of D): the
                          // delta rule acts on the columns of H independently, so each
                          // (sequence, head) runs as nsplit CTAs of D / nsplit columns
    int states_ready = 0; // tt, sk, mk, hs already hold Tt, S^K_r, M_r, H_r (from the forward)
    int *status = nullptr; // status word of the tensor-core products' bounded waits (TC kernels)
};

__device__ __forceinline__ size_t tok_row(const GdnBwdArgs &a, int b, int t, int h) {
    return (static_cast<size_t>(b) * a.T + t) * a.H + h;
}

// Load the rows of chunk r of a [B][T][H][D] tensor into dst[64][D] (zero past T).
template <int D, typename Tin>
__device__ __forceinline__ void load_tile(float *dst, const void *src, const GdnBwdArgs &a, int b, int h, int r) {
    const Tin *s = static_cast<const Tin *>(src);
    GBWD_FOR(idx, kC * D) {
        const int i = idx / D, c = idx % D, t = r * kC + i;
        dst[idx] = t < a.T ? to_f(s[tok_row(a, b, t, h) * D + c]) : 0.f;
    }
}

// Per-row inverse norms (phase) of a [64][D] tile: 1/max(|x|, 1e-6), 0 for an all-zero row
// (which normalises to itself and passes no gradient), or 1 when disabled.
template <int D>
__device__ __forceinline__ void row_rnorm(const float *x, float *rn, int l2norm) {
    GBWD_FOR(i, kC) {
        float ss = 0.f;
        for (int c = 0; c < D; ++c) ss += x[i * D + c] * x[i * D + c];
        rn[i] = !l2norm ? 1.f : (ss > 0.f ? 1.f / sqrtf(fmaxf(ss, 1e-12f)) : 0.f);
    }
}

// Gate scalars (phase, one thread): in-chunk cumulative log decay of the first n rows,
// held constant past them.
__device__ __forceinline__ void gate_prefix(const float *graw, float *gc) {
    if (threadIdx.x == 0) {
        float acc = 0.f;
        for (int i = 0; i < kC; ++i) {
            acc += graw[i];
            gc[i] = acc;
        }
    }
}

// An element-wise pass over total items whose loads come from global memory: the thread's
// items go U at a time, all U loads issued before the first store (the last, fewer than U, the
// same way), so that a thread keeps U loads in flight instead of one.  ld(e) loads item e,
// st(e, x) stores it.
template <int U, typename L, typename S>
__device__ __forceinline__ void stream_u(int total, L ld, S st) {
    using X = decltype(ld(0));
    const int stride = static_cast<int>(blockDim.x);
    int idx = static_cast<int>(threadIdx.x);
    for (; idx + (U - 1) * stride < total; idx += U * stride) {
        X x[U];
#pragma unroll
        for (int u = 0; u < U; ++u) x[u] = ld(idx + u * stride);
#pragma unroll
        for (int u = 0; u < U; ++u) st(idx + u * stride, x[u]);
    }
    X x[U];
#pragma unroll
    for (int u = 0; u < U; ++u)
        if (idx + u * stride < total) x[u] = ld(idx + u * stride);
#pragma unroll
    for (int u = 0; u < U; ++u)
        if (idx + u * stride < total) st(idx + u * stride, x[u]);
}
template <typename L, typename S>
__device__ __forceinline__ void stream8(int total, L ld, S st) {
    stream_u<8>(total, ld, st);
}

// 16-byte chunks of a [rows][CPR chunks] row-major array: chunk c is (row, column chunk).  With
// CPR a multiple of 8 (rows a multiple of 4) the eight lanes of a warp quarter take consecutive
// chunks of one row (128 contiguous bytes) and the four quarters four consecutive rows, so that
// stores into a tile of odd row stride hit 32 different banks; narrower rows go in row order.
template <int CPR>
__device__ __forceinline__ void chunk_rc(int c, int &row, int &col_chunk) {
    if constexpr (CPR % 8 == 0) {
        const int w = c >> 5;
        row = 4 * (w / (CPR / 8)) + ((c >> 3) & 3);
        col_chunk = 8 * (w % (CPR / 8)) + (c & 7);
    } else {
        row = c / CPR;
        col_chunk = c % CPR;
    }
}

// Unpack 16 bytes holding 16 / sizeof(T) values of type T into floats.
template <typename T>
__device__ __forceinline__ void unpack16(const uint4 &u, float (&f)[16 / sizeof(T)]) {
    T e[16 / sizeof(T)];
    memcpy(e, &u, 16);
#pragma unroll
    for (int x = 0; x < static_cast<int>(16 / sizeof(T)); ++x) f[x] = to_f(e[x]);
}

// Load the rows of chunk r of a [B][T][H][D] tensor, times scale, into dst[64][ld] (zero past T):
// 16-byte loads, all of a thread's issued before its stores.
template <int D, typename Tin>
__device__ __forceinline__ void load_tile_ld(float *dst, int ld, const void *src, const GdnBwdArgs &a, int b, int h,
                                             int r, float scale = 1.f) {
    constexpr int V = 16 / sizeof(Tin), CPR = D / V;
    const Tin *s = static_cast<const Tin *>(src);
    stream_u<4>(kC * CPR, [&](int c) {
        int i, cc;
        chunk_rc<CPR>(c, i, cc);
        const int t = r * kC + i;
        uint4 u = make_uint4(0u, 0u, 0u, 0u);
        if (t < a.T) u = *reinterpret_cast<const uint4 *>(s + tok_row(a, b, t, h) * D + cc * V);
        return u;
    }, [&](int c, uint4 u) {
        int i, cc;
        chunk_rc<CPR>(c, i, cc);
        float f[V];
        unpack16<Tin>(u, f);
        float *d = dst + i * ld + cc * V;
#pragma unroll
        for (int x = 0; x < V; ++x) d[x] = scale * f[x];
    });
}

// load_tile_ld for three tensors at once (all of a thread's loads of the three issued before its
// stores): the rows of chunk r of s0, s1, s2 into d0, d1, d2.
template <int D, typename Tin>
__device__ __forceinline__ void load_tiles3_ld(float *d0, float *d1, float *d2, int ld, const void *s0,
                                               const void *s1, const void *s2, const GdnBwdArgs &a, int b, int h,
                                               int r) {
    constexpr int V = 16 / sizeof(Tin), CPR = D / V, PER = kC * CPR;
    constexpr int U = 3 * ((PER + kBwdThreads - 1) / kBwdThreads);
    stream_u<U>(3 * PER, [&](int c) {
        const int tix = c / PER;
        int i, cc;
        chunk_rc<CPR>(c - tix * PER, i, cc);
        const Tin *sp = static_cast<const Tin *>(tix == 0 ? s0 : (tix == 1 ? s1 : s2));
        const int t = r * kC + i;
        uint4 u = make_uint4(0u, 0u, 0u, 0u);
        if (t < a.T) u = *reinterpret_cast<const uint4 *>(sp + tok_row(a, b, t, h) * D + cc * V);
        return u;
    }, [&](int c, uint4 u) {
        const int tix = c / PER;
        int i, cc;
        chunk_rc<CPR>(c - tix * PER, i, cc);
        float f[V];
        unpack16<Tin>(u, f);
        float *d = (tix == 0 ? d0 : (tix == 1 ? d1 : d2)) + i * ld + cc * V;
#pragma unroll
        for (int x = 0; x < V; ++x) d[x] = f[x];
    });
}

// A pass over rows [0, rows) and columns [0, COLS) of an fp32 array in global memory with row
// stride sld (floats), 16 bytes at a time (src and sld 16-byte aligned, rows a multiple of 4), all
// of a thread's loads issued before its stores: f(i, j0, x) gets row i, columns [j0, j0 + 4).
template <int COLS, typename F>
__device__ __forceinline__ void rows4(const float *src, int sld, int rows, F f) {
    constexpr int CPR = COLS / 4;
    stream_u<8>(rows * CPR, [&](int c) {
        int i, cc;
        chunk_rc<CPR>(c, i, cc);
        return *reinterpret_cast<const float4 *>(src + static_cast<size_t>(i) * sld + 4 * cc);
    }, [&](int c, float4 x) {
        int i, cc;
        chunk_rc<CPR>(c, i, cc);
        f(i, 4 * cc, x);
    });
}

// dst[rows][ld] <- src[rows][COLS] (fp32, e.g. a workspace tile into shared memory; src 16-byte
// aligned, rows a multiple of 4).
template <int COLS>
__device__ __forceinline__ void copy_rows(float *dst, int ld, const float *src, int rows) {
    rows4<COLS>(src, COLS, rows, [&](int i, int j0, float4 x) {
        float *d = dst + i * ld + j0;
        d[0] = x.x;
        d[1] = x.y;
        d[2] = x.z;
        d[3] = x.w;
    });
}

// row_rnorm over a [64][ld] tile.
template <int D>
__device__ __forceinline__ void row_rnorm_ld(const float *x, int ld, float *rn, int l2norm) {
    GBWD_FOR(i, kC) {
        float ss = 0.f;
        for (int c = 0; c < D; ++c) ss += x[i * ld + c] * x[i * ld + c];
        rn[i] = !l2norm ? 1.f : (ss > 0.f ? 1.f / sqrtf(fmaxf(ss, 1e-12f)) : 0.f);
    }
}

struct Pair4 {
    float4 a, b;
};

// Row sums over the 64 rows of a chunk: out[i] += sum_{c < ncols} f(i, c), as eight work items a
// row (a warp's items on 32 consecutive rows, so reads of a tile with odd row stride are free of
// bank conflicts) combined by shared-memory atomics.  out must be zero before the preceding
// barrier; the sums are complete after the next one.
template <typename F>
__device__ __forceinline__ void row_sums(float *out, int ncols, F f) {
    GBWD_FOR(w, 8 * kC) {
        const int i = w & (kC - 1), part = w / kC;
        float acc = 0.f;
        for (int c2 = part; c2 < ncols; c2 += 8) acc += f(i, c2);
        atomicAdd(&out[i], acc);
    }
}

// The l2 normalisation factor of a row from its sum of squares: 1/max(|x|, 1e-6), 0 for an
// all-zero row (which normalises to itself and passes no gradient), or 1 when disabled.
__device__ __forceinline__ float rnorm_of(float ss, int l2norm) {
    return !l2norm ? 1.f : (ss > 0.f ? 1.f / sqrtf(fmaxf(ss, 1e-12f)) : 0.f);
}

// Register-tiled product of two operands in shared memory, computed by VT virtual threads
// (the CTA's threads stride over them) of TM x TN outputs each, on a (VT / GN) x GN grid:
//   out(m, n) = sum_{k<K} A[m ars + k acs] B[k brs + n bcs],   m < (VT / GN) TM, n < GN TN,
// virtual thread (tm, tn) holding rows tm + (VT / GN) i and columns tn + GN j, so that a warp's
// loads of B for one j are GN consecutive columns and its loads of A 32 / GN rows (broadcasts);
// a B column stride bcs and an A row stride ars that are odd (or 1) keep them free of bank
// conflicts.  ep(m, n, value) consumes every output once, in the thread that computed it.
// (Rows at or past mlim are skipped: a product with fewer rows than the grid, TM = 1.)
template <int TM, int TN, int GN = 16, int VT = 256, typename Ep>
__device__ __forceinline__ void tile_mm(const float *A, int ars, int acs, const float *B, int brs, int bcs, int K,
                                        Ep ep, int mlim = 1 << 30) {
    constexpr int GM = VT / GN;
    for (int vt = static_cast<int>(threadIdx.x); vt < VT; vt += static_cast<int>(blockDim.x)) {
        const int tm = vt / GN, tn = vt % GN;
        if (tm >= mlim) continue;
        float acc[TM][TN];
#pragma unroll
        for (int i = 0; i < TM; ++i)
#pragma unroll
            for (int j = 0; j < TN; ++j) acc[i][j] = 0.f;
        const float *a0 = A + tm * ars, *b0 = B + tn * bcs;
#pragma unroll 2
        for (int k = 0; k < K; ++k) {
            float av[TM], bv[TN];
#pragma unroll
            for (int i = 0; i < TM; ++i) av[i] = a0[GM * i * ars + k * acs];
#pragma unroll
            for (int j = 0; j < TN; ++j) bv[j] = b0[k * brs + GN * j * bcs];
#pragma unroll
            for (int i = 0; i < TM; ++i)
#pragma unroll
                for (int j = 0; j < TN; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
        }
#pragma unroll
        for (int i = 0; i < TM; ++i)
#pragma unroll
            for (int j = 0; j < TN; ++j) ep(tm + GM * i, tn + GN * j, acc[i][j]);
    }
}

// The grid of an M x N product for VT virtual threads: 32 columns a row of the grid for N >= 128
// with 512 threads, 16 otherwise (N itself below 16).
template <int M, int N, int VT>
struct MmShape {
    static constexpr int GN = (N >= 128 && VT >= 512) ? 32 : (N >= 16 ? 16 : N);
    static constexpr int TN = N / GN, GM = VT / GN, TM = M / GM > 0 ? M / GM : 1;
};
template <int M, int N, int VT, typename Ep>
__device__ __forceinline__ void mm(const float *A, int ars, int acs, const float *B, int brs, int bcs, int K, Ep ep) {
    using S = MmShape<M, N, VT>;
    tile_mm<S::TM, S::TN, S::GN, VT>(A, ars, acs, B, brs, bcs, K, ep, M);
}

// An M x N x K product of the per-chunk kernels: on the tensor core (tc_mm, bf16 operands) in
// their TC instantiation, else tile_mm on the CUDA cores.
template <bool TC, int M, int N, int K, typename Ep>
__device__ __forceinline__ void gmm(TcEng &e, const float *A, int ars, int acs, const float *B, int brs, int bcs,
                                    Ep ep) {
    if constexpr (TC) {
        tc_mm<M, N, K>(e, A, ars, acs, B, brs, bcs, ep);
    } else {
        (void)e;
        mm<M, N, kBwdThreads>(A, ars, acs, B, brs, bcs, K, ep);
    }
}

// Staging-buffer bytes of the two per-chunk kernels' tensor-core products (the local kernel's
// D x D products, M = 128 when D = 128, stage 16 reduction steps at a time).
template <int D> constexpr int local_tc_stage() {
    return tc_stage_bytes(kC, D, kTcSliceK) > tc_stage_bytes(D, D, D == 128 ? 16 : kTcSliceK)
               ? tc_stage_bytes(kC, D, kTcSliceK) : tc_stage_bytes(D, D, D == 128 ? 16 : kTcSliceK);
}
template <int D> constexpr int kv_tc_stage() { return tc_stage_bytes(kC, D, kTcSliceK); }

// v[0..NV) to dst[0..NV) in the tensor's type as 16-byte stores (dst 16-byte aligned, NV a
// multiple of 8).
template <typename T, int NV>
__device__ __forceinline__ void st_row_t(T *dst, const float (&v)[NV]) {
    constexpr int E = 16 / sizeof(T);
#pragma unroll
    for (int q = 0; q < NV / E; ++q) {
        T e[E];
#pragma unroll
        for (int x = 0; x < E; ++x) e[x] = from_f<T>(v[E * q + x]);
        uint4 u;
        memcpy(&u, e, 16);
        reinterpret_cast<uint4 *>(dst)[q] = u;
    }
}

// v[0..NV) to dst[0..NV) as 16-byte stores (dst 16-byte aligned, NV a multiple of 4).
template <int NV>
__device__ __forceinline__ void st_row(float *dst, const float (&v)[NV]) {
    float4 *d4 = reinterpret_cast<float4 *>(dst);
#pragma unroll
    for (int q = 0; q < NV / 4; ++q) d4[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
}

// ---------------------------------------------------------------------------------------------
// Per chunk: Tt = (I + A)^{-1} by forward substitution, and the chunk's key statistics (the
// products KK and Kbar^T Kbar as tile_mm over padded tiles).
template <int D, typename Tin>
__global__ void __launch_bounds__(256) gdn_bwd_prep_kernel(const GdnBwdArgs a) {
    extern __shared__ float4 gbwd_smem4[];
    constexpr int LD = D + 1, LC = kC + 1, TD = D / 16;
    float *sm = reinterpret_cast<float *>(gbwd_smem4);
    float *Kb = sm;                // [64][LD]
    float *A = Kb + kC * LD;       // [64][LC]
    float *Tt = A + kC * LC;       // [64][LC]
    float *graw = Tt + kC * LC;    // [64]
    float *gc = graw + kC;
    float *be = gc + kC;
    float *rk = be + kC;

    const int ch = blockIdx.x, r = ch % a.NC, bh = ch / a.NC, b = bh / a.H, h = bh % a.H;
    load_tile_ld<D, Tin>(Kb, LD, a.k, a, b, h, r);
    GBWD_FOR(i, kC) {
        const int t = r * kC + i;
        const size_t row = tok_row(a, b, t < a.T ? t : 0, h);
        graw[i] = t < a.T ? a.g[row] : 0.f;
        be[i] = t < a.T ? a.beta[row] : 0.f;
    }
    __syncthreads();
    row_rnorm_ld<D>(Kb, LD, rk, a.l2norm);
    gate_prefix(graw, gc);
    __syncthreads();
    GBWD_FOR(idx, kC * D) Kb[(idx / D) * LD + idx % D] *= rk[idx / D];
    __syncthreads();
    // A_ij = beta_i e^{gc_i - gc_j} kbar_i . kbar_j for j < i
    tile_mm<4, 4>(Kb, LD, 1, Kb, 1, LD, D, [&](int i, int j, float v) {
        A[i * LC + j] = j < i ? be[i] * expf(gc[i] - gc[j]) * v : 0.f;
    });
    __syncthreads();
    // (I + A) Tt = I with A strictly lower: row i of Tt needs rows 0..i-1.
    for (int i = 0; i < kC; ++i) {
        GBWD_FOR(j, kC) {
            float v = i == j ? 1.f : 0.f;
            for (int l = j; l < i; ++l) v -= A[i * LC + l] * Tt[l * LC + j];
            Tt[i * LC + j] = v;
        }
        __syncthreads();
    }
    float *tt = a.tt + static_cast<size_t>(ch) * kC * kC;
    GBWD_FOR(idx, kC * kC) tt[idx] = Tt[(idx / kC) * LC + idx % kC];
    float *sk = a.sk + static_cast<size_t>(ch) * D * D;
    tile_mm<TD, TD>(Kb, 1, LD, Kb, LD, 1, kC, [&](int p, int c, float v) { sk[p * D + c] = v; });
    float *mk = a.mk + static_cast<size_t>(ch) * D;
    GBWD_FOR(c, D) {
        float acc = 0.f;
        for (int i = 0; i < kC; ++i) acc += Kb[i * LD + c];
        mk[c] = acc;
    }
}

// Exclusive prefix over the chunks of each sequence and head: sk[r] <- C0 + sum_{s<r} sk[s],
// mk[r] <- m0 + sum_{s<r} mk[s].  One thread per (sequence-head, element).
template <int D>
__global__ void __launch_bounds__(256) gdn_bwd_prefix_kernel(const GdnBwdArgs a) {
    const long long per = static_cast<long long>(D) * D + D;
    const long long gid = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (gid >= per * a.B * a.H) return;
    const int bh = static_cast<int>(gid / per);
    const int e = static_cast<int>(gid % per);
    const bool isC = e < D * D;
    float *base = isC ? a.sk + static_cast<size_t>(bh) * a.NC * D * D + e
                      : a.mk + static_cast<size_t>(bh) * a.NC * D + (e - D * D);
    const size_t stride = isC ? static_cast<size_t>(D) * D : static_cast<size_t>(D);
    float acc = 0.f;
    if (isC && a.C0) acc = a.C0[static_cast<size_t>(bh) * D * D + e];
    if (!isC && a.m0) acc = a.m0[static_cast<size_t>(bh) * D + (e - D * D)];
    // eight chunks' loads in flight before their stores
    int r = 0;
    for (; r + 8 <= a.NC; r += 8) {
        float x[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) x[u] = base[(r + u) * stride];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            base[(r + u) * stride] = acc;
            acc += x[u];
        }
    }
    for (; r < a.NC; ++r) {
        const float x = base[r * stride];
        base[r * stride] = acc;
        acc += x;
    }
}

// Per sequence and head, chunks in order: the state entering every chunk (and, when hT is
// set, the final state).  CTA (sequence-head, s) carries the value columns [s DC, (s+1) DC),
// DC = D / NS, of H; a chunk's three products run as tile_mm over padded tiles.
template <int D, typename Tin, int NS>
__global__ void __launch_bounds__(512) gdn_bwd_fstate_kernel(const GdnBwdArgs a) {
    extern __shared__ float4 gbwd_smem4[];
    constexpr int DC = D / NS, LD = D + 1, LDC = DC + 1, LC = kC + 1;
    constexpr int GN = DC < 16 ? DC : 16, GM = 256 / GN, TMD = D / GM > 0 ? D / GM : 1;
    float *sm = reinterpret_cast<float *>(gbwd_smem4);
    float *Hs = sm;                // [D][LDC]
    float *Kb = Hs + D * LDC;      // [64][LD]
    float *R = Kb + kC * LD;       // [64][LDC]
    float *U = R + kC * LDC;       // [64][LDC] diag(ed) U
    float *Tt = U + kC * LDC;      // [64][LC] Tt diag(beta)
    float *graw = Tt + kC * LC;    // [64]
    float *gc = graw + kC, *be = gc + kC, *rk = be + kC, *E = rk + kC, *ed = E + kC;

    const int bh = blockIdx.x / NS, c0 = (blockIdx.x % NS) * DC, b = bh / a.H, h = bh % a.H;
    const Tin *vin = static_cast<const Tin *>(a.v);
    stream8(D * DC, [&](int idx) {
        return a.S0 ? a.S0[(static_cast<size_t>(bh) * D + idx / DC) * D + c0 + idx % DC] : 0.f;
    }, [&](int idx, float x) { Hs[(idx / DC) * LDC + idx % DC] = x; });
    __syncthreads();
    for (int r = 0; r < a.NC; ++r) {
        const size_t ch = static_cast<size_t>(bh) * a.NC + r;
        float *hs = a.hs + ch * D * D;
        GBWD_FOR(idx, D * DC) hs[(idx / DC) * D + c0 + idx % DC] = Hs[(idx / DC) * LDC + idx % DC];
        load_tile_ld<D, Tin>(Kb, LD, a.k, a, b, h, r);
        stream8(kC * DC, [&](int idx) {
            const int t = r * kC + idx / DC;
            return t < a.T ? to_f(vin[tok_row(a, b, t, h) * D + c0 + idx % DC]) : 0.f;
        }, [&](int idx, float x) { R[(idx / DC) * LDC + idx % DC] = x; });
        const float *tt = a.tt + ch * kC * kC;
        stream8(kC * kC, [&](int idx) { return tt[idx]; }, [&](int idx, float x) { Tt[(idx / kC) * LC + idx % kC] = x; });
        GBWD_FOR(i, kC) {
            const int t = r * kC + i;
            const size_t row = tok_row(a, b, t < a.T ? t : 0, h);
            graw[i] = t < a.T ? a.g[row] : 0.f;
            be[i] = t < a.T ? a.beta[row] : 0.f;
        }
        __syncthreads();
        row_rnorm_ld<D>(Kb, LD, rk, a.l2norm);
        gate_prefix(graw, gc);
        __syncthreads();
        GBWD_FOR(idx, kC * D) Kb[(idx / D) * LD + idx % D] *= rk[idx / D];
        GBWD_FOR(idx, kC * kC) Tt[(idx / kC) * LC + idx % kC] *= be[idx % kC];
        GBWD_FOR(i, kC) {
            E[i] = expf(gc[i]);
            ed[i] = expf(gc[kC - 1] - gc[i]);
        }
        __syncthreads();
        // R = V - diag(E) Kbar H
        tile_mm<kC / GM, DC / GN, GN>(Kb, LD, 1, Hs, LDC, 1, D, [&](int i, int j, float v) { R[i * LDC + j] -= E[i] * v; });
        __syncthreads();
        // diag(ed) U = diag(ed) Tt diag(beta) R
        tile_mm<kC / GM, DC / GN, GN>(Tt, LC, 1, R, LDC, 1, kC, [&](int i, int j, float v) { U[i * LDC + j] = ed[i] * v; });
        __syncthreads();
        // H <- e^{gc_last} H + Kd^T U = e^{gc_last} H + Kbar^T diag(ed) U
        const float elast = expf(gc[kC - 1]);
        tile_mm<TMD, DC / GN, GN>(Kb, 1, LD, U, LDC, 1, kC, [&](int l, int j, float v) {
            Hs[l * LDC + j] = elast * Hs[l * LDC + j] + v;
        }, D);
        __syncthreads();
    }
    if (a.hT)
        GBWD_FOR(idx, D * DC)
            a.hT[(static_cast<size_t>(bh) * D + idx / DC) * D + c0 + idx % DC] = Hs[(idx / DC) * LDC + idx % DC];
}

// Per chunk, everything that does not need dH: z, qc, R, U, dqc, dq, dlambda, the CCQ
// increments of DC and Dm, P^T D and (diag(E) Qc)^T D.  Products as in gdn_bwd_kv_kernel
// (gmm over [64][D + 1] and [64][65] tiles); the D x D operands H and S^K are staged a row
// block at a time through a tile that is free at that point, and z waits in the W slot of the
// workspace while its tile holds D.
template <int D, typename Tin, bool TC = false>
__global__ void __launch_bounds__(kBwdThreads, 1) gdn_bwd_local_kernel(const GdnBwdArgs a) {
    extern __shared__ float4 gbwd_smem4[];
    constexpr int LD = D + 1, LC = kC + 1, VT = kBwdThreads;
    constexpr int RB = D < 64 ? D : 64, NH = D / RB;      // row blocks of 64 (k-blocks)
    constexpr int RN = D < 32 ? D : 32, NN = D / RN;      // row blocks of 32 (n-blocks, in sB)
    float *sm = reinterpret_cast<float *>(gbwd_smem4);
    float *Qb = sm;                // [64][LD] qbar
    float *Kb = Qb + kC * LD;      // [64][LD] kbar
    float *Rq = Kb + kC * LD;      // [64][LD] V, then R, then S^K blocks, then qc, then S^K blocks
    float *Zw = Rq + kC * LD;      // [64][LD] H blocks, then z, then D (scaled by E), then W
    float *Ud = Zw + kC * LD;      // [64][LD] U, then dqc, then dqbar
    float *sA = Ud + kC * LD;      // [64][LC] (Qbar Kbar^T) o causal, then dP
    float *sB = sA + kC * LC;      // [64][LC] Tt diag(beta), then P, then H blocks, then (W Kbar^T) o causal
    float *graw = sB + kC * LC;
    float *gc = graw + kC, *E = gc + kC, *be = E + kC, *lam = be + kC, *tinv = lam + kC;
    float *rq = tinv + kC, *rk = rq + kC, *cq = rk + kC, *cz = cq + kC, *gqh = cz + kC;
    float *rdot = gqh + kC;
    float *M = rdot + kC;          // [D] the key sum M_r entering the chunk
    float *ssq = M + D, *ssk = ssq + kC, *dls = ssk + kC;  // row sums of squares, -dlambda
    float *segs = dls + kC;        // [4][D] sums of kbar over the four 16-row segments
    float *dMs = segs + 4 * D;     // [D] the Dm increment, accumulated
    TcEng eng{};                   // TC: the tensor-core products' state, behind dMs
    if constexpr (TC) tc_setup(eng, reinterpret_cast<uint8_t *>(dMs + D), local_tc_stage<D>(), kTcBufLocal, a.status);

    const int ch = blockIdx.x, r = ch % a.NC, bh = ch / a.NC, b = bh / a.H, h = bh % a.H;
    const int n = min(kC, a.T - r * kC);
    const float c = a.centered ? 1.f : 0.f;
    const float *H = a.hs + static_cast<size_t>(ch) * D * D;
    const float *SK = a.sk + static_cast<size_t>(ch) * D * D;
    const float *Mg = a.mk + static_cast<size_t>(ch) * D;
    const float *Tt = a.tt + static_cast<size_t>(ch) * kC * kC;
    const size_t t64 = static_cast<size_t>(ch) * kC * D;
    float *Wg = a.w + t64;
    const float t_start = static_cast<float>((a.t0 ? a.t0[b] : 0) + static_cast<int64_t>(r) * kC);

    load_tiles3_ld<D, Tin>(Qb, Kb, Rq, LD, a.q, a.k, a.v, a, b, h, r);
    GBWD_FOR(i, kC) {
        const int t = r * kC + i;
        const size_t row = tok_row(a, b, t < a.T ? t : 0, h);
        graw[i] = i < n ? a.g[row] : 0.f;
        be[i] = i < n ? a.beta[row] : 0.f;
        lam[i] = i < n ? a.lambda[row] : 0.f;
        tinv[i] = 1.f / (t_start + 1.f + static_cast<float>(i));
        gqh[i] = cq[i] = cz[i] = rdot[i] = ssq[i] = ssk[i] = dls[i] = 0.f;
    }
    GBWD_FOR(j, D) {
        M[j] = Mg[j];
        dMs[j] = 0.f;
    }
    __syncthreads();
    row_sums(ssq, D, [&](int i, int l) { return Qb[i * LD + l] * Qb[i * LD + l]; });
    row_sums(ssk, D, [&](int i, int l) { return Kb[i * LD + l] * Kb[i * LD + l]; });
    gate_prefix(graw, gc);
    __syncthreads();
    GBWD_FOR(i, kC) {
        E[i] = expf(gc[i]);
        rq[i] = rnorm_of(ssq[i], a.l2norm);
        rk[i] = rnorm_of(ssk[i], a.l2norm);
    }
    __syncthreads();
    GBWD_FOR(idx, kC * D) {
        const int i = idx / D, j = idx % D;
        Qb[i * LD + j] *= rq[i];
        Kb[i * LD + j] *= rk[i];
    }
    // Tt diag(beta) for U (be is visible after the barrier above)
    stream8(kC * kC, [&](int idx) { return Tt[idx]; },
            [&](int idx, float x) { sB[(idx / kC) * LC + idx % kC] = x * be[idx % kC]; });
    __syncthreads();
    // the segment sums of kbar, for CumK_i = M + sum_{j<=i} kbar_j
    GBWD_FOR(w, 4 * D) {
        const int j = w % D, sg = w / D;
        float acc = 0.f;
        for (int i = 16 * sg; i < 16 * sg + 16; ++i) acc += Kb[i * LD + j];
        segs[sg * D + j] = acc;
    }
    // (Qbar Kbar^T) o causal;  R = V - diag(E) Kbar H over the row blocks of H
    gmm<TC, kC, kC, D>(eng, Qb, LD, 1, Kb, 1, LD, [&](int i, int j, float v) { sA[i * LC + j] = j <= i ? v : 0.f; });
    for (int hf = 0; hf < NH; ++hf) {
        __syncthreads();
        copy_rows<D>(Zw, LD, H + static_cast<size_t>(RB * hf) * D, RB);
        __syncthreads();
        if constexpr (TC)  // the row blocks' products sum in TMEM, read back once
            tc_mma<kC, D, RB>(eng, Kb + RB * hf, LD, 1, Zw, LD, 1, hf > 0);
        else
            mm<kC, D, VT>(Kb + RB * hf, LD, 1, Zw, LD, 1, RB, [&](int i, int j, float v) { Rq[i * LD + j] -= E[i] * v; });
    }
    if constexpr (TC) tc_read_elem<kC, D>(eng, [&](int i, int j, float v) { Rq[i * LD + j] -= E[i] * v; });
    __syncthreads();
    // cq_i = CumK_i . qbar_i with CumK_i = M + sum_{j<=i} kbar_j;  U = Tt diag(beta) R
    row_sums(cq, D + kC, [&](int i, int l) {
        return l < D ? M[l] * Qb[i * LD + l] : (l - D <= i ? sA[i * LC + l - D] : 0.f);
    });
    {
        float *Rg = a.r + t64;
        float *Ug = a.u + t64;
        if constexpr (TC) {
            tc_mm_rows<kC, D, kC>(eng, sB, LC, 1, Rq, LD, 1, [&](int i, int j0, const auto &v) {
#pragma unroll
                for (int c = 0; c < static_cast<int>(sizeof(v) / sizeof(float)); ++c) Ud[i * LD + j0 + c] = v[c];
                st_row(Ug + i * D + j0, v);
            });
        } else {
            mm<kC, D, VT>(sB, LC, 1, Rq, LD, 1, kC, [&](int i, int j, float v) {
                Ud[i * LD + j] = v;
                Ug[i * D + j] = v;
            });
        }
        GBWD_FOR(idx, kC * D) Rg[idx] = Rq[(idx / D) * LD + idx % D];
    }
    // z = Sigma_t qbar (App. B form): (Qbar S^K + ((Qbar Kbar^T) o causal) Kbar) / t - c CumK cq / t^2
    __syncthreads();
    if constexpr (TC)
        tc_mma<kC, D, kC>(eng, sA, LC, 1, Kb, LD, 1, false);
    else
        mm<kC, D, VT>(sA, LC, 1, Kb, LD, 1, kC, [&](int i, int j, float v) { Zw[i * LD + j] = v; });
    for (int hf = 0; hf < NH; ++hf) {
        __syncthreads();
        copy_rows<D>(Rq, LD, SK + static_cast<size_t>(RB * hf) * D, RB);
        __syncthreads();
        if constexpr (TC)
            tc_mma<kC, D, RB>(eng, Qb + RB * hf, LD, 1, Rq, LD, 1, true);
        else
            mm<kC, D, VT>(Qb + RB * hf, LD, 1, Rq, LD, 1, RB, [&](int i, int j, float v) { Zw[i * LD + j] += v; });
    }
    if constexpr (TC) tc_read_elem<kC, D>(eng, [&](int i, int j, float v) { Zw[i * LD + j] = v; });
    __syncthreads();
    GBWD_FOR(w, 4 * D) {
        const int j = w % D, sg = w / D;
        float cum = M[j];
        for (int s2 = 0; s2 < sg; ++s2) cum += segs[s2 * D + j];
        for (int i = 16 * sg; i < 16 * sg + 16; ++i) {
            cum += Kb[i * LD + j];
            const float z = Zw[i * LD + j] * tinv[i] - c * cum * cq[i] * tinv[i] * tinv[i];
            Zw[i * LD + j] = z;
            Wg[i * D + j] = z;  // z waits in the W slot until dlambda
        }
    }
    __syncthreads();
    // qc = qbar - lambda z (Eq. clean)
    {
        float *Qg = a.qb + t64;
        float *Qcg = a.qc + t64;
        GBWD_FOR(idx, kC * D) {
            const int i = idx / D, j = idx % D;
            const float v = Qb[i * LD + j] - lam[i] * Zw[i * LD + j];
            Rq[i * LD + j] = v;
            Qcg[idx] = v;
            Qg[idx] = Qb[i * LD + j];
        }
    }
    __syncthreads();
    // P = (Qc Kbar^T) o Gamma o causal;  D (the scaled output adjoint) into z's tile
    gmm<TC, kC, kC, D>(eng, Rq, LD, 1, Kb, 1, LD, [&](int i, int j, float v) {
        sB[i * LC + j] = j <= i ? v * expf(gc[i] - gc[j]) : 0.f;
    });
    load_tile_ld<D, Tin>(Zw, LD, a.dout, a, b, h, r, a.scale);
    __syncthreads();
    // P^T D for the state pass;  dP = (D U^T) o Gamma o causal
    {
        float *X1 = a.x1 + t64;
        if constexpr (TC)
            tc_mm_rows<kC, D, kC>(eng, sB, 1, LC, Zw, LD, 1, [&](int i, int j0, const auto &v) { st_row(X1 + i * D + j0, v); });
        else
            mm<kC, D, VT>(sB, 1, LC, Zw, LD, 1, kC, [&](int i, int j, float v) { X1[i * D + j] = v; });
        gmm<TC, kC, kC, D>(eng, Zw, LD, 1, Ud, 1, LD, [&](int i, int j, float v) {
            sA[i * LC + j] = (j <= i && i < n) ? v * expf(gc[i] - gc[j]) : 0.f;
        });
    }
    __syncthreads();
    GBWD_FOR(idx, kC * D) Zw[(idx / D) * LD + idx % D] *= E[idx / D];  // diag(E) D
    __syncthreads();
    // (diag(E) Qc)^T D = Qc^T (diag(E) D) for the state pass;  dqc = dP Kbar + (diag(E) D) H^T
    // (over row blocks of H in sB);  gqh_i = E_i rowsum((Qc H) o D)_i = sum_j qc_ij ((E D) H^T)_ij
    {
        float *Y1 = a.y1 + static_cast<size_t>(ch) * D * D;
        if constexpr (TC)
            tc_mm_rows<D, D, kC>(eng, Rq, 1, LD, Zw, LD, 1, [&](int p, int j0, const auto &v) { st_row(Y1 + p * D + j0, v); });
        else
            mm<D, D, VT>(Rq, 1, LD, Zw, LD, 1, kC, [&](int p, int j, float v) { Y1[p * D + j] = v; });
        gmm<TC, kC, D, kC>(eng, sA, LC, 1, Kb, LD, 1, [&](int i, int j, float v) { Ud[i * LD + j] = v; });
    }
    if constexpr (TC) {
        // 64 rows of H at a time through the S/dP pair (free now), one N = 64 product each
        for (int nb = 0; nb < D / 64; ++nb) {
            __syncthreads();
            copy_rows<D>(sA, LD, H + static_cast<size_t>(64 * nb) * D, 64);
            __syncthreads();
            tc_mm_rows<kC, 64, D>(eng, Zw, LD, 1, sA, 1, LD, [&](int i, int j0, const auto &v) {
                float acc = 0.f;
#pragma unroll
                for (int c = 0; c < static_cast<int>(sizeof(v) / sizeof(float)); ++c) {
                    const int jg = 64 * nb + j0 + c;
                    Ud[i * LD + jg] += v[c];
                    acc += Rq[i * LD + jg] * v[c];
                }
                if (i < n) atomicAdd(&gqh[i], acc);
            });
        }
    } else {
        for (int nb = 0; nb < NN; ++nb) {
            __syncthreads();
            copy_rows<D>(sB, LD, H + static_cast<size_t>(RN * nb) * D, RN);
            __syncthreads();
            mm<kC, RN, VT>(Zw, LD, 1, sB, 1, LD, D, [&](int i, int j, float v) {
                const int jg = RN * nb + j;
                Ud[i * LD + jg] += v;
                if (i < n) atomicAdd(&gqh[i], Rq[i * LD + jg] * v);
            });
        }
    }
    __syncthreads();
    copy_rows<D>(Zw, LD, Wg, kC);  // z back from the W slot
    __syncthreads();
    // dlambda_i = -z_i . dqc_i
    row_sums(dls, D, [&](int i, int j) { return Zw[i * LD + j] * Ud[i * LD + j]; });
    __syncthreads();
    GBWD_FOR(i, kC)
        if (i < n && a.dlambda) a.dlambda[tok_row(a, b, r * kC + i, h)] = -dls[i];
    // W = dz / t with dz = -lambda dqc
    GBWD_FOR(idx, kC * D) {
        const int i = idx / D, j = idx % D;
        const float wv = -lam[i] * Ud[i * LD + j] * tinv[i];
        Zw[i * LD + j] = wv;
        Wg[idx] = wv;
    }
    __syncthreads();
    // (W Kbar^T) o causal
    gmm<TC, kC, kC, D>(eng, Zw, LD, 1, Kb, 1, LD, [&](int i, int j, float v) { sB[i * LC + j] = j <= i ? v : 0.f; });
    __syncthreads();
    // cz_i = CumK_i . dz_i = t_i (M . W_i + sum_{j<=i} W_i . kbar_j)
    row_sums(cz, D + kC, [&](int i, int l) {
        return (l < D ? M[l] * Zw[i * LD + l] : (l - D <= i ? sB[i * LC + l - D] : 0.f)) / tinv[i];
    });
    // dqbar = dqc + W S^K + ((W Kbar^T) o causal) Kbar - c CumK cz / t^2 (in place);
    // the chunk's increments DC += W^T Qbar and Dm += sum_i dCum_i,
    // dCum_i = -c (dz_i cq_i + qbar_i cz_i) / t_i^2
    if constexpr (TC)
        tc_mma<kC, D, kC>(eng, sB, LC, 1, Kb, LD, 1, false);
    else
        mm<kC, D, VT>(sB, LC, 1, Kb, LD, 1, kC, [&](int i, int j, float v) { Ud[i * LD + j] += v; });
    for (int hf = 0; hf < NH; ++hf) {
        __syncthreads();
        copy_rows<D>(Rq, LD, SK + static_cast<size_t>(RB * hf) * D, RB);
        __syncthreads();
        if constexpr (TC)
            tc_mma<kC, D, RB>(eng, Zw + RB * hf, LD, 1, Rq, LD, 1, true);
        else
            mm<kC, D, VT>(Zw + RB * hf, LD, 1, Rq, LD, 1, RB, [&](int i, int j, float v) { Ud[i * LD + j] += v; });
    }
    if constexpr (TC) tc_read_elem<kC, D>(eng, [&](int i, int j, float v) { Ud[i * LD + j] += v; });
    __syncthreads();
    {
        float *dC = a.dc + static_cast<size_t>(ch) * D * D;
        GBWD_FOR(w, 4 * D) {
            const int j = w % D, sg = w / D;
            float cum = M[j], acc = 0.f;
            for (int s2 = 0; s2 < sg; ++s2) cum += segs[s2 * D + j];
            for (int i = 16 * sg; i < 16 * sg + 16; ++i) {
                cum += Kb[i * LD + j];
                Ud[i * LD + j] -= c * cum * cz[i] * tinv[i] * tinv[i];
                acc += (Zw[i * LD + j] * cq[i] / tinv[i] + Qb[i * LD + j] * cz[i]) * tinv[i] * tinv[i];
            }
            atomicAdd(&dMs[j], acc);
        }
        if constexpr (TC)
            tc_mm_rows<D, D, kC>(eng, Zw, 1, LD, Qb, LD, 1, [&](int p, int j0, const auto &v) { st_row(dC + p * D + j0, v); });
        else
            mm<D, D, VT>(Zw, 1, LD, Qb, LD, 1, kC, [&](int p, int j, float v) { dC[p * D + j] = v; });
        float *vec = a.vec + static_cast<size_t>(ch) * 4 * kC;
        GBWD_FOR(i, kC) {
            vec[i] = cq[i];
            vec[kC + i] = cz[i];
            vec[2 * kC + i] = gqh[i];
            vec[3 * kC + i] = 0.f;
        }
    }
    __syncthreads();
    row_sums(rdot, D, [&](int i, int j) { return a.l2norm ? Qb[i * LD + j] * Ud[i * LD + j] : 0.f; });
    GBWD_FOR(j, D) a.dm[static_cast<size_t>(ch) * D + j] = -c * dMs[j];
    __syncthreads();
    {
        Tin *dq = static_cast<Tin *>(a.dq);
        GBWD_FOR(idx, kC * D) {
            const int i = idx / D, j = idx % D;
            if (i < n)
                dq[tok_row(a, b, r * kC + i, h) * D + j] = from_f<Tin>((Ud[i * LD + j] - Qb[i * LD + j] * rdot[i]) * rq[i]);
        }
    }
    if constexpr (TC) tc_teardown(eng);
}

// Per sequence and head, chunks last to first: the adjoint dH of the state leaving every
// chunk (stored), then carried into the chunk: dU = P^T D + Kd dH, dR = diag(beta) Tt^T dU,
// dH <- e^{gc_last} dH + (diag(E) Qc)^T D - (diag(E) Kbar)^T dR.  Writes dS0.  Like the
// forward pass, CTA (sequence-head, s) carries the value columns [s DC, (s+1) DC), DC = D / NS.
template <int D, typename Tin, int NS>
__global__ void __launch_bounds__(512) gdn_bwd_dstate_kernel(const GdnBwdArgs a) {
    extern __shared__ float4 gbwd_smem4[];
    constexpr int DC = D / NS, LD = D + 1, LDC = DC + 1, LC = kC + 1;
    constexpr int GN = DC < 16 ? DC : 16, GM = 256 / GN, TMD = D / GM > 0 ? D / GM : 1;
    float *sm = reinterpret_cast<float *>(gbwd_smem4);
    float *dH = sm;                // [D][LDC]
    float *Yb = dH + D * LDC;      // [D][LDC] the chunk's (diag(E) Qc)^T D columns
    float *Kb = Yb + D * LDC;      // [64][LD]
    float *dU = Kb + kC * LD;      // [64][LDC]
    float *dR = dU + kC * LDC;     // [64][LDC] diag(E) dR
    float *Tt = dR + kC * LDC;     // [64][LC]
    float *graw = Tt + kC * LC;    // [64]
    float *gc = graw + kC, *be = gc + kC, *rk = be + kC, *E = rk + kC, *ed = E + kC;

    const int bh = blockIdx.x / NS, c0 = (blockIdx.x % NS) * DC, b = bh / a.H, h = bh % a.H;
    stream8(D * DC, [&](int idx) {
        return a.dST ? a.dST[(static_cast<size_t>(bh) * D + idx / DC) * D + c0 + idx % DC] : 0.f;
    }, [&](int idx, float x) { dH[(idx / DC) * LDC + idx % DC] = x; });
    __syncthreads();
    for (int r = a.NC - 1; r >= 0; --r) {
        const size_t ch = static_cast<size_t>(bh) * a.NC + r;
        float *dhg = a.dh + ch * D * D;
        GBWD_FOR(idx, D * DC) dhg[(idx / DC) * D + c0 + idx % DC] = dH[(idx / DC) * LDC + idx % DC];
        load_tile_ld<D, Tin>(Kb, LD, a.k, a, b, h, r);
        const float *tt = a.tt + ch * kC * kC;
        stream8(kC * kC, [&](int idx) { return tt[idx]; }, [&](int idx, float x) { Tt[(idx / kC) * LC + idx % kC] = x; });
        const float *X1 = a.x1 + ch * kC * D;
        stream8(kC * DC, [&](int idx) { return X1[(idx / DC) * D + c0 + idx % DC]; },
                [&](int idx, float x) { dU[(idx / DC) * LDC + idx % DC] = x; });
        const float *Y1 = a.y1 + ch * D * D;
        stream8(D * DC, [&](int idx) { return Y1[(idx / DC) * D + c0 + idx % DC]; },
                [&](int idx, float x) { Yb[(idx / DC) * LDC + idx % DC] = x; });
        GBWD_FOR(i, kC) {
            const int t = r * kC + i;
            const size_t row = tok_row(a, b, t < a.T ? t : 0, h);
            graw[i] = t < a.T ? a.g[row] : 0.f;
            be[i] = t < a.T ? a.beta[row] : 0.f;
        }
        __syncthreads();
        row_rnorm_ld<D>(Kb, LD, rk, a.l2norm);
        gate_prefix(graw, gc);
        __syncthreads();
        GBWD_FOR(idx, kC * D) Kb[(idx / D) * LD + idx % D] *= rk[idx / D];
        GBWD_FOR(i, kC) {
            E[i] = expf(gc[i]);
            ed[i] = expf(gc[kC - 1] - gc[i]);
        }
        __syncthreads();
        // dU = P^T D + diag(ed) Kbar dH
        tile_mm<kC / GM, DC / GN, GN>(Kb, LD, 1, dH, LDC, 1, D, [&](int i, int j, float v) { dU[i * LDC + j] += ed[i] * v; });
        __syncthreads();
        // diag(E) dR = diag(E beta) Tt^T dU
        tile_mm<kC / GM, DC / GN, GN>(Tt, 1, LC, dU, LDC, 1, kC, [&](int i, int j, float v) {
            dR[i * LDC + j] = E[i] * be[i] * v;
        });
        __syncthreads();
        // dH <- e^{gc_last} dH + (diag(E) Qc)^T D - Kbar^T diag(E) dR
        const float elast = expf(gc[kC - 1]);
        tile_mm<TMD, DC / GN, GN>(Kb, 1, LD, dR, LDC, 1, kC, [&](int p, int j, float v) {
            dH[p * LDC + j] = elast * dH[p * LDC + j] + Yb[p * LDC + j] - v;
        }, D);
        __syncthreads();
    }
    if (a.dS0)
        GBWD_FOR(idx, D * DC)
            a.dS0[(static_cast<size_t>(bh) * D + idx / DC) * D + c0 + idx % DC] = dH[(idx / DC) * LDC + idx % DC];
}

// Exclusive suffix over the chunks of each sequence and head of the CCQ increments:
// dc[r] <- dC_T + sum_{s>r} dc[s], dm[r] <- dm_T + sum_{s>r} dm[s]; the full sums are dC0, dm0.
template <int D>
__global__ void __launch_bounds__(256) gdn_bwd_suffix_kernel(const GdnBwdArgs a) {
    const long long per = static_cast<long long>(D) * D + D;
    const long long gid = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (gid >= per * a.B * a.H) return;
    const int bh = static_cast<int>(gid / per);
    const int e = static_cast<int>(gid % per);
    const bool isC = e < D * D;
    const int em = e - D * D;
    float *base = isC ? a.dc + static_cast<size_t>(bh) * a.NC * D * D + e
                      : a.dm + static_cast<size_t>(bh) * a.NC * D + em;
    const size_t stride = isC ? static_cast<size_t>(D) * D : static_cast<size_t>(D);
    float acc = 0.f;
    if (isC && a.dCT) acc = a.dCT[static_cast<size_t>(bh) * D * D + e];
    if (!isC && a.dmT) acc = a.dmT[static_cast<size_t>(bh) * D + em];
    // eight chunks' loads in flight before their stores
    int r = a.NC - 1;
    for (; r - 7 >= 0; r -= 8) {
        float x[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) x[u] = base[(r - u) * stride];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            base[(r - u) * stride] = acc;
            acc += x[u];
        }
    }
    for (; r >= 0; --r) {
        const float x = base[r * stride];
        base[r * stride] = acc;
        acc += x;
    }
    if (isC && a.dC0) a.dC0[static_cast<size_t>(bh) * D * D + e] = acc;
    if (!isC && a.dm0) a.dm0[static_cast<size_t>(bh) * D + em] = acc;
}

// Per chunk: dv, dk, dbeta, dg from the chunk's forward quantities (gdn_bwd_local_kernel),
// the entering state H_r, the adjoint dH of the leaving state, and DC_{r+1}, Dm_{r+1}.
// Every product runs through gmm (tile_mm on the CUDA cores, or tc_mm on the tensor cores when
// TC) over shared-memory operands; the [64][D] tiles have the odd row stride D + 1 and the
// [64][64] ones 65, and the workspace operands are staged through BF (and, for the D x D ones,
// 64 rows at a time through the S/dP pair).  With TC the kernel reads Tt from the workspace.
template <int D, typename Tin, bool TC = false>
__global__ void __launch_bounds__(kBwdThreads, 1) gdn_bwd_kv_kernel(const GdnBwdArgs a) {
    extern __shared__ float4 gbwd_smem4[];
    constexpr int LD = D + 1, LC = kC + 1, VT = kBwdThreads;
    constexpr int RB = D < 64 ? D : 64, NH = D / RB;  // row blocks of the D x D operands
    float *sm = reinterpret_cast<float *>(gbwd_smem4);
    float *Kb = sm;                // [64][LD] kbar
    float *dU = Kb + kC * LD;      // [64][LD] dU, then the reverse sums of dCum
    float *dR = dU + kC * LD;      // [64][LD] dR, then W
    float *dK = dR + kC * LD;      // [64][LD] dkbar (accumulated)
    float *BF = dK + kC * LD;      // [64][LD] staging: Qc, D, U, R, Qbar, DC + DC^T
    float *sA = BF + kC * LD;      // [64][LC] S, then dTb, then dA, then (Qbar Kbar^T) o causal
    float *sB = sA + kC * LC;      // [64][LC] dP, then M2, then dKK, then (W Kbar^T) o causal
    float *B2 = sA;                // sA and sB together: [64][LD] staging of 64 rows of dH or H
    // [64][LC] Tt (TC: read from the workspace instead, which leaves room for the engine)
    float *Tt = TC ? nullptr : sB + kC * LC;
    float *graw = sB + (TC ? 1 : 2) * kC * LC;
    float *gc = graw + kC, *E = gc + kC, *ed = E + kC, *be = ed + kC, *tinv = be + kC;
    float *rk = tinv + kC, *prs = rk + kC, *pcs = prs + kC, *kd = pcs + kC, *gkh = kd + kC;
    float *rs = gkh + kC, *cs = rs + kC, *db1 = cs + kC, *rdot = db1 + kC, *dgc = rdot + kC;
    float *scal = dgc + kC;        // [4]: <dH, H>
    float *ssk = scal + 4;         // row sums of squares of k
    float *segs = ssk + kC;        // [4][D] segment sums of the reverse cumulative sums below
    TcEng eng{};                   // TC: the tensor-core products' state, behind segs
    if constexpr (TC) tc_setup(eng, reinterpret_cast<uint8_t *>(segs + 4 * D), kv_tc_stage<D>(), kTcBufKv, a.status);

    const int ch = blockIdx.x, r = ch % a.NC, bh = ch / a.NC, b = bh / a.H, h = bh % a.H;
    const int n = min(kC, a.T - r * kC);
    const float c = a.centered ? 1.f : 0.f;
    const size_t t64 = static_cast<size_t>(ch) * kC * D;
    const float *H = a.hs + static_cast<size_t>(ch) * D * D;
    const float *dHg = a.dh + static_cast<size_t>(ch) * D * D;
    const float *DC = a.dc + static_cast<size_t>(ch) * D * D;
    const float *Dm = a.dm + static_cast<size_t>(ch) * D;
    const float *X1 = a.x1 + t64;
    const float *Qbg = a.qb + t64, *Qcg = a.qc + t64, *Ug = a.u + t64, *Rg = a.r + t64, *Wg = a.w + t64;
    const float *vec = a.vec + static_cast<size_t>(ch) * 4 * kC;
    const float *cq = vec, *cz = vec + kC, *gqh = vec + 2 * kC;
    const float *ttg = a.tt + static_cast<size_t>(ch) * kC * kC;
    const float *TtS = TC ? ttg : Tt;  // Tt as the products and the dbeta sums read it
    constexpr int tld = TC ? kC : LC;
    const float t_start = static_cast<float>((a.t0 ? a.t0[b] : 0) + static_cast<int64_t>(r) * kC);

    load_tile_ld<D, Tin>(Kb, LD, a.k, a, b, h, r);
    if constexpr (!TC)
        stream8(kC * kC, [&](int idx) { return ttg[idx]; }, [&](int idx, float x) { Tt[(idx / kC) * LC + idx % kC] = x; });
    GBWD_FOR(i, kC) {
        const int t = r * kC + i;
        const size_t row = tok_row(a, b, t < a.T ? t : 0, h);
        graw[i] = i < n ? a.g[row] : 0.f;
        be[i] = i < n ? a.beta[row] : 0.f;
        tinv[i] = 1.f / (t_start + 1.f + static_cast<float>(i));
        prs[i] = pcs[i] = kd[i] = gkh[i] = rs[i] = cs[i] = db1[i] = rdot[i] = ssk[i] = 0.f;
    }
    if (threadIdx.x == 0) scal[0] = 0.f;
    copy_rows<D>(BF, LD, Qcg, kC);
    __syncthreads();
    row_sums(ssk, D, [&](int i, int l) { return Kb[i * LD + l] * Kb[i * LD + l]; });
    gate_prefix(graw, gc);
    __syncthreads();
    GBWD_FOR(i, kC) {
        E[i] = expf(gc[i]);
        ed[i] = expf(gc[kC - 1] - gc[i]);
        rk[i] = rnorm_of(ssk[i], a.l2norm);
    }
    __syncthreads();
    GBWD_FOR(idx, kC * D) Kb[(idx / D) * LD + idx % D] *= rk[idx / D];
    __syncthreads();
    // dU = P^T D + Kd dH = X1 + diag(ed) Kbar dH, over the row blocks of dH
    for (int hf = 0; hf < NH; ++hf) {
        __syncthreads();
        copy_rows<D>(B2, LD, dHg + static_cast<size_t>(RB * hf) * D, RB);
        __syncthreads();
        if constexpr (TC)
            tc_mma<kC, D, RB>(eng, Kb + RB * hf, LD, 1, B2, LD, 1, hf > 0);
        else
            mm<kC, D, VT>(Kb + RB * hf, LD, 1, B2, LD, 1, RB, [&](int i, int j, float v) {
                dU[i * LD + j] = (hf ? dU[i * LD + j] : 0.f) + v;
            });
    }
    if constexpr (TC) tc_read_elem<kC, D>(eng, [&](int i, int j, float v) { dU[i * LD + j] = v; });
    __syncthreads();
    // S = Qc Kbar^T (Qc in BF; S in the S/dP pair, free once the staging of dH is read)
    gmm<TC, kC, kC, D>(eng, BF, LD, 1, Kb, 1, LD, [&](int i, int j, float v) { sA[i * LC + j] = v; });
    // dU = X1 + diag(ed) t with t = Kbar dH, which also waits in dR for kd
    rows4<D>(X1, D, kC, [&](int i, int j0, float4 x4) {
        const float xs[4] = {x4.x, x4.y, x4.z, x4.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float t = dU[i * LD + j0 + e];
            dR[i * LD + j0 + e] = t;
            dU[i * LD + j0 + e] = xs[e] + ed[i] * t;
        }
    });
    __syncthreads();
    // D (scaled output adjoint) and U for dP
    load_tile_ld<D, Tin>(BF, LD, a.dout, a, b, h, r, a.scale);
    copy_rows<D>(dK, LD, Ug, kC);
    __syncthreads();
    // kd_i = rowsum(Kd o U dH^T)_i = U_i . (dU - P^T D)_i = ed_i U_i . t_i
    row_sums(kd, D, [&](int i, int l) { return ed[i] * dK[i * LD + l] * dR[i * LD + l]; });
    __syncthreads();
    // dv = dR = diag(beta) Tt^T dU;  dP = (D U^T) o Gamma o causal
    {
        Tin *dv = static_cast<Tin *>(a.dv);
        if constexpr (TC) {
            tc_mm_rows<kC, D, kC>(eng, TtS, 1, tld, dU, LD, 1, [&](int i, int j0, const auto &v) {
                constexpr int nv = static_cast<int>(sizeof(v) / sizeof(float));
                float x[nv];
#pragma unroll
                for (int c = 0; c < nv; ++c) {
                    x[c] = be[i] * v[c];
                    dR[i * LD + j0 + c] = x[c];
                }
                if (i < n) st_row_t<Tin>(dv + tok_row(a, b, r * kC + i, h) * D + j0, x);
            });
        } else {
            mm<kC, D, VT>(Tt, 1, LC, dU, LD, 1, kC, [&](int i, int j, float v) {
                const float x = be[i] * v;
                dR[i * LD + j] = x;
                if (i < n) dv[tok_row(a, b, r * kC + i, h) * D + j] = from_f<Tin>(x);
            });
        }
        gmm<TC, kC, kC, D>(eng, BF, LD, 1, dK, 1, LD, [&](int i, int j, float v) {
            sB[i * LC + j] = (j <= i && i < n) ? v * expf(gc[i] - gc[j]) : 0.f;
        });
    }
    __syncthreads();
    // V - R (= diag(E) Kbar H) into BF for gkh;  <dH, H>
    load_tile_ld<D, Tin>(BF, LD, a.v, a, b, h, r);
    __syncthreads();
    rows4<D>(Rg, D, kC, [&](int i, int j0, float4 x4) {
        float *d = BF + i * LD + j0;
        d[0] -= x4.x;
        d[1] -= x4.y;
        d[2] -= x4.z;
        d[3] -= x4.w;
    });
    __syncthreads();
    // row and column sums of dP o S;  gkh_i = (V - R)_i . dR_i
    row_sums(prs, kC, [&](int i, int j) { return sB[i * LC + j] * sA[i * LC + j]; });
    row_sums(pcs, kC, [&](int i, int j) { return sB[j * LC + i] * sA[j * LC + i]; });
    row_sums(gkh, D, [&](int i, int l) { return BF[i * LD + l] * dR[i * LD + l]; });
    __syncthreads();
    // dK = dP^T Qc + diag(ed) U dH^T - diag(E) dR H^T (the last two over row blocks of dH, H)
    copy_rows<D>(BF, LD, Qcg, kC);
    __syncthreads();
    gmm<TC, kC, D, kC>(eng, sB, 1, LC, BF, LD, 1, [&](int i, int j, float v) { dK[i * LD + j] = v; });
    __syncthreads();
    copy_rows<D>(BF, LD, Ug, kC);
    for (int hf = 0; hf < NH; ++hf) {
        __syncthreads();
        copy_rows<D>(B2, LD, dHg + static_cast<size_t>(RB * hf) * D, RB);
        __syncthreads();
        gmm<TC, kC, RB, D>(eng, BF, LD, 1, B2, 1, LD, [&](int i, int j, float v) { dK[i * LD + RB * hf + j] += ed[i] * v; });
        __syncthreads();
        {
            // these rows of H, and their part of <dH, H> (the rows of dH again, from L2)
            constexpr int CPR = D / 4;
            const float *Hb = H + static_cast<size_t>(RB * hf) * D, *dHb = dHg + static_cast<size_t>(RB * hf) * D;
            float part = 0.f;
            stream_u<4>(RB * CPR, [&](int c) {
                int i, cc;
                chunk_rc<CPR>(c, i, cc);
                float4 x[2];
                x[0] = *reinterpret_cast<const float4 *>(Hb + i * D + 4 * cc);
                x[1] = *reinterpret_cast<const float4 *>(dHb + i * D + 4 * cc);
                return Pair4{x[0], x[1]};
            }, [&](int c, Pair4 p) {
                int i, cc;
                chunk_rc<CPR>(c, i, cc);
                float *d = B2 + i * LD + 4 * cc;
                d[0] = p.a.x;
                d[1] = p.a.y;
                d[2] = p.a.z;
                d[3] = p.a.w;
                part += p.a.x * p.b.x + p.a.y * p.b.y + p.a.z * p.b.z + p.a.w * p.b.w;
            });
            atomicAdd(&scal[0], part);
        }
        __syncthreads();
        gmm<TC, kC, RB, D>(eng, dR, LD, 1, B2, 1, LD, [&](int i, int j, float v) { dK[i * LD + RB * hf + j] -= E[i] * v; });
    }
    __syncthreads();
    copy_rows<D>(BF, LD, Rg, kC);
    __syncthreads();
    // dTb = dU R^T
    gmm<TC, kC, kC, D>(eng, dU, LD, 1, BF, 1, LD, [&](int i, int j, float v) { sA[i * LC + j] = v; });
    __syncthreads();
    // dbeta (the Tb = Tt diag(beta) factor) = column sums of dTb o Tt;  M2 = Tt^T (dTb diag(beta))
    row_sums(db1, kC, [&](int j, int i) { return sA[i * LC + j] * TtS[i * tld + j]; });
    gmm<TC, kC, kC, kC>(eng, TtS, 1, tld, sA, LC, 1, [&](int i, int j, float v) { sB[i * LC + j] = v * be[j]; });
    __syncthreads();
    // dA = strict_lower(-M2 Tt^T)
    gmm<TC, kC, kC, kC>(eng, sB, LC, 1, TtS, 1, tld, [&](int i, int j, float v) { sA[i * LC + j] = j < i ? -v : 0.f; });
    __syncthreads();
    // dKK = diag(beta) (dA o Gamma);  rs_i = sum_j dA_ij Gamma_ij KK_ij (the dbeta of A);
    // rowsum(dA o A)_i = beta_i rs_i;  cs_j = colsum(dA o A)_j
    if constexpr (TC) {
        // the terms x of rs and cs wait in dU (free between dTb and the reverse sums below)
        tc_mm<kC, kC, D>(eng, Kb, LD, 1, Kb, 1, LD, [&](int i, int j, float kk) {
            float v = 0.f, x = 0.f;
            if (j < i) {
                const float gm = expf(gc[i] - gc[j]);
                x = sA[i * LC + j] * gm * kk;
                v = sA[i * LC + j] * be[i] * gm;
            }
            sB[i * LC + j] = v;
            dU[i * LD + j] = x;
        });
        row_sums(rs, kC, [&](int i, int j) { return dU[i * LD + j]; });
        row_sums(cs, kC, [&](int j, int i) { return be[i] * dU[i * LD + j]; });
    } else {
        mm<kC, kC, VT>(Kb, LD, 1, Kb, 1, LD, D, [&](int i, int j, float kk) {
            float v = 0.f;
            if (j < i) {
                const float gm = expf(gc[i] - gc[j]);
                const float x = sA[i * LC + j] * gm * kk;
                atomicAdd(&rs[i], x);
                atomicAdd(&cs[j], be[i] * x);
                v = sA[i * LC + j] * be[i] * gm;
            }
            sB[i * LC + j] = v;
        });
    }
    __syncthreads();
    GBWD_FOR(idx, kC * kC) {
        const int i = idx / kC, j = idx % kC;
        sA[i * LC + j] = sB[i * LC + j] + sB[j * LC + i];
    }
    __syncthreads();
    // dK += (dKK + dKK^T) Kbar
    gmm<TC, kC, D, kC>(eng, sA, LC, 1, Kb, LD, 1, [&](int i, int j, float v) { dK[i * LD + j] += v; });
    __syncthreads();
    // CCQ terms: (Qbar Kbar^T) o causal and (W Kbar^T) o causal
    copy_rows<D>(BF, LD, Qbg, kC);
    copy_rows<D>(dR, LD, Wg, kC);
    __syncthreads();
    gmm<TC, kC, kC, D>(eng, BF, LD, 1, Kb, 1, LD, [&](int i, int j, float v) { sA[i * LC + j] = j <= i ? v : 0.f; });
    gmm<TC, kC, kC, D>(eng, dR, LD, 1, Kb, 1, LD, [&](int i, int j, float v) { sB[i * LC + j] = j <= i ? v : 0.f; });
    // reverse cumulative sums G_ij = sum_{l>=i} dCum_lj / (-c), dCum_l = -c (dz_l cq_l + qbar_l cz_l) / t_l^2,
    // dz_l = t_l W_l
    auto dcum = [&](int l, int j) {
        return (dR[l * LD + j] * cq[l] / tinv[l] + BF[l * LD + j] * cz[l]) * tinv[l] * tinv[l];
    };
    GBWD_FOR(w, 4 * D) {  // four 16-row segments: their sums, then the suffix sums within them
        const int j = w % D, sg = w / D;
        float acc = 0.f;
        for (int l = 16 * sg; l < 16 * sg + 16; ++l) acc += dcum(l, j);
        segs[sg * D + j] = acc;
    }
    __syncthreads();
    GBWD_FOR(w, 4 * D) {
        const int j = w % D, sg = w / D;
        float acc = 0.f;
        for (int s2 = sg + 1; s2 < 4; ++s2) acc += segs[s2 * D + j];
        for (int l = 16 * sg + 15; l >= 16 * sg; --l) {
            acc += dcum(l, j);
            dU[l * LD + j] = acc;
        }
    }
    __syncthreads();
    // dK += QKc^T W + WKc^T Qbar + Dm - c G
    if constexpr (TC) {
        tc_mma<kC, D, kC>(eng, sA, 1, LC, dR, LD, 1, false);
        tc_mma<kC, D, kC>(eng, sB, 1, LC, BF, LD, 1, true);
        tc_read_elem<kC, D>(eng, [&](int i, int j, float v) { dK[i * LD + j] += v + Dm[j] - c * dU[i * LD + j]; });
    } else {
        mm<kC, D, VT>(sA, 1, LC, dR, LD, 1, kC, [&](int i, int j, float v) { dK[i * LD + j] += v; });
        mm<kC, D, VT>(sB, 1, LC, BF, LD, 1, kC, [&](int i, int j, float v) {
            dK[i * LD + j] += v + Dm[j] - c * dU[i * LD + j];
        });
    }
    // dK += Kbar (DC + DC^T), over the row blocks p of DC
    for (int hf = 0; hf < NH; ++hf) {
        __syncthreads();
        copy_rows<D>(B2, LD, DC + static_cast<size_t>(RB * hf) * D, RB);
        __syncthreads();
        rows4<RB>(DC + RB * hf, D, D, [&](int j, int p0, float4 x4) {
            B2[p0 * LD + j] += x4.x;
            B2[(p0 + 1) * LD + j] += x4.y;
            B2[(p0 + 2) * LD + j] += x4.z;
            B2[(p0 + 3) * LD + j] += x4.w;
        });
        __syncthreads();
        if constexpr (TC)
            tc_mma<kC, D, RB>(eng, Kb + RB * hf, LD, 1, B2, LD, 1, hf > 0);
        else
            mm<kC, D, VT>(Kb + RB * hf, LD, 1, B2, LD, 1, RB, [&](int i, int j, float v) { dK[i * LD + j] += v; });
    }
    if constexpr (TC) tc_read_elem<kC, D>(eng, [&](int i, int j, float v) { dK[i * LD + j] += v; });
    __syncthreads();
    row_sums(rdot, D, [&](int i, int j) { return a.l2norm ? Kb[i * LD + j] * dK[i * LD + j] : 0.f; });
    GBWD_FOR(i, kC) {
        float x = be[i] * rs[i] - cs[i] + prs[i] - pcs[i] + gqh[i] - kd[i] - gkh[i];
        if (i == n - 1) {
            float sk = 0.f;
            for (int l = 0; l < kC; ++l) sk += kd[l];
            x += expf(gc[kC - 1]) * scal[0] + sk;
        }
        dgc[i] = x;
        if (i < n) a.dbeta[tok_row(a, b, r * kC + i, h)] = db1[i] + rs[i];
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        float acc = 0.f;
        for (int i = n - 1; i >= 0; --i) {
            acc += dgc[i];
            a.dg[tok_row(a, b, r * kC + i, h)] = acc;
        }
    }
    {
        Tin *dk = static_cast<Tin *>(a.dk);
        GBWD_FOR(idx, kC * D) {
            const int i = idx / D, j = idx % D;
            if (i < n)
                dk[tok_row(a, b, r * kC + i, h) * D + j] = from_f<Tin>((dK[i * LD + j] - Kb[i * LD + j] * rdot[i]) * rk[i]);
        }
    }
    if constexpr (TC) tc_teardown(eng);
}

// Shared-memory bytes of each kernel.
template <int D> constexpr size_t prep_smem() { return sizeof(float) * (kC * (D + 1) + 2 * kC * (kC + 1) + 4 * kC); }
template <int D, int NS> constexpr size_t fstate_smem() {
    return sizeof(float) * (D * (D / NS + 1) + kC * (D + 1) + 2 * kC * (D / NS + 1) + kC * (kC + 1) + 6 * kC);
}
template <int D, bool TC = false> constexpr size_t local_smem() {
    return sizeof(float) * (5 * kC * (D + 1) + 2 * kC * (kC + 1) + 15 * kC + 6 * D) +
           (TC ? tc_smem_bytes(local_tc_stage<D>(), kTcBufLocal) : 0);
}
static_assert(local_smem<128, true>() <= 232448, "local kernel shared memory");
template <int D, int NS> constexpr size_t dstate_smem() {
    return sizeof(float) * (2 * D * (D / NS + 1) + kC * (D + 1) + 2 * kC * (D / NS + 1) + kC * (kC + 1) + 6 * kC);
}

// Value-column blocks of the sequential passes: the most (up to 4) that keep the CTAs within
// about two per SM of a 152-SM GPU.
inline int seq_split(int B, int H) {
    int ns = 1;
    while (ns < 4 && static_cast<long long>(B) * H * ns * 2 <= 304) ns *= 2;
    return ns;
}
template <int D, bool TC = false> constexpr size_t kv_smem() {
    return sizeof(float) * (5 * kC * (D + 1) + (TC ? 2 : 3) * kC * (kC + 1) + 17 * kC + 4 + 4 * D) +
           (TC ? tc_smem_bytes(kv_tc_stage<D>(), kTcBufKv) : 0);
}
static_assert(kv_smem<128, true>() <= 232448, "kv kernel shared memory");

}  // namespace gbwd
}  // namespace ccq
