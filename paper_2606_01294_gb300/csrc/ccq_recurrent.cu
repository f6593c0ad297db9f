// ccq_recurrent.cu -- token-by-token CCQ kernel on CUDA cores (fp32 arithmetic).
//
// One CTA per (batch, head) keeps the three recurrent states of Algorithm 2 --
// the backbone state S (stored transposed, [Dk][Dv]), the key second-moment
// sum C [Dk][Dk] and the key sum m [Dk] -- in registers, streams the tokens,
// and writes the states back once.  With T = 1 this is the decode step
// (Algorithm 2, one token, the cache read and written exactly once); with
// T > 1 it is the fp32 forward path.
//
// Per token (Algorithm 2, Eq. clean, Eq. read):
//   qbar, kbar = l2-normalised q, k;   t += 1
//   C += kbar kbar^T;  m += kbar
//   Sigma qbar = C qbar / t - m (m . qbar) / t^2   (second term only when centred)
//   q_clean = qbar - lambda Sigma qbar
//   GLA: S[i][:] = alpha_i S[i][:] + kbar_i v
//   GDN: S[i][:] = alpha (S[i][:] - beta kbar_i (kbar^T S)) + beta kbar_i v
//   o = scale * S^T q_clean
//
// Thread layout (256 threads = 8 warps): warp w owns state rows
// [w*DK/8, (w+1)*DK/8); lane l owns columns [l*DV/32, (l+1)*DV/32) of S and
// [l*DK/32, (l+1)*DK/32) of C, so each row is read with one coalesced
// vector access per warp.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "ccq_internal.h"

namespace ccq {

namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;

template <typename T>
__device__ __forceinline__ float to_f(T x);
template <>
__device__ __forceinline__ float to_f<float>(float x) { return x; }
template <>
__device__ __forceinline__ float to_f<__nv_bfloat16>(__nv_bfloat16 x) { return __bfloat162float(x); }

template <typename T>
__device__ __forceinline__ T from_f(float x);
template <>
__device__ __forceinline__ float from_f<float>(float x) { return x; }
template <>
__device__ __forceinline__ __nv_bfloat16 from_f<__nv_bfloat16>(float x) { return __float2bfloat16_rn(x); }

__device__ __forceinline__ float warp_sum(float x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}

// Load/store N consecutive floats (N in {1, 2, 4}) with one vector access.
template <int N>
__device__ __forceinline__ void ldv(const float *p, float (&r)[N]) {
    if constexpr (N == 4) {
        float4 x = *reinterpret_cast<const float4 *>(p);
        r[0] = x.x; r[1] = x.y; r[2] = x.z; r[3] = x.w;
    } else if constexpr (N == 2) {
        float2 x = *reinterpret_cast<const float2 *>(p);
        r[0] = x.x; r[1] = x.y;
    } else {
        r[0] = *p;
    }
}
template <int N>
__device__ __forceinline__ void stv(float *p, const float (&r)[N]) {
    if constexpr (N == 4) {
        *reinterpret_cast<float4 *>(p) = make_float4(r[0], r[1], r[2], r[3]);
    } else if constexpr (N == 2) {
        *reinterpret_cast<float2 *>(p) = make_float2(r[0], r[1]);
    } else {
        *p = r[0];
    }
}

template <int DK, int DV, int BACKBONE, typename IT, typename GT>
__global__ void __launch_bounds__(kThreads, 1)
recurrent_kernel(RecurrentArgs a) {
    constexpr int RS = DK / kWarps;  // state rows per warp
    constexpr int CS = DV / 32;      // S columns per lane
    constexpr int CK = DK / 32;      // C columns per lane

    __shared__ float qs[DK], ks[DK], vs[DV], gs[DK], qcs[DK], ms[DK];
    __shared__ float red0[kWarps][DV], red1[kWarps][DV];
    __shared__ float scal[8];  // 0 rq, 1 rk, 2 lambda, 3 alpha, 4 beta, 5 m.q, 6 qc.k

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int bh = blockIdx.x, b = bh / a.H, h = bh % a.H;
    const size_t sbase = static_cast<size_t>(bh);

    // ---- load the states once (registers), zero when no initial state
    float S[RS][CS], C[RS][CK];
#pragma unroll
    for (int rr = 0; rr < RS; ++rr) {
        const int r = warp * RS + rr;
        if (a.S0) {
            ldv<CS>(a.S0 + (sbase * DK + r) * DV + lane * CS, S[rr]);
        } else {
#pragma unroll
            for (int c = 0; c < CS; ++c) S[rr][c] = 0.f;
        }
        if (a.C0) {
            ldv<CK>(a.C0 + (sbase * DK + r) * DK + lane * CK, C[rr]);
        } else {
#pragma unroll
            for (int c = 0; c < CK; ++c) C[rr][c] = 0.f;
        }
    }
    if (tid < DK) ms[tid] = a.m0 ? a.m0[sbase * DK + tid] : 0.f;
    int64_t t = a.t0 ? a.t0[b] : 0;
    const float scale = a.scale;

    const IT *q = static_cast<const IT *>(a.q);
    const IT *k = static_cast<const IT *>(a.k);
    const IT *v = static_cast<const IT *>(a.v);
    IT *o = static_cast<IT *>(a.o);

    for (int tl = 0; tl < a.T; ++tl) {
        const size_t row = (static_cast<size_t>(b) * a.T + tl) * a.H + h;
        // ---- inputs of this token
        if (tid < DK) {
            qs[tid] = to_f(q[row * DK + tid]);
            ks[tid] = to_f(k[row * DK + tid]);
            if (BACKBONE == 0) gs[tid] = __expf(to_f(static_cast<const GT *>(a.gate)[row * DK + tid]));
        }
        if (tid < DV) vs[tid] = to_f(v[row * DV + tid]);
        if (tid == 0) {
            scal[2] = a.lambda[row];
            if (BACKBONE == 1) {
                scal[3] = __expf(static_cast<const float *>(a.gate)[row]);
                scal[4] = a.beta[row];
            }
        }
        __syncthreads();
        // ---- l2 norms (Algorithms 1, 2)
        if (warp < 2) {
            const float *x = warp == 0 ? qs : ks;
            float s = 0.f;
#pragma unroll
            for (int c = 0; c < CK; ++c) s += x[lane * CK + c] * x[lane * CK + c];
            s = warp_sum(s);
            if (lane == 0) scal[warp] = a.l2norm ? rsqrtf(fmaxf(s, 1e-12f)) : 1.f;
        }
        __syncthreads();
        if (tid < DK) {
            qs[tid] *= scal[0];
            ks[tid] *= scal[1];
            ms[tid] += ks[tid];  // m_t = m_{t-1} + kbar_t
        }
        t += 1;
        __syncthreads();
        // ---- C_t = C_{t-1} + kbar kbar^T and the row sums of C_t qbar
        float kc[CK], qv[CK];
#pragma unroll
        for (int c = 0; c < CK; ++c) {
            kc[c] = ks[lane * CK + c];
            qv[c] = qs[lane * CK + c];
        }
        if (warp == 0) {
            // m . qbar and (later) q_clean . kbar
            float s = 0.f;
#pragma unroll
            for (int c = 0; c < CK; ++c) s += ms[lane * CK + c] * qv[c];
            s = warp_sum(s);
            if (lane == 0) scal[5] = s;
        }
        float cq[RS];
#pragma unroll
        for (int rr = 0; rr < RS; ++rr) {
            const float kr = ks[warp * RS + rr];
            float s = 0.f;
#pragma unroll
            for (int c = 0; c < CK; ++c) {
                C[rr][c] = fmaf(kr, kc[c], C[rr][c]);
                s = fmaf(C[rr][c], qv[c], s);
            }
            cq[rr] = warp_sum(s);
        }
        __syncthreads();
        // ---- Eq. clean: q_clean = qbar - lambda (C qbar / t - m (m.qbar) / t^2)
        {
            const float tf = static_cast<float>(t);
            const float inv_t = 1.f / tf;
            const float mq = scal[5], lam = scal[2];
            if (lane < RS) {
                float cqv = 0.f;
#pragma unroll
                for (int rr = 0; rr < RS; ++rr)
                    if (rr == lane) cqv = cq[rr];
                const int r = warp * RS + lane;
                float sig = cqv * inv_t;
                if (a.centered) sig -= ms[r] * mq * inv_t * inv_t;
                qcs[r] = qs[r] - lam * sig;
            }
        }
        __syncthreads();
        if (BACKBONE == 1 && warp == 0) {
            float s = 0.f;
#pragma unroll
            for (int c = 0; c < CK; ++c) s += qcs[lane * CK + c] * kc[c];
            s = warp_sum(s);
            if (lane == 0) scal[6] = s;
        }
        // ---- backbone write and read
        float vv[CS];
#pragma unroll
        for (int c = 0; c < CS; ++c) vv[c] = vs[lane * CS + c];
        if (BACKBONE == 0) {
            float po[CS];
#pragma unroll
            for (int c = 0; c < CS; ++c) po[c] = 0.f;
#pragma unroll
            for (int rr = 0; rr < RS; ++rr) {
                const int r = warp * RS + rr;
                const float al = gs[r], kr = ks[r], qr = qcs[r];
#pragma unroll
                for (int c = 0; c < CS; ++c) {
                    S[rr][c] = fmaf(al, S[rr][c], kr * vv[c]);
                    po[c] = fmaf(S[rr][c], qr, po[c]);
                }
            }
#pragma unroll
            for (int c = 0; c < CS; ++c) red0[warp][lane * CS + c] = po[c];
            __syncthreads();
            if (tid < DV) {
                float s = 0.f;
#pragma unroll
                for (int w = 0; w < kWarps; ++w) s += red0[w][tid];
                o[row * DV + tid] = from_f<IT>(scale * s);
            }
        } else {
            float pk[CS], pq[CS];
#pragma unroll
            for (int c = 0; c < CS; ++c) pk[c] = pq[c] = 0.f;
#pragma unroll
            for (int rr = 0; rr < RS; ++rr) {
                const int r = warp * RS + rr;
                const float kr = ks[r], qr = qcs[r];
#pragma unroll
                for (int c = 0; c < CS; ++c) {
                    pk[c] = fmaf(kr, S[rr][c], pk[c]);
                    pq[c] = fmaf(qr, S[rr][c], pq[c]);
                }
            }
#pragma unroll
            for (int c = 0; c < CS; ++c) {
                red0[warp][lane * CS + c] = pk[c];
                red1[warp][lane * CS + c] = pq[c];
            }
            __syncthreads();
            if (tid < DV) {
                float sk = 0.f, sq = 0.f;
#pragma unroll
                for (int w = 0; w < kWarps; ++w) {
                    sk += red0[w][tid];
                    sq += red1[w][tid];
                }
                red0[0][tid] = sk;  // kbar^T S (old state)
                const float al = scal[3], be = scal[4], qk = scal[6];
                // o = S_new^T q_clean expanded in the old state
                o[row * DV + tid] =
                    from_f<IT>(scale * (al * sq - al * be * qk * sk + be * qk * vs[tid]));
            }
            __syncthreads();
            const float al = scal[3], be = scal[4];
            float ksv[CS];
#pragma unroll
            for (int c = 0; c < CS; ++c) ksv[c] = red0[0][lane * CS + c];
#pragma unroll
            for (int rr = 0; rr < RS; ++rr) {
                const float kr = ks[warp * RS + rr];
#pragma unroll
                for (int c = 0; c < CS; ++c)
                    S[rr][c] = al * (S[rr][c] - be * kr * ksv[c]) + be * kr * vv[c];
            }
        }
        __syncthreads();
    }

    // ---- final states
#pragma unroll
    for (int rr = 0; rr < RS; ++rr) {
        const int r = warp * RS + rr;
        if (a.ST) stv<CS>(a.ST + (sbase * DK + r) * DV + lane * CS, S[rr]);
        if (a.CT) stv<CK>(a.CT + (sbase * DK + r) * DK + lane * CK, C[rr]);
    }
    if (a.mT && tid < DK) a.mT[sbase * DK + tid] = ms[tid];
}

// The decode step (T = 1) as a streaming pass: the cache of one (batch, head)
// is read and written once, C first (rank-one update, row dots C qbar, stored
// back at once), then S (update, read with q_clean, stored back), so only one
// of the two 64 KB states is live in registers at a time.  At about half the
// registers of recurrent_kernel two CTAs share an SM and one CTA's loads overlap
// the other's arithmetic and stores.  Same arithmetic as recurrent_kernel with
// T = 1 (Algorithm 2, Eq. clean, Eq. read).
template <int DK, int DV, int BACKBONE, typename IT, typename GT>
__global__ void __launch_bounds__(kThreads, 2)
decode_kernel(RecurrentArgs a) {
    constexpr int RS = DK / kWarps;  // state rows per warp
    constexpr int CS = DV / 32;      // S columns per lane
    constexpr int CK = DK / 32;      // C columns per lane

    __shared__ float qs[DK], ks[DK], vs[DV], gs[DK], qcs[DK], ms[DK], cqs[DK];
    __shared__ float red0[kWarps][DV], red1[kWarps][DV];
    __shared__ float scal[8];  // 0 rq, 1 rk, 2 lambda, 3 alpha, 4 beta, 5 m.q, 6 qc.k

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int bh = blockIdx.x, b = bh / a.H, h = bh % a.H;
    const size_t sbase = static_cast<size_t>(bh);
    const size_t row = static_cast<size_t>(b) * a.H + h;  // T = 1

    // ---- C rows first: their loads are in flight while the token is prepared
    float C[RS][CK];
#pragma unroll
    for (int rr = 0; rr < RS; ++rr) {
        const int r = warp * RS + rr;
        if (a.C0) ldv<CK>(a.C0 + (sbase * DK + r) * DK + lane * CK, C[rr]);
        else
#pragma unroll
            for (int c = 0; c < CK; ++c) C[rr][c] = 0.f;
    }
    const IT *q = static_cast<const IT *>(a.q);
    const IT *k = static_cast<const IT *>(a.k);
    const IT *v = static_cast<const IT *>(a.v);
    IT *o = static_cast<IT *>(a.o);
    if (tid < DK) {
        qs[tid] = to_f(q[row * DK + tid]);
        ks[tid] = to_f(k[row * DK + tid]);
        if (BACKBONE == 0) gs[tid] = __expf(to_f(static_cast<const GT *>(a.gate)[row * DK + tid]));
        ms[tid] = a.m0 ? a.m0[sbase * DK + tid] : 0.f;
    }
    if (tid < DV) vs[tid] = to_f(v[row * DV + tid]);
    if (tid == 0) {
        scal[2] = a.lambda[row];
        if (BACKBONE == 1) {
            scal[3] = __expf(static_cast<const float *>(a.gate)[row]);
            scal[4] = a.beta[row];
        }
    }
    const int64_t t = (a.t0 ? a.t0[b] : 0) + 1;
    __syncthreads();
    if (warp < 2) {
        const float *x = warp == 0 ? qs : ks;
        float s = 0.f;
#pragma unroll
        for (int c = 0; c < CK; ++c) s += x[lane * CK + c] * x[lane * CK + c];
        s = warp_sum(s);
        if (lane == 0) scal[warp] = a.l2norm ? rsqrtf(fmaxf(s, 1e-12f)) : 1.f;
    }
    __syncthreads();
    if (tid < DK) {
        qs[tid] *= scal[0];
        ks[tid] *= scal[1];
        ms[tid] += ks[tid];  // m_t = m_{t-1} + kbar_t
    }
    __syncthreads();
    // ---- C_t = C_{t-1} + kbar kbar^T, its row dots with qbar, and C_t written back
    float kc[CK], qv[CK];
#pragma unroll
    for (int c = 0; c < CK; ++c) {
        kc[c] = ks[lane * CK + c];
        qv[c] = qs[lane * CK + c];
    }
    if (warp == 0) {
        float s = 0.f;
#pragma unroll
        for (int c = 0; c < CK; ++c) s += ms[lane * CK + c] * qv[c];
        s = warp_sum(s);
        if (lane == 0) scal[5] = s;
    }
#pragma unroll
    for (int rr = 0; rr < RS; ++rr) {
        const int r = warp * RS + rr;
        const float kr = ks[r];
        float s = 0.f;
#pragma unroll
        for (int c = 0; c < CK; ++c) {
            C[rr][c] = fmaf(kr, kc[c], C[rr][c]);
            s = fmaf(C[rr][c], qv[c], s);
        }
        if (a.CT) stv<CK>(a.CT + (sbase * DK + r) * DK + lane * CK, C[rr]);
        s = warp_sum(s);
        if (lane == 0) cqs[r] = s;
    }
    // ---- S rows: loads issued before q_clean is formed
    float S[RS][CS];
#pragma unroll
    for (int rr = 0; rr < RS; ++rr) {
        const int r = warp * RS + rr;
        if (a.S0) ldv<CS>(a.S0 + (sbase * DK + r) * DV + lane * CS, S[rr]);
        else
#pragma unroll
            for (int c = 0; c < CS; ++c) S[rr][c] = 0.f;
    }
    __syncthreads();
    // ---- Eq. clean: q_clean = qbar - lambda (C qbar / t - m (m.qbar) / t^2)
    if (tid < DK) {
        const float inv_t = 1.f / static_cast<float>(t);
        float sig = cqs[tid] * inv_t;
        if (a.centered) sig -= ms[tid] * scal[5] * inv_t * inv_t;
        qcs[tid] = qs[tid] - scal[2] * sig;
    }
    __syncthreads();
    if (BACKBONE == 1 && warp == 0) {
        float s = 0.f;
#pragma unroll
        for (int c = 0; c < CK; ++c) s += qcs[lane * CK + c] * kc[c];
        s = warp_sum(s);
        if (lane == 0) scal[6] = s;
    }
    float vv[CS];
#pragma unroll
    for (int c = 0; c < CS; ++c) vv[c] = vs[lane * CS + c];
    if (BACKBONE == 0) {
        float po[CS];
#pragma unroll
        for (int c = 0; c < CS; ++c) po[c] = 0.f;
#pragma unroll
        for (int rr = 0; rr < RS; ++rr) {
            const int r = warp * RS + rr;
            const float al = gs[r], kr = ks[r], qr = qcs[r];
#pragma unroll
            for (int c = 0; c < CS; ++c) {
                S[rr][c] = fmaf(al, S[rr][c], kr * vv[c]);
                po[c] = fmaf(S[rr][c], qr, po[c]);
            }
            if (a.ST) stv<CS>(a.ST + (sbase * DK + r) * DV + lane * CS, S[rr]);
        }
#pragma unroll
        for (int c = 0; c < CS; ++c) red0[warp][lane * CS + c] = po[c];
        __syncthreads();
        if (tid < DV) {
            float s = 0.f;
#pragma unroll
            for (int w = 0; w < kWarps; ++w) s += red0[w][tid];
            o[row * DV + tid] = from_f<IT>(a.scale * s);
        }
    } else {
        float pk[CS], pq[CS];
#pragma unroll
        for (int c = 0; c < CS; ++c) pk[c] = pq[c] = 0.f;
#pragma unroll
        for (int rr = 0; rr < RS; ++rr) {
            const int r = warp * RS + rr;
            const float kr = ks[r], qr = qcs[r];
#pragma unroll
            for (int c = 0; c < CS; ++c) {
                pk[c] = fmaf(kr, S[rr][c], pk[c]);
                pq[c] = fmaf(qr, S[rr][c], pq[c]);
            }
        }
#pragma unroll
        for (int c = 0; c < CS; ++c) {
            red0[warp][lane * CS + c] = pk[c];
            red1[warp][lane * CS + c] = pq[c];
        }
        __syncthreads();
        if (tid < DV) {
            float sk = 0.f, sq = 0.f;
#pragma unroll
            for (int w = 0; w < kWarps; ++w) {
                sk += red0[w][tid];
                sq += red1[w][tid];
            }
            red0[0][tid] = sk;  // kbar^T S (old state)
            const float al = scal[3], be = scal[4], qk = scal[6];
            o[row * DV + tid] = from_f<IT>(a.scale * (al * sq - al * be * qk * sk + be * qk * vs[tid]));
        }
        __syncthreads();
        const float al = scal[3], be = scal[4];
        float ksv[CS];
#pragma unroll
        for (int c = 0; c < CS; ++c) ksv[c] = red0[0][lane * CS + c];
#pragma unroll
        for (int rr = 0; rr < RS; ++rr) {
            const int r = warp * RS + rr;
            const float kr = ks[r];
#pragma unroll
            for (int c = 0; c < CS; ++c) S[rr][c] = al * (S[rr][c] - be * kr * ksv[c]) + be * kr * vv[c];
            if (a.ST) stv<CS>(a.ST + (sbase * DK + r) * DV + lane * CS, S[rr]);
        }
    }
    if (a.mT && tid < DK) a.mT[sbase * DK + tid] = ms[tid];
}

template <int DK, int DV, int BB, typename IT>
cudaError_t launch_gate(const RecurrentArgs &a, cudaStream_t s) {
    const bool gbf = BB == 0 && a.gate_dtype == 0;
    if (a.T == 1) {
        if (gbf) decode_kernel<DK, DV, BB, IT, __nv_bfloat16><<<a.B * a.H, kThreads, 0, s>>>(a);
        else decode_kernel<DK, DV, BB, IT, float><<<a.B * a.H, kThreads, 0, s>>>(a);
        return cudaGetLastError();
    }
    if (gbf)
        recurrent_kernel<DK, DV, BB, IT, __nv_bfloat16><<<a.B * a.H, kThreads, 0, s>>>(a);
    else
        recurrent_kernel<DK, DV, BB, IT, float><<<a.B * a.H, kThreads, 0, s>>>(a);
    return cudaGetLastError();
}

template <int DK, int DV, int BB>
cudaError_t launch_in(const RecurrentArgs &a, cudaStream_t s) {
    if (a.in_dtype == 0) return launch_gate<DK, DV, BB, __nv_bfloat16>(a, s);
    return launch_gate<DK, DV, BB, float>(a, s);
}

template <int DK, int DV>
cudaError_t launch_bb(const RecurrentArgs &a, cudaStream_t s) {
    if (a.backbone == 0) return launch_in<DK, DV, 0>(a, s);
    return launch_in<DK, DV, 1>(a, s);
}

__global__ void t_update_kernel(const int64_t *t0, int64_t *tT, int B, int T) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i < B) tT[i] = (t0 ? t0[i] : 0) + T;
}

__global__ void t_update_varlen_kernel(const int64_t *t0, int64_t *tT, const int64_t *cu, int n) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i < n) tT[i] = (t0 ? t0[i] : 0) + (cu[i + 1] - cu[i]);
}

}  // namespace

cudaError_t launch_t_update(const int64_t *t0, int64_t *tT, int B, int T, cudaStream_t s) {
    if (!tT || B == 0) return cudaSuccess;
    t_update_kernel<<<(B + 255) / 256, 256, 0, s>>>(t0, tT, B, T);
    return cudaGetLastError();
}

cudaError_t launch_t_update_varlen(const int64_t *t0, int64_t *tT, const int64_t *cu, int num_seqs,
                                   cudaStream_t s) {
    if (!tT || num_seqs == 0) return cudaSuccess;
    t_update_varlen_kernel<<<(num_seqs + 255) / 256, 256, 0, s>>>(t0, tT, cu, num_seqs);
    return cudaGetLastError();
}

cudaError_t launch_recurrent(const RecurrentArgs &a, cudaStream_t s) {
    if (a.B * a.H == 0) return cudaSuccess;
    if (a.Dk == 128 && a.Dv == 128) return launch_bb<128, 128>(a, s);
    if (a.Dk == 64 && a.Dv == 64) return launch_bb<64, 64>(a, s);
    return cudaErrorInvalidValue;
}

}  // namespace ccq
