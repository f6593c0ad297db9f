// ccq_gla_segment.cu -- sequence-segment parallelism for long CCQ-GLA sequences.
//
// With few (batch, head) sequences (B*H well below the SM count), each sequence
// is cut into `nseg` segments of whole chunks.  Every recurrent state of the
// layer composes across a segment boundary in closed form:
//   GLA state   S_out = Diag(D) S_in + dS,     D = e^{sum of the segment's log gates}
//   second moment  C_out = C_in + dC,  key sum  m_out = m_in + dm  (undecayed, App. B)
// so three launches replace one long sequential walk:
//   1. gla_segment_state_kernel: per segment, from a zero state, the deltas
//      (dS, dC, dm, D) -- no read, no output.  Chunks are visited last to first so
//      each chunk's write is scaled by the decay of the chunks after it and
//      accumulates straight into TMEM: dS = sum_r (kbar e^{Gtot_r - G} * Dsuf_r)^T V.
//   2. gla_segment_combine_kernel: per sequence, an exclusive scan over its
//      segments that replaces each delta with that segment's initial state.
//   3. gla_chunk_kernel with one CTA per (sequence, segment), started from those
//      states (ccq_gla_chunk.cu).
// Workspace per (sequence, segment): S [128][128], C [128][128], m [128], D [128] fp32.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "ccq_internal.h"
#include "sm100_ptx.cuh"

namespace ccq {

namespace {

constexpr int kC = 64;
constexpr int kD = 128;
constexpr int kThreads = 256;
constexpr float kLog2e = 1.4426950408889634f;

// shared memory: two slots of {k 16K, v 16K, gates 32K, Ku 16K}
constexpr uint32_t SL_BYTES = 81920;
constexpr uint32_t SL_K = 0, SL_V = 16384, SL_G = 32768, SL_KU = 65536;
constexpr uint32_t OFF_MISC = 2 * SL_BYTES;  // 163840
constexpr uint32_t M_DSUF = 0;     // [128] decay of the chunks already visited (later ones)
constexpr uint32_t M_MSUM = 512;   // [128] key sum
constexpr uint32_t M_GP = 1024;    // [4][128] gate sums of the four token quarters
constexpr uint32_t M_DM = 3072;    // [4][128] key sums of the four token quarters
constexpr uint32_t M_RK = 5120;    // [64]
constexpr uint32_t M_BAR = 5376;   // 4 mbarriers: in[2], mma[2]
constexpr uint32_t M_TMEM = 5408, M_ABORT = 5412;
constexpr uint32_t kSmem = OFF_MISC + 6144 + 1024;
static_assert(kSmem <= 232448, "smem");

__global__ void __launch_bounds__(kThreads, 1)
gla_segment_state_kernel(const __grid_constant__ CUtensorMap map_k, const __grid_constant__ CUtensorMap map_v,
                         const __grid_constant__ CUtensorMap map_g, const ChunkArgs a) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = smem_align1024(smem_raw);
    const uint32_t sb = smem_addr(sm);
    uint8_t *misc = sm + OFF_MISC;
    float *dsuf = reinterpret_cast<float *>(misc + M_DSUF);
    float *msum = reinterpret_cast<float *>(misc + M_MSUM);
    float *gp = reinterpret_cast<float *>(misc + M_GP);
    float *dm = reinterpret_cast<float *>(misc + M_DM);
    float *rk = reinterpret_cast<float *>(misc + M_RK);
    uint64_t *bar = reinterpret_cast<uint64_t *>(misc + M_BAR);
    uint32_t *tslot = reinterpret_cast<uint32_t *>(misc + M_TMEM);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(misc + M_ABORT);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int seq = blockIdx.x / a.nseg, seg = blockIdx.x % a.nseg;
    const int b = seq / a.H, h = seq % a.H;
    const int NCt = (a.T + kC - 1) / kC;
    const int cb = seg * a.seg_chunks, ce = min(NCt, cb + a.seg_chunks);
    const int n = ce - cb;  // chunks of this segment (>= 1)
    const bool gate_f32 = a.gate_dtype != 0;
    const uint32_t g_bytes = gate_f32 ? kC * kD * 4 : kC * kD * 2;
    int *status = a.status;

    if (tid == 0) {
        for (int i = 0; i < 4; ++i) mbar_init(&bar[i], 1);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 0) tmem_alloc(tslot, 256);
    if (tid < kD) {
        dsuf[tid] = 1.f;
        msum[tid] = 0.f;
    }
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *tslot;
    // visit chunks last to first: local step i handles global chunk ce - 1 - i
    auto issue = [&](int i) {
        const int s = i & 1, cg = ce - 1 - i;
        uint8_t *base = sm + s * SL_BYTES;
        mbar_arrive_expect_tx(&bar[s], 4 * 8192 + g_bytes);
        tma_load_4d(base + SL_K, &map_k, &bar[s], 0, h, cg * kC, b);
        tma_load_4d(base + SL_K + 8192, &map_k, &bar[s], 64, h, cg * kC, b);
        tma_load_4d(base + SL_V, &map_v, &bar[s], 0, h, cg * kC, b);
        tma_load_4d(base + SL_V + 8192, &map_v, &bar[s], 64, h, cg * kC, b);
        tma_load_4d(base + SL_G, &map_g, &bar[s], 0, h, cg * kC, b);
    };
    if (tid == 0) issue(0);
    if (tid == 0 && n > 1) issue(1);
    for (int i = 0; i < n; ++i) {
        const int s = i & 1;
        const uint32_t par = (i >> 1) & 1;
        uint8_t *slot = sm + s * SL_BYTES;
        // refill the other slot with chunk step i + 1 once the products of step i - 1 (which
        // read it) are done; they ran under that step's tail, so this rarely waits
        if (tid == 0 && i >= 1 && i + 1 < n && !*abort_flag) {
            mbar_wait(&bar[2 + (s ^ 1)], ((i - 1) >> 1) & 1, abort_flag, status);
            issue(i + 1);
        }
        mbar_wait(&bar[s], par, abort_flag, status);
        // k row norms: two threads per row (one T64 tile each), eight partial sums in pairs
        if (tid < 128) {
            const int j = tid >> 1, hh = tid & 1;
            uint64_t s0 = 0, s1 = 0;
#pragma unroll
            for (int cc = 0; cc < 8; ++cc) {
                const uint4 v = *reinterpret_cast<const uint4 *>(slot + SL_K + hh * 8192 + t64_chunk(j, cc));
                const uint64_t p0 = f2_from_bf16x2(v.x), p1 = f2_from_bf16x2(v.y), p2 = f2_from_bf16x2(v.z),
                               p3 = f2_from_bf16x2(v.w);
                s0 = f2_fma(p0, p0, s0); s1 = f2_fma(p1, p1, s1);
                s0 = f2_fma(p2, p2, s0); s1 = f2_fma(p3, p3, s1);
            }
            const float2 sv = f2_split(f2_add(s0, s1));
            float ss = sv.x + sv.y;
            ss += __shfl_xor_sync(0xffffffffu, ss, 1);
            if (hh == 0) rk[j] = a.l2norm ? rsqrtf(fmaxf(ss, 1e-12f)) : 1.f;
        }
        // thread = (key-dim pair (d0, d0 + 1), token quarter): gate prefix over its 16 tokens
        const int p = tid & 63, qq = tid >> 6, d0 = 2 * p;
        uint64_t gl[16];
        {
            uint64_t run = 0;
#pragma unroll
            for (int u = 0; u < 16; ++u) {
                const int j = 16 * qq + u;
                uint64_t g2;
                if (gate_f32) {
                    const float2 f = *reinterpret_cast<const float2 *>(slot + SL_G + (j * kD + d0) * 4);
                    g2 = f2_make(f.x, f.y);
                } else {
                    g2 = f2_from_bf16x2(*reinterpret_cast<const uint32_t *>(slot + SL_G + (j * kD + d0) * 2));
                }
                run = f2_add(run, g2);
                gl[u] = run;
            }
            const float2 rv = f2_split(run);
            gp[qq * kD + d0] = rv.x;
            gp[qq * kD + d0 + 1] = rv.y;
        }
        __syncthreads();
        {
            // Ku_j = kbar_j Dsuf e^{Gtot - G_j}: the exponent is (Gtot - quarter offset) - prefix
            float offx = 0.f, offy = 0.f, totx = 0.f, toty = 0.f;
#pragma unroll
            for (int q2 = 0; q2 < 4; ++q2) {
                const float gx = gp[q2 * kD + d0], gy = gp[q2 * kD + d0 + 1];
                totx += gx; toty += gy;
                if (q2 < qq) { offx += gx; offy += gy; }
            }
            const uint64_t base2 = f2_make(totx - offx, toty - offy);
            const uint64_t l2 = f2_make(kLog2e, kLog2e);
            const uint64_t ds2 = f2_make(dsuf[d0], dsuf[d0 + 1]);
            const uint32_t tcol = (d0 >> 6) * 8192;
            uint32_t kraw[16];
            float rkv[16];
#pragma unroll
            for (int u = 0; u < 16; ++u) kraw[u] = *reinterpret_cast<const uint32_t *>(slot + SL_K + tcol + t64_offset(16 * qq + u, d0 & 63));
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const float4 r4 = *reinterpret_cast<const float4 *>(rk + 16 * qq + 4 * u);
                rkv[4 * u] = r4.x; rkv[4 * u + 1] = r4.y; rkv[4 * u + 2] = r4.z; rkv[4 * u + 3] = r4.w;
            }
            uint64_t dm2 = 0;
#pragma unroll
            for (int u = 0; u < 16; ++u) {
                const uint32_t o = tcol + t64_offset(16 * qq + u, d0 & 63);
                const uint64_t kb2 = f2_mul(f2_from_bf16x2(kraw[u]), f2_make(rkv[u], rkv[u]));
                const float2 x = f2_split(f2_mul(f2_add(base2, f2_make(-f2_split(gl[u]).x, -f2_split(gl[u]).y)), l2));
                const uint64_t ku2 = f2_mul(f2_mul(kb2, ds2), f2_make(fast_exp2(x.x), fast_exp2(x.y)));
                *reinterpret_cast<uint32_t *>(slot + SL_K + o) = bf16x2_from_f2(kb2);
                *reinterpret_cast<uint32_t *>(slot + SL_KU + o) = bf16x2_from_f2(ku2);
                dm2 = f2_add(dm2, kb2);
            }
            const float2 dv = f2_split(dm2);
            dm[qq * kD + d0] = dv.x;
            dm[qq * kD + d0 + 1] = dv.y;
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        if (tid == 0 && !*abort_flag) {
            tc_fence_after();
            const uint32_t ss = sb + s * SL_BYTES;
            const uint64_t dku = make_desc(ss + SL_KU, 8192, 1024);
            const uint64_t dv = make_desc(ss + SL_V, 8192, 1024);
            const uint64_t dk = make_desc(ss + SL_K, 8192, 1024);
            const uint32_t id = make_idesc(128, 128, 1, 1);
            for (int k = 0; k < 4; ++k) mma_bf16(tbase, dku + k * 128, dv + k * 128, id, (i | k) != 0);
            for (int k = 0; k < 4; ++k) mma_bf16(tbase + 128, dk + k * 128, dk + k * 128, id, (i | k) != 0);
            mma_commit(&bar[2 + s]);
        }
        if (tid < kD) {
            dsuf[tid] *= fast_exp2(((gp[tid] + gp[kD + tid]) + (gp[2 * kD + tid] + gp[3 * kD + tid])) * kLog2e);
            msum[tid] += (dm[tid] + dm[kD + tid]) + (dm[2 * kD + tid] + dm[3 * kD + tid]);
        }
        __syncthreads();
    }
    // wait for the last products of both slots
    if (n >= 1) mbar_wait(&bar[2 + ((n - 1) & 1)], ((n - 1) >> 1) & 1, abort_flag, status);
    if (n >= 2) mbar_wait(&bar[2 + ((n - 2) & 1)], ((n - 2) >> 1) & 1, abort_flag, status);
    tc_fence_after();
    float *out = a.seg_ws + static_cast<size_t>(blockIdx.x) * kSegFloats;
    {
        const int lq = warp & 3, ch = warp >> 2;  // 8 warps: lane quadrant, column half
        const int row = 32 * lq + lane;
        const uint32_t tl = tbase + (static_cast<uint32_t>(32 * lq) << 16);
#pragma unroll
        for (int m = 0; m < 2; ++m) {
#pragma unroll
            for (int c = 0; c < 2; ++c) {
                const int col = 64 * ch + 32 * c;
                float x[32];
                tmem_ld32(tl + 128 * m + col, x);
                float4 *dst = reinterpret_cast<float4 *>(out + m * kD * kD + row * kD + col);
#pragma unroll
                for (int e = 0; e < 8; ++e) dst[e] = make_float4(x[4 * e], x[4 * e + 1], x[4 * e + 2], x[4 * e + 3]);
            }
        }
    }
    if (tid < kD) {
        out[2 * kD * kD + tid] = msum[tid];
        out[2 * kD * kD + kD + tid] = dsuf[tid];
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tbase, 256);
    }
}

// Exclusive scan over the segments of each sequence: the delta stored in slot s
// is replaced by the state entering segment s.  Elementwise, so the grid spans
// (sequence, 1024-element block) and every thread walks the segments of 4 elements.
constexpr int kCombineBlock = 1024;

__global__ void __launch_bounds__(256)
gla_segment_combine_kernel(const ChunkArgs a) {
    const int nblk = (kSegFloats - kD + kCombineBlock - 1) / kCombineBlock;  // D is not scanned
    const int seq = blockIdx.x / nblk, blk = blockIdx.x % nblk;
    const size_t sq = static_cast<size_t>(seq);
    constexpr int kSS = kD * kD;  // S block, then C block, then m
    float cur[4];
    int el[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        const int e = blk * kCombineBlock + u * 256 + threadIdx.x;
        el[u] = e;
        float x = 0.f;
        if (e < kSS) x = a.S0 ? a.S0[sq * kSS + e] : 0.f;
        else if (e < 2 * kSS) x = a.C0 ? a.C0[sq * kSS + e - kSS] : 0.f;
        else if (e < 2 * kSS + kD) x = a.m0 ? a.m0[sq * kD + e - 2 * kSS] : 0.f;
        cur[u] = x;
    }
    // segments in groups of kGroup: every load of a group is issued before its scan steps
    // (the loads do not depend on the scan), so the group costs one memory round trip
    constexpr int kGroup = 8;
    for (int s0 = 0; s0 < a.nseg; s0 += kGroup) {
        const int ns = min(kGroup, a.nseg - s0);
        float dv[kGroup][4], Dv[kGroup][4];
#pragma unroll
        for (int g = 0; g < kGroup; ++g) {
            if (g < ns) {
                const float *slot = a.seg_ws + (sq * a.nseg + s0 + g) * kSegFloats;
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int e = el[u];
                    const bool live = e < 2 * kSS + kD;
                    dv[g][u] = live ? slot[e] : 0.f;
                    Dv[g][u] = (e < kSS) ? slot[2 * kSS + kD + (e >> 7)] : 1.f;
                }
            }
        }
#pragma unroll
        for (int g = 0; g < kGroup; ++g) {
            if (g < ns) {
                float *slot = a.seg_ws + (sq * a.nseg + s0 + g) * kSegFloats;
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int e = el[u];
                    if (e >= 2 * kSS + kD) continue;
                    slot[e] = cur[u];
                    cur[u] = Dv[g][u] * cur[u] + dv[g][u];
                }
            }
        }
    }
}

}  // namespace

cudaError_t launch_gla_segments(const ChunkArgs &a, const ChunkMaps &m, cudaStream_t s) {
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(gla_segment_state_kernel,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(kSmem));
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    gla_segment_state_kernel<<<a.B * a.H * a.nseg, kThreads, kSmem, s>>>(m.k, m.v, m.g, a);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const int nblk = (kSegFloats - kD + kCombineBlock - 1) / kCombineBlock;
    gla_segment_combine_kernel<<<a.B * a.H * nblk, 256, 0, s>>>(a);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    return launch_gla_chunk(a, m, s);
}

}  // namespace ccq
