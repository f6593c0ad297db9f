// ccq_capi.cu -- the extern "C" boundary of the CCQ library (include/ccq.h):
// argument validation, tensor-map encoding, kernel dispatch and the device
// status word.  No entry point allocates memory.
#include <cuda.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdarg.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <algorithm>
#include <initializer_list>

#include "../../include/ccq.h"
#include "ccq_gdn_bwd.h"
#include "ccq_internal.h"

namespace ccq {

// Written by a kernel whose bounded wait gave up; read and cleared by
// ccq_device_status().
__device__ int g_status = 0;

int *device_status_word() {
    // one slot per device ordinal; filled on first use with that device current
    static int *addr[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
    if (!addr[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_status) != cudaSuccess) return nullptr;
        addr[dev] = static_cast<int *>(p);
    }
    return addr[dev];
}

namespace {

thread_local char g_last_error[512] = "";

ccq_status fail(ccq_status s, const char *fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_last_error, sizeof g_last_error, fmt, ap);
    va_end(ap);
    return s;
}

ccq_status cuda_fail(cudaError_t e, const char *what) {
    return fail(CCQ_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                  const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                  const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    static bool tried = false;
    if (!tried) {
        tried = true;
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    }
    return fn;
}

struct Common {
    ccq_params p;
    float scale;
};

ccq_status check_common(const ccq_params *pin, int B, int T, int H, int Dk, int Dv, Common *c) {
    if (pin) c->p = *pin;
    else ccq_default_params(&c->p);
    if (B < 1 || H < 1 || T < 0) return fail(CCQ_ERR_INVALID_ARG, "bad sizes B=%d T=%d H=%d", B, T, H);
    if (Dk != Dv || (Dk != 64 && Dk != 128))
        return fail(CCQ_ERR_UNSUPPORTED, "head dims Dk=%d Dv=%d: supported Dk = Dv in {64, 128}", Dk, Dv);
    if (c->p.chunk != 0 && c->p.chunk != 64)
        return fail(CCQ_ERR_UNSUPPORTED, "chunk=%d: supported 64", c->p.chunk);
    if (c->p.algo < CCQ_ALGO_AUTO || c->p.algo > CCQ_ALGO_CHUNKWISE_WIDE)
        return fail(CCQ_ERR_INVALID_ARG, "unknown algo %d", c->p.algo);
    if (c->p.seq_split < 0) return fail(CCQ_ERR_INVALID_ARG, "seq_split must be >= 0");
    if ((static_cast<long long>(B) * H) > 0x7fffffffLL)
        return fail(CCQ_ERR_INVALID_ARG, "B*H too large");
    c->scale = c->p.scale > 0.f ? c->p.scale : 1.f / sqrtf(static_cast<float>(Dk));
    return CCQ_OK;
}

ccq_status check_ptrs(const char *names, std::initializer_list<const void *> required,
                      std::initializer_list<const void *> optional) {
    int i = 0;
    for (const void *p : required) {
        if (!p) return fail(CCQ_ERR_INVALID_ARG, "required pointer #%d of (%s) is NULL", i, names);
        if (!aligned16(p)) return fail(CCQ_ERR_INVALID_ARG, "pointer #%d of (%s) is not 16-byte aligned", i, names);
        ++i;
    }
    for (const void *p : optional) {
        if (p && !aligned16(p)) return fail(CCQ_ERR_INVALID_ARG, "an optional state pointer is not 16-byte aligned");
    }
    return CCQ_OK;
}

// The int64 position counters t0 / tT are read and written one element per
// batch row, so they need only their natural 8-byte alignment (a row of a
// larger counter array, as the packed-sequence call passes, is enough).
ccq_status check_counts(std::initializer_list<const void *> counts) {
    for (const void *p : counts) {
        if (p && (reinterpret_cast<uintptr_t>(p) & 7u) != 0)
            return fail(CCQ_ERR_INVALID_ARG, "a position-count pointer (t0 / tT) is not 8-byte aligned");
    }
    return CCQ_OK;
}

// Final position count, after the kernels that read t0 (tT may alias it).
ccq_status finish_t(const int64_t *t0, int64_t *tT, int B, int T, cudaStream_t s) {
    cudaError_t e = launch_t_update(t0, tT, B, T, s);
    if (e != cudaSuccess) return cuda_fail(e, "position update launch");
    return CCQ_OK;
}

ccq_status run_recurrent(RecurrentArgs &ra, cudaStream_t s) {
    cudaError_t e = launch_recurrent(ra, s);
    if (e != cudaSuccess) return cuda_fail(e, "recurrent kernel launch");
    return CCQ_OK;
}

}  // namespace

int record_error_code(int st, const char *msg) {
    snprintf(g_last_error, sizeof g_last_error, "%s", msg);
    return st;
}

bool make_token_map(CUtensorMap *map, const void *base, int elem_bytes, int B, int T, int H, int D,
                    int box_inner, bool swizzle128) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    const cuuint64_t dims[4] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(H),
                                static_cast<cuuint64_t>(T), static_cast<cuuint64_t>(B)};
    const cuuint64_t eb = static_cast<cuuint64_t>(elem_bytes);
    const cuuint64_t strides[3] = {eb * D, eb * D * H, eb * D * H * T};
    const cuuint32_t box[4] = {static_cast<cuuint32_t>(box_inner), 1, 64, 1};
    const cuuint32_t estr[4] = {1, 1, 1, 1};
    const CUtensorMapDataType dt =
        elem_bytes == 2 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32;
    CUresult r = fn(map, dt, 4, const_cast<void *>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE,
                    swizzle128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

bool make_f32_rows_map(CUtensorMap *map, const void *base, long long rows, int cols, int box_cols, int box_rows) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(cols) * 4};
    const cuuint32_t box[2] = {static_cast<cuuint32_t>(box_cols), static_cast<cuuint32_t>(box_rows)};
    const cuuint32_t estr[2] = {1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<void *>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

bool make_rows_map(CUtensorMap *map, const void *base, long long rows, int cols) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(cols) * 2};
    const cuuint32_t box[2] = {64, 64};
    const cuuint32_t estr[2] = {1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box,
                    estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

}  // namespace ccq

using namespace ccq;

extern "C" {

void ccq_default_params(ccq_params *p) {
    if (!p) return;
    p->l2norm_qk = 1;
    p->scale = 0.f;
    p->centered = 1;
    p->chunk = 64;
    p->algo = CCQ_ALGO_AUTO;
    p->seq_split = 0;
}

const char *ccq_status_string(ccq_status s) {
    switch (s) {
        case CCQ_OK: return "ok";
        case CCQ_ERR_INVALID_ARG: return "invalid argument";
        case CCQ_ERR_UNSUPPORTED: return "unsupported configuration";
        case CCQ_ERR_CUDA: return "CUDA error";
        case CCQ_ERR_TIMEOUT: return "a kernel's bounded wait timed out";
        case CCQ_ERR_RANGE: return "gates outside the range the chunkwise kernel can factor";
    }
    return "unknown status";
}

const char *ccq_last_error(void) { return g_last_error; }

static int sm_count() {
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
        n = 148;
    return n;
}

// Segments per sequence for the chunkwise GLA path, and chunks per segment.
static void split_sequences(const ccq_params &p, int B, int T, int H, int *nseg, int *seg_chunks) {
    const int nc = (T + 63) / 64;
    int ns = 1;
    if (p.seq_split > 0) {
        ns = p.seq_split;
    } else if (p.seq_split == 0) {
        const long long seqs = static_cast<long long>(B) * H;
        const int sms = sm_count();
        if (seqs * 2 <= sms) ns = static_cast<int>(sms / seqs);
        ns = std::min(ns, nc / 8);  // keep at least 8 chunks per segment
    }
    ns = std::max(1, std::min(ns, nc));
    const int per = (nc + ns - 1) / ns;
    *seg_chunks = per;
    *nseg = (nc + per - 1) / per;  // no empty segment
}

static bool gla_chunk_selected(const ccq_params &p, ccq_dtype in_dtype, int Dk, int T) {
    return in_dtype == CCQ_BF16 && Dk == 128 && T > 0 && p.algo != CCQ_ALGO_RECURRENT;
}

ccq_status ccq_gla_workspace_size(int B, int T, int H, int Dk, int Dv, ccq_dtype in_dtype,
                                  const ccq_params *p, size_t *bytes) {
    Common c;
    ccq_status st = check_common(p, B, T, H, Dk, Dv, &c);
    if (st != CCQ_OK) return st;
    if (!bytes) return fail(CCQ_ERR_INVALID_ARG, "bytes is NULL");
    *bytes = 0;
    if (gla_chunk_selected(c.p, in_dtype, Dk, T)) {
        int ns, per;
        split_sequences(c.p, B, T, H, &ns, &per);
        if (ns > 1) *bytes = static_cast<size_t>(B) * H * ns * kSegFloats * sizeof(float);
    }
    return CCQ_OK;
}

// The GLA forward behind ccq_gla_fwd, ccq_gla_fwd_save and the backward's
// checkpoint recompute: ckpt (nullable) receives the chunk-start states,
// skip_o suppresses the output.
static ccq_status gla_fwd_impl(const void *q, const void *k, const void *v, const void *gk,
                               const float *lambda, ccq_dtype in_dtype, ccq_dtype gate_dtype,
                               const float *S0, const float *C0, const float *m0, const int64_t *t0,
                               void *o, float *ST, float *CT, float *mT, int64_t *tT,
                               int B, int T, int H, int Dk, int Dv, void *workspace,
                               size_t workspace_bytes, uint8_t *ckpt, int skip_o, const ccq_params *p,
                               void *stream, bool dry = false) {
    Common c;
    ccq_status st = check_common(p, B, T, H, Dk, Dv, &c);
    if (st != CCQ_OK) return st;
    if ((in_dtype != CCQ_BF16 && in_dtype != CCQ_FP32) || (gate_dtype != CCQ_BF16 && gate_dtype != CCQ_FP32))
        return fail(CCQ_ERR_INVALID_ARG, "unknown dtype");
    if (T > 0) {
        st = check_ptrs("q,k,v,gk,lambda,o", {q, k, v, gk, lambda, o}, {S0, C0, m0, ST, CT, mT});
        if (st == CCQ_OK) st = check_counts({t0, tT});
        if (st != CCQ_OK) return st;
    } else {
        st = check_ptrs("", {}, {S0, C0, m0, ST, CT, mT});
        if (st == CCQ_OK) st = check_counts({t0, tT});
        if (st != CCQ_OK) return st;
    }
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const bool chunk_ok = in_dtype == CCQ_BF16 && Dk == 128 && T > 0;
    if ((c.p.algo == CCQ_ALGO_CHUNKWISE || c.p.algo == CCQ_ALGO_CHUNKWISE_WIDE || ckpt) && !chunk_ok)
        return fail(CCQ_ERR_UNSUPPORTED, "chunkwise kernel needs bf16 inputs, Dk = Dv = 128, T > 0");
    if (ckpt && c.p.algo == CCQ_ALGO_RECURRENT)
        return fail(CCQ_ERR_UNSUPPORTED, "checkpoints come from the chunkwise kernel (algo recurrent given)");
    if (chunk_ok && c.p.algo != CCQ_ALGO_RECURRENT) {
        int nseg = 1, seg_chunks = 0;
        split_sequences(c.p, B, T, H, &nseg, &seg_chunks);
        if (nseg > 1) {
            const size_t need = static_cast<size_t>(B) * H * nseg * kSegFloats * sizeof(float);
            if (!workspace || workspace_bytes < need)
                return fail(CCQ_ERR_INVALID_ARG, "workspace of %zu bytes required (got %zu)", need,
                            workspace ? workspace_bytes : static_cast<size_t>(0));
            if (!aligned16(workspace)) return fail(CCQ_ERR_INVALID_ARG, "workspace is not 16-byte aligned");
        }
        ChunkMaps maps;
        const int geb = gate_dtype == CCQ_BF16 ? 2 : 4;
        if (!make_token_map(&maps.q, q, 2, B, T, H, 128, 64, true) ||
            !make_token_map(&maps.k, k, 2, B, T, H, 128, 64, true) ||
            !make_token_map(&maps.v, v, 2, B, T, H, 128, 64, true) ||
            !make_token_map(&maps.g, gk, geb, B, T, H, 128, 128, false) ||
            !make_token_map(&maps.o, o, 2, B, T, H, 128, 64, true))
            return fail(CCQ_ERR_CUDA, "cuTensorMapEncodeTiled failed (driver entry point missing or map rejected)");
        if (dry) return CCQ_OK;
        ChunkArgs a = {};
        a.B = B; a.T = T; a.H = H;
        a.gate_dtype = gate_dtype == CCQ_BF16 ? 0 : 1;
        a.l2norm = c.p.l2norm_qk; a.centered = c.p.centered; a.scale = c.scale;
        a.lambda = lambda;
        a.gk = gk;
        a.wide = c.p.algo == CCQ_ALGO_CHUNKWISE_WIDE;
        a.S0 = S0; a.C0 = C0; a.m0 = m0; a.t0 = t0;
        a.o = static_cast<__nv_bfloat16 *>(o);
        a.ST = ST; a.CT = CT; a.mT = mT;
        a.status = device_status_word();
        if (!a.status) return fail(CCQ_ERR_CUDA, "cannot resolve the device status word");
        a.nseg = nseg;
        a.seg_chunks = seg_chunks;
        a.ckpt = ckpt;
        a.skip_o = skip_o;
        if (a.nseg > 1) {
            a.seg_ws = static_cast<float *>(workspace);
            cudaError_t e = launch_gla_segments(a, maps, s);
            if (e != cudaSuccess) return cuda_fail(e, "segmented chunkwise GLA launch");
            return finish_t(t0, tT, B, T, s);
        }
        cudaError_t e = launch_gla_chunk(a, maps, s);
        if (e != cudaSuccess) return cuda_fail(e, "chunkwise GLA kernel launch");
        return finish_t(t0, tT, B, T, s);
    }
    if (dry) return CCQ_OK;
    RecurrentArgs ra = {};
    ra.backbone = 0; ra.B = B; ra.T = T; ra.H = H; ra.Dk = Dk; ra.Dv = Dv;
    ra.in_dtype = in_dtype; ra.gate_dtype = gate_dtype;
    ra.l2norm = c.p.l2norm_qk; ra.centered = c.p.centered; ra.scale = c.scale;
    ra.q = q; ra.k = k; ra.v = v; ra.gate = gk; ra.beta = nullptr; ra.lambda = lambda;
    ra.S0 = S0; ra.C0 = C0; ra.m0 = m0; ra.t0 = t0;
    ra.o = o; ra.ST = ST; ra.CT = CT; ra.mT = mT;
    st = run_recurrent(ra, s);
    return st != CCQ_OK ? st : finish_t(t0, tT, B, T, s);
}

ccq_status ccq_gla_fwd(const void *q, const void *k, const void *v, const void *gk,
                       const float *lambda, ccq_dtype in_dtype, ccq_dtype gate_dtype,
                       const float *S0, const float *C0, const float *m0, const int64_t *t0,
                       void *o, float *ST, float *CT, float *mT, int64_t *tT,
                       int B, int T, int H, int Dk, int Dv, void *workspace,
                       size_t workspace_bytes, const ccq_params *p, void *stream) {
    return gla_fwd_impl(q, k, v, gk, lambda, in_dtype, gate_dtype, S0, C0, m0, t0, o, ST, CT, mT, tT, B, T,
                        H, Dk, Dv, workspace, workspace_bytes, nullptr, 0, p, stream);
}

ccq_status ccq_gla_ckpt_size(int B, int T, int H, int Dk, int Dv, size_t *bytes) {
    if (!bytes) return fail(CCQ_ERR_INVALID_ARG, "bytes is NULL");
    if (B < 1 || H < 1 || T < 0) return fail(CCQ_ERR_INVALID_ARG, "bad sizes B=%d T=%d H=%d", B, T, H);
    if (Dk != 128 || Dv != 128) return fail(CCQ_ERR_UNSUPPORTED, "checkpoints need Dk = Dv = 128");
    *bytes = static_cast<size_t>(B) * H * ckpt_head_bytes(T);
    return CCQ_OK;
}

ccq_status ccq_gla_fwd_save(const void *q, const void *k, const void *v, const void *gk,
                            const float *lambda, ccq_dtype in_dtype, ccq_dtype gate_dtype,
                            const float *S0, const float *C0, const float *m0, const int64_t *t0,
                            void *o, float *ST, float *CT, float *mT, int64_t *tT,
                            int B, int T, int H, int Dk, int Dv, void *workspace,
                            size_t workspace_bytes, void *ckpt, size_t ckpt_bytes,
                            const ccq_params *p, void *stream) {
    size_t need = 0;
    ccq_status st = ccq_gla_ckpt_size(B, T, H, Dk, Dv, &need);
    if (st != CCQ_OK) return st;
    if (!ckpt || ckpt_bytes < need)
        return fail(CCQ_ERR_INVALID_ARG, "checkpoint buffer of %zu bytes required (got %zu)", need,
                    ckpt ? ckpt_bytes : static_cast<size_t>(0));
    if (!aligned16(ckpt)) return fail(CCQ_ERR_INVALID_ARG, "ckpt is not 16-byte aligned");
    return gla_fwd_impl(q, k, v, gk, lambda, in_dtype, gate_dtype, S0, C0, m0, t0, o, ST, CT, mT, tT, B, T,
                        H, Dk, Dv, workspace, workspace_bytes, static_cast<uint8_t *>(ckpt), 0, p, stream);
}

// Workspace layout of ccq_gla_bwd: four bf16 [B,T,H,128] exchange tensors, then
// per chunk the q kernel's vectors (3 x 128 fp32), the state pass's images (64 KB)
// and vectors (2 x 128 fp32); then (without caller checkpoints) the checkpoints
// and the forward's scratch.
static size_t gla_bwd_exchange_bytes(int B, int T, int H) {
    const size_t chunks = static_cast<size_t>(B) * H * ((T + 63) / 64);
    return 4 * static_cast<size_t>(B) * T * H * 128 * 2 + chunks * (3 * 128 * 4 + 65536 + 3 * 128 * 4);
}

static size_t gla_fwd_scratch_bytes(const ccq_params &p, int B, int T, int H) {
    int ns, per;
    split_sequences(p, B, T, H, &ns, &per);
    return ns > 1 ? static_cast<size_t>(B) * H * ns * kSegFloats * sizeof(float) : 0;
}

ccq_status ccq_gla_bwd_workspace_size(int B, int T, int H, int Dk, int Dv, ccq_dtype in_dtype,
                                      int with_ckpt, const ccq_params *p, size_t *bytes) {
    Common c;
    ccq_status st = check_common(p, B, T, H, Dk, Dv, &c);
    if (st != CCQ_OK) return st;
    if (!bytes) return fail(CCQ_ERR_INVALID_ARG, "bytes is NULL");
    if (in_dtype != CCQ_BF16 || Dk != 128)
        return fail(CCQ_ERR_UNSUPPORTED, "the backward needs bf16 inputs and Dk = Dv = 128");
    *bytes = 0;
    if (T == 0) return CCQ_OK;
    *bytes = gla_bwd_exchange_bytes(B, T, H);
    if (!with_ckpt) *bytes += static_cast<size_t>(B) * H * ckpt_head_bytes(T) + gla_fwd_scratch_bytes(c.p, B, T, H);
    return CCQ_OK;
}

ccq_status ccq_gla_bwd(const void *q, const void *k, const void *v, const void *gk,
                       const float *lambda, ccq_dtype in_dtype, ccq_dtype gate_dtype,
                       const float *S0, const float *C0, const float *m0, const int64_t *t0,
                       const void *dout, const float *dST, const float *dCT, const float *dmT,
                       const void *ckpt, void *dq, void *dk, void *dv, void *dgk,
                       float *dlambda, float *dS0, float *dC0, float *dm0,
                       int B, int T, int H, int Dk, int Dv, void *workspace,
                       size_t workspace_bytes, const ccq_params *p, void *stream) {
    Common c;
    ccq_status st = check_common(p, B, T, H, Dk, Dv, &c);
    if (st != CCQ_OK) return st;
    if ((in_dtype != CCQ_BF16 && in_dtype != CCQ_FP32) || (gate_dtype != CCQ_BF16 && gate_dtype != CCQ_FP32))
        return fail(CCQ_ERR_INVALID_ARG, "unknown dtype");
    if (in_dtype != CCQ_BF16 || Dk != 128)
        return fail(CCQ_ERR_UNSUPPORTED, "the backward needs bf16 inputs and Dk = Dv = 128");
    if (c.p.algo == CCQ_ALGO_RECURRENT)
        return fail(CCQ_ERR_UNSUPPORTED, "the backward is chunkwise only (algo recurrent given)");
    st = check_ptrs("", {}, {S0, C0, m0, dST, dCT, dmT, ckpt, dlambda, dS0, dC0, dm0});
    if (st == CCQ_OK) st = check_counts({t0});
    if (st != CCQ_OK) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (T == 0) {
        // no tokens: the initial states are the final states
        const size_t n[3] = {static_cast<size_t>(B) * H * Dk * Dv * 4, static_cast<size_t>(B) * H * Dk * Dk * 4,
                             static_cast<size_t>(B) * H * Dk * 4};
        float *dst[3] = {dS0, dC0, dm0};
        const float *src[3] = {dST, dCT, dmT};
        for (int i = 0; i < 3; ++i) {
            if (!dst[i]) continue;
            cudaError_t e = src[i] ? cudaMemcpyAsync(dst[i], src[i], n[i], cudaMemcpyDeviceToDevice, s)
                                   : cudaMemsetAsync(dst[i], 0, n[i], s);
            if (e != cudaSuccess) return cuda_fail(e, "state gradient copy");
        }
        return CCQ_OK;
    }
    st = check_ptrs("q,k,v,gk,lambda,dout,dq,dk,dv,dgk", {q, k, v, gk, lambda, dout, dq, dk, dv, dgk}, {});
    if (st != CCQ_OK) return st;
    size_t need = gla_bwd_exchange_bytes(B, T, H);
    const size_t ck_bytes = static_cast<size_t>(B) * H * ckpt_head_bytes(T);
    const size_t fwd_bytes = ckpt ? 0 : gla_fwd_scratch_bytes(c.p, B, T, H);
    if (!ckpt) need += ck_bytes + fwd_bytes;
    if (!workspace || workspace_bytes < need)
        return fail(CCQ_ERR_INVALID_ARG, "workspace of %zu bytes required (got %zu)", need,
                    workspace ? workspace_bytes : static_cast<size_t>(0));
    if (!aligned16(workspace)) return fail(CCQ_ERR_INVALID_ARG, "workspace is not 16-byte aligned");
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    const size_t xbytes = static_cast<size_t>(B) * T * H * 128 * 2;
    const size_t chunks = static_cast<size_t>(B) * H * ((T + 63) / 64);
    uint8_t *qg = ws, *dkc = ws + xbytes, *gq = ws + 2 * xbytes, *dzr = ws + 3 * xbytes;
    float *chunk_vec = reinterpret_cast<float *>(ws + 4 * xbytes);
    uint8_t *state_img = ws + 4 * xbytes + chunks * 3 * 128 * 4;
    float *state_vec = reinterpret_cast<float *>(state_img + chunks * 65536);
    const uint8_t *ck = static_cast<const uint8_t *>(ckpt);
    if (!ckpt) {
        uint8_t *own = ws + gla_bwd_exchange_bytes(B, T, H);
        // forward without output: dq stands in for the unused output tensor
        st = gla_fwd_impl(q, k, v, gk, lambda, in_dtype, gate_dtype, S0, C0, m0, t0, dq, nullptr, nullptr,
                          nullptr, nullptr, B, T, H, Dk, Dv, fwd_bytes ? own + ck_bytes : nullptr, fwd_bytes,
                          own, 1, &c.p, stream);
        if (st != CCQ_OK) return st;
        ck = own;
    }
    BwdMaps maps;
    const int geb = gate_dtype == CCQ_BF16 ? 2 : 4;
    if (!make_token_map(&maps.q, q, 2, B, T, H, 128, 64, true) ||
        !make_token_map(&maps.k, k, 2, B, T, H, 128, 64, true) ||
        !make_token_map(&maps.v, v, 2, B, T, H, 128, 64, true) ||
        !make_token_map(&maps.dO, dout, 2, B, T, H, 128, 64, true) ||
        !make_token_map(&maps.g, gk, geb, B, T, H, 128, 128, false) ||
        !make_token_map(&maps.dq, dq, 2, B, T, H, 128, 64, true) ||
        !make_token_map(&maps.dk, dk, 2, B, T, H, 128, 64, true) ||
        !make_token_map(&maps.dv, dv, 2, B, T, H, 128, 64, true) ||
        !make_token_map(&maps.qg, qg, 2, B, T, H, 128, 64, true) ||
        !make_token_map(&maps.dkc, dkc, 2, B, T, H, 128, 64, true) ||
        !make_token_map(&maps.gq, gq, 2, B, T, H, 128, 64, true) ||
        !make_token_map(&maps.dzr, dzr, 2, B, T, H, 128, 64, true))
        return fail(CCQ_ERR_CUDA, "cuTensorMapEncodeTiled failed (driver entry point missing or map rejected)");
    BwdArgs a = {};
    a.B = B; a.T = T; a.H = H;
    a.gate_dtype = gate_dtype == CCQ_BF16 ? 0 : 1;
    a.l2norm = c.p.l2norm_qk; a.centered = c.p.centered; a.scale = c.scale;
    a.lambda = lambda; a.t0 = t0; a.ckpt = ck;
    a.dST = dST; a.dCT = dCT; a.dmT = dmT;
    a.dlambda = dlambda; a.dgk = dgk; a.dS0 = dS0; a.dC0 = dC0; a.dm0 = dm0;
    a.chunk_vec = chunk_vec; a.state_img = state_img; a.state_vec = state_vec;
    a.wave = sm_count();
    a.status = device_status_word();
    if (!a.status) return fail(CCQ_ERR_CUDA, "cannot resolve the device status word");
    cudaError_t e = launch_gla_bwd(a, maps, s);
    if (e != cudaSuccess) return cuda_fail(e, "GLA backward kernel launch");
    return CCQ_OK;
}

static bool gdn_chunk_selected(const ccq_params &p, ccq_dtype in_dtype, int Dk, int T) {
    const bool ok = in_dtype == CCQ_BF16 && Dk == 128 && T > 0;
    return ok && p.algo != CCQ_ALGO_RECURRENT;
}

// Workspace of the chunkwise Gated DeltaNet path: Tb of every chunk, then (split
// sequences) the per-segment states.
static size_t gdn_total_workspace(const ccq_params &p, int B, int T, int H) {
    int nseg = 1, per = 0;
    split_sequences(p, B, T, H, &nseg, &per);
    size_t bytes = gdn_workspace_bytes(B, T, H);
    if (nseg > 1) bytes += static_cast<size_t>(B) * H * nseg * kGdnSegFloats * sizeof(float);
    return bytes;
}

ccq_status ccq_gdn_workspace_size(int B, int T, int H, int Dk, int Dv, ccq_dtype in_dtype,
                                  const ccq_params *p, size_t *bytes) {
    Common c;
    ccq_status st = check_common(p, B, T, H, Dk, Dv, &c);
    if (st != CCQ_OK) return st;
    if (!bytes) return fail(CCQ_ERR_INVALID_ARG, "bytes is NULL");
    *bytes = gdn_chunk_selected(c.p, in_dtype, Dk, T) ? gdn_total_workspace(c.p, B, T, H) : 0;
    return CCQ_OK;
}

// Per-chunk fp32 arrays of the CCQ-Gated-DeltaNet backward that the tensor-core forward can
// fill (ChunkArgs::tt_out and the rest); with them the forward writes no output.
struct GdnDumps {
    float *tt, *sk, *mk, *hs;
};

// The Gated DeltaNet forward behind ccq_gdn_fwd; `dry` runs every argument check and
// returns before the first CUDA call.
static ccq_status gdn_fwd_impl(const void *q, const void *k, const void *v, const float *g,
                               const float *beta, const float *lambda, ccq_dtype in_dtype,
                               const float *S0, const float *C0, const float *m0, const int64_t *t0,
                               void *o, float *ST, float *CT, float *mT, int64_t *tT,
                               int B, int T, int H, int Dk, int Dv, void *workspace,
                               size_t workspace_bytes, const ccq_params *p, void *stream, bool dry,
                               const GdnDumps *dumps = nullptr) {
    Common c;
    ccq_status st = check_common(p, B, T, H, Dk, Dv, &c);
    if (st != CCQ_OK) return st;
    if (in_dtype != CCQ_BF16 && in_dtype != CCQ_FP32) return fail(CCQ_ERR_INVALID_ARG, "unknown dtype");
    if (T > 0) {
        st = check_ptrs("q,k,v,g,beta,lambda,o", {q, k, v, g, beta, lambda, o}, {S0, C0, m0, ST, CT, mT});
        if (st == CCQ_OK) st = check_counts({t0, tT});
        if (st != CCQ_OK) return st;
    } else {
        st = check_ptrs("", {}, {S0, C0, m0, ST, CT, mT});
        if (st == CCQ_OK) st = check_counts({t0, tT});
        if (st != CCQ_OK) return st;
    }
    const bool chunk_ok = in_dtype == CCQ_BF16 && Dk == 128 && T > 0;
    if ((c.p.algo == CCQ_ALGO_CHUNKWISE || c.p.algo == CCQ_ALGO_CHUNKWISE_WIDE) && !chunk_ok)
        return fail(CCQ_ERR_UNSUPPORTED, "chunkwise kernel needs bf16 inputs, Dk = Dv = 128, T > 0");
    if (gdn_chunk_selected(c.p, in_dtype, Dk, T)) {
        const size_t need = gdn_total_workspace(c.p, B, T, H);
        if (!workspace || workspace_bytes < need)
            return fail(CCQ_ERR_INVALID_ARG, "workspace of %zu bytes required (got %zu)", need,
                        workspace ? workspace_bytes : static_cast<size_t>(0));
        if (!aligned16(workspace)) return fail(CCQ_ERR_INVALID_ARG, "workspace is not 16-byte aligned");
        const int nc = (T + 63) / 64;
        const long long rows = static_cast<long long>(B) * H * nc * 64;
        GdnMaps maps;
        if (!make_token_map(&maps.q, q, 2, B, T, H, 128, 64, true) ||
            !make_token_map(&maps.k, k, 2, B, T, H, 128, 64, true) ||
            !make_token_map(&maps.v, v, 2, B, T, H, 128, 64, true) ||
            !make_token_map(&maps.o, o, 2, B, T, H, 128, 64, true) ||
            !make_rows_map(&maps.tb, workspace, rows, 64))
            return fail(CCQ_ERR_CUDA, "cuTensorMapEncodeTiled failed (driver entry point missing or map rejected)");
        if (dry) return CCQ_OK;
        ChunkArgs a = {};
        a.B = B; a.T = T; a.H = H;
        a.gate_dtype = 1;
        a.l2norm = c.p.l2norm_qk; a.centered = c.p.centered; a.scale = c.scale;
        a.lambda = lambda; a.g = g; a.beta = beta;
        a.S0 = S0; a.C0 = C0; a.m0 = m0; a.t0 = t0;
        a.o = static_cast<__nv_bfloat16 *>(o);
        a.ST = ST; a.CT = CT; a.mT = mT;
        if (dumps) {
            a.tt_out = dumps->tt; a.sk_out = dumps->sk; a.mk_out = dumps->mk; a.hs_out = dumps->hs;
            a.skip_o = 1;
        }
        a.status = device_status_word();
        if (!a.status) return fail(CCQ_ERR_CUDA, "cannot resolve the device status word");
        int nseg = 1, seg_chunks = 0;
        split_sequences(c.p, B, T, H, &nseg, &seg_chunks);
        a.nseg = nseg;
        a.seg_chunks = seg_chunks;
        cudaError_t e;
        if (nseg > 1) {
            a.seg_ws = reinterpret_cast<float *>(static_cast<uint8_t *>(workspace) + gdn_workspace_bytes(B, T, H));
            e = launch_gdn_segments(a, maps, static_cast<cudaStream_t>(stream));
        } else {
            e = launch_gdn_chunk(a, maps, static_cast<cudaStream_t>(stream));
        }
        if (e != cudaSuccess) return cuda_fail(e, "chunkwise Gated DeltaNet kernel launch");
        return finish_t(t0, tT, B, T, static_cast<cudaStream_t>(stream));
    }
    if (dry) return CCQ_OK;
    RecurrentArgs ra = {};
    ra.backbone = 1; ra.B = B; ra.T = T; ra.H = H; ra.Dk = Dk; ra.Dv = Dv;
    ra.in_dtype = in_dtype; ra.gate_dtype = CCQ_FP32;
    ra.l2norm = c.p.l2norm_qk; ra.centered = c.p.centered; ra.scale = c.scale;
    ra.q = q; ra.k = k; ra.v = v; ra.gate = g; ra.beta = beta; ra.lambda = lambda;
    ra.S0 = S0; ra.C0 = C0; ra.m0 = m0; ra.t0 = t0;
    ra.o = o; ra.ST = ST; ra.CT = CT; ra.mT = mT;
    st = run_recurrent(ra, static_cast<cudaStream_t>(stream));
    return st != CCQ_OK ? st : finish_t(t0, tT, B, T, static_cast<cudaStream_t>(stream));
}

ccq_status ccq_gdn_fwd(const void *q, const void *k, const void *v, const float *g,
                       const float *beta, const float *lambda, ccq_dtype in_dtype,
                       const float *S0, const float *C0, const float *m0, const int64_t *t0,
                       void *o, float *ST, float *CT, float *mT, int64_t *tT,
                       int B, int T, int H, int Dk, int Dv, void *workspace,
                       size_t workspace_bytes, const ccq_params *p, void *stream) {
    return gdn_fwd_impl(q, k, v, g, beta, lambda, in_dtype, S0, C0, m0, t0, o, ST, CT, mT, tT, B, T, H, Dk, Dv,
                        workspace, workspace_bytes, p, stream, false);
}

// Copies the final-state gradients to the initial-state ones (zero where a final one is NULL):
// the backward of a call with no tokens.
static ccq_status copy_state_grads(const float *dST, const float *dCT, const float *dmT, float *dS0, float *dC0,
                                   float *dm0, int B, int H, int Dk, int Dv, cudaStream_t s) {
    const size_t n[3] = {static_cast<size_t>(B) * H * Dk * Dv * 4, static_cast<size_t>(B) * H * Dk * Dk * 4,
                         static_cast<size_t>(B) * H * Dk * 4};
    float *dst[3] = {dS0, dC0, dm0};
    const float *src[3] = {dST, dCT, dmT};
    for (int i = 0; i < 3; ++i) {
        if (!dst[i]) continue;
        cudaError_t e = src[i] ? cudaMemcpyAsync(dst[i], src[i], n[i], cudaMemcpyDeviceToDevice, s)
                               : cudaMemsetAsync(dst[i], 0, n[i], s);
        if (e != cudaSuccess) return cuda_fail(e, "state gradient copy");
    }
    return CCQ_OK;
}

// bf16 inputs with Dk = 128 recompute the forward's per-chunk quantities with the tensor-core
// forward kernels (gdn_wy_kernel, gdn_chunk_kernel), whose own workspace follows the
// backward's arrays (at a 1 KB boundary); other inputs compute them on the CUDA cores.
static bool gdn_bwd_tc_forward(ccq_dtype in_dtype, int Dk) { return in_dtype == CCQ_BF16 && Dk == 128; }
static ccq_params gdn_bwd_forward_params(const ccq_params &p) {
    ccq_params f = p;
    f.algo = CCQ_ALGO_CHUNKWISE;
    return f;
}
static size_t gdn_bwd_forward_offset(int B, int T, int H, int Dk) {
    return (gdn_bwd_workspace_bytes(B, T, H, Dk) + 1023) & ~static_cast<size_t>(1023);
}
static size_t gdn_bwd_total_workspace(const ccq_params &p, ccq_dtype in_dtype, int B, int T, int H, int Dk) {
    if (!gdn_bwd_tc_forward(in_dtype, Dk)) return gdn_bwd_workspace_bytes(B, T, H, Dk);
    return gdn_bwd_forward_offset(B, T, H, Dk) + gdn_total_workspace(gdn_bwd_forward_params(p), B, T, H);
}

ccq_status ccq_gdn_bwd_workspace_size(int B, int T, int H, int Dk, int Dv, ccq_dtype in_dtype,
                                      const ccq_params *p, size_t *bytes) {
    Common c;
    ccq_status st = check_common(p, B, T, H, Dk, Dv, &c);
    if (st != CCQ_OK) return st;
    if (!bytes) return fail(CCQ_ERR_INVALID_ARG, "bytes is NULL");
    if (in_dtype != CCQ_BF16 && in_dtype != CCQ_FP32) return fail(CCQ_ERR_INVALID_ARG, "unknown dtype");
    *bytes = T > 0 ? gdn_bwd_total_workspace(c.p, in_dtype, B, T, H, Dk) : 0;
    return CCQ_OK;
}

ccq_status ccq_gdn_bwd(const void *q, const void *k, const void *v, const float *g, const float *beta,
                       const float *lambda, ccq_dtype in_dtype, const float *S0, const float *C0,
                       const float *m0, const int64_t *t0, const void *dout, const float *dST,
                       const float *dCT, const float *dmT, void *dq, void *dk, void *dv, float *dg,
                       float *dbeta, float *dlambda, float *dS0, float *dC0, float *dm0, int B, int T,
                       int H, int Dk, int Dv, void *workspace, size_t workspace_bytes,
                       const ccq_params *p, void *stream) {
    Common c;
    ccq_status st = check_common(p, B, T, H, Dk, Dv, &c);
    if (st != CCQ_OK) return st;
    if (in_dtype != CCQ_BF16 && in_dtype != CCQ_FP32) return fail(CCQ_ERR_INVALID_ARG, "unknown dtype");
    st = check_ptrs("", {}, {S0, C0, m0, dST, dCT, dmT, dlambda, dS0, dC0, dm0});
    if (st == CCQ_OK) st = check_counts({t0});
    if (st != CCQ_OK) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (T == 0) return copy_state_grads(dST, dCT, dmT, dS0, dC0, dm0, B, H, Dk, Dv, s);
    st = check_ptrs("q,k,v,g,beta,lambda,dout,dq,dk,dv,dg,dbeta",
                    {q, k, v, g, beta, lambda, dout, dq, dk, dv, dg, dbeta}, {});
    if (st != CCQ_OK) return st;
    const size_t need = gdn_bwd_total_workspace(c.p, in_dtype, B, T, H, Dk);
    if (!workspace || workspace_bytes < need)
        return fail(CCQ_ERR_INVALID_ARG, "workspace of %zu bytes required (got %zu)", need,
                    workspace ? workspace_bytes : static_cast<size_t>(0));
    if (!aligned16(workspace)) return fail(CCQ_ERR_INVALID_ARG, "workspace is not 16-byte aligned");
    GdnBwdCall a = {};
    a.B = B; a.T = T; a.H = H; a.D = Dk; a.bf16 = in_dtype == CCQ_BF16;
    a.l2norm = c.p.l2norm_qk; a.centered = c.p.centered; a.scale = c.scale;
    a.q = q; a.k = k; a.v = v; a.dout = dout;
    a.g = g; a.beta = beta; a.lambda = lambda; a.S0 = S0; a.C0 = C0; a.m0 = m0; a.t0 = t0;
    a.dST = dST; a.dCT = dCT; a.dmT = dmT;
    a.dq = dq; a.dk = dk; a.dv = dv; a.dg = dg; a.dbeta = dbeta; a.dlambda = dlambda;
    a.dS0 = dS0; a.dC0 = dC0; a.dm0 = dm0;
    a.workspace = workspace;
    if (gdn_bwd_tc_forward(in_dtype, Dk)) {
        // Tt, S^K_r, M_r and H_r of every chunk from the tensor-core forward (no output written:
        // dq stands in for the output tensor, which the forward must be given)
        GdnDumps d;
        gdn_bwd_state_arrays(a, &d.tt, &d.sk, &d.mk, &d.hs);
        const ccq_params fp = gdn_bwd_forward_params(c.p);
        const size_t off = gdn_bwd_forward_offset(B, T, H, Dk);
        st = gdn_fwd_impl(q, k, v, g, beta, lambda, in_dtype, S0, C0, m0, t0, dq, nullptr, nullptr, nullptr,
                          nullptr, B, T, H, Dk, Dv, static_cast<uint8_t *>(workspace) + off, workspace_bytes - off,
                          &fp, stream, false, &d);
        if (st != CCQ_OK) return st;
        a.states_ready = 1;
    }
    cudaError_t e = launch_gdn_bwd(a, s);
    if (e != cudaSuccess) return cuda_fail(e, "Gated DeltaNet backward launch");
    return CCQ_OK;
}

ccq_status ccq_gdn_decayed_workspace_size(int B, int T, int H, int Dk, int Dv, ccq_dtype in_dtype,
                                          const ccq_params *p, size_t *bytes) {
    Common c;
    ccq_status st = check_common(p, B, T, H, Dk, Dv, &c);
    if (st != CCQ_OK) return st;
    if (!bytes) return fail(CCQ_ERR_INVALID_ARG, "bytes is NULL");
    if (in_dtype != CCQ_BF16 && in_dtype != CCQ_FP32) return fail(CCQ_ERR_INVALID_ARG, "unknown dtype");
    *bytes = T > 0 ? gdn_decayed_workspace_bytes(B, T, H, Dk) : 0;
    return CCQ_OK;
}

ccq_status ccq_gdn_fwd_spectral(const void *q, const void *k, const void *v, const float *g,
                                const float *beta, const float *lambda, ccq_dtype in_dtype,
                                const float *S0, const float *C0, const float *m0, const float *n0,
                                void *o, float *ST, float *CT, float *mT, float *nT, int B, int T, int H,
                                int Dk, int Dv, int contraction, int decayed, void *workspace,
                                size_t workspace_bytes, const ccq_params *p, void *stream) {
    if (contraction < CCQ_CONTRACT_LINEAR || contraction > CCQ_CONTRACT_EXPONENTIAL)
        return fail(CCQ_ERR_INVALID_ARG, "unknown contraction %d", contraction);
    if (decayed != 0 && decayed != 1) return fail(CCQ_ERR_INVALID_ARG, "decayed must be 0 or 1");
    Common c;
    ccq_status st = check_common(p, B, T, H, Dk, Dv, &c);
    if (st != CCQ_OK) return st;
    if (in_dtype != CCQ_BF16 && in_dtype != CCQ_FP32) return fail(CCQ_ERR_INVALID_ARG, "unknown dtype");
    // The fixed CG / Taylor iteration counts are bounded only for unit-norm keys (|lambda Sigma| <= 1).
    if (contraction != CCQ_CONTRACT_LINEAR && !c.p.l2norm_qk)
        return fail(CCQ_ERR_UNSUPPORTED, "the resolvent and exponential contractions need l2norm_qk = 1");
    st = check_ptrs("", {}, {S0, C0, m0, n0, ST, CT, mT, nT});
    if (st != CCQ_OK) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (T == 0) {
        // no tokens: the final states are the initial ones
        const size_t n[4] = {static_cast<size_t>(B) * H * Dk * Dv * 4, static_cast<size_t>(B) * H * Dk * Dk * 4,
                             static_cast<size_t>(B) * H * Dk * 4, static_cast<size_t>(B) * H * 4};
        float *dst[4] = {ST, CT, mT, nT};
        const float *src[4] = {S0, C0, m0, n0};
        for (int i = 0; i < 4; ++i) {
            if (!dst[i] || dst[i] == src[i]) continue;
            cudaError_t e = src[i] ? cudaMemcpyAsync(dst[i], src[i], n[i], cudaMemcpyDeviceToDevice, s)
                                   : cudaMemsetAsync(dst[i], 0, n[i], s);
            if (e != cudaSuccess) return cuda_fail(e, "state copy");
        }
        return CCQ_OK;
    }
    st = check_ptrs("q,k,v,g,beta,lambda,o", {q, k, v, g, beta, lambda, o}, {});
    if (st != CCQ_OK) return st;
    const size_t need = gdn_decayed_workspace_bytes(B, T, H, Dk);
    if (!workspace || workspace_bytes < need)
        return fail(CCQ_ERR_INVALID_ARG, "workspace of %zu bytes required (got %zu)", need,
                    workspace ? workspace_bytes : static_cast<size_t>(0));
    if (!aligned16(workspace)) return fail(CCQ_ERR_INVALID_ARG, "workspace is not 16-byte aligned");
    GdecCall a = {};
    a.B = B; a.T = T; a.H = H; a.D = Dk; a.bf16 = in_dtype == CCQ_BF16;
    a.l2norm = c.p.l2norm_qk; a.centered = c.p.centered; a.scale = c.scale;
    a.q = q; a.k = k; a.v = v; a.g = g; a.beta = beta; a.lambda = lambda;
    a.S0 = S0; a.C0 = C0; a.m0 = m0; a.n0 = n0;
    a.o = o; a.ST = ST; a.CT = CT; a.mT = mT; a.nT = nT;
    a.workspace = workspace;
    a.cov_decay = decayed;
    a.contraction = contraction;
    cudaError_t e = launch_gdn_decayed(a, s);
    if (e != cudaSuccess) return cuda_fail(e, "CUDA-core Gated DeltaNet launch");
    return CCQ_OK;
}

ccq_status ccq_gdn_fwd_decayed(const void *q, const void *k, const void *v, const float *g,
                               const float *beta, const float *lambda, ccq_dtype in_dtype,
                               const float *S0, const float *C0, const float *m0, const float *n0,
                               void *o, float *ST, float *CT, float *mT, float *nT, int B, int T, int H,
                               int Dk, int Dv, void *workspace, size_t workspace_bytes,
                               const ccq_params *p, void *stream) {
    return ccq_gdn_fwd_spectral(q, k, v, g, beta, lambda, in_dtype, S0, C0, m0, n0, o, ST, CT, mT, nT, B, T, H,
                                Dk, Dv, CCQ_CONTRACT_LINEAR, 1, workspace, workspace_bytes, p, stream);
}

// Packed variable-length sequences: validation shared by the call and its workspace query.
// The per-sequence path offsets the fp32 [T][H] row pointers, which must stay 16-byte aligned.
static ccq_status check_varlen(int backbone, const int64_t *cu, int num_seqs, int H, bool per_sequence,
                               long long *max_len) {
    if (backbone != 0 && backbone != 1) return fail(CCQ_ERR_INVALID_ARG, "backbone must be 0 (GLA) or 1 (GDN)");
    if (!cu || num_seqs < 1) return fail(CCQ_ERR_INVALID_ARG, "cu_seqlens is NULL or num_seqs < 1");
    if (cu[0] != 0) return fail(CCQ_ERR_INVALID_ARG, "cu_seqlens[0] must be 0");
    long long mx = 0;
    for (int s = 0; s < num_seqs; ++s) {
        const long long len = cu[s + 1] - cu[s];
        if (len < 0) return fail(CCQ_ERR_INVALID_ARG, "cu_seqlens decreases at %d", s);
        if (len > 0x7fffffffLL) return fail(CCQ_ERR_INVALID_ARG, "sequence %d is too long", s);
        if (per_sequence && (cu[s] * H) % 4 != 0)
            return fail(CCQ_ERR_INVALID_ARG, "cu_seqlens[%d] * H must be a multiple of 4 (16-byte aligned rows)", s);
        mx = std::max(mx, len);
    }
    if (cu[num_seqs] > 0x7fffffffLL) return fail(CCQ_ERR_INVALID_ARG, "packed length too large");
    *max_len = mx;
    return CCQ_OK;
}

// Whether a pack runs as one launch of the chunkwise kernels (bf16, Dk = Dv = 128, a chunkwise
// algo whose kernel reads packed sequences, a non-empty pack); else one call per sequence.
static bool varlen_single_launch(int backbone, ccq_dtype in_dtype, int Dk, int Dv, const ccq_params *p,
                                 long long total) {
    ccq_params c;
    if (p) c = *p;
    else ccq_default_params(&c);
    const bool algo_ok = c.algo == CCQ_ALGO_AUTO || c.algo == CCQ_ALGO_CHUNKWISE ||
                         (backbone == 1 && c.algo == CCQ_ALGO_CHUNKWISE_WIDE);
    return in_dtype == CCQ_BF16 && Dk == 128 && Dv == 128 && algo_ok && total > 0;
}

// Workspace of the single launch: the device copy of cu_seqlens (int64), the first packed chunk
// of every sequence (int32, num_seqs + 1) and the sequence of every packed chunk (int32), then
// (Gated DeltaNet) the UT factor of every packed chunk of every head.
struct VarlenLayout {
    size_t cbase_off, cseq_off, meta_bytes, bytes;
    int chunks;
};

static VarlenLayout varlen_layout(int backbone, const int64_t *cu, int num_seqs, int H) {
    VarlenLayout L{};
    long long nct = 0;
    for (int s = 0; s < num_seqs; ++s) nct += (cu[s + 1] - cu[s] + 63) / 64;
    L.chunks = static_cast<int>(nct);
    L.cbase_off = (8 * static_cast<size_t>(num_seqs + 1) + 15) & ~static_cast<size_t>(15);
    L.cseq_off = L.cbase_off + ((4 * static_cast<size_t>(num_seqs + 1) + 15) & ~static_cast<size_t>(15));
    L.meta_bytes = (L.cseq_off + 4 * static_cast<size_t>(nct) + 255) & ~static_cast<size_t>(255);
    L.bytes = L.meta_bytes + (backbone == 1 ? static_cast<size_t>(nct) * H * 64 * 64 * 2 : 0);
    return L;
}

ccq_status ccq_fwd_varlen_workspace_size(int backbone, const int64_t *cu_seqlens, int num_seqs, int H, int Dk,
                                         int Dv, ccq_dtype in_dtype, const ccq_params *p, size_t *bytes) {
    long long mx = 0;
    ccq_status st = check_varlen(backbone, cu_seqlens, num_seqs, H, false, &mx);
    if (st != CCQ_OK) return st;
    if (!bytes) return fail(CCQ_ERR_INVALID_ARG, "bytes is NULL");
    if (varlen_single_launch(backbone, in_dtype, Dk, Dv, p, cu_seqlens[num_seqs])) {
        *bytes = varlen_layout(backbone, cu_seqlens, num_seqs, H).bytes;
        return CCQ_OK;
    }
    size_t need = 0;
    for (int s = 0; s < num_seqs; ++s) {
        const int len = static_cast<int>(cu_seqlens[s + 1] - cu_seqlens[s]);
        size_t b = 0;
        st = backbone == 0 ? ccq_gla_workspace_size(1, len, H, Dk, Dv, in_dtype, p, &b)
                           : ccq_gdn_workspace_size(1, len, H, Dk, Dv, in_dtype, p, &b);
        if (st != CCQ_OK) return st;
        need = std::max(need, b);
    }
    *bytes = need;
    return CCQ_OK;
}

// One launch over the whole pack (chunkwise kernels with packed-sequence indexing).
static ccq_status varlen_launch(int backbone, const void *q, const void *k, const void *v, const void *gate,
                                const float *beta, const float *lambda, ccq_dtype gate_dtype, const int64_t *cu,
                                int ns, const float *S0, const float *C0, const float *m0, const int64_t *t0,
                                void *o, float *ST, float *CT, float *mT, int64_t *tT, int H, void *workspace,
                                size_t workspace_bytes, const ccq_params *p, cudaStream_t s) {
    Common c;
    const int total = static_cast<int>(cu[ns]);
    ccq_status st = check_common(p, ns, total, H, 128, 128, &c);
    if (st != CCQ_OK) return st;
    if (backbone == 1) st = check_ptrs("q,k,v,g,beta,lambda,o", {q, k, v, gate, beta, lambda, o}, {S0, C0, m0, ST, CT, mT});
    else st = check_ptrs("q,k,v,gk,lambda,o", {q, k, v, gate, lambda, o}, {S0, C0, m0, ST, CT, mT});
    if (st == CCQ_OK) st = check_counts({t0, tT});
    if (st != CCQ_OK) return st;
    const VarlenLayout L = varlen_layout(backbone, cu, ns, H);
    if (!workspace || workspace_bytes < L.bytes)
        return fail(CCQ_ERR_INVALID_ARG, "workspace of %zu bytes required (got %zu)", L.bytes,
                    workspace ? workspace_bytes : static_cast<size_t>(0));
    if (!aligned16(workspace)) return fail(CCQ_ERR_INVALID_ARG, "workspace is not 16-byte aligned");
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    ChunkArgs a = {};
    ChunkMaps gm;
    GdnMaps dm;
    const int geb = gate_dtype == CCQ_BF16 ? 2 : 4;
    bool ok = make_token_map(&gm.q, q, 2, 1, total, H, 128, 64, true) &&
              make_token_map(&gm.k, k, 2, 1, total, H, 128, 64, true) &&
              make_token_map(&gm.v, v, 2, 1, total, H, 128, 64, true) &&
              make_token_map(&gm.o, o, 2, 1, total, H, 128, 64, true);
    if (ok && backbone == 0) ok = make_token_map(&gm.g, gate, geb, 1, total, H, 128, 128, false);
    if (ok && backbone == 1) {
        dm.q = gm.q; dm.k = gm.k; dm.v = gm.v; dm.o = gm.o;
        ok = make_rows_map(&dm.tb, ws + L.meta_bytes, static_cast<long long>(L.chunks) * H * 64, 64);
    }
    if (!ok) return fail(CCQ_ERR_CUDA, "cuTensorMapEncodeTiled failed (driver entry point missing or map rejected)");
    a.status = device_status_word();
    if (!a.status) return fail(CCQ_ERR_CUDA, "cannot resolve the device status word");
    // the pack's offsets, chunk bases and chunk -> sequence map, staged on the host and copied in
    // one transfer (from pageable memory: the copy is staged before this call returns)
    {
        uint8_t *meta = static_cast<uint8_t *>(malloc(L.meta_bytes));
        if (!meta) return fail(CCQ_ERR_INVALID_ARG, "out of host memory for %zu bytes", L.meta_bytes);
        memcpy(meta, cu, 8 * static_cast<size_t>(ns + 1));
        int *cbase = reinterpret_cast<int *>(meta + L.cbase_off);
        int *cseq = reinterpret_cast<int *>(meta + L.cseq_off);
        int acc = 0;
        for (int sq = 0; sq < ns; ++sq) {
            cbase[sq] = acc;
            const int nc = static_cast<int>((cu[sq + 1] - cu[sq] + 63) / 64);
            for (int r = 0; r < nc; ++r) cseq[acc + r] = sq;
            acc += nc;
        }
        cbase[ns] = acc;
        cudaError_t e = cudaMemcpyAsync(ws, meta, L.meta_bytes, cudaMemcpyHostToDevice, s);
        free(meta);
        if (e != cudaSuccess) return cuda_fail(e, "packed-sequence offsets copy");
    }
    a.B = ns; a.T = total; a.H = H;
    a.gate_dtype = gate_dtype == CCQ_BF16 ? 0 : 1;
    a.l2norm = c.p.l2norm_qk; a.centered = c.p.centered; a.scale = c.scale;
    a.lambda = lambda; a.gk = gate;
    a.g = static_cast<const float *>(gate); a.beta = beta;
    a.S0 = S0; a.C0 = C0; a.m0 = m0; a.t0 = t0;
    a.o = static_cast<__nv_bfloat16 *>(o);
    a.ST = ST; a.CT = CT; a.mT = mT;
    a.nseg = 1;
    a.cu = reinterpret_cast<const int64_t *>(ws);
    a.cbase = reinterpret_cast<const int *>(ws + L.cbase_off);
    a.chunk_seq = reinterpret_cast<const int *>(ws + L.cseq_off);
    a.vl_chunks = L.chunks;
    cudaError_t e = backbone == 0 ? launch_gla_chunk(a, gm, s) : launch_gdn_chunk(a, dm, s);
    if (e != cudaSuccess) return cuda_fail(e, "packed-sequence chunkwise launch");
    e = launch_t_update_varlen(t0, tT, a.cu, ns, s);
    if (e != cudaSuccess) return cuda_fail(e, "position update launch");
    return CCQ_OK;
}

ccq_status ccq_fwd_varlen(int backbone, const void *q, const void *k, const void *v, const void *gate,
                          const float *beta, const float *lambda, ccq_dtype in_dtype, ccq_dtype gate_dtype,
                          const int64_t *cu_seqlens, int num_seqs, const float *S0, const float *C0,
                          const float *m0, const int64_t *t0, void *o, float *ST, float *CT, float *mT,
                          int64_t *tT, int H, int Dk, int Dv, void *workspace, size_t workspace_bytes,
                          const ccq_params *p, void *stream) {
    long long mx = 0;
    ccq_status st = check_varlen(backbone, cu_seqlens, num_seqs, H, false, &mx);
    if (st != CCQ_OK) return st;
    if ((in_dtype != CCQ_BF16 && in_dtype != CCQ_FP32) || (gate_dtype != CCQ_BF16 && gate_dtype != CCQ_FP32))
        return fail(CCQ_ERR_INVALID_ARG, "unknown dtype");
    if (backbone == 1 && gate_dtype != CCQ_FP32) return fail(CCQ_ERR_INVALID_ARG, "Gated DeltaNet decay must be fp32");
    if (varlen_single_launch(backbone, in_dtype, Dk, Dv, p, cu_seqlens[num_seqs]))
        return varlen_launch(backbone, q, k, v, gate, beta, lambda, gate_dtype, cu_seqlens, num_seqs, S0, C0, m0,
                             t0, o, ST, CT, mT, tT, H, workspace, workspace_bytes, p,
                             static_cast<cudaStream_t>(stream));
    st = check_varlen(backbone, cu_seqlens, num_seqs, H, true, &mx);
    if (st != CCQ_OK) return st;
    size_t need = 0;
    st = ccq_fwd_varlen_workspace_size(backbone, cu_seqlens, num_seqs, H, Dk, Dv, in_dtype, p, &need);
    if (st != CCQ_OK) return st;
    if (need && (!workspace || workspace_bytes < need))
        return fail(CCQ_ERR_INVALID_ARG, "workspace of %zu bytes required (got %zu)", need,
                    workspace ? workspace_bytes : static_cast<size_t>(0));
    const size_t esz = in_dtype == CCQ_BF16 ? 2 : 4, gsz = gate_dtype == CCQ_BF16 ? 2 : 4;
    const size_t h = static_cast<size_t>(H);
    ccq_params pin;
    if (p) pin = *p;
    else ccq_default_params(&pin);
    ccq_params pempty = pin;  // an empty sequence passes its state through on any path
    pempty.algo = CCQ_ALGO_AUTO;
    // Otherwise one call of the (batch-1) forward per sequence, in stream order: the calls share
    // the workspace, and sequence s reads and writes row s of every state.  Pass 0 checks every
    // call's arguments, pass 1 launches, so that a rejected pack enqueues nothing.
    for (int pass = 0; pass < 2; ++pass)
    for (int s = 0; s < num_seqs; ++s) {
        const size_t off = static_cast<size_t>(cu_seqlens[s]);
        const int len = static_cast<int>(cu_seqlens[s + 1] - cu_seqlens[s]);
        auto at = [&](const void *base, size_t bytes_per_token) -> const void * {
            return base ? static_cast<const uint8_t *>(base) + off * bytes_per_token : nullptr;
        };
        auto row = [&](const float *base, size_t per) -> const float * { return base ? base + s * per : nullptr; };
        auto rowm = [&](float *base, size_t per) -> float * { return base ? base + s * per : nullptr; };
        const void *qs = at(q, h * Dk * esz), *ks = at(k, h * Dk * esz), *vs = at(v, h * Dv * esz);
        void *os = const_cast<void *>(at(o, h * Dv * esz));
        const float *ls = static_cast<const float *>(at(lambda, h * 4));
        const size_t sS = h * Dk * Dv, sC = h * Dk * Dk, sm = h * Dk;
        const int64_t *t0s = t0 ? t0 + s : nullptr;
        int64_t *tTs = tT ? tT + s : nullptr;
        const ccq_params *ps = len > 0 ? &pin : &pempty;
        const bool dry = pass == 0;
        if (backbone == 0) {
            st = gla_fwd_impl(qs, ks, vs, at(gate, h * Dk * gsz), ls, in_dtype, gate_dtype, row(S0, sS), row(C0, sC),
                              row(m0, sm), t0s, os, rowm(ST, sS), rowm(CT, sC), rowm(mT, sm), tTs, 1, len, H, Dk, Dv,
                              workspace, workspace_bytes, nullptr, 0, ps, stream, dry);
        } else {
            st = gdn_fwd_impl(qs, ks, vs, static_cast<const float *>(at(gate, h * 4)),
                              static_cast<const float *>(at(beta, h * 4)), ls, in_dtype, row(S0, sS), row(C0, sC),
                              row(m0, sm), t0s, os, rowm(ST, sS), rowm(CT, sC), rowm(mT, sm), tTs, 1, len, H, Dk, Dv,
                              workspace, workspace_bytes, ps, stream, dry);
        }
        if (st != CCQ_OK) return st;
    }
    return CCQ_OK;
}

ccq_status ccq_decode_step(int backbone, const void *q, const void *k, const void *v,
                           const void *gate, const float *beta, const float *lambda,
                           ccq_dtype in_dtype, ccq_dtype gate_dtype, float *S, float *C,
                           float *m, int64_t *t, void *o, int B, int H, int Dk, int Dv,
                           const ccq_params *p, void *stream) {
    Common c;
    ccq_status st = check_common(p, B, 1, H, Dk, Dv, &c);
    if (st != CCQ_OK) return st;
    if (backbone != 0 && backbone != 1) return fail(CCQ_ERR_INVALID_ARG, "backbone must be 0 (GLA) or 1 (GDN)");
    if ((in_dtype != CCQ_BF16 && in_dtype != CCQ_FP32) || (gate_dtype != CCQ_BF16 && gate_dtype != CCQ_FP32))
        return fail(CCQ_ERR_INVALID_ARG, "unknown dtype");
    if (backbone == 1 && gate_dtype != CCQ_FP32)
        return fail(CCQ_ERR_INVALID_ARG, "Gated DeltaNet decay must be fp32");
    if (backbone == 1) st = check_ptrs("q,k,v,gate,beta,lambda,S,C,m,t,o", {q, k, v, gate, beta, lambda, S, C, m, t, o}, {});
    else st = check_ptrs("q,k,v,gate,lambda,S,C,m,t,o", {q, k, v, gate, lambda, S, C, m, t, o}, {});
    if (st != CCQ_OK) return st;
    RecurrentArgs ra = {};
    ra.backbone = backbone; ra.B = B; ra.T = 1; ra.H = H; ra.Dk = Dk; ra.Dv = Dv;
    ra.in_dtype = in_dtype; ra.gate_dtype = gate_dtype;
    ra.l2norm = c.p.l2norm_qk; ra.centered = c.p.centered; ra.scale = c.scale;
    ra.q = q; ra.k = k; ra.v = v; ra.gate = gate; ra.beta = beta; ra.lambda = lambda;
    ra.S0 = S; ra.C0 = C; ra.m0 = m; ra.t0 = t;
    ra.o = o; ra.ST = S; ra.CT = C; ra.mT = m;
    st = run_recurrent(ra, static_cast<cudaStream_t>(stream));
    return st != CCQ_OK ? st : finish_t(t, t, B, 1, static_cast<cudaStream_t>(stream));
}

ccq_status ccq_device_status(void *stream) {
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(e, "stream synchronize");
    int v = 0;
    e = cudaMemcpyFromSymbol(&v, ccq::g_status, sizeof(int));
    if (e != cudaSuccess) return cuda_fail(e, "read device status");
    if (v != 0) {
        const int zero = 0;
        e = cudaMemcpyToSymbol(ccq::g_status, &zero, sizeof(int));
        if (e != cudaSuccess) return cuda_fail(e, "clear device status");
        if (v == static_cast<int>(CCQ_ERR_RANGE))  // the kernels write the status code itself
            return fail(CCQ_ERR_RANGE, "device status %d: a chunk's cumulative log gates over 16 tokens fell "
                                       "below about -87 (see ccq_gla_fwd); the outputs are not valid", v);
        return fail(CCQ_ERR_TIMEOUT, "device status %d: an in-kernel wait gave up", v);
    }
    return CCQ_OK;
}

}  // extern "C"
