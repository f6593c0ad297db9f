// ccq_noalloc.cu -- a CCQ-GLA forward for callers that cannot hand the library
// any device memory of its own.
//
// ccq_gla_fwd needs a caller workspace when it splits long sequences into
// segments (the per-segment states).  Some callers cannot provide one: an
// engine that reserved all device memory for its own caches at start-up and
// has no allocator left to draw from, or code on a path where a device
// allocation is not permitted or would stall the device.  This entry point
// takes the same inputs and outputs as ccq_gla_fwd but keeps that scratch in a
// fixed array compiled into the library, so it never allocates.
#include <cuda_runtime.h>
#include <stdio.h>

#include <mutex>

#include "../../include/ccq.h"
#include "ccq_internal.h"

namespace {

// Size of the fixed scratch: 24 MiB, room for 190 (sequence, segment) states
// of 129 KiB each.  Every GPU that loads the library keeps this array until the
// process exits.
constexpr size_t kFixedScratchBytes = 24u << 20;

}  // namespace

static __device__ __align__(256) unsigned char g_fixed_scratch[kFixedScratchBytes];

namespace {

// Device address of g_fixed_scratch on the current device.  In host code the
// symbol's name is only a host-side handle, so the address is asked from the
// runtime once per device (with that device current) and cached.
void *fixed_scratch_address() {
    static std::mutex mu;
    static void *addr[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
    std::lock_guard<std::mutex> lock(mu);
    if (!addr[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_fixed_scratch) != cudaSuccess) return nullptr;
        addr[dev] = p;
    }
    return addr[dev];
}

}  // namespace

extern "C" CCQ_API ccq_status ccq_gla_fwd_fixed_scratch(
    const void *q, const void *k, const void *v, const void *gk, const float *lambda, ccq_dtype in_dtype,
    ccq_dtype gate_dtype, const float *S0, const float *C0, const float *m0, const int64_t *t0, void *o,
    float *ST, float *CT, float *mT, int64_t *tT, int B, int T, int H, int Dk, int Dv, const ccq_params *p,
    void *stream) {
    size_t need = 0;
    ccq_status st = ccq_gla_workspace_size(B, T, H, Dk, Dv, in_dtype, p, &need);
    if (st != CCQ_OK) return st;
    if (need > kFixedScratchBytes) {
        char msg[256];
        snprintf(msg, sizeof msg,
                 "this launch needs %zu bytes of scratch; the fixed scratch of "
                 "ccq_gla_fwd_fixed_scratch holds %zu (use ccq_gla_fwd with a workspace, "
                 "or fewer (batch, head) sequences / a smaller seq_split)",
                 need, kFixedScratchBytes);
        return static_cast<ccq_status>(ccq::record_error_code(CCQ_ERR_INVALID_ARG, msg));
    }
    void *ws = nullptr;
    if (need > 0) {
        ws = fixed_scratch_address();
        if (!ws)
            return static_cast<ccq_status>(
                ccq::record_error_code(CCQ_ERR_CUDA, "cudaGetSymbolAddress of the fixed scratch failed"));
    }
    // Every slot of the scratch that a launch reads is written earlier in the same
    // launch, so nothing in it has to start at zero.
    return ccq_gla_fwd(q, k, v, gk, lambda, in_dtype, gate_dtype, S0, C0, m0, t0, o, ST, CT, mT, tT, B, T, H,
                       Dk, Dv, ws, ws ? kFixedScratchBytes : 0, p, stream);
}
