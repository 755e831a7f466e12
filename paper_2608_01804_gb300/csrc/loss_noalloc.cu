// leap_grpo_loss_fwd_noalloc: the clipped-surrogate forward (+ fused dlogits)
// for callers that cannot allocate device memory at the call site, e.g. a C
// program that links only this library and has no device allocator of its
// own, or a process whose device-memory budget is fixed up front by a pool
// that forbids further cudaMalloc.  Its scratch lives in a file-scope device
// array instead of a caller-provided workspace.  The paper has no
// counterpart: this is a property of the library's interface only.
#include "../../include/leap.h"
#include "leap_internal.h"

#include <cuda_runtime.h>
#include <mutex>

namespace {

constexpr int64_t kNoAllocMaxRows = LEAP_NOALLOC_MAX_ROWS;
constexpr size_t kNoAllocBytes = (size_t)1 << 20;  // >= the workspace of kNoAllocMaxRows rows

// One copy per device that loads the library, held until the process exits.
// Every call shares it; see leap.h for the consequences.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocBytes];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void* g_scratch_ptr[kMaxDevices] = {};

// Device address of g_noalloc_scratch on the current device.  In host code the
// array's name is only a host-side stand-in, so the address is looked up once
// per device with that device current, and cached.
void* scratch_on_current_device() {
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_scratch_ptr[dev]) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return nullptr;
        g_scratch_ptr[dev] = p;
    }
    return g_scratch_ptr[dev];
}

}  // namespace

extern "C" leap_status_t leap_grpo_loss_fwd_noalloc(
    const leap_loss_params_t* params, const uint16_t* logits, int64_t ld, const int32_t* ids,
    const float* old_logp, const float* adv, const float* w, int64_t N, int32_t V, float* loss, float* logp,
    float* lse, float* ell, uint16_t* dlogits, leap_loss_stats_t* stats, void* stream) {
    if (N < 0 || N > kNoAllocMaxRows) return LEAP_ERR_INVALID_ARG;
    if (leap::loss_workspace_bytes(N) > kNoAllocBytes) return LEAP_ERR_INVALID_ARG;
    void* scratch = scratch_on_current_device();
    if (!scratch) return LEAP_ERR_CUDA;
    return leap_grpo_loss_fwd(params, logits, ld, ids, old_logp, adv, w, N, V, loss, logp, lse, ell, dlogits,
                              scratch, kNoAllocBytes, stats, stream);
}
