// C ABI of libleap: argument validation, launch selection, error mapping.
// Every entry point is declared and documented in include/leap.h.
#include "../../include/leap.h"
#include "leap_internal.h"

#include <cuda_runtime.h>
#include <math.h>
#include <mutex>

namespace leap {

// Sticky per-device status word (LEAP_DEV_* bits).
__device__ unsigned int g_leap_status;

namespace {

constexpr int kMaxDevices = 64;

std::mutex g_mu;
unsigned int* g_status_ptr[kMaxDevices] = {};
int g_sm_count[kMaxDevices] = {};

int current_device() {
    int d = 0;
    if (cudaGetDevice(&d) != cudaSuccess || d < 0 || d >= kMaxDevices) return -1;
    return d;
}

// Device address of g_leap_status on the current device (host code may not
// use the symbol itself as a pointer).
unsigned int* status_ptr() {
    const int d = current_device();
    if (d < 0) return nullptr;
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_status_ptr[d]) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_leap_status) != cudaSuccess) return nullptr;
        g_status_ptr[d] = static_cast<unsigned int*>(p);
    }
    return g_status_ptr[d];
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

leap_status_t from_cuda(cudaError_t e) {
    if (e == cudaSuccess) return LEAP_OK;
    if (e == cudaErrorNotSupported) return LEAP_ERR_UNSUPPORTED;
    return LEAP_ERR_CUDA;
}

bool finite(float x) { return isfinite(x) != 0; }

// Common checks of a bf16 logits matrix and its per-row vectors.
bool rows_ok(const uint16_t* logits, int64_t ld, const int32_t* ids, int64_t N, int32_t V) {
    if (N < 0 || V < 1 || ld < V || (ld & 7) != 0) return false;
    if (N > 0 && (!logits || !ids || !aligned16(logits))) return false;
    if (N > (int64_t)0x7fffffff) return false;
    return true;
}

}  // namespace

unsigned int* device_status_ptr() { return status_ptr(); }

int device_sm_count() {
    const int d = current_device();
    if (d < 0) return 132;
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_sm_count[d]) {
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, d) != cudaSuccess || n <= 0) n = 132;
        g_sm_count[d] = n;
    }
    return g_sm_count[d];
}

}  // namespace leap

using namespace leap;

extern "C" {

const char* leap_status_string(leap_status_t s) {
    switch (s) {
        case LEAP_OK: return "LEAP_OK";
        case LEAP_ERR_INVALID_ARG: return "LEAP_ERR_INVALID_ARG";
        case LEAP_ERR_UNSUPPORTED: return "LEAP_ERR_UNSUPPORTED";
        case LEAP_ERR_CUDA: return "LEAP_ERR_CUDA";
        case LEAP_ERR_TIMEOUT: return "LEAP_ERR_TIMEOUT";
        case LEAP_ERR_BAD_INDEX: return "LEAP_ERR_BAD_INDEX";
    }
    return "LEAP_ERR_UNKNOWN";
}

int32_t leap_version(void) { return 100; }

leap_status_t leap_get_device_status(uint32_t* host_flags, void* stream) {
    if (!host_flags) return LEAP_ERR_INVALID_ARG;
    unsigned int* p = status_ptr();
    if (!p) return LEAP_ERR_CUDA;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    unsigned int v = 0;
    cudaError_t e = cudaMemcpyAsync(&v, p, sizeof(v), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(p, 0, sizeof(unsigned int), s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return LEAP_ERR_CUDA;
    *host_flags = v;
    return v ? LEAP_ERR_BAD_INDEX : LEAP_OK;
}

leap_status_t leap_group_rank_advantages(const leap_rank_params_t* p, const int8_t* pass_turn,
                                         const int8_t* num_turns, const float* speedup, const int32_t* ntokens,
                                         const uint8_t* gate_in, uint8_t* gate_out, uint8_t* r_out,
                                         int32_t* n_worse, int32_t* n_better, float* R, float* A,
                                         float* turn_adv, uint8_t* T_eff, leap_rank_stats_t* stats,
                                         void* stream) {
    if (!p) return LEAP_ERR_INVALID_ARG;
    if (p->num_groups < 0 || p->G < 2 || p->G > 1024 || p->M < 1 || p->M > 8) return LEAP_ERR_INVALID_ARG;
    if (!gate_in && (p->tau_min < 0 || p->tau_min > p->tau_max || p->tau_max > p->G)) return LEAP_ERR_INVALID_ARG;
    if (!finite(p->gamma) || !(p->gamma > 0.f) || p->gamma > 1.f) return LEAP_ERR_INVALID_ARG;
    if (!finite(p->eps_std) || p->eps_std < 0.f) return LEAP_ERR_INVALID_ARG;
    if (p->norm != LEAP_ADVNORM_GRPO_STD && p->norm != LEAP_ADVNORM_NONE) return LEAP_ERR_INVALID_ARG;
    if (p->std_unbiased != 0 && p->std_unbiased != 1) return LEAP_ERR_INVALID_ARG;
    if (p->cmp != LEAP_CMP_PAPER && p->cmp != LEAP_CMP_LEXI) return LEAP_ERR_INVALID_ARG;
    if (p->reward != LEAP_REWARD_RANK && p->reward != LEAP_REWARD_STATIC) return LEAP_ERR_INVALID_ARG;
    if (!finite(p->static_c) || p->static_c < 0.f || p->static_c > 1.f) return LEAP_ERR_INVALID_ARG;
    if (p->num_groups > 0 && (!pass_turn || !num_turns || !turn_adv || !T_eff)) return LEAP_ERR_INVALID_ARG;
    if (p->num_groups > 0 && p->cmp == LEAP_CMP_LEXI && (!speedup || !ntokens)) return LEAP_ERR_INVALID_ARG;
    RankArgs a;
    a.num_groups = p->num_groups;
    a.G = p->G;
    a.M = p->M;
    a.tau_min = p->tau_min;
    a.tau_max = p->tau_max;
    a.gamma = p->gamma;
    a.eps_std = p->eps_std;
    a.cmp = p->cmp;
    a.norm = p->norm;
    a.std_unbiased = p->std_unbiased;
    a.reward = p->reward;
    a.static_c = p->static_c;
    a.stats = stats;
    a.pass_turn = pass_turn;
    a.num_turns = num_turns;
    a.speedup = speedup;
    a.ntokens = ntokens;
    a.gate_in = gate_in;
    a.gate_out = gate_out;
    a.r_out = r_out;
    a.n_worse = n_worse;
    a.n_better = n_better;
    a.R = R;
    a.A = A;
    a.turn_adv = turn_adv;
    a.T_eff = T_eff;
    a.status = status_ptr();
    if (!a.status) return LEAP_ERR_CUDA;
    return from_cuda(launch_rank_advantages(a, static_cast<cudaStream_t>(stream)));
}

static bool seg_args_ok(int64_t N, int32_t n_rollouts, int32_t M, const int32_t* seg_offsets,
                        const int32_t* seg_rollout, const int8_t* seg_turn, int32_t num_segs, const uint8_t* T_eff) {
    if (N < 0 || N > (int64_t)0x7fffffff || n_rollouts < 0 || M < 1 || M > 8 || num_segs < 0) return false;
    if (num_segs > 0 && (!seg_offsets || !seg_rollout || !seg_turn)) return false;
    if (n_rollouts > 0 && !T_eff) return false;
    return true;
}

leap_status_t leap_rollout_token_counts(int64_t N, int32_t n_rollouts, int32_t M, const int32_t* seg_offsets,
                                        const int32_t* seg_rollout, const int8_t* seg_turn, int32_t num_segs,
                                        const uint8_t* T_eff, int32_t* L, int64_t* totals, void* stream) {
    if (!seg_args_ok(N, n_rollouts, M, seg_offsets, seg_rollout, seg_turn, num_segs, T_eff)) return LEAP_ERR_INVALID_ARG;
    if (!totals || (n_rollouts > 0 && !L)) return LEAP_ERR_INVALID_ARG;
    SegArgs a = {};
    a.N = N;
    a.n_rollouts = n_rollouts;
    a.M = M;
    a.num_segs = num_segs;
    a.seg_offsets = seg_offsets;
    a.seg_rollout = seg_rollout;
    a.seg_turn = seg_turn;
    a.T_eff = T_eff;
    a.L_out = L;
    a.totals_out = totals;
    a.status = status_ptr();
    if (!a.status) return LEAP_ERR_CUDA;
    return from_cuda(launch_token_counts(a, static_cast<cudaStream_t>(stream)));
}

leap_status_t leap_scatter_turn_advantages(int64_t N, int32_t n_rollouts, int32_t M, const int32_t* seg_offsets,
                                           const int32_t* seg_rollout, const int8_t* seg_turn, int32_t num_segs,
                                           const float* turn_adv, const uint8_t* T_eff, const int32_t* L,
                                           const int64_t* totals, int32_t agg, float* adv_out, float* w_out,
                                           void* stream) {
    if (!seg_args_ok(N, n_rollouts, M, seg_offsets, seg_rollout, seg_turn, num_segs, T_eff)) return LEAP_ERR_INVALID_ARG;
    if (agg != LEAP_AGG_SEQ_MEAN_TOKEN_MEAN && agg != LEAP_AGG_TOKEN_MEAN) return LEAP_ERR_INVALID_ARG;
    if (N > 0 && (!adv_out || !w_out || !totals)) return LEAP_ERR_INVALID_ARG;
    if (n_rollouts > 0 && (!turn_adv || !L)) return LEAP_ERR_INVALID_ARG;
    SegArgs a = {};
    a.N = N;
    a.n_rollouts = n_rollouts;
    a.M = M;
    a.num_segs = num_segs;
    a.seg_offsets = seg_offsets;
    a.seg_rollout = seg_rollout;
    a.seg_turn = seg_turn;
    a.T_eff = T_eff;
    a.turn_adv = turn_adv;
    a.L_in = L;
    a.totals_in = totals;
    a.agg = agg;
    a.adv_out = adv_out;
    a.w_out = w_out;
    a.status = status_ptr();
    if (!a.status) return LEAP_ERR_CUDA;
    return from_cuda(launch_scatter(a, static_cast<cudaStream_t>(stream)));
}

leap_status_t leap_token_advantages(int64_t N, int32_t n_rollouts, int32_t M, const int32_t* seg_offsets,
                                    const int32_t* seg_rollout, const int8_t* seg_turn, int32_t num_segs,
                                    const float* turn_adv, const uint8_t* T_eff, int32_t agg, int32_t* L,
                                    int64_t* totals, float* adv_out, float* w_out, void* stream) {
    if (!seg_args_ok(N, n_rollouts, M, seg_offsets, seg_rollout, seg_turn, num_segs, T_eff)) return LEAP_ERR_INVALID_ARG;
    if (agg != LEAP_AGG_SEQ_MEAN_TOKEN_MEAN && agg != LEAP_AGG_TOKEN_MEAN) return LEAP_ERR_INVALID_ARG;
    if (!totals || (n_rollouts > 0 && (!L || !turn_adv)) || (N > 0 && (!adv_out || !w_out)))
        return LEAP_ERR_INVALID_ARG;
    SegArgs a = {};
    a.N = N;
    a.n_rollouts = n_rollouts;
    a.M = M;
    a.num_segs = num_segs;
    a.seg_offsets = seg_offsets;
    a.seg_rollout = seg_rollout;
    a.seg_turn = seg_turn;
    a.T_eff = T_eff;
    a.turn_adv = turn_adv;
    a.L_out = L;
    a.totals_out = totals;
    a.agg = agg;
    a.adv_out = adv_out;
    a.w_out = w_out;
    a.status = status_ptr();
    if (!a.status) return LEAP_ERR_CUDA;
    return from_cuda(launch_token_advantages(a, static_cast<cudaStream_t>(stream)));
}

leap_status_t leap_token_logprobs(const uint16_t* logits, int64_t ld, const int32_t* ids, int64_t N, int32_t V,
                                  float inv_temp, float* logp, float* lse, void* stream) {
    if (!rows_ok(logits, ld, ids, N, V)) return LEAP_ERR_INVALID_ARG;
    if (!finite(inv_temp) || !(inv_temp > 0.f)) return LEAP_ERR_INVALID_ARG;
    if (N > 0 && !logp) return LEAP_ERR_INVALID_ARG;
    RowArgs a = {};
    a.logits = logits;
    a.ld = ld;
    a.ids = ids;
    a.N = N;
    a.V = V;
    a.inv_temp = inv_temp;
    a.logp = logp;
    a.lse = lse;
    a.status = status_ptr();
    if (!a.status) return LEAP_ERR_CUDA;
    return from_cuda(launch_row_stream(a, 0, static_cast<cudaStream_t>(stream)));
}

static bool loss_params_ok(const leap_loss_params_t* p) {
    if (!p) return false;
    if (!finite(p->eps_low) || !finite(p->eps_high) || p->eps_low < 0.f || p->eps_high < 0.f) return false;
    if (!finite(p->inv_temp) || !(p->inv_temp > 0.f) || !finite(p->grad_scale)) return false;
    if (p->flags & ~(LEAP_LOSS_ACCUMULATE | LEAP_LOSS_SINGLE_READ | LEAP_LOSS_INTERLEAVED_ROWS)) return false;
    return true;
}

size_t leap_grpo_loss_workspace_size(int64_t N, int32_t V) {
    (void)V;
    if (N < 0) return 0;
    return loss_workspace_bytes(N);
}

leap_status_t leap_grpo_loss_fwd(const leap_loss_params_t* p, const uint16_t* logits, int64_t ld,
                                 const int32_t* ids, const float* old_logp, const float* adv, const float* w,
                                 int64_t N, int32_t V, float* loss, float* logp, float* lse, float* ell,
                                 uint16_t* dlogits, void* workspace, size_t ws_bytes, leap_loss_stats_t* stats,
                                 void* stream) {
    if (!loss_params_ok(p) || !rows_ok(logits, ld, ids, N, V)) return LEAP_ERR_INVALID_ARG;
    if (!loss) return LEAP_ERR_INVALID_ARG;
    if (N > 0 && (!old_logp || !adv || !w)) return LEAP_ERR_INVALID_ARG;
    if (dlogits && !aligned16(dlogits)) return LEAP_ERR_INVALID_ARG;
    if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return LEAP_ERR_INVALID_ARG;
    if (ws_bytes < loss_workspace_bytes(N)) return LEAP_ERR_INVALID_ARG;
    // Rows of at most kShortRowMaxV columns take the short-row kernel whatever
    // the flag (a group of warps holds each row on chip, read once), where the
    // pipelined kernel's 16 KB staging chunks would be mostly empty.
    const bool single_read = (p->flags & LEAP_LOSS_SINGLE_READ) != 0 || V <= kShortRowMaxV;
    if (dlogits && single_read && (int64_t)V > fused_max_vocab()) return LEAP_ERR_UNSUPPORTED;
    const LossWorkspace ws = carve_loss_workspace(workspace, N);
    RowArgs a = {};
    a.logits = logits;
    a.ld = ld;
    a.ids = ids;
    a.old_logp = old_logp;
    a.adv = adv;
    a.w = w;
    a.N = N;
    a.V = V;
    a.eps_low = p->eps_low;
    a.eps_high = p->eps_high;
    a.inv_temp = p->inv_temp;
    a.grad_scale = p->grad_scale;
    a.logp = logp;
    a.lse = lse;
    a.ell = ell;
    a.dlogits = dlogits;
    a.ws_contrib = ws.contrib;
    a.ws_rho = ws.rho;
    a.ws_flag = ws.flag;
    a.row_streams = (p->flags & LEAP_LOSS_INTERLEAVED_ROWS) ? 2 : 1;
    a.status = status_ptr();
    if (!a.status) return LEAP_ERR_CUDA;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = dlogits ? launch_fused_loss(a, single_read, s) : launch_row_stream(a, 1, s);
    if (e != cudaSuccess) return from_cuda(e);
    return from_cuda(launch_loss_reduce(ws, N, loss, stats, (p->flags & LEAP_LOSS_ACCUMULATE) != 0, s));
}

leap_status_t leap_grpo_loss_bwd(const leap_loss_params_t* p, const uint16_t* logits, int64_t ld,
                                 const int32_t* ids, const float* old_logp, const float* adv, const float* w,
                                 const float* lse, int64_t N, int32_t V, uint16_t* dlogits, void* stream) {
    if (!loss_params_ok(p) || !rows_ok(logits, ld, ids, N, V)) return LEAP_ERR_INVALID_ARG;
    if (N > 0 && (!old_logp || !adv || !w || !lse || !dlogits)) return LEAP_ERR_INVALID_ARG;
    if (dlogits && !aligned16(dlogits)) return LEAP_ERR_INVALID_ARG;
    RowArgs a = {};
    a.logits = logits;
    a.ld = ld;
    a.ids = ids;
    a.old_logp = old_logp;
    a.adv = adv;
    a.w = w;
    a.lse_in = lse;
    a.N = N;
    a.V = V;
    a.eps_low = p->eps_low;
    a.eps_high = p->eps_high;
    a.inv_temp = p->inv_temp;
    a.grad_scale = p->grad_scale;
    a.dlogits = dlogits;
    a.status = status_ptr();
    if (!a.status) return LEAP_ERR_CUDA;
    return from_cuda(launch_split_bwd(a, static_cast<cudaStream_t>(stream)));
}

}  // extern "C"
