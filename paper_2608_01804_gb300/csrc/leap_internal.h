// Internal launch interface between the C-ABI layer (leap_api.cu) and the
// kernel translation units.  Host arguments are already validated here.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace leap {

struct RankArgs {
    int32_t num_groups, G, M, tau_min, tau_max;
    float gamma, eps_std;
    int32_t cmp, norm, std_unbiased, reward;
    float static_c;
    const int8_t* pass_turn;
    const int8_t* num_turns;
    const float* speedup;
    const int32_t* ntokens;
    const uint8_t* gate_in;
    uint8_t* gate_out;
    uint8_t* r_out;
    int32_t* n_worse;
    int32_t* n_better;
    float* R;
    float* A;
    float* turn_adv;
    uint8_t* T_eff;
    void* stats;  // leap_rank_stats_t*, accumulated
    unsigned int* status;
};

struct SegArgs {
    int64_t N;
    int32_t n_rollouts, M, num_segs;
    const int32_t* seg_offsets;
    const int32_t* seg_rollout;
    const int8_t* seg_turn;
    const uint8_t* T_eff;
    const float* turn_adv;
    int32_t* L_out;
    const int32_t* L_in;
    int64_t* totals_out;
    const int64_t* totals_in;
    int32_t agg;
    float* adv_out;
    float* w_out;
    unsigned int* status;
};

// Per-row loss-path arguments.  Any output pointer may be null.
struct RowArgs {
    const uint16_t* logits;
    int64_t ld;
    const int32_t* ids;
    const float* old_logp;
    const float* adv;
    const float* w;
    const float* lse_in;  // split backward only
    int64_t N;
    int32_t V;
    float eps_low, eps_high, inv_temp, grad_scale;
    float* logp;
    float* lse;
    float* ell;
    uint16_t* dlogits;
    // per-row partials of the loss reduction (workspace)
    double* ws_contrib;
    float* ws_rho;
    uint8_t* ws_flag;
    unsigned int* status;
    int32_t row_streams;  // pipelined fused kernel: 1 = rows in stream order, 2 = live rows spread among masked
};

// Workspace carve-up of leap_grpo_loss_fwd.
struct LossWorkspace {
    double* contrib;
    float* rho;
    uint8_t* flag;
    double* part_loss;
    double* part_rho;
    long long* part_live;
    long long* part_clip;
    int64_t nblk;
};
constexpr int64_t kReduceRowsPerBlock = 512;
size_t loss_workspace_bytes(int64_t N);
LossWorkspace carve_loss_workspace(void* base, int64_t N);

cudaError_t launch_rank_advantages(const RankArgs& a, cudaStream_t s);
cudaError_t launch_token_counts(const SegArgs& a, cudaStream_t s);
cudaError_t launch_scatter(const SegArgs& a, cudaStream_t s);
// Counts (to L_out, totals_out) and scatter with those local totals, in one
// launch when the segment table fits on chip.
cudaError_t launch_token_advantages(const SegArgs& a, cudaStream_t s);

// mode: 0 = log-probs only, 1 = loss forward (no dlogits).
cudaError_t launch_row_stream(const RowArgs& a, int mode, cudaStream_t s);
// Fused forward + backward: the row-pipelined two-pass kernel, or with
// single_read the cluster-resident one (cudaErrorNotSupported if V is too
// large for it).
cudaError_t launch_fused_loss(const RowArgs& a, bool single_read, cudaStream_t s);
cudaError_t launch_split_bwd(const RowArgs& a, cudaStream_t s);
// Fused forward + backward with the two passes of consecutive rows overlapped
// on each SM through bulk-copy rings (loss_pipe.cu).
cudaError_t launch_pipe_loss(const RowArgs& a, cudaStream_t s);
// Fused forward + backward for rows of V <= kShortRowMaxV (short_rows.cu).
constexpr int32_t kShortRowMaxV = 32768;
cudaError_t launch_short_row_loss(const RowArgs& a, cudaStream_t s);
cudaError_t launch_loss_reduce(const LossWorkspace& ws, int64_t N, float* loss, void* stats,
                               bool accumulate, cudaStream_t s);
int64_t fused_max_vocab();

int device_sm_count();
// Device address of the sticky status word on the current device (null on error).
unsigned int* device_status_ptr();

}  // namespace leap
