/*
 * libleap: GB300 (sm_103a) kernels for the data-parallel hot path of one LEAP
 * training step (LEAP: Lean Environment-Feedback via Adaptive Pruning,
 * arXiv 2608.01804): rank-based tournament advantages gated by
 * Difficulty-Conditioned Pruning, per-turn discounted token advantages, token
 * log-probs over a large vocabulary, and the clipped GRPO surrogate with its
 * dlogits backward; and, on the tensor cores (tcgen05), the same loss
 * straight from the hidden states through the lm-head with its gradients
 * with respect to the hidden states and the lm-head weight.
 *
 * Conventions for every entry point
 * ---------------------------------
 *  - Plain C ABI.  Every array argument is a DEVICE pointer owned by the
 *    caller; libleap allocates no device memory and frees none.  Outputs are
 *    written, never read (except where "accumulate" is stated).
 *  - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *    stream).  Every call is asynchronous on that stream; it returns once the
 *    kernels are enqueued.  No call synchronises, except
 *    leap_get_device_status().
 *  - Argument errors (bad sizes, NULL required pointers, misalignment) are
 *    detected on the host before any launch and return LEAP_ERR_INVALID_ARG
 *    (or LEAP_ERR_UNSUPPORTED for a valid but unimplemented combination);
 *    nothing is enqueued then.  A failed launch returns LEAP_ERR_CUDA.
 *  - Data errors that only the device can see (a token id outside [0, V), an
 *    outcome field out of range, a malformed segment) never cause an
 *    out-of-bounds access: the offending item is treated as masked and a
 *    sticky bit (LEAP_DEV_*) is OR-ed into a per-device status word that
 *    leap_get_device_status() reads and clears.
 *  - bf16 tensors are passed as uint16_t bit patterns.  Row-major matrices
 *    have a leading dimension `ld` (elements); bf16 matrices need a 16-byte
 *    aligned base and ld % 8 == 0.
 *  - No kernel waits on another launch.  The single-read fused loss kernel
 *    waits on its own asynchronous copies and on the other CTAs of its
 *    cluster, the tensor-core GEMM on its own TMA loads, MMAs and epilogue,
 *    all through mbarriers; every such wait is bounded and, if it ever gave
 *    up, the kernel would set LEAP_DEV_TIMEOUT and finish instead of hanging.
 */
#ifndef LEAP_H_
#define LEAP_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    LEAP_OK = 0,
    LEAP_ERR_INVALID_ARG = 1,
    LEAP_ERR_UNSUPPORTED = 2,
    LEAP_ERR_CUDA = 3,
    LEAP_ERR_TIMEOUT = 4,     /* reserved (a wait that gave up is reported as LEAP_DEV_TIMEOUT) */
    LEAP_ERR_BAD_INDEX = 5    /* returned by leap_get_device_status() when a bit is set */
} leap_status_t;

/* Sticky device status bits (see leap_get_device_status). */
#define LEAP_DEV_BAD_ID 1u      /* a token id with nonzero weight lay outside [0, V) */
#define LEAP_DEV_BAD_OUTCOME 2u /* pass_turn / num_turns out of range or inconsistent */
#define LEAP_DEV_BAD_SEGMENT 4u /* segment offsets, rollout or turn out of range */
#define LEAP_DEV_TIMEOUT 8u     /* a bounded wait inside a kernel gave up (results undefined) */

/* Human-readable name of a status code (static storage). */
const char* leap_status_string(leap_status_t status);

/* Library version, major*10000 + minor*100 + patch. */
int32_t leap_version(void);

/*
 * Reads and clears the sticky status word of the CURRENT device after all
 * work already enqueued on `stream` (synchronises `stream`).  *host_flags
 * receives the OR of LEAP_DEV_* bits seen since the last call.  Returns
 * LEAP_OK when no bit is set, LEAP_ERR_BAD_INDEX when one is, LEAP_ERR_CUDA
 * on a CUDA error.
 */
leap_status_t leap_get_device_status(uint32_t* host_flags, void* stream);

/* ------------------------------------------------------------------------
 * 1. Rank-based advantages per rollout group (Sec. 3.1 Eqs. 1-2; Sec. 3.2
 *    Eqs. 4-6 and the final GRPO step; Sec. 3.3 discount).
 * ------------------------------------------------------------------------ */
typedef enum {
    LEAP_CMP_PAPER = 0,  /* Eq. 4: order by turns-to-pass only (tier r) */
    LEAP_CMP_LEXI = 1    /* tier r, then higher speedup, then fewer tokens (extension) */
} leap_cmp_t;

typedef enum {
    LEAP_ADVNORM_GRPO_STD = 0,  /* A = (R - mean R) / (std R + eps_std) over the group */
    LEAP_ADVNORM_NONE = 1       /* A = R */
} leap_advnorm_t;

typedef enum {
    LEAP_REWARD_RANK = 0,    /* Eq. 6: tournament reward (the method) */
    LEAP_REWARD_STATIC = 1   /* static-scalar baseline the paper compares against (Sec. 3.2,
                                Table 6 "GRPO-MT"): 1 for a turn-1 pass, static_c for a later
                                pass, 0 for a failure */
} leap_reward_t;

/* Training-observability counters of a leap_group_rank_advantages call
 * (activated groups and recovery rates: Table 5, Sec. 4.3; turns per pass:
 * Table 2, Sec. 4.2).  Device struct, ACCUMULATED (+=): zero it first.
 *   activated-group rate  = gated_groups / groups
 *   per-rollout recovery  = later_passes / failed_first_turn_in_gated
 *   per-group recovery    = groups_with_recovery / gated_groups
 *   turns per pass        = total_turns / (first_turn_passes + later_passes) */
#define LEAP_PASS_BUCKETS 10
/* Rollout composition (Fig. 4, Sec. 4.5).  A group's observed pass rate is its
 * first-turn pass rate p = (G - N_fail) / G (Eq. 1's count, the quantity the
 * DCP gate sees); it falls in bucket b = min(9, floor(10 p)), computed exactly
 * as min(9, (10 (G - N_fail)) div G), i.e. ten equal-width buckets with p = 1
 * in the last.  Each rollout with A != 0 is counted in
 * composition[b][type][sign]: type 0 = immediate pass (tier r = M, a turn-1
 * pass), 1 = debug-assisted pass (0 < r < M, a pass at a later turn of an
 * expanded group), 2 = failure (r = 0, including later passes a gated-off
 * group never ran); sign 0 = A > 0, 1 = A < 0.  Fig. 4's per-bucket
 * percentages are composition[b][.][.] over its sum for bucket b. */
typedef struct {
    int64_t groups, gated_groups;
    int64_t rollouts, nonzero_adv_rollouts;
    int64_t first_turn_passes;          /* passes at turn 1 (any group) */
    int64_t later_passes;               /* passes at turn > 1 in gated groups (recoveries) */
    int64_t groups_with_recovery;       /* gated groups with at least one recovery */
    int64_t failed_first_turn_in_gated; /* rollouts of gated groups that failed turn 1 */
    int64_t total_turns;                /* sum of the effective turn counts */
    int64_t passes_by_turn[8];          /* [m - 1]: passes at turn m (turn 1 from any group) */
    int64_t composition[LEAP_PASS_BUCKETS][3][2]; /* nonzero-advantage rollouts, see above */
    int64_t groups_by_bucket[LEAP_PASS_BUCKETS];  /* groups per observed-pass-rate bucket */
} leap_rank_stats_t;

typedef struct {
    int32_t num_groups;   /* prompts q in this call, >= 0 */
    int32_t G;            /* rollouts per group, 2 .. 1024 (Eq. 6 divides by G - 1) */
    int32_t M;            /* maximum turns, 1 .. 8 */
    int32_t tau_min;      /* Eq. 2 bounds, inclusive: 0 <= tau_min <= tau_max <= G; */
    int32_t tau_max;      /*   ignored when gate_in != NULL */
    float gamma;          /* Sec. 3.3 discount, in (0, 1] */
    float eps_std;        /* >= 0, added to the group std */
    int32_t cmp;          /* leap_cmp_t */
    int32_t norm;         /* leap_advnorm_t */
    int32_t std_unbiased; /* 1: std divides by G - 1; 0: by G */
    int32_t reward;       /* leap_reward_t */
    float static_c;       /* in [0, 1]: LEAP_REWARD_STATIC's later-pass reward */
} leap_rank_params_t;

/*
 * Per group of G rollouts (rollout i of group g at index g*G + i):
 *   N_fail  = rollouts that did not pass on turn 1                 (Eq. 1)
 *   gate    = gate_in[g] != 0 if gate_in, else tau_min <= N_fail <= tau_max (Eq. 2)
 *   r_i     = M - m + 1 for a first pass at turn m, 0 if never passed (Sec. 3.2);
 *             a gated-off group ran one turn only: r_i = M on a turn-1 pass else 0,
 *             and T_eff_i = 1; otherwise T_eff_i = num_turns_i
 *   n_worse_i / n_better_i = peers with strictly lower / higher r   (Eq. 5)
 *   R_i     = (n_worse_i - n_better_i) / (G - 1)                     (Eq. 6)
 *   A_i     = R_i / (std_g R + eps_std)  (mean_g R is exactly 0)     (GRPO step)
 *   turn_adv[i*M + t] = beta_i^(T_eff_i - t - 1) * A_i for t < T_eff_i, else 0,
 *             beta_i = gamma if A_i >= 0 else 1                     (Sec. 3.3)
 * With LEAP_CMP_LEXI (an extension, not in the paper) a tie of tiers between
 * two passing rollouts is broken by the higher speedup, then by fewer tokens;
 * failures tie among themselves.  With LEAP_REWARD_STATIC, R is the static
 * baseline reward and A its standard GRPO advantage (general mean; a group
 * with all rewards equal gets A = 0).
 * Inputs  pass_turn int8 [n]: 0 = never passed, 1..M = turn of the first pass;
 *         num_turns int8 [n]: generated turns T_i, 1..M, >= pass_turn if passed;
 *         speedup f32 [n], ntokens int32 [n]: required for LEAP_CMP_LEXI, else ignored;
 *         gate_in u8 [num_groups] or NULL; stats: leap_rank_stats_t or NULL.
 * Outputs (n = num_groups*G): gate_out u8 [num_groups], r_out u8 [n],
 *         n_worse, n_better int32 [n], R, A f32 [n] - each may be NULL;
 *         turn_adv f32 [n*M] and T_eff u8 [n] are required.
 * A rollout with an out-of-range outcome sets LEAP_DEV_BAD_OUTCOME and is
 * ranked as a failure (r = 0) with T_eff = 0 (no tokens).
 */
leap_status_t leap_group_rank_advantages(
    const leap_rank_params_t* params,
    const int8_t* pass_turn, const int8_t* num_turns,
    const float* speedup, const int32_t* ntokens,
    const uint8_t* gate_in,
    uint8_t* gate_out, uint8_t* r_out, int32_t* n_worse, int32_t* n_better,
    float* R, float* A, float* turn_adv, uint8_t* T_eff,
    leap_rank_stats_t* stats,
    void* stream);

/* ------------------------------------------------------------------------
 * 2. Per-token advantages and loss weights over the packed token stream
 *    (Sec. 3.3 token sets M_{i,t}; Sec. 4.1 sample-level loss aggregation).
 *
 * Segments: segment s covers tokens [seg_offsets[s], seg_offsets[s+1]) of the
 * packed stream of N tokens (cu_seqlens convention, offsets non-decreasing,
 * within [0, N]).  seg_rollout[s] is the rollout index (0 .. n_rollouts-1)
 * and seg_turn[s] the generated-turn index t (0 .. M-1) of a segment of
 * model-generated tokens; seg_turn[s] < 0 marks prompt, environment-feedback
 * or padding tokens.  Tokens in no segment are masked.
 * ------------------------------------------------------------------------ */
typedef enum {
    LEAP_AGG_SEQ_MEAN_TOKEN_MEAN = 0, /* w = 1 / (R_valid * L_i) */
    LEAP_AGG_TOKEN_MEAN = 1           /* w = 1 / N_valid */
} leap_agg_t;

/*
 * L[i] = number of tokens of rollout i in generated turns t < T_eff[i]
 * (written for every i < n_rollouts); totals[0] = sum_i L[i] (N_valid),
 * totals[1] = #{i : L[i] > 0} (R_valid).  For data-parallel training,
 * all-reduce(sum) `totals` across ranks before leap_scatter_turn_advantages.
 * A segment with decreasing or out-of-range offsets, rollout >= n_rollouts or
 * turn >= M sets LEAP_DEV_BAD_SEGMENT and is skipped.
 */
leap_status_t leap_rollout_token_counts(
    int64_t N, int32_t n_rollouts, int32_t M,
    const int32_t* seg_offsets, const int32_t* seg_rollout, const int8_t* seg_turn,
    int32_t num_segs, const uint8_t* T_eff,
    int32_t* L, int64_t* totals,
    void* stream);

/*
 * adv_out[k] = turn_adv[i*M + t] and w_out[k] = aggregation weight for every
 * token k of a generated segment (rollout i, turn t < T_eff[i]); 0 and 0 for
 * every other token.  `L` and `totals` come from leap_rollout_token_counts
 * (totals possibly all-reduced: they are the GLOBAL normalisers, so shards
 * and chunks of one batch sum to the batch loss).  agg is a leap_agg_t.
 */
leap_status_t leap_scatter_turn_advantages(
    int64_t N, int32_t n_rollouts, int32_t M,
    const int32_t* seg_offsets, const int32_t* seg_rollout, const int8_t* seg_turn,
    int32_t num_segs, const float* turn_adv, const uint8_t* T_eff,
    const int32_t* L, const int64_t* totals, int32_t agg,
    float* adv_out, float* w_out,
    void* stream);

/*
 * leap_rollout_token_counts followed by leap_scatter_turn_advantages with
 * this call's own totals (no exchange in between), in one launch: every block
 * builds the counts and each segment's advantage and weight in shared memory,
 * then scatters its share of the tokens.  Same arguments and results as the
 * two calls (L, totals, adv_out, w_out written; malformed segments flagged
 * and skipped alike).  For one process (or one rank holding the whole batch).
 * When the batch is split over data-parallel ranks the totals must be
 * all-reduced between counting and scattering: use the two calls.  The one
 * launch serves tables of up to 768 segments (every block rebuilds the table,
 * which pays off on small batches only); larger ones take the two calls'
 * kernels.
 */
leap_status_t leap_token_advantages(
    int64_t N, int32_t n_rollouts, int32_t M,
    const int32_t* seg_offsets, const int32_t* seg_rollout, const int8_t* seg_turn,
    int32_t num_segs, const float* turn_adv, const uint8_t* T_eff, int32_t agg,
    int32_t* L, int64_t* totals, float* adv_out, float* w_out,
    void* stream);

/* ------------------------------------------------------------------------
 * 3. Token log-probabilities under pi_theta (the log pi terms of Eq. 3's
 *    surrogate): lse_k = log sum_v exp(inv_temp * z_kv),
 *    logp_k = inv_temp * z_k[ids_k] - lse_k.
 * logits bf16 [N x ld] (row k = token k), 1 <= V <= ld; ids int32 [N].
 * logp f32 [N] required, lse f32 [N] optional.  An id outside [0, V) sets
 * LEAP_DEV_BAD_ID and yields logp = 0 (lse is still the row's).
 * ------------------------------------------------------------------------ */
leap_status_t leap_token_logprobs(
    const uint16_t* logits, int64_t ld, const int32_t* ids,
    int64_t N, int32_t V, float inv_temp,
    float* logp, float* lse,
    void* stream);

/* ------------------------------------------------------------------------
 * 4. Clipped-ratio surrogate of Eq. 3 (KL term skipped, Fig. 2) with masked
 *    reduction, and its backward.
 *   rho_k  = exp(logp_k - old_logp_k)
 *   ell_k  = -min(rho_k A_k, clip(rho_k, 1 - eps_low, 1 + eps_high) A_k)
 *   loss   = sum_k w_k ell_k      (deterministic: fixed-order fp64 sum)
 *   g_k    = -w_k A_k rho_k if the unclipped term is active (A >= 0 and
 *            rho <= 1 + eps_high, or A < 0 and rho >= 1 - eps_low), else 0
 *   dlogits_kv = grad_scale * g_k * inv_temp * (1[v = ids_k] - softmax_kv)
 * Rows with w_k == 0 (or a bad id) are masked: their logits are not read,
 * logp/lse/ell are written as 0 and their dlogits row as zeros.
 * ------------------------------------------------------------------------ */
#define LEAP_LOSS_ACCUMULATE 1u  /* loss[0] += this call's sum (chunked passes) */
/* Fused backward through the cluster kernel: each logits row is split over 8
 * CTAs that hold it in registers, so it is read from HBM exactly once whatever
 * else is using L2 (supports V <= 262,144).  The default kernel reads a row
 * twice, the second time from L2, which is faster when the loss pass has the
 * GPU's L2 to itself.  Rows of V <= 32,768 take a third kernel with or
 * without the flag: a group of 1-16 warps holds each row in registers (read
 * once) and reduces it with warp shuffles. */
#define LEAP_LOSS_SINGLE_READ 2u
/* A scheduling hint for the default fused kernel (rows of V > 32,768 with
 * dlogits; ignored elsewhere): each persistent CTA spreads its live rows
 * evenly among its masked ones instead of visiting them in stream order, so
 * that long runs of masked rows (prompts and environment feedback in a packed
 * multi-turn stream) and of live rows overlap on every SM instead of
 * alternating.  Results are the same bit for bit; measured on the packed
 * multi-turn workload 0.934 -> 0.950 of the copy bandwidth, on a padded
 * single-turn batch (short runs) 0.951 -> 0.945. */
#define LEAP_LOSS_INTERLEAVED_ROWS 4u

typedef struct {
    float eps_low;     /* >= 0 */
    float eps_high;    /* >= 0 */
    float inv_temp;    /* > 0; 1 / sampling temperature */
    float grad_scale;  /* multiplies dlogits */
    uint32_t flags;    /* LEAP_LOSS_* bits */
} leap_loss_params_t;

/* Optional side outputs of leap_grpo_loss_fwd (device struct, overwritten,
 * or accumulated under LEAP_LOSS_ACCUMULATE). */
typedef struct {
    double loss_sum;        /* same value as loss[0], in fp64 */
    double rho_sum;         /* sum of rho over live tokens */
    int64_t live_tokens;    /* tokens with w != 0 and a valid id */
    int64_t clipped_tokens; /* live tokens whose gradient is clipped to 0 */
} leap_loss_stats_t;

/* Bytes of device workspace leap_grpo_loss_fwd needs for N tokens. */
size_t leap_grpo_loss_workspace_size(int64_t N, int32_t V);

/*
 * Forward (and, if dlogits != NULL, the fused backward in the same pass: each
 * logits row is read from HBM once and dlogits written once).
 * logits bf16 [N x ld]; ids int32 [N]; old_logp, adv, w f32 [N].
 * Outputs: loss f32 [1] (required); logp, lse, ell f32 [N] (optional);
 * dlogits bf16 [N x ld] (optional; columns >= V untouched); stats optional.
 * workspace: >= leap_grpo_loss_workspace_size(N, V) bytes, 256-byte aligned,
 * contents ignored on entry.  Requires 1 <= V.  With LEAP_LOSS_SINGLE_READ
 * the fused backward supports V up to 262,144 (LEAP_ERR_UNSUPPORTED beyond).
 */
leap_status_t leap_grpo_loss_fwd(
    const leap_loss_params_t* params,
    const uint16_t* logits, int64_t ld, const int32_t* ids,
    const float* old_logp, const float* adv, const float* w,
    int64_t N, int32_t V,
    float* loss, float* logp, float* lse, float* ell,
    uint16_t* dlogits,
    void* workspace, size_t ws_bytes,
    leap_loss_stats_t* stats,
    void* stream);

/*
 * leap_grpo_loss_fwd without a workspace argument, for callers that cannot
 * allocate device memory where they call the loss: a C program that links
 * only libleap and has no device allocator of its own, or a process whose
 * device memory is carved up front by a pool that forbids further
 * cudaMalloc.  The paper has no counterpart; this is an interface variant.
 * Same arguments and results as leap_grpo_loss_fwd, minus workspace/ws_bytes.
 * Its scratch is a file-scope device array of 1 MiB, enough for
 * N <= LEAP_NOALLOC_MAX_ROWS rows; larger N returns LEAP_ERR_INVALID_ARG
 * (split the batch into chunks and use LEAP_LOSS_ACCUMULATE).  Each device
 * that loads libleap holds its own copy until the process exits.  The first
 * call on a device looks the array's device address up (a host-side
 * cudaGetSymbolAddress with that device current); make that first call
 * before any stream capture.  Nothing is allocated or freed by any call.
 * All calls on a device share the one array: calls whose work overlaps on
 * the GPU (different streams, or host threads) race and give wrong results;
 * serialise them.  No state carries over between calls: every call writes
 * all of the scratch it later reads, so nothing needs clearing.
 */
#define LEAP_NOALLOC_MAX_ROWS 65536

leap_status_t leap_grpo_loss_fwd_noalloc(
    const leap_loss_params_t* params,
    const uint16_t* logits, int64_t ld, const int32_t* ids,
    const float* old_logp, const float* adv, const float* w,
    int64_t N, int32_t V,
    float* loss, float* logp, float* lse, float* ell,
    uint16_t* dlogits,
    leap_loss_stats_t* stats,
    void* stream);

/*
 * Split backward: dlogits from logits and the lse saved by the forward
 * (reads logits once more: 2V bytes read + 2V written per live row).
 * Same argument meanings as leap_grpo_loss_fwd; lse f32 [N] required.
 */
leap_status_t leap_grpo_loss_bwd(
    const leap_loss_params_t* params,
    const uint16_t* logits, int64_t ld, const int32_t* ids,
    const float* old_logp, const float* adv, const float* w, const float* lse,
    int64_t N, int32_t V,
    uint16_t* dlogits,
    void* stream);

/* ------------------------------------------------------------------------
 * 5. Fused lm-head: token log-probs straight from the hidden states, logits =
 *    hidden . W^T computed tile by tile on the tensor cores (tcgen05) and
 *    reduced in tensor memory, never stored; the same clipped surrogate as
 *    section 4; and its gradients with respect to the hidden states and
 *    the lm-head weight.  The paper trains the policy through Eq. 3; these
 *    are that objective's gradients for the last layer, by the chain rule.
 * ------------------------------------------------------------------------ */

/*
 * Plain GEMM building block: C[M x N] = A[M x K] . B[N x K]^T with bf16
 * inputs, fp32 accumulation on tcgen05 and bf16 output (round to nearest).
 * A, B, C row-major with leading dimensions lda, ldb >= K and ldc >= N, all
 * multiples of 8 elements; 16-byte aligned bases.
 */
leap_status_t leap_gemm_bf16_nt(const uint16_t* A, int64_t lda, const uint16_t* B, int64_t ldb,
                                uint16_t* C, int64_t ldc, int32_t M, int32_t N, int32_t K,
                                void* stream);

/*
 * Weight-gradient GEMM building block: C[M x N] = A^T . B (accumulate == 0)
 * or C += A^T . B (accumulate != 0), with A bf16 [K x M] and B bf16 [K x N]
 * row-major (so both operands are read MN-major: the contraction runs over
 * their rows, e.g. tokens), fp32 accumulation on tcgen05 and an fp32 C
 * [M x N] with leading dimension ldc.  lda >= M and ldb >= N multiples of 8
 * elements, ldc >= N a multiple of 4; 16-byte aligned bases.  K == 0 sets
 * C = 0 (or leaves it unchanged when accumulating).  This is the shape of
 * dW = dlogits^T . hidden in section 5.
 */
leap_status_t leap_gemm_bf16_tn_f32(const uint16_t* A, int64_t lda, const uint16_t* B, int64_t ldb,
                                    float* C, int64_t ldc, int32_t M, int32_t N, int32_t K,
                                    int32_t accumulate, void* stream);

/* Gradients the fused lm-head is asked for (the `grads` bit set of
 * leap_fused_lmhead_workspace_size). */
#define LEAP_LMHEAD_DHIDDEN 1
#define LEAP_LMHEAD_DW 2

/* Bytes of workspace leap_fused_lmhead_logprobs needs for the gradients in
 * `grads` (0: forward only).  Either gradient adds one chunk of bf16 dlogits
 * (min(N, 16,384) x V: 5 GB at V = 151,936). */
size_t leap_fused_lmhead_workspace_size(int64_t N, int32_t H, int32_t V, int32_t grads);

/*
 * hidden bf16 [N x H] (row-major), W bf16 [V x H] (the lm-head weight,
 * row-major); H % 8 == 0, 16-byte aligned bases.  logits z = hidden . W^T,
 * then exactly leap_grpo_loss_fwd's outputs (loss, logp, lse, ell, stats;
 * ids, old_logp, adv, w as there; params->flags may hold
 * LEAP_LOSS_ACCUMULATE).  Gradients of the loss (chain rule through z,
 * from bf16 dlogits recomputed for 16,384-token chunks):
 *   dhidden  bf16 [N x H], nullable: d loss / d hidden = dlogits . W;
 *   dW       fp32 [V x H], nullable, 16-byte aligned: d loss / d W =
 *            dlogits^T . hidden, summed over all N tokens in fp32 (chunk by
 *            chunk).  With LEAP_LOSS_ACCUMULATE the sum is added into dW
 *            (gradient accumulation over micro-batches); otherwise dW is
 *            overwritten (set to 0 when N == 0).
 * workspace: >= leap_fused_lmhead_workspace_size(N, H, V, grads) bytes for
 * the gradients requested, 256-byte aligned.
 */
leap_status_t leap_fused_lmhead_logprobs(
    const leap_loss_params_t* params,
    const uint16_t* hidden, const uint16_t* W, int64_t N, int32_t H, int32_t V,
    const int32_t* ids, const float* old_logp, const float* adv, const float* w,
    float* loss, float* logp, float* lse, float* ell,
    uint16_t* dhidden, float* dW,
    void* workspace, size_t ws_bytes,
    leap_loss_stats_t* stats,
    void* stream);

/* ------------------------------------------------------------------------
 * 6. Self-test of the failure path (library diagnostics; the paper has no
 *    counterpart).
 * ------------------------------------------------------------------------ */

/*
 * Every wait inside a libleap kernel (on its own asynchronous copies, its
 * tensor-core work or its cluster peers) is bounded: if it ever gave up, the
 * kernel would set LEAP_DEV_TIMEOUT and return instead of hanging the GPU.
 * This call exercises that give-up path on purpose: one thread of a tiny
 * kernel waits, through the same bounded wait, on a barrier that nothing
 * completes, for limit_ns nanoseconds of GPU wall time (1,000 .. 10^10),
 * then sets LEAP_DEV_TIMEOUT and returns; leap_get_device_status() then
 * reports it.  waited_ns (device uint64, nullable) receives the time the wait
 * took before giving up.  Nothing is in flight when it gives up, so the
 * context stays usable.  Returns LEAP_ERR_INVALID_ARG for a limit out of
 * range, LEAP_ERR_CUDA if the launch fails.
 */
leap_status_t leap_selftest_bounded_wait(uint64_t limit_ns, uint64_t* waited_ns, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* LEAP_H_ */
