"""Plain, slow fp64 CPU oracle for the LEAP GRPO-loss hot path.

TEST INFRASTRUCTURE ONLY.  Nothing on the product path may import this module:
only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` use it.  It shares no code with the
CUDA library (``paper_2608_01804_gb300``) and imports nothing from it.

Every function follows the paper (LEAP: Lean Environment-Feedback via Adaptive
Pruning, arXiv 2608.01804) in its own order and notation, in float64, with
numpy used only for whole-array primitives (max, exp, log, sum, matmul).
Where the paper is silent the function states the reading it takes.

Pins (what checks this oracle against something other than itself) live in
``tests/test_oracle_*.py``.  No function here is "parity unpinned".

Conventions shared with the library's contract (not the paper's):
  * outcomes are per rollout: ``pass_turn`` = 1-based turn of the first passing
    verification (0 = never passed), ``num_turns`` = generated turns T_i;
  * a rollout whose outcome fields are out of range is treated as a failure
    (r = 0) that contributes no tokens (T_eff = 0), and is reported in the
    returned ``bad_outcome`` mask;
  * a token whose id lies outside [0, V) is treated as masked (w = 0) and is
    reported in ``bad_id``;
  * rows with w == 0 are not read: their logp, lse, ell and dlogits are 0.
"""

from __future__ import annotations

import numpy as np

AGG_SEQ_MEAN_TOKEN_MEAN = 0
AGG_TOKEN_MEAN = 1
ADVNORM_GRPO_STD = 0
ADVNORM_NONE = 1
CMP_PAPER = 0
CMP_LEXI = 1
REWARD_RANK = 0
REWARD_STATIC = 1


# ---------------------------------------------------------------------------
# Sec. 3.1 (DCP), Eq. 1-2, and Sec. 3.2 (rank tiers), Eq. 4 and the tier rule.
# ---------------------------------------------------------------------------
def tiers_and_gate(pass_turn, num_turns, M, tau_min, tau_max, gate_in=None):
    """Failure count, DCP gate, rank tier r and effective turn count per rollout.

    Eq. 1: N_fail(q) = sum_i I(o_i failed).  Reading: "failed" is judged on the
    first turn, because the gate decides whether turn 2 is generated at all.
    Eq. 2: G(q) = 1 iff tau_min <= N_fail <= tau_max (both bounds inclusive).
    Tier rule (Sec. 3.2): pass at turn m -> r = M - m + 1; never passed -> r = 0.
    A gated-off group (G(q) = 0) never ran turns after the first, so its
    outcomes are truncated to turn 1: r = M on a first-turn pass, else 0, and
    T_eff = 1.  ``gate_in`` (if given) replaces Eq. 2 with a recorded gate.

    Arrays are [num_groups, G].  Returns (n_fail, gate, r, T_eff, bad_outcome).
    """
    pass_turn = np.asarray(pass_turn, dtype=np.int64)
    num_turns = np.asarray(num_turns, dtype=np.int64)
    m, T = pass_turn, num_turns

    bad = (m < 0) | (m > M) | (T < 1) | (T > M) | ((m >= 1) & (m > T))
    # Eq. 1 over first-turn outcomes (a malformed rollout counts as failed).
    n_fail = np.sum(bad | (m != 1), axis=1).astype(np.int64)
    if gate_in is not None:
        gate = (np.asarray(gate_in) != 0).astype(np.uint8)
    else:
        gate = ((tau_min <= n_fail) & (n_fail <= tau_max)).astype(np.uint8)    # Eq. 2
    on = gate[:, None] == 1
    r_on = np.where(m >= 1, M - m + 1, 0)          # tier rule, expanded group
    r_off = np.where(m == 1, M, 0)                 # truncated to turn 1
    r = np.where(bad, 0, np.where(on, r_on, r_off)).astype(np.int64)
    T_eff = np.where(bad, 0, np.where(on, T, 1)).astype(np.int64)
    return n_fail, gate, r, T_eff, bad


# ---------------------------------------------------------------------------
# Sec. 3.2, Eq. 5: the complete pairwise tournament, literally.
# ---------------------------------------------------------------------------
def tournament(r):
    """N_worse(o_i) = #{j != i : r_i > r_j},  N_better(o_i) = #{j != i : r_i < r_j}.

    Strict inequalities: a tie counts in neither.  This is the O(G^2) double
    loop of Eq. 5 (vectorised over j for speed; the comparison is the same).
    """
    r = np.asarray(r, dtype=np.int64)
    num_groups, G = r.shape
    n_worse = np.zeros((num_groups, G), dtype=np.int64)
    n_better = np.zeros((num_groups, G), dtype=np.int64)
    for i in range(G):
        ri = r[:, i:i + 1]
        others = np.ones(G, dtype=bool)
        others[i] = False
        n_worse[:, i] = np.sum((ri > r) & others, axis=1)
        n_better[:, i] = np.sum((ri < r) & others, axis=1)
    return n_worse, n_better


def tournament_lexi(r, speedup, ntokens):
    """Extension of Eq. 5 with tie-breaks (not in the paper): rollout i beats j
    if its tier is higher, or the tiers are equal, both passed (r > 0), and i
    has the higher speedup, or the same speedup and fewer tokens.  Failures
    (r = 0) carry no speedup and tie among themselves; exact ties count in
    neither direction.  Pairwise double loop, vectorised over groups."""
    r = np.asarray(r, dtype=np.int64)
    sp = np.asarray(speedup, dtype=np.float64)
    tk = np.asarray(ntokens, dtype=np.int64)
    num_groups, G = r.shape
    n_worse = np.zeros((num_groups, G), dtype=np.int64)
    n_better = np.zeros((num_groups, G), dtype=np.int64)

    def beats(a, b):
        ra, rb = r[:, a:a + 1], r[:, b]
        sa, sb = sp[:, a:a + 1], sp[:, b]
        ta, tb = tk[:, a:a + 1], tk[:, b]
        return (ra > rb) | ((ra == rb) & (ra > 0) & ((sa > sb) | ((sa == sb) & (ta < tb))))

    allj = np.arange(G)
    for i in range(G):
        others = allj != i
        n_worse[:, i] = np.sum(beats(i, allj) & others, axis=1)
        # j beats i, for every j: evaluate with j as the first argument
        better = (r > r[:, i:i + 1]) | ((r == r[:, i:i + 1]) & (r > 0) &
                                        ((sp > sp[:, i:i + 1]) | ((sp == sp[:, i:i + 1]) & (tk < tk[:, i:i + 1]))))
        n_better[:, i] = np.sum(better & others, axis=1)
    return n_worse, n_better


def static_reward(r, M, c):
    """The static-scalar multi-turn reward the paper compares against (Sec. 3.2,
    "GRPO-MT" in Table 6): 1 for a first-turn pass, the constant c for a pass
    at a later turn, 0 for a failure."""
    r = np.asarray(r, dtype=np.int64)
    return np.where(r == M, 1.0, np.where(r > 0, float(c), 0.0))


def tournament_reward(n_worse, n_better, G):
    """Eq. 6: R_i = (N_worse(o_i) - N_better(o_i)) / (G - 1), in [-1, 1]."""
    if G < 2:
        raise ValueError("Eq. 6 divides by G - 1: G must be at least 2")
    return (np.asarray(n_worse, np.float64) - np.asarray(n_better, np.float64)) / (G - 1)


def grpo_advantage(R, eps_std=1e-6, norm=ADVNORM_GRPO_STD, std_unbiased=True):
    """Sec. 3.2, last step: the final advantage A_i by "the standard GRPO formulation".

    Reading: A_i = (R_i - mean_g R) / (std_g R + eps_std) over the rollout group,
    std with the (G - 1) divisor by default.  A group whose rewards are all
    equal (std = 0) carries no preference signal: its advantages are 0, also
    when eps_std = 0 (where the formula would read 0/0).  ``ADVNORM_NONE``
    returns R as is.
    """
    R = np.asarray(R, dtype=np.float64)
    if norm == ADVNORM_NONE:
        return R.copy()
    G = R.shape[1]
    mean = R.sum(axis=1, keepdims=True) / G
    dev = R - mean
    ddof = 1 if std_unbiased else 0
    std = np.sqrt((dev * dev).sum(axis=1, keepdims=True) / (G - ddof))
    flat = np.all(R == R[:, :1], axis=1, keepdims=True)
    return np.where(flat, 0.0, dev / np.where(flat, 1.0, std + eps_std))


def turn_advantages(A, T_eff, gamma, M):
    """Sec. 3.3: discounted per-turn advantage.

    beta_i = gamma if A_i >= 0 else 1;  A_hat_{i,t} = beta_i^(T_i - t - 1) * A_i
    for generated turns t = 0 .. T_i - 1 (T_i = the effective turn count after
    DCP).  Turns t >= T_i get 0.  Returns [num_groups, G, M].
    """
    A = np.asarray(A, dtype=np.float64)
    T_eff = np.asarray(T_eff, dtype=np.int64)
    beta = np.where(A >= 0, gamma, 1.0)
    out = np.zeros(A.shape + (M,), dtype=np.float64)
    for t in range(M):
        exponent = T_eff - t - 1
        out[..., t] = np.where(t < T_eff, beta ** np.maximum(exponent, 0) * A, 0.0)
    return out


def rank_advantages(pass_turn, num_turns, M, tau_min, tau_max, gamma,
                    eps_std=1e-6, norm=ADVNORM_GRPO_STD, std_unbiased=True,
                    gate_in=None, cmp=CMP_PAPER, speedup=None, ntokens=None,
                    reward=REWARD_RANK, static_c=0.5):
    """Sec. 3.1-3.3 end to end for every group: gate, tiers, tournament, R, A, A_hat.

    reward = REWARD_STATIC replaces the tournament reward by the static-scalar
    baseline (tiers and counts are still reported)."""
    pass_turn = np.asarray(pass_turn)
    G = pass_turn.shape[1]
    n_fail, gate, r, T_eff, bad = tiers_and_gate(pass_turn, num_turns, M,
                                                 tau_min, tau_max, gate_in)
    if cmp == CMP_LEXI:
        n_worse, n_better = tournament_lexi(r, np.asarray(speedup).reshape(r.shape),
                                            np.asarray(ntokens).reshape(r.shape))
    else:
        n_worse, n_better = tournament(r)
    if reward == REWARD_STATIC:
        R = static_reward(r, M, static_c)
    else:
        R = tournament_reward(n_worse, n_better, G)
    A = grpo_advantage(R, eps_std, norm, std_unbiased)
    turn_adv = turn_advantages(A, T_eff, gamma, M)
    return dict(n_fail=n_fail, gate=gate, r=r, T_eff=T_eff, bad_outcome=bad,
                n_worse=n_worse, n_better=n_better, R=R, A=A, turn_adv=turn_adv)


def rank_stats(out, pass_turn, M):
    """Training-observability counters (Table 5, Sec. 4.3; turns per pass:
    Table 2, Sec. 4.2) from rank_advantages' results: activated groups, per-rollout and per-group recovery, passes by
    turn, total effective turns and passed samples (turns per pass)."""
    gate = np.asarray(out["gate"]).astype(bool)
    T_eff = np.asarray(out["T_eff"])
    bad = np.asarray(out["bad_outcome"])
    pt = np.where(bad, 0, np.asarray(pass_turn, dtype=np.int64))
    on = gate[:, None] & ~bad
    first = (pt == 1) & ~bad
    later = on & (pt >= 2)                              # recovered after a first-turn failure
    failed_first_on = on & (pt != 1)
    passes_by_turn = [int(np.sum(first)) if m == 1 else int(np.sum(later & (pt == m))) for m in range(1, 9)]
    composition, groups_by_bucket = rank_composition(out, M)
    return dict(groups=int(gate.size), gated_groups=int(gate.sum()), rollouts=int(pt.size),
                nonzero_adv_rollouts=int(np.count_nonzero(np.abs(out["A"]) > 1e-9)),
                first_turn_passes=int(first.sum()), later_passes=int(later.sum()),
                groups_with_recovery=int(np.sum(np.any(later, axis=1))),
                failed_first_turn_in_gated=int(failed_first_on.sum()),
                total_turns=int(T_eff.sum()), passes_by_turn=passes_by_turn,
                composition=composition.tolist(), groups_by_bucket=groups_by_bucket.tolist())


PASS_BUCKETS = 10


def rank_composition(out, M, buckets=PASS_BUCKETS):
    """Rollout composition of Fig. 4 (Sec. 4.5) from rank_advantages' results.

    Readings (the figure itself is not in the text):
      * a group's "observed pass rate" is its first-turn pass rate
        p = (G - N_fail) / G, with N_fail of Eq. 1 (the quantity the DCP gate
        sees, defined alike for LEAP and for multi-turn GRPO);
      * the buckets are ten equal-width bins of p, b = min(9, floor(10 p)),
        taken in exact integer arithmetic as min(9, (10 (G - N_fail)) // G);
      * outcome type from the effective tier r: immediate pass (r = M, a pass
        at turn 1), debug-assisted pass (0 < r < M, a later pass of an expanded
        group), failure (r = 0; later passes of a gated-off group never ran);
      * only rollouts with a nonzero advantage count (|A| > 1e-9 in fp64), split
        by the sign of A (0: positive, 1: negative).
    Returns (composition int64 [buckets, 3, 2], groups per bucket int64 [buckets]).
    """
    r = np.asarray(out["r"], dtype=np.int64)
    A = np.asarray(out["A"], dtype=np.float64)
    n_fail = np.asarray(out["n_fail"], dtype=np.int64)
    num_groups, G = r.shape
    bucket = np.minimum(buckets - 1, (buckets * (G - n_fail)) // G)
    groups_by_bucket = np.bincount(bucket, minlength=buckets).astype(np.int64)
    kind = np.where(r == M, 0, np.where(r > 0, 1, 2))
    sign = np.where(A > 0, 0, 1)
    counted = np.abs(A) > 1e-9
    b_full = np.broadcast_to(bucket[:, None], r.shape)
    flat = (b_full * 3 + kind) * 2 + sign
    composition = np.bincount(flat[counted], minlength=buckets * 6).astype(np.int64)
    return composition.reshape(buckets, 3, 2), groups_by_bucket


# ---------------------------------------------------------------------------
# Sec. 3.3 (token sets M_{i,t}) and Sec. 4.1 (sample-level aggregation).
# ---------------------------------------------------------------------------
def rollout_token_counts(seg_offsets, seg_rollout, seg_turn, T_eff_flat):
    """L_i = number of optimised tokens of rollout i = sum of |M_{i,t}| over t < T_eff_i.

    Segments are consecutive ranges [seg_offsets[s], seg_offsets[s+1]) of the
    packed token stream.  seg_turn < 0 (prompt, feedback, padding) or a turn at
    or beyond T_eff (pruned by DCP) contributes nothing (Sec. 3.3: tokens
    outside the generated turns get zero advantage and are excluded).
    Returns (L [n], n_valid_tokens, n_valid_rollouts).
    """
    n = len(T_eff_flat)
    L = np.zeros(n, dtype=np.int64)
    for s in range(len(seg_rollout)):
        i, t = int(seg_rollout[s]), int(seg_turn[s])
        if t < 0 or i < 0 or i >= n:
            continue
        if t < T_eff_flat[i]:
            L[i] += int(seg_offsets[s + 1]) - int(seg_offsets[s])
    return L, int(L.sum()), int(np.count_nonzero(L))


def token_advantages(N, seg_offsets, seg_rollout, seg_turn, turn_adv_flat, T_eff_flat,
                     M, agg, L, n_valid_tokens, n_valid_rollouts):
    """Per-token advantage A_hat_k and loss weight w_k.

    Sec. 3.3: every token of generated turn t of rollout i carries A_hat_{i,t};
    every other token carries 0 and weight 0.
    Sec. 4.1 ("sample-level loss objective"), reading: each rollout's loss is
    the mean over its own tokens, and the batch loss the mean over rollouts
    with at least one token, so w_k = 1 / (R_valid * L_i).  TOKEN_MEAN instead
    averages over all valid tokens: w_k = 1 / N_valid.  The normalisers are
    global (passed in) so that shards and chunks sum to the whole.
    """
    adv = np.zeros(N, dtype=np.float64)
    w = np.zeros(N, dtype=np.float64)
    for s in range(len(seg_rollout)):
        i, t = int(seg_rollout[s]), int(seg_turn[s])
        if t < 0 or i < 0 or t >= T_eff_flat[i]:
            continue
        a, b = int(seg_offsets[s]), int(seg_offsets[s + 1])
        adv[a:b] = turn_adv_flat[i * M + t]
        if agg == AGG_TOKEN_MEAN:
            w[a:b] = 1.0 / float(n_valid_tokens)
        else:
            w[a:b] = 1.0 / (float(n_valid_rollouts) * float(L[i]))
    return adv, w


# ---------------------------------------------------------------------------
# Token log-probabilities under pi_theta (Eq. 3's surrogate needs log pi).
# ---------------------------------------------------------------------------
def bf16_bits_to_f64(bits):
    """bf16 bit patterns (uint16) -> exact float64 values."""
    u = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return u.view(np.float32).astype(np.float64)


def f64_to_bf16_bits(x):
    """Round float64 to the nearest bf16 (ties to even) via float32; returns uint16 bits.

    Used only to present the oracle's fp64 dlogits in the library's output type.
    """
    f = np.asarray(x, dtype=np.float64).astype(np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    nan = np.isnan(f)
    rounding = ((u >> np.uint64(16)) & np.uint64(1)) + np.uint64(0x7FFF)
    out = ((u + rounding) >> np.uint64(16)).astype(np.uint16)
    out[nan] = np.uint16(0x7FC0)
    return out


def log_softmax_rows(z, ids, inv_temp=1.0):
    """lse_k = log sum_v exp(inv_temp * z_kv);  logp_k = inv_temp * z_k[y_k] - lse_k.

    z is float64 [rows, V]; the max is subtracted before exp (same value, no
    overflow).  Returns (lse, logp).
    """
    x = np.asarray(z, dtype=np.float64) * inv_temp
    m = x.max(axis=1)
    s = np.exp(x - m[:, None]).sum(axis=1)
    lse = m + np.log(s)
    ids = np.asarray(ids, dtype=np.int64)
    logp = x[np.arange(x.shape[0]), ids] - lse
    return lse, logp


# ---------------------------------------------------------------------------
# Eq. 3: the clipped-ratio surrogate L_surr (KL skipped, Fig. 2 caption) and
# its gradient with respect to the logits.
# ---------------------------------------------------------------------------
def grpo_loss_rows(z, ids, old_logp, adv, w, eps_low=0.2, eps_high=0.2, inv_temp=1.0,
                   grad_scale=1.0, want_dlogits=True):
    """Clipped surrogate per token and its dlogits, for float64 logits z [rows, V].

    Reading of L_surr (standard PPO/GRPO clip, no dual clip):
      rho_k   = exp(logp_k - old_k)
      ell_k   = -min(rho_k * A_k, clip(rho_k, 1 - eps_low, 1 + eps_high) * A_k)
      loss    = sum_k w_k * ell_k
    Gradient: d(w_k ell_k)/d logp_k = -w_k A_k rho_k where the unclipped term is
    the active one (A >= 0 and rho <= 1 + eps_high, or A < 0 and rho >= 1 - eps_low;
    the closed interval counts as unclipped), else 0; then
      dlogits_kv = grad_scale * g_k * inv_temp * (1[v = y_k] - softmax_v).
    Rows with w_k == 0 or an id outside [0, V) are masked: every output is 0.
    Returns dict(logp, lse, ell, g, rho, active, loss, dlogits, bad_id).
    """
    z = np.asarray(z, dtype=np.float64)
    rows, V = z.shape
    ids = np.asarray(ids, dtype=np.int64)
    old_logp = np.asarray(old_logp, dtype=np.float64)
    adv = np.asarray(adv, dtype=np.float64)
    w = np.asarray(w, dtype=np.float64)

    bad_id = (w != 0) & ((ids < 0) | (ids >= V))
    live = (w != 0) & ~bad_id
    safe_ids = np.where(live, ids, 0)

    lse = np.zeros(rows)
    logp = np.zeros(rows)
    if live.any():
        l_lse, l_logp = log_softmax_rows(z[live], safe_ids[live], inv_temp)
        lse[live], logp[live] = l_lse, l_logp

    rho = np.where(live, np.exp(logp - old_logp), 0.0)
    clipped = np.clip(rho, 1.0 - eps_low, 1.0 + eps_high)
    ell = np.where(live, -np.minimum(rho * adv, clipped * adv), 0.0)
    active = live & (((adv >= 0) & (rho <= 1.0 + eps_high)) | ((adv < 0) & (rho >= 1.0 - eps_low)))
    g = np.where(active, -w * adv * rho, 0.0)
    loss = 0.0
    for k in range(rows):                      # plain sequential sum
        loss += w[k] * ell[k]

    dlogits = None
    if want_dlogits:
        dlogits = np.zeros((rows, V))
        for k in np.nonzero(live)[0]:
            p = np.exp(z[k] * inv_temp - lse[k])
            onehot = np.zeros(V)
            onehot[safe_ids[k]] = 1.0
            dlogits[k] = grad_scale * g[k] * inv_temp * (onehot - p)
    return dict(logp=logp, lse=lse, ell=ell, g=g, rho=rho, active=active, live=live,
                loss=loss, dlogits=dlogits, bad_id=bad_id)


# ---------------------------------------------------------------------------
# Fused lm-head variant: logits = hidden . W^T, never stored by the library.
# ---------------------------------------------------------------------------
def lmhead_loss_rows(hidden, W, ids, old_logp, adv, w, eps_low=0.2, eps_high=0.2,
                     inv_temp=1.0, grad_scale=1.0, want_dhidden=True, want_dW=False, dW_rows=None):
    """The same surrogate on logits z = hidden W^T (fp64), plus its gradients
    with respect to both factors of the product (chain rule through z):

        dhidden = dlogits . W          [rows, H]
        dW      = dlogits^T . hidden   [V, H]   (sum over the given rows)

    hidden float64 [rows, H], W float64 [V, H].  Returns the grpo_loss_rows dict
    with 'dhidden' and, if asked, 'dW' added; with ``dW_rows`` (vocabulary
    indices) 'dW' holds only those rows of dW, in that order.  Rows with
    w == 0 have zero dlogits, so they add nothing to dW: dW over a subset of
    token rows that holds every row with w != 0 is dW over all rows.
    """
    hidden = np.asarray(hidden, dtype=np.float64)
    W = np.asarray(W, dtype=np.float64)
    z = hidden @ W.T
    out = grpo_loss_rows(z, ids, old_logp, adv, w, eps_low, eps_high, inv_temp,
                         grad_scale, want_dlogits=want_dhidden or want_dW)
    if want_dhidden:
        out["dhidden"] = out["dlogits"] @ W
    if want_dW:
        dl = out["dlogits"] if dW_rows is None else out["dlogits"][:, np.asarray(dW_rows)]
        out["dW"] = dl.T @ hidden
    return out
