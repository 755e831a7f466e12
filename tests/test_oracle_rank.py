"""Pins for the oracle's rank-based advantage path (Sec. 3.1-3.3), CPU only.

Each test checks the oracle against something other than itself: the paper's
closed forms (Eqs. 7-9, hand-worked fixtures under tests/golden/), its stated
bounds and regime laws (Eqs. 10-11), a library ranking routine for the
tournament counts, a textbook closed form for GRPO on binary rewards, and
exhaustive enumeration of small groups.
"""
import itertools
import json
import os
from fractions import Fraction

import numpy as np
import pytest
from scipy.stats import rankdata

from oracle import leap_oracle as O


def _tiers_to_pass_turn(tiers, M):
    """Tier index k (0 = first-turn pass ... M-1 = M-th-turn pass, M = failure)."""
    return [(k + 1) if k < M else 0 for k in tiers]


def _run(pass_turn, M, gate_in=None, tau=(0, 10 ** 6), gamma=1.0, num_turns=None, **kw):
    pt = np.asarray(pass_turn, dtype=np.int64).reshape(1, -1)
    if num_turns is None:
        nt = np.where(pt >= 1, pt, M)
    else:
        nt = np.asarray(num_turns, dtype=np.int64).reshape(1, -1)
    gi = None if gate_in is None else np.asarray([gate_in])
    return O.rank_advantages(pt, nt, M, tau[0], tau[1], gamma, gate_in=gi, **kw)


def test_closed_form_three_tier_golden(golden_dir):
    """Eqs. 7-9 (M = 2): every hand-worked case, exactly (R compared as fractions)."""
    with open(os.path.join(golden_dir, "three_tier_closed_form.json")) as f:
        fx = json.load(f)
    M = fx["M"]
    for case in fx["cases"]:
        tiers = [0] * case["N1"] + [1] * case["N2"] + [2] * case["N3"]
        G = len(tiers)
        out = _run(_tiers_to_pass_turn(tiers, M), M)
        for i, k in enumerate(tiers):
            num, den = case["R_O%d" % (k + 1)]
            assert Fraction(int(out["n_worse"][0, i] - out["n_better"][0, i]), G - 1) == Fraction(num, den)
            assert out["R"][0, i] == pytest.approx(num / den, abs=1e-15)


def test_closed_form_three_tier_exhaustive():
    """Eqs. 7-9 for every (N1, N2, N3) with G <= 9, in random positions in the group."""
    rng = np.random.default_rng(1)
    for G in range(2, 10):
        for N1 in range(G + 1):
            for N2 in range(G + 1 - N1):
                N3 = G - N1 - N2
                tiers = np.array([0] * N1 + [1] * N2 + [2] * N3)
                rng.shuffle(tiers)
                out = _run(_tiers_to_pass_turn(tiers, 2), 2)
                expect = {0: (N2 + N3) / (G - 1), 1: (N3 - N1) / (G - 1), 2: -(N1 + N2) / (G - 1)}
                for i, k in enumerate(tiers):
                    assert out["R"][0, i] == pytest.approx(expect[int(k)], abs=1e-15)


def test_tournament_counts_match_competition_ranking():
    """Eq. 5 vs a library routine: N_better + 1 is the 'min' competition rank of -r,
    N_worse + 1 the 'min' rank of r (ties share the lowest rank)."""
    rng = np.random.default_rng(2)
    for G in (2, 3, 8, 16, 64, 257):
        r = rng.integers(0, 4, size=(5, G))
        nw, nb = O.tournament(r)
        for g in range(5):
            np.testing.assert_array_equal(nb[g], rankdata(-r[g], method="min").astype(int) - 1)
            np.testing.assert_array_equal(nw[g], rankdata(r[g], method="min").astype(int) - 1)


def test_reward_bounds_and_extremes():
    """Eq. 6 bounds: R in [-1, 1]; a sole winner gets +1, a sole loser -1."""
    for M in (1, 2, 3):
        for G in range(2, 8):
            for tiers in itertools.combinations_with_replacement(range(M + 1), G):
                out = _run(_tiers_to_pass_turn(tiers, M), M)
                R = out["R"][0]
                assert np.all(R >= -1.0) and np.all(R <= 1.0)
                best, worst = min(tiers), max(tiers)
                if tiers.count(best) == 1 and best != worst:
                    assert R[tiers.index(best)] == 1.0
                if tiers.count(worst) == 1 and best != worst:
                    assert R[tiers.index(worst)] == -1.0


def test_reward_zero_sum_and_all_tied():
    """Each strict pair adds +1 and -1, so sum_i R_i = 0; an all-tied group gets R = A = 0."""
    rng = np.random.default_rng(3)
    r = rng.integers(0, 4, size=(50, 16))
    nw, nb = O.tournament(r)
    np.testing.assert_array_equal((nw - nb).sum(axis=1), 0)
    for M in (1, 2, 3):
        for k in range(M + 1):
            for eps in (1e-6, 0.0):
                out = _run(_tiers_to_pass_turn([k] * 6, M), M, eps_std=eps)
                assert np.all(out["R"] == 0.0) and np.all(out["A"] == 0.0)


def test_regime_laws_of_the_intermediate_tier():
    """Eqs. 10-11 and the partial-derivative claim: sign R(O2) = sign(N3 - N1);
    moving one rollout from O1 to O3 raises R(O2) by 2/(G-1)."""
    for G in range(3, 12):
        for N1 in range(G):
            for N3 in range(G - N1):
                N2 = G - N1 - N3
                if N2 < 1:
                    continue
                tiers = [0] * N1 + [1] * N2 + [2] * N3
                R2 = _run(_tiers_to_pass_turn(tiers, 2), 2)["R"][0, N1]
                assert np.sign(R2) == np.sign(N3 - N1)
                if N1 >= 1:
                    tiers_b = [0] * (N1 - 1) + [1] * N2 + [2] * (N3 + 1)
                    R2b = _run(_tiers_to_pass_turn(tiers_b, 2), 2)["R"][0, N1 - 1]
                    assert R2b - R2 == pytest.approx(2.0 / (G - 1), abs=1e-14)


def test_permutation_equivariance_and_scale_free():
    """Permuting a group permutes R and A; relabelling tiers by any strictly
    increasing map (another M, other gaps) leaves R and A unchanged."""
    rng = np.random.default_rng(4)
    for _ in range(40):
        G = int(rng.integers(2, 40))
        r = rng.integers(0, 4, size=(1, G))
        nw, nb = O.tournament(r)
        R = O.tournament_reward(nw, nb, G)
        A = O.grpo_advantage(R)
        perm = rng.permutation(G)
        nw2, nb2 = O.tournament(r[:, perm])
        R2 = O.tournament_reward(nw2, nb2, G)
        np.testing.assert_array_equal(R2, R[:, perm])
        np.testing.assert_allclose(O.grpo_advantage(R2), A[:, perm], rtol=0, atol=1e-12)
        relabel = np.array([0, 5, 6, 40])           # strictly increasing
        nw3, nb3 = O.tournament(relabel[r])
        np.testing.assert_array_equal(O.tournament_reward(nw3, nb3, G), R)


def test_grpo_advantage_binary_closed_form():
    """Single turn (M = 1): R is an affine map of the binary pass reward, so the
    standard GRPO advantage (unbiased std, eps -> 0) has the textbook closed form
    A_pass = sqrt((G-k)(G-1)/(G k)), A_fail = -sqrt(k (G-1)/(G (G-k)))."""
    for G in (2, 3, 8, 16, 64):
        for k in range(1, G):
            tiers = [0] * k + [1] * (G - k)
            out = _run(_tiers_to_pass_turn(tiers, 1), 1, eps_std=0.0)
            A = out["A"][0]
            a_pass = np.sqrt((G - k) * (G - 1) / (G * k))
            a_fail = -np.sqrt(k * (G - 1) / (G * (G - k)))
            np.testing.assert_allclose(A[:k], a_pass, rtol=1e-12)
            np.testing.assert_allclose(A[k:], a_fail, rtol=1e-12)
    # Biased-std variant: A_pass = sqrt((G-k)/k).
    out = _run(_tiers_to_pass_turn([0, 0, 1, 1, 1, 1, 1, 1], 1), 1, eps_std=0.0, std_unbiased=False)
    np.testing.assert_allclose(out["A"][0, :2], np.sqrt(6 / 2), rtol=1e-12)


def test_grpo_advantage_none_mode_and_scale_invariance():
    rng = np.random.default_rng(5)
    R = rng.uniform(-1, 1, size=(3, 9))
    np.testing.assert_array_equal(O.grpo_advantage(R, norm=O.ADVNORM_NONE), R)
    np.testing.assert_allclose(O.grpo_advantage(3.7 * R, eps_std=0.0), O.grpo_advantage(R, eps_std=0.0),
                               rtol=1e-12)


def test_dcp_gate_truth_table(golden_dir):
    """Eqs. 1-2, hand-worked truth table (inclusive bounds, first-turn failures)."""
    with open(os.path.join(golden_dir, "dcp_gate.json")) as f:
        fx = json.load(f)
    for case in fx["cases"]:
        out = _run(case["pass_turn"], fx["M"], tau=case["tau"])
        assert out["n_fail"][0] == case["n_fail"]
        assert out["gate"][0] == case["gate"]


def test_gated_off_groups_are_truncated_to_turn_one():
    """A gated-off group never ran turn 2: a turn-2 pass is a failure, T_eff = 1."""
    M = 3
    pt = [1, 2, 3, 0]
    nt = [1, 2, 3, 3]
    off = _run(pt, M, gate_in=0, num_turns=nt)
    np.testing.assert_array_equal(off["r"][0], [3, 0, 0, 0])
    np.testing.assert_array_equal(off["T_eff"][0], [1, 1, 1, 1])
    on = _run(pt, M, gate_in=1, num_turns=nt)
    np.testing.assert_array_equal(on["r"][0], [3, 2, 1, 0])
    np.testing.assert_array_equal(on["T_eff"][0], nt)
    # Gated off, only the first-turn pass beats the rest.
    np.testing.assert_allclose(off["R"][0], [1.0, -1 / 3, -1 / 3, -1 / 3])


def test_bad_outcomes_are_failures_without_tokens():
    out = _run([1, 5, -1, 2], 2, num_turns=[1, 2, 2, 1])   # 5 > M, -1 < 0, pass at 2 > T = 1
    np.testing.assert_array_equal(out["bad_outcome"][0], [False, True, True, True])
    np.testing.assert_array_equal(out["r"][0], [2, 0, 0, 0])
    np.testing.assert_array_equal(out["T_eff"][0], [1, 0, 0, 0])


def test_turn_discount_golden(golden_dir):
    """Sec. 3.3 discount, hand-worked cases."""
    with open(os.path.join(golden_dir, "turn_discount.json")) as f:
        fx = json.load(f)
    M = 4
    for case in fx["cases"]:
        A = np.array([[case["A"]]])
        T = np.array([[case["T"]]])
        out = O.turn_advantages(A, T, case["gamma"], M)[0, 0]
        np.testing.assert_allclose(out[:case["T"]], case["A_hat"], rtol=0, atol=1e-15)
        assert np.all(out[case["T"]:] == 0.0)


def test_turn_discount_properties():
    """Last turn keeps A; consecutive turns differ by the factor gamma when A >= 0;
    A < 0 gives equal turns; gamma = 1 is a plain broadcast."""
    rng = np.random.default_rng(6)
    A = rng.normal(size=(4, 16))
    T = rng.integers(1, 4, size=(4, 16))
    for gamma in (1.0, 0.9, 0.5):
        ta = O.turn_advantages(A, T, gamma, 3)
        for g in range(4):
            for i in range(16):
                t_last = T[g, i] - 1
                assert ta[g, i, t_last] == A[g, i]
                for t in range(t_last):
                    if A[g, i] >= 0:
                        assert ta[g, i, t] == pytest.approx(gamma * ta[g, i, t + 1], rel=1e-14)
                    else:
                        assert ta[g, i, t] == A[g, i]
                assert np.all(ta[g, i, T[g, i]:] == 0)


# ---- extensions: lexicographic tie-breaks, static-scalar baseline, counters ----

def _lexi_brute(r, sp, tk):
    """Python tuple ordering as an independent formulation of the tie-broken
    tournament: passing rollouts carry (r, speedup, -tokens), failures (0,)."""
    keys = [(int(a), float(b), -int(c)) if a > 0 else (0,) for a, b, c in zip(r, sp, tk)]
    nw = [sum(1 for j, kj in enumerate(keys) if j != i and ki > kj) for i, ki in enumerate(keys)]
    nb = [sum(1 for j, kj in enumerate(keys) if j != i and ki < kj) for i, ki in enumerate(keys)]
    return np.array(nw), np.array(nb)


def test_lexi_tournament_against_tuple_ordering():
    rng = np.random.default_rng(21)
    for G in (2, 5, 8, 33):
        r = rng.integers(0, 4, size=(6, G))
        sp = rng.choice([0.5, 1.0, 1.5], size=(6, G))          # many exact ties
        tk = rng.choice([100, 200], size=(6, G))
        nw, nb = O.tournament_lexi(r, sp, tk)
        for g in range(6):
            bw, bb = _lexi_brute(r[g], sp[g], tk[g])
            np.testing.assert_array_equal(nw[g], bw)
            np.testing.assert_array_equal(nb[g], bb)
        np.testing.assert_array_equal(nw.sum(axis=1), nb.sum(axis=1))


def test_lexi_reduces_to_paper_comparator_without_tie_breaks():
    rng = np.random.default_rng(22)
    r = rng.integers(0, 4, size=(10, 16))
    nw, nb = O.tournament_lexi(r, np.ones_like(r, dtype=float), np.full(r.shape, 7))
    pw, pb = O.tournament(r)
    np.testing.assert_array_equal(nw, pw)
    np.testing.assert_array_equal(nb, pb)


def test_static_reward_baseline_by_hand():
    """GRPO-MT baseline, G = 4, M = 2, c = 0.5: outcomes (turn-1 pass, turn-2
    pass, fail, fail) -> R = (1, 0.5, 0, 0), mean 0.375, unbiased std
    sqrt(0.6875 / 3); A worked out by hand."""
    out = _run([1, 2, 0, 0], 2, reward=O.REWARD_STATIC, static_c=0.5, eps_std=0.0)
    np.testing.assert_allclose(out["R"][0], [1.0, 0.5, 0.0, 0.0])
    std = np.sqrt(0.6875 / 3)
    np.testing.assert_allclose(out["A"][0], np.array([0.625, 0.125, -0.375, -0.375]) / std, rtol=1e-12)
    # Single turn: the static reward is the binary reward, so A equals the rank-based A.
    a = _run([1, 0, 1, 1, 0], 1, reward=O.REWARD_STATIC, eps_std=0.0)["A"]
    b = _run([1, 0, 1, 1, 0], 1, eps_std=0.0)["A"]
    np.testing.assert_allclose(a, b, rtol=1e-12)


def test_rank_stats_by_hand():
    """Two groups of 4, M = 3.  Group 0 gated on: turn-1 pass, turn-2 pass,
    turn-3 pass, fail (T = 1, 2, 3, 3).  Group 1 gated off: pass, fail, fail,
    turn-2 pass truncated to a failure."""
    pt = np.array([[1, 2, 3, 0], [1, 0, 0, 2]])
    nt = np.array([[1, 2, 3, 3], [1, 1, 1, 2]])
    out = O.rank_advantages(pt, nt, 3, 0, 4, 0.9, gate_in=np.array([1, 0]))
    st = O.rank_stats(out, pt, 3)
    assert (st["groups"], st["gated_groups"], st["rollouts"]) == (2, 1, 8)
    assert (st["first_turn_passes"], st["later_passes"]) == (2, 2)
    assert (st["groups_with_recovery"], st["failed_first_turn_in_gated"]) == (1, 3)
    assert st["total_turns"] == 1 + 2 + 3 + 3 + 4
    assert st["passes_by_turn"][:3] == [2, 1, 1]


def test_rank_composition_by_hand():
    """Fig. 4 counts (Sec. 4.5) on four groups of G = 4, M = 3, worked by hand.
    Group 0, expanded: turn-1 pass x2, turn-2 pass, failure; 2 of 4 passed turn 1
    (bucket 5); r = 3, 3, 2, 0 so d = 2, 2, -1, -3.  Group 1, not expanded: its
    turn-2 pass never ran (a failure), one turn-1 pass; 1 of 4 (bucket 2);
    r = 0, 0, 0, 3 so d = -1, -1, -1, 3.  Group 2: all fail (bucket 0), group 3:
    all pass at turn 1 (bucket 9); both all-tied, so A = 0 and nothing counts."""
    pt = np.array([[1, 1, 2, 0], [2, 0, 0, 1], [0, 0, 0, 0], [1, 1, 1, 1]])
    nt = np.array([[1, 1, 2, 3], [2, 1, 1, 1], [1, 1, 1, 1], [1, 1, 1, 1]])
    gate = np.array([1, 0, 0, 0])
    expect = np.zeros((10, 3, 2), dtype=np.int64)
    expect[5, 0, 0] = 2      # immediate passes, A > 0
    expect[5, 1, 1] = 1      # debug-assisted pass, A < 0 (beaten by both turn-1 passes)
    expect[5, 2, 1] = 1      # failure, A < 0
    expect[2, 0, 0] = 1
    expect[2, 2, 1] = 3      # includes the truncated turn-2 pass
    groups = [1, 0, 1, 0, 0, 1, 0, 0, 0, 1]
    for reward in (O.REWARD_RANK, O.REWARD_STATIC):   # static 1 / 0.5 / 0 gives the same signs here
        out = O.rank_advantages(pt, nt, 3, 0, 4, 0.9, gate_in=gate, reward=reward, static_c=0.5)
        comp, gb = O.rank_composition(out, 3)
        np.testing.assert_array_equal(comp, expect)
        assert gb.tolist() == groups
        st = O.rank_stats(out, pt, 3)
        assert st["composition"] == expect.tolist() and st["groups_by_bucket"] == groups
        assert int(comp.sum()) == st["nonzero_adv_rollouts"] == 8


def test_rank_composition_invariants():
    """On a random batch: every nonzero-advantage rollout is counted once, every
    group sits in one bucket, groups whose rollouts all pass turn 1 land in the
    last bucket and those with none in the first, and with M = 1 there is no
    debug-assisted pass."""
    rng = np.random.default_rng(5)
    for G, M in ((8, 3), (16, 1), (64, 3), (5, 2)):
        n = 300
        T = rng.integers(1, M + 1, size=(n, G))
        pt = np.where(rng.random((n, G)) < 0.5, rng.integers(1, M + 1, size=(n, G)), 0)
        pt = np.minimum(pt, T)
        pt[0] = 1
        pt[1] = 0
        out = O.rank_advantages(pt, T, M, 2, G - 2, 0.9)
        comp, gb = O.rank_composition(out, M)
        st = O.rank_stats(out, pt, M)
        assert int(comp.sum()) == st["nonzero_adv_rollouts"]
        assert int(gb.sum()) == n
        b = np.minimum(9, (10 * (G - out["n_fail"])) // G)
        assert b[0] == 9 and b[1] == 0
        np.testing.assert_array_equal(np.bincount(b, minlength=10), gb)
        if M == 1:
            assert comp[:, 1, :].sum() == 0
