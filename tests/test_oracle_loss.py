"""Pins for the oracle's token path: log-probs, clipped surrogate, dlogits,
per-token advantages/weights and the fused lm-head variant.  CPU only.

Pins: closed forms (uniform logits, rho = 1, hand-built clip branches), a
library routine (scipy's log_softmax), central finite differences of the
oracle's own loss (which catch a wrong sign, branch, temperature or scale in
the gradient), and invariants (sum of weights, chunked sums, row sums).
"""
import numpy as np
import pytest
from scipy.special import log_softmax as sp_log_softmax

from oracle import leap_oracle as O


def test_log_softmax_uniform_and_library():
    V = 1000
    lse, logp = O.log_softmax_rows(np.full((3, V), 2.5), [0, 7, 999])
    np.testing.assert_allclose(logp, -np.log(V), rtol=0, atol=1e-13)
    np.testing.assert_allclose(lse, 2.5 + np.log(V), rtol=1e-15)
    rng = np.random.default_rng(7)
    z = rng.normal(0, 3, size=(5, 257))
    ids = rng.integers(0, 257, size=5)
    for inv_temp in (1.0, 0.7, 1.3):
        _, logp = O.log_softmax_rows(z, ids, inv_temp)
        ref = sp_log_softmax(z * inv_temp, axis=1)[np.arange(5), ids]
        np.testing.assert_allclose(logp, ref, rtol=0, atol=1e-12)
    # Shift invariance and one dominant logit.
    _, a = O.log_softmax_rows(z, ids)
    _, b = O.log_softmax_rows(z + 123.0, ids)
    np.testing.assert_allclose(a, b, atol=1e-12)
    zd = np.zeros((1, 64))
    zd[0, 5] = 20.0
    _, lp = O.log_softmax_rows(zd, [5, ])
    assert lp[0] == pytest.approx(-np.log1p(63 * np.exp(-20.0)), rel=1e-6)
    _, lp = O.log_softmax_rows(zd, [6])
    assert lp[0] == pytest.approx(-20.0, rel=1e-6)


def test_bf16_round_trip():
    vals = np.array([0.0, 1.0, -2.5, 3.140625, 1e-3, 65504.0, -1e30])
    bits = O.f64_to_bf16_bits(vals)
    back = O.bf16_bits_to_f64(bits)
    np.testing.assert_allclose(back, vals, rtol=2 ** -8)
    # Ties round to even: 1 + 2^-8 sits halfway between 1 and 1 + 2^-7.
    assert O.f64_to_bf16_bits(np.array([1.0 + 2 ** -8]))[0] == 0x3F80
    assert O.f64_to_bf16_bits(np.array([1.0 + 3 * 2 ** -8]))[0] == 0x3F82


def test_loss_rho_one_closed_form():
    """old = new => rho = 1, nothing clipped, loss = -sum_k w_k A_k."""
    rng = np.random.default_rng(8)
    z = rng.normal(0, 2, size=(20, 50))
    ids = rng.integers(0, 50, size=20)
    _, logp = O.log_softmax_rows(z, ids)
    adv = rng.normal(size=20)
    w = rng.uniform(0, 1, size=20)
    out = O.grpo_loss_rows(z, ids, logp, adv, w)
    assert out["loss"] == pytest.approx(-(w * adv).sum(), rel=1e-12)
    np.testing.assert_allclose(out["rho"], 1.0, rtol=1e-12)
    assert out["active"].all()


def test_loss_clip_branches_hand_built():
    """One token per branch, values by hand: log-probs are set through old_logp
    so that rho takes chosen values."""
    z = np.zeros((5, 4))          # uniform: logp = -log 4 for every id
    ids = np.zeros(5, dtype=int)
    lp = -np.log(4.0)
    rho = np.array([1.5, 0.5, 1.1, 0.5, 1.5])
    adv = np.array([2.0, -1.0, 1.0, 3.0, -2.0])
    old = lp - np.log(rho)
    w = np.ones(5)
    out = O.grpo_loss_rows(z, ids, old, adv, w, eps_low=0.2, eps_high=0.2)
    # A>0, rho>1.2: clipped at 1.2 -> ell = -1.2*2 ; A<0, rho<0.8: -(0.8*-1) ;
    # inside: -rho*A ; A>0, rho<0.8: min(0.5*3, 0.8*3) -> -1.5 ; A<0, rho>1.2: -(1.5*-2) = 3
    np.testing.assert_allclose(out["ell"], [-2.4, 0.8, -1.1, -1.5, 3.0], rtol=1e-12)
    np.testing.assert_array_equal(out["active"], [False, False, True, True, True])
    np.testing.assert_allclose(out["g"], [0.0, 0.0, -1.1, -1.5, 3.0], rtol=1e-12)


def test_loss_asymmetric_clip_hand_built():
    """Asymmetric clip range eps_low = 0.1, eps_high = 0.28 (Eq. 3 with the two
    edges 0.9 and 1.28), values by hand; tokens 0 and 1 sit where swapping the
    two epsilons, or using 0.2 for both, would change their branch."""
    z = np.zeros((4, 8))          # uniform: logp = -log 8
    ids = np.zeros(4, dtype=int)
    lp = -np.log(8.0)
    rho = np.array([1.25, 0.85, 1.35, 0.95])
    adv = np.array([1.0, -2.0, 0.5, -1.0])
    old = lp - np.log(rho)
    w = np.array([1.0, 0.5, 2.0, 1.0])
    out = O.grpo_loss_rows(z, ids, old, adv, w, eps_low=0.1, eps_high=0.28)
    # A>0, rho=1.25 <= 1.28: unclipped, ell = -1.25 ; A<0, rho=0.85 < 0.9: clipped,
    # ell = -min(-1.7, -1.8) = 1.8 ; A>0, rho=1.35 > 1.28: ell = -1.28*0.5 = -0.64 ;
    # A<0, rho=0.95 >= 0.9: unclipped, ell = 0.95.
    np.testing.assert_allclose(out["ell"], [-1.25, 1.8, -0.64, 0.95], rtol=1e-12)
    np.testing.assert_array_equal(out["active"], [True, False, False, True])
    np.testing.assert_allclose(out["g"], [-1.25, 0.0, 0.0, 0.95], rtol=1e-12)
    np.testing.assert_allclose(out["loss"], -1.25 + 0.9 - 1.28 + 0.95, rtol=1e-12)
    # The symmetric 0.2 range decides tokens 0 and 1 the other way.
    sym = O.grpo_loss_rows(z, ids, old, adv, w, eps_low=0.2, eps_high=0.2)
    np.testing.assert_array_equal(sym["active"], [False, True, False, True])


def _fd_check(z, ids, old, adv, w, inv_temp, grad_scale, eps_low=0.2, eps_high=0.28):
    out = O.grpo_loss_rows(z, ids, old, adv, w, eps_low, eps_high, inv_temp, grad_scale)
    h = 1e-6
    fd = np.zeros_like(z)
    for k in range(z.shape[0]):
        for v in range(z.shape[1]):
            zp, zm = z.copy(), z.copy()
            zp[k, v] += h
            zm[k, v] -= h
            lp = O.grpo_loss_rows(zp, ids, old, adv, w, eps_low, eps_high, inv_temp, grad_scale,
                                  want_dlogits=False)["loss"]
            lm = O.grpo_loss_rows(zm, ids, old, adv, w, eps_low, eps_high, inv_temp, grad_scale,
                                  want_dlogits=False)["loss"]
            fd[k, v] = grad_scale * (lp - lm) / (2 * h)
    return out, fd


def test_dlogits_central_finite_differences():
    """dlogits = d(sum_k w_k ell_k)/dz (times grad_scale), checked numerically on
    tokens away from the clip edges, for several temperatures and scales."""
    rng = np.random.default_rng(9)
    rows, V = 12, 17
    z = rng.normal(0, 2, size=(rows, V))
    ids = rng.integers(0, V, size=rows)
    _, logp = O.log_softmax_rows(z, ids, 0.8)
    old = logp + rng.normal(0, 0.4, size=rows)
    adv = rng.normal(size=rows)
    w = rng.uniform(0.1, 1, size=rows)
    w[3] = 0.0
    for inv_temp, grad_scale in ((1.0, 1.0), (0.8, 2.5)):
        _, logp = O.log_softmax_rows(z, ids, inv_temp)
        rho = np.exp(logp - old)
        keep = (np.abs(rho - 0.8) > 1e-3) & (np.abs(rho - 1.28) > 1e-3)
        out, fd = _fd_check(z, ids, old, adv, w, inv_temp, grad_scale)
        np.testing.assert_allclose(out["dlogits"][keep], fd[keep], rtol=0, atol=1e-7)
        assert (~out["active"]).any() and out["active"].any()   # both branches covered
        np.testing.assert_allclose(out["dlogits"].sum(axis=1), 0.0, atol=1e-14)
        assert np.all(out["dlogits"][3] == 0.0)
        assert np.all(out["dlogits"][~out["active"]] == 0.0)


def test_masked_and_bad_rows():
    z = np.ones((4, 8))
    ids = np.array([1, 9, -1, 2])
    w = np.array([1.0, 1.0, 1.0, 0.0])
    out = O.grpo_loss_rows(z, ids, np.zeros(4), np.ones(4), w)
    np.testing.assert_array_equal(out["bad_id"], [False, True, True, False])
    np.testing.assert_array_equal(out["live"], [True, False, False, False])
    for key in ("logp", "lse", "ell", "g"):
        assert np.all(out[key][1:] == 0.0)
    assert np.all(out["dlogits"][1:] == 0.0)


def _tiny_layout():
    """Two groups of 2 rollouts, M = 2, packed stream of 40 tokens, by hand.

    rollout 0: turn 0 [0,5), feedback [5,8), turn 1 [8,12)
    rollout 1: turn 0 [12,15)                          (passed at turn 1)
    rollout 2: turn 0 [15,20), feedback [20,22), turn 1 [22,30) (turn 1 pruned: T_eff = 1)
    rollout 3: prompt-like masked [30,33), turn 0 [33,38), padding [38,40)
    """
    seg_offsets = np.array([0, 5, 8, 12, 15, 20, 22, 30, 33, 38, 40])
    seg_rollout = np.array([0, 0, 0, 1, 2, 2, 2, -1, 3, -1])
    seg_turn = np.array([0, -1, 1, 0, 0, -1, 1, -1, 0, -1])
    T_eff = np.array([2, 1, 1, 1])
    return seg_offsets, seg_rollout, seg_turn, T_eff


def test_token_counts_and_weights_by_hand():
    so, sr, st, T_eff = _tiny_layout()
    L, nv, rv = O.rollout_token_counts(so, sr, st, T_eff)
    np.testing.assert_array_equal(L, [9, 3, 5, 5])
    assert (nv, rv) == (22, 4)
    M = 2
    turn_adv = np.array([0.5, 1.0, -2.0, 0.0, 3.0, 7.0, 4.0, 0.0])   # [rollout, turn]
    adv, w = O.token_advantages(40, so, sr, st, turn_adv, T_eff, M, O.AGG_SEQ_MEAN_TOKEN_MEAN, L, nv, rv)
    exp_adv = np.zeros(40)
    exp_adv[0:5], exp_adv[8:12], exp_adv[12:15], exp_adv[15:20], exp_adv[33:38] = 0.5, 1.0, -2.0, 3.0, 4.0
    np.testing.assert_array_equal(adv, exp_adv)
    exp_w = np.zeros(40)
    exp_w[0:5] = exp_w[8:12] = 1 / 36
    exp_w[12:15] = 1 / 12
    exp_w[15:20] = 1 / 20
    exp_w[33:38] = 1 / 20
    np.testing.assert_allclose(w, exp_w, rtol=1e-15)
    adv2, w2 = O.token_advantages(40, so, sr, st, turn_adv, T_eff, M, O.AGG_TOKEN_MEAN, L, nv, rv)
    np.testing.assert_array_equal(adv2, exp_adv)
    np.testing.assert_allclose(w2, np.where(exp_w > 0, 1 / 22, 0.0), rtol=1e-15)


def test_weights_sum_to_one_and_chunks_sum_to_whole():
    rng = np.random.default_rng(10)
    n, M, N = 30, 3, 0
    so, sr, st = [0], [], []
    T_eff = rng.integers(0, 4, size=n)
    for i in range(n):
        for t in range(3):
            ln = int(rng.integers(1, 20))
            N += ln
            so.append(N), sr.append(i), st.append(t)
            ln = int(rng.integers(0, 5))
            if ln:
                N += ln
                so.append(N), sr.append(i), st.append(-1)
    so, sr, st = np.array(so), np.array(sr), np.array(st)
    L, nv, rv = O.rollout_token_counts(so, sr, st, T_eff)
    turn_adv = rng.normal(size=n * M)
    for agg in (O.AGG_SEQ_MEAN_TOKEN_MEAN, O.AGG_TOKEN_MEAN):
        adv, w = O.token_advantages(N, so, sr, st, turn_adv, T_eff, M, agg, L, nv, rv)
        assert w.sum() == pytest.approx(1.0, rel=1e-12)
        V = 11
        z = rng.normal(size=(N, V))
        ids = rng.integers(0, V, size=N)
        old = rng.normal(-2.4, 0.3, size=N)
        whole = O.grpo_loss_rows(z, ids, old, adv, w, want_dlogits=False)["loss"]
        parts = 0.0
        for a in range(0, N, 37):
            b = min(N, a + 37)
            parts += O.grpo_loss_rows(z[a:b], ids[a:b], old[a:b], adv[a:b], w[a:b],
                                      want_dlogits=False)["loss"]
        assert parts == pytest.approx(whole, rel=1e-12)


def test_lmhead_dhidden_finite_differences():
    rng = np.random.default_rng(11)
    rows, H, V = 5, 6, 13
    hidden = rng.normal(size=(rows, H))
    W = rng.normal(0, 0.5, size=(V, H))
    ids = rng.integers(0, V, size=rows)
    z = hidden @ W.T
    _, logp = O.log_softmax_rows(z, ids)
    old = logp + rng.normal(0, 0.1, size=rows)
    adv = rng.normal(size=rows)
    w = np.full(rows, 0.2)
    out = O.lmhead_loss_rows(hidden, W, ids, old, adv, w)
    h = 1e-6
    fd = np.zeros_like(hidden)
    for k in range(rows):
        for j in range(H):
            hp, hm = hidden.copy(), hidden.copy()
            hp[k, j] += h
            hm[k, j] -= h
            lp = O.lmhead_loss_rows(hp, W, ids, old, adv, w, want_dhidden=False)["loss"]
            lm = O.lmhead_loss_rows(hm, W, ids, old, adv, w, want_dhidden=False)["loss"]
            fd[k, j] = (lp - lm) / (2 * h)
    np.testing.assert_allclose(out["dhidden"], fd, rtol=0, atol=1e-7)


def test_lmhead_dW_finite_differences():
    """dW = dlogits^T . hidden against central differences of the loss in W,
    including one masked row (w = 0) and two rows sharing a target id."""
    rng = np.random.default_rng(12)
    rows, H, V = 6, 5, 11
    hidden = rng.normal(size=(rows, H))
    W = rng.normal(0, 0.5, size=(V, H))
    ids = rng.integers(0, V, size=rows)
    ids[3] = ids[1]
    z = hidden @ W.T
    _, logp = O.log_softmax_rows(z, ids)
    old = logp + rng.normal(0, 0.1, size=rows)
    adv = rng.normal(size=rows)
    w = np.full(rows, 0.2)
    w[4] = 0.0
    out = O.lmhead_loss_rows(hidden, W, ids, old, adv, w, want_dW=True)
    assert out["dW"].shape == (V, H)
    h = 1e-6
    fd = np.zeros_like(W)
    for v in range(V):
        for j in range(H):
            Wp, Wm = W.copy(), W.copy()
            Wp[v, j] += h
            Wm[v, j] -= h
            lp = O.lmhead_loss_rows(hidden, Wp, ids, old, adv, w, want_dhidden=False)["loss"]
            lm = O.lmhead_loss_rows(hidden, Wm, ids, old, adv, w, want_dhidden=False)["loss"]
            fd[v, j] = (lp - lm) / (2 * h)
    np.testing.assert_allclose(out["dW"], fd, rtol=0, atol=1e-7)
    # Masked rows add nothing: dW over the live rows alone is the same.
    live = w != 0
    sub = O.lmhead_loss_rows(hidden[live], W, ids[live], old[live], adv[live], w[live], want_dW=True)
    np.testing.assert_allclose(sub["dW"], out["dW"], rtol=0, atol=1e-15)
    # Selected vocabulary rows of dW are those rows of the whole.
    pick = [7, 0, ids[1], V - 1]
    part = O.lmhead_loss_rows(hidden, W, ids, old, adv, w, want_dW=True, dW_rows=pick)
    np.testing.assert_allclose(part["dW"], out["dW"][pick], rtol=1e-13, atol=1e-15)
