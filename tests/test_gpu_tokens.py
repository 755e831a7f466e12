"""GPU parity: per-rollout token counts, per-token advantages and loss
weights over packed segments (Sec. 3.3, Sec. 4.1)."""
import numpy as np
import pytest
import torch

from harness import O, TOL_ADV, leap, oracle_rank, oracle_tokens, to_dev
from paper_2608_01804_gb300 import synth

pytestmark = pytest.mark.gpu


def _gpu_tokens(b, turn_adv, T_eff, agg):
    L = leap()
    so, sr, st = to_dev(b.seg_offsets, torch.int32), to_dev(b.seg_rollout, torch.int32), to_dev(b.seg_turn, torch.int8)
    ta = to_dev(turn_adv, torch.float32)
    te = to_dev(T_eff, torch.uint8)
    Lc, tot = L.leap_rollout_token_counts(b.N, so, sr, st, te, M=b.M)
    adv, w = L.leap_scatter_turn_advantages(b.N, so, sr, st, ta, te, Lc, tot, M=b.M, agg=agg)
    return Lc.cpu().numpy(), tot.cpu().numpy(), adv.cpu().numpy(), w.cpu().numpy()


@pytest.mark.parametrize("maker", [synth.tiny_batch, synth.single_turn_batch, synth.multiturn_dcp_batch])
@pytest.mark.parametrize("agg", [O.AGG_SEQ_MEAN_TOKEN_MEAN, O.AGG_TOKEN_MEAN])
def test_counts_and_scatter(maker, agg):
    b = maker()
    orc = oracle_rank(b, gamma=0.9)
    # Same fp32 turn advantages and T_eff on both sides (the rank step is tested on its own).
    ta32 = orc["turn_adv"].reshape(-1).astype(np.float32)
    T_eff = orc["T_eff"].reshape(-1)
    Lc, tot, adv, w = _gpu_tokens(b, ta32, T_eff, agg)
    L_o, nv, rv, adv_o, w_o = oracle_tokens(b, ta32.astype(np.float64), T_eff, agg)
    np.testing.assert_array_equal(Lc, L_o)
    assert tuple(tot) == (nv, rv)
    np.testing.assert_array_equal(adv, adv_o.astype(np.float32))
    np.testing.assert_array_equal(w, w_o.astype(np.float32))      # 1/(R L) in fp64, rounded once
    assert abs(w.astype(np.float64).sum() - 1.0) < 1e-5


def test_counts_past_the_one_block_limit():
    """More rollouts than the one-block count keeps in shared memory (12,000):
    the three-launch count path, against the oracle."""
    b = synth.single_turn_batch(seed=5, num_prompts=1600)      # 12,800 rollouts, 3.3 M tokens
    assert b.n > 12000
    orc = oracle_rank(b, gamma=0.9)
    ta32 = orc["turn_adv"].reshape(-1).astype(np.float32)
    T_eff = orc["T_eff"].reshape(-1)
    Lc, tot, adv, w = _gpu_tokens(b, ta32, T_eff, O.AGG_SEQ_MEAN_TOKEN_MEAN)
    L_o, nv, rv, adv_o, w_o = oracle_tokens(b, ta32.astype(np.float64), T_eff, O.AGG_SEQ_MEAN_TOKEN_MEAN)
    np.testing.assert_array_equal(Lc, L_o)
    assert tuple(tot) == (nv, rv)
    np.testing.assert_array_equal(adv, adv_o.astype(np.float32))
    np.testing.assert_array_equal(w, w_o.astype(np.float32))


def test_dcp_pruned_turns_have_zero_weight():
    b = synth.tiny_batch()
    orc = oracle_rank(b, gamma=0.9)
    ta32 = orc["turn_adv"].reshape(-1).astype(np.float32)
    T_eff = orc["T_eff"].reshape(-1)
    _, _, adv, w = _gpu_tokens(b, ta32, T_eff, O.AGG_SEQ_MEAN_TOKEN_MEAN)
    for s in range(len(b.seg_rollout)):
        i, t = b.seg_rollout[s], b.seg_turn[s]
        a0, a1 = b.seg_offsets[s], b.seg_offsets[s + 1]
        if t < 0 or t >= T_eff[i]:
            assert np.all(w[a0:a1] == 0) and np.all(adv[a0:a1] == 0)


def test_bad_segments_flagged():
    L = leap()
    L.leap_get_device_status()
    M = 2
    so = np.array([0, 4, 2, 10], dtype=np.int32)      # decreasing offsets in segment 1
    sr = np.array([0, 1, 5], dtype=np.int32)           # rollout 5 out of range
    st = np.array([0, 0, 1], dtype=np.int8)
    T_eff = np.array([1, 1], dtype=np.uint8)
    ta = np.array([0.5, 0.0, -1.0, 0.0], dtype=np.float32)
    Lc, tot = L.leap_rollout_token_counts(10, to_dev(so, torch.int32), to_dev(sr, torch.int32),
                                          to_dev(st, torch.int8), to_dev(T_eff, torch.uint8), M=M)
    assert L.leap_get_device_status() & L.LEAP_DEV_BAD_SEGMENT
    np.testing.assert_array_equal(Lc.cpu().numpy(), [4, 0])
    adv, w = L.leap_scatter_turn_advantages(10, to_dev(so, torch.int32), to_dev(sr, torch.int32),
                                            to_dev(st, torch.int8), to_dev(ta, torch.float32),
                                            to_dev(T_eff, torch.uint8), Lc, tot, M=M)
    np.testing.assert_array_equal(adv.cpu().numpy()[:4], 0.5)
    assert np.all(w.cpu().numpy()[4:] == 0)


def test_empty_stream():
    L = leap()
    z32 = torch.zeros(1, dtype=torch.int32, device="cuda")
    e32 = torch.empty(0, dtype=torch.int32, device="cuda")
    e8 = torch.empty(0, dtype=torch.int8, device="cuda")
    te = torch.ones(3, dtype=torch.uint8, device="cuda")
    Lc, tot = L.leap_rollout_token_counts(0, z32, e32, e8, te, M=2)
    assert tot.cpu().tolist() == [0, 0] and Lc.cpu().tolist() == [0, 0, 0]
    adv, w = L.leap_scatter_turn_advantages(0, z32, e32, e8, torch.zeros(6, device="cuda"), te, Lc, tot, M=2)
    assert adv.numel() == 0


def _fused_vs_two_calls(b, ta32, T_eff, agg):
    L = leap()
    so, sr, st = to_dev(b.seg_offsets, torch.int32), to_dev(b.seg_rollout, torch.int32), to_dev(b.seg_turn, torch.int8)
    ta = to_dev(ta32, torch.float32)
    te = to_dev(T_eff, torch.uint8)
    Lc, tot = L.leap_rollout_token_counts(b.N, so, sr, st, te, M=b.M)
    adv, w = L.leap_scatter_turn_advantages(b.N, so, sr, st, ta, te, Lc, tot, M=b.M, agg=agg)
    Lf, totf, advf, wf = L.leap_token_advantages(b.N, so, sr, st, ta, te, M=b.M, agg=agg)
    assert torch.equal(Lf, Lc) and torch.equal(totf, tot)
    assert torch.equal(advf, adv) and torch.equal(wf, w)
    return Lf, totf, advf, wf


@pytest.mark.parametrize("maker", [synth.tiny_batch, synth.single_turn_batch, synth.multiturn_dcp_batch])
@pytest.mark.parametrize("agg", [O.AGG_SEQ_MEAN_TOKEN_MEAN, O.AGG_TOKEN_MEAN])
def test_one_launch_counts_and_scatter(maker, agg):
    """leap_token_advantages (counts + scatter in one launch) equals the two
    calls bit for bit, and the oracle."""
    b = maker()
    orc = oracle_rank(b, gamma=0.9)
    ta32 = orc["turn_adv"].reshape(-1).astype(np.float32)
    T_eff = orc["T_eff"].reshape(-1)
    Lf, totf, advf, wf = _fused_vs_two_calls(b, ta32, T_eff, agg)
    L_o, nv, rv, adv_o, w_o = oracle_tokens(b, ta32.astype(np.float64), T_eff, agg)
    np.testing.assert_array_equal(Lf.cpu().numpy(), L_o)
    assert tuple(totf.cpu().numpy()) == (nv, rv)
    np.testing.assert_array_equal(advf.cpu().numpy(), adv_o.astype(np.float32))
    np.testing.assert_array_equal(wf.cpu().numpy(), w_o.astype(np.float32))


def test_one_launch_fallback_for_large_tables():
    """12,800 rollouts and 25,600 segments do not fit the one-launch kernel's
    shared memory: the call takes the two kernels' path and still matches."""
    b = synth.single_turn_batch(seed=5, num_prompts=1600)
    assert 4 * b.n + 16 * len(b.seg_rollout) > 96 * 1024
    orc = oracle_rank(b, gamma=0.9)
    _fused_vs_two_calls(b, orc["turn_adv"].reshape(-1).astype(np.float32), orc["T_eff"].reshape(-1),
                        O.AGG_SEQ_MEAN_TOKEN_MEAN)


def test_one_launch_bad_segments_and_empty():
    L = leap()
    L.leap_get_device_status()
    so = np.array([0, 4, 2, 10], dtype=np.int32)
    sr = np.array([0, 1, 5], dtype=np.int32)
    st = np.array([0, 0, 1], dtype=np.int8)
    T_eff = np.array([1, 1], dtype=np.uint8)
    ta = np.array([0.5, 0.0, -1.0, 0.0], dtype=np.float32)
    Lf, totf, advf, wf = L.leap_token_advantages(10, to_dev(so, torch.int32), to_dev(sr, torch.int32),
                                                 to_dev(st, torch.int8), to_dev(ta, torch.float32),
                                                 to_dev(T_eff, torch.uint8), M=2)
    assert L.leap_get_device_status() & L.LEAP_DEV_BAD_SEGMENT
    np.testing.assert_array_equal(Lf.cpu().numpy(), [4, 0])
    np.testing.assert_array_equal(advf.cpu().numpy()[:4], 0.5)
    assert np.all(wf.cpu().numpy()[4:] == 0)
    # Empty stream and no segments: counts and totals still written.
    z32 = torch.zeros(1, dtype=torch.int32, device="cuda")
    e32 = torch.empty(0, dtype=torch.int32, device="cuda")
    e8 = torch.empty(0, dtype=torch.int8, device="cuda")
    te = torch.ones(3, dtype=torch.uint8, device="cuda")
    Lc = torch.full((3,), 7, dtype=torch.int32, device="cuda")
    tot = torch.full((2,), 7, dtype=torch.int64, device="cuda")
    L.leap_token_advantages(0, z32, e32, e8, torch.zeros(6, device="cuda"), te, M=2, L=Lc, totals=tot)
    assert tot.cpu().tolist() == [0, 0] and Lc.cpu().tolist() == [0, 0, 0]
