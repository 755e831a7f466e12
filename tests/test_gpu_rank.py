"""GPU parity: rank-based advantages (Sec. 3.1-3.3) against the oracle.

Integers, the gate and R are compared bit for bit; A and the per-turn
advantages within 1e-5 absolute."""
import numpy as np
import pytest
import torch

from harness import O, TOL_ADV, leap, oracle_rank, to_dev
from paper_2608_01804_gb300 import synth

pytestmark = pytest.mark.gpu


def _run_gpu(pass_turn, num_turns, G, M, tau, gamma, gate_in=None, **kw):
    L = leap()
    return L.leap_group_rank_advantages(to_dev(pass_turn, torch.int8), to_dev(num_turns, torch.int8), G=G, M=M,
                                        tau_min=tau[0], tau_max=tau[1], gamma=gamma,
                                        gate_in=None if gate_in is None else to_dev(gate_in, torch.uint8), **kw)


def _compare(gpu, orc, M, strict_A=True):
    n = orc["r"].size
    np.testing.assert_array_equal(gpu["gate"].cpu().numpy(), orc["gate"])
    np.testing.assert_array_equal(gpu["r"].cpu().numpy(), orc["r"].reshape(-1))
    np.testing.assert_array_equal(gpu["T_eff"].cpu().numpy(), orc["T_eff"].reshape(-1))
    np.testing.assert_array_equal(gpu["n_worse"].cpu().numpy(), orc["n_worse"].reshape(-1))
    np.testing.assert_array_equal(gpu["n_better"].cpu().numpy(), orc["n_better"].reshape(-1))
    R32 = orc["R"].reshape(-1).astype(np.float32)
    np.testing.assert_array_equal(gpu["R"].cpu().numpy(), R32)
    A = gpu["A"].cpu().numpy().astype(np.float64)
    assert np.max(np.abs(A - orc["A"].reshape(-1))) <= TOL_ADV
    ta = gpu["turn_adv"].cpu().numpy().astype(np.float64).reshape(n, M)
    assert np.max(np.abs(ta - orc["turn_adv"].reshape(n, M))) <= TOL_ADV
    # Signs decide the discount base: they must agree wherever the net score is
    # nonzero (there |A| >= 1/((G-1)(std+eps)); a zero net score leaves only
    # rounding noise of the oracle's fp64 mean).
    nz = np.abs(orc["A"].reshape(-1)) > 1e-9
    assert np.all(np.sign(A[nz]) == np.sign(orc["A"].reshape(-1)[nz]))


def test_tiny_batch_recorded_gate():
    b = synth.tiny_batch()
    gpu = _run_gpu(b.pass_turn, b.num_turns, b.G, b.M, (0, b.G), 0.9, gate_in=b.gate_in)
    orc = oracle_rank(b, gamma=0.9)
    _compare(gpu, orc, b.M)
    # Turn 2 of the gated-off prompts 0 and 1 is pruned.
    assert np.all(gpu["T_eff"].cpu().numpy()[:16] == 1)


@pytest.mark.parametrize("tau", [(4, 7), (0, 8), (8, 8), (0, 0)])
def test_tiny_batch_computed_gate(tau):
    b = synth.tiny_batch(seed=5)
    gpu = _run_gpu(b.pass_turn, b.num_turns, b.G, b.M, tau, 0.5)
    orc = oracle_rank(b, tau=tau, gamma=0.5, use_gate_in=False)
    _compare(gpu, orc, b.M)


def test_tournament_stress_full_size():
    """65,536 groups x G = 64, M = 3, ~10% exact duplicate tuples: bit-exact counts."""
    pt, nt, sp, tok = synth.tournament_outcomes()
    G, M = 64, 3
    gpu = _run_gpu(pt, nt, G, M, (50, 56), 0.9)
    orc = O.rank_advantages(pt.reshape(-1, G), nt.reshape(-1, G), M, 50, 56, 0.9)
    _compare(gpu, orc, M)
    assert 0.2 < orc["gate"].mean() < 0.9


@pytest.mark.parametrize("G", [2, 3, 31, 32, 33, 64, 100, 257, 1024])
@pytest.mark.parametrize("M", [1, 3, 8])
def test_group_sizes_and_turns(G, M):
    rng = np.random.default_rng(G * 10 + M)
    groups = max(1, 4096 // G)
    nt = rng.integers(1, M + 1, size=groups * G).astype(np.int8)
    pt = np.where(rng.random(groups * G) < 0.5, rng.integers(1, M + 1, size=groups * G), 0)
    pt = np.minimum(pt, nt).astype(np.int8)
    tau = (G // 4, (3 * G) // 4)
    gpu = _run_gpu(pt, nt, G, M, tau, 0.8)
    orc = O.rank_advantages(pt.reshape(-1, G), nt.reshape(-1, G), M, tau[0], tau[1], 0.8)
    _compare(gpu, orc, M)


@pytest.mark.parametrize("norm,unbiased,eps", [(O.ADVNORM_NONE, 1, 1e-6), (O.ADVNORM_GRPO_STD, 0, 1e-6),
                                                (O.ADVNORM_GRPO_STD, 1, 0.0), (O.ADVNORM_GRPO_STD, 1, 0.1)])
def test_norm_modes(norm, unbiased, eps):
    b = synth.multiturn_dcp_batch(seed=7)
    gpu = _run_gpu(b.pass_turn, b.num_turns, b.G, b.M, (0, b.G), 0.9, gate_in=b.gate_in, norm=norm,
                   std_unbiased=bool(unbiased), eps_std=eps)
    orc = oracle_rank(b, gamma=0.9, eps_std=eps, norm=norm, std_unbiased=bool(unbiased))
    _compare(gpu, orc, b.M)


def test_bad_outcomes_flagged_and_ranked_as_failures():
    L = leap()
    L.leap_get_device_status()
    G, M = 8, 2
    pt = np.array([1, 2, 0, 5, 1, 1, -1, 2], dtype=np.int8)
    nt = np.array([1, 2, 2, 2, 1, 1, 1, 1], dtype=np.int8)   # index 7: pass at 2 > T = 1
    gpu = _run_gpu(pt, nt, G, M, (0, G), 0.9)
    orc = O.rank_advantages(pt.reshape(1, G), nt.reshape(1, G), M, 0, G, 0.9)
    _compare(gpu, orc, M)
    assert L.leap_get_device_status() & L.LEAP_DEV_BAD_OUTCOME
    assert L.leap_get_device_status() == 0   # cleared by the read


def test_empty_and_gamma_one():
    L = leap()
    empty = torch.empty(0, dtype=torch.int8, device="cuda")
    out = L.leap_group_rank_advantages(empty, empty, G=8, M=2, tau_max=8)
    assert out["A"].numel() == 0
    b = synth.tiny_batch(seed=9)
    gpu = _run_gpu(b.pass_turn, b.num_turns, b.G, b.M, (0, b.G), 1.0, gate_in=b.gate_in)
    ta = gpu["turn_adv"].cpu().numpy().reshape(-1, b.M)
    T = gpu["T_eff"].cpu().numpy()
    A = gpu["A"].cpu().numpy()
    for i in range(ta.shape[0]):
        assert np.all(ta[i, :T[i]] == A[i]) and np.all(ta[i, T[i]:] == 0)


# ---- extensions: tie-broken comparator, static-scalar baseline, counters ----

def test_lexi_tournament_stress_full_size():
    """65,536 groups x 64 with ~10% exact duplicate tuples: the tie-broken
    tournament, bit-exact."""
    pt, nt, sp, tok = synth.tournament_outcomes()
    G, M = 64, 3
    L = leap()
    gpu = L.leap_group_rank_advantages(to_dev(pt, torch.int8), to_dev(nt, torch.int8), G=G, M=M, tau_min=50,
                                       tau_max=56, gamma=0.9, cmp=L.LEAP_CMP_LEXI,
                                       speedup=to_dev(sp, torch.float32), ntokens=to_dev(tok, torch.int32))
    orc = O.rank_advantages(pt.reshape(-1, G), nt.reshape(-1, G), M, 50, 56, 0.9, cmp=O.CMP_LEXI,
                            speedup=sp.reshape(-1, G), ntokens=tok.reshape(-1, G))
    _compare(gpu, orc, M)
    assert np.any(orc["n_worse"] + orc["n_better"] < G - 1)   # exact ties occurred


@pytest.mark.parametrize("G,M", [(8, 2), (64, 3), (100, 4), (1024, 3)])
def test_lexi_group_sizes(G, M):
    rng = np.random.default_rng(G + M)
    groups = max(1, 2048 // G)
    n = groups * G
    nt = rng.integers(1, M + 1, size=n).astype(np.int8)
    pt = np.minimum(np.where(rng.random(n) < 0.6, rng.integers(1, M + 1, size=n), 0), nt).astype(np.int8)
    sp = rng.choice([0.5, 1.0, 2.0], size=n).astype(np.float32)
    tok = rng.choice([128, 256], size=n).astype(np.int32)
    L = leap()
    gpu = L.leap_group_rank_advantages(to_dev(pt, torch.int8), to_dev(nt, torch.int8), G=G, M=M, tau_max=G,
                                       gamma=0.8, cmp=L.LEAP_CMP_LEXI, speedup=to_dev(sp, torch.float32),
                                       ntokens=to_dev(tok, torch.int32))
    orc = O.rank_advantages(pt.reshape(-1, G), nt.reshape(-1, G), M, 0, G, 0.8, cmp=O.CMP_LEXI,
                            speedup=sp.reshape(-1, G), ntokens=tok.reshape(-1, G))
    _compare(gpu, orc, M)


@pytest.mark.parametrize("c,eps", [(0.5, 1e-6), (0.2, 0.0), (1.0, 1e-6)])
def test_static_reward_baseline(c, eps):
    b = synth.multiturn_dcp_batch(seed=9)
    L = leap()
    gpu = L.leap_group_rank_advantages(to_dev(b.pass_turn, torch.int8), to_dev(b.num_turns, torch.int8), G=b.G,
                                       M=b.M, tau_max=b.G, gamma=0.9, gate_in=to_dev(b.gate_in, torch.uint8),
                                       reward=L.LEAP_REWARD_STATIC, static_c=c, eps_std=eps)
    orc = O.rank_advantages(b.pass_turn.reshape(-1, b.G), b.num_turns.reshape(-1, b.G), b.M, 0, b.G, 0.9,
                            eps_std=eps, gate_in=b.gate_in, reward=O.REWARD_STATIC, static_c=c)
    np.testing.assert_array_equal(gpu["n_worse"].cpu().numpy(), orc["n_worse"].reshape(-1))
    np.testing.assert_allclose(gpu["R"].cpu().numpy(), orc["R"].reshape(-1), rtol=0, atol=1e-7)
    assert np.max(np.abs(gpu["A"].cpu().numpy() - orc["A"].reshape(-1))) <= TOL_ADV
    ta = gpu["turn_adv"].cpu().numpy().reshape(-1, b.M)
    assert np.max(np.abs(ta - orc["turn_adv"].reshape(-1, b.M))) <= TOL_ADV


@pytest.mark.parametrize("maker,tau", [(synth.multiturn_dcp_batch, (8, 15)), (synth.tiny_batch, (3, 6))])
def test_rank_stats_match_oracle(maker, tau):
    b = maker()
    L = leap()
    st = L.rank_stats_tensor("cuda")
    gpu = L.leap_group_rank_advantages(to_dev(b.pass_turn, torch.int8), to_dev(b.num_turns, torch.int8), G=b.G,
                                       M=b.M, tau_min=tau[0], tau_max=tau[1], gamma=0.9, stats=st)
    orc = O.rank_advantages(b.pass_turn.reshape(-1, b.G), b.num_turns.reshape(-1, b.G), b.M, tau[0], tau[1], 0.9)
    exp = O.rank_stats(orc, b.pass_turn.reshape(-1, b.G), b.M)
    got = L.read_rank_stats(st)
    assert got == exp
    # accumulate: a second call doubles every counter
    L.leap_group_rank_advantages(to_dev(b.pass_turn, torch.int8), to_dev(b.num_turns, torch.int8), G=b.G, M=b.M,
                                 tau_min=tau[0], tau_max=tau[1], gamma=0.9, stats=st)
    got2 = L.read_rank_stats(st)
    assert got2["total_turns"] == 2 * exp["total_turns"] and got2["groups"] == 2 * exp["groups"]


def test_rank_stats_full_size_tournament():
    pt, nt, sp, tok = synth.tournament_outcomes()
    G, M = 64, 3
    L = leap()
    st = L.rank_stats_tensor("cuda")
    L.leap_group_rank_advantages(to_dev(pt, torch.int8), to_dev(nt, torch.int8), G=G, M=M, tau_min=50, tau_max=56,
                                 gamma=0.9, stats=st)
    orc = O.rank_advantages(pt.reshape(-1, G), nt.reshape(-1, G), M, 50, 56, 0.9)
    assert L.read_rank_stats(st) == O.rank_stats(orc, pt.reshape(-1, G), M)


@pytest.mark.parametrize("G,M,groups,reward,tau", [(64, 3, 65536, 0, (20, 44)), (64, 3, 65536, 1, (20, 44)),
                                                    (33, 2, 4000, 0, (10, 25)), (100, 3, 2000, 1, (30, 80)),
                                                    (8, 1, 8000, 0, (0, 8))])
def test_rank_composition_matches_oracle(G, M, groups, reward, tau):
    """Fig. 4 counters (pass-rate bucket x outcome type x sign of A) and the
    other training counters, pair kernel and generic kernel, tournament and
    static-scalar rewards (the two reward definitions the figure compares),
    equal to the oracle."""
    pt, nt, _, _ = synth.tournament_outcomes(seed=G + M, num_groups=groups, G=G, M=M)
    L = leap()
    st = L.rank_stats_tensor("cuda")
    L.leap_group_rank_advantages(to_dev(pt, torch.int8), to_dev(nt, torch.int8), G=G, M=M, tau_min=tau[0],
                                 tau_max=tau[1], gamma=0.9, stats=st, reward=reward, static_c=0.5)
    orc = O.rank_advantages(pt.reshape(-1, G), nt.reshape(-1, G), M, tau[0], tau[1], 0.9, reward=reward,
                            static_c=0.5)
    exp = O.rank_stats(orc, pt.reshape(-1, G), M)
    got = L.read_rank_stats(st)
    assert got["composition"] == exp["composition"]
    assert got["groups_by_bucket"] == exp["groups_by_bucket"]
    assert got == exp
    assert sum(sum(sum(x) for x in b) for b in got["composition"]) == got["nonzero_adv_rollouts"]


@pytest.mark.parametrize("G,M", [(64, 3), (16, 2), (2, 8)])
def test_pair_and_generic_kernels_agree(G, M):
    """Even G <= 64 with the paper's comparator runs the pair kernel (vector
    loads and stores); outputs that are not 8-byte aligned send the same call
    to the generic kernel.  Both equal the oracle and each other, bit for bit."""
    rng = np.random.default_rng(7 * G + M)
    groups = 2048 // G + 3
    n = groups * G
    nt = rng.integers(1, M + 1, size=n).astype(np.int8)
    pt = np.minimum(np.where(rng.random(n) < 0.5, rng.integers(1, M + 1, size=n), 0), nt).astype(np.int8)
    pt[5] = M + 1                                   # one malformed outcome
    L = leap()
    dev = torch.device("cuda")
    pt_d, nt_d = torch.as_tensor(pt, device=dev), torch.as_tensor(nt, device=dev)
    tau = (G // 4, (3 * G) // 4)
    L.leap_get_device_status()                      # clears the sticky flags
    aligned = L.leap_group_rank_advantages(pt_d, nt_d, G=G, M=M, tau_min=tau[0], tau_max=tau[1], gamma=0.8)
    off = lambda k, dt: torch.empty(k + 1, dtype=dt, device=dev)[1:]    # 4-byte offset: generic kernel
    out = dict(gate=off(groups, torch.uint8), r=off(n, torch.uint8), n_worse=off(n, torch.int32),
               n_better=off(n, torch.int32), R=off(n, torch.float32), A=off(n, torch.float32),
               turn_adv=off(n * M, torch.float32), T_eff=off(n, torch.uint8))
    generic = L.leap_group_rank_advantages(pt_d, nt_d, G=G, M=M, tau_min=tau[0], tau_max=tau[1], gamma=0.8,
                                           out=out)
    torch.cuda.synchronize()
    assert L.leap_get_device_status() & L.LEAP_DEV_BAD_OUTCOME
    for k in aligned:
        assert torch.equal(aligned[k], generic[k]), k
    orc = O.rank_advantages(pt.reshape(-1, G), nt.reshape(-1, G), M, tau[0], tau[1], 0.8)
    _compare(aligned, orc, M)


@pytest.mark.parametrize("G", [8, 64, 100, 300])
def test_lexi_special_keys(G):
    """Tie-breaks on edge values: +0 and -0 speedups (equal), infinities,
    negative and extreme token counts, and NaN speedups in some groups (a NaN
    compares false both ways, so those groups take the peer-by-peer path)."""
    rng = np.random.default_rng(3 * G)
    groups = max(4, 2048 // G)
    n = groups * G
    M = 3
    nt = rng.integers(1, M + 1, size=n).astype(np.int8)
    pt = np.minimum(np.where(rng.random(n) < 0.7, rng.integers(1, M + 1, size=n), 0), nt).astype(np.int8)
    sp = rng.choice(np.array([0.0, -0.0, 1.0, np.inf, -np.inf, 2.5, -3.0], dtype=np.float32), size=n)
    tok = rng.choice(np.array([0, 1, -5, 2 ** 31 - 1, -2 ** 31, 128], dtype=np.int64), size=n).astype(np.int32)
    sp[G * 1 + 3] = np.nan                       # group 1 has a NaN
    sp[G * 2: G * 2 + G // 2] = np.nan           # group 2 half NaN
    L = leap()
    gpu = L.leap_group_rank_advantages(to_dev(pt, torch.int8), to_dev(nt, torch.int8), G=G, M=M, tau_max=G,
                                       gamma=0.8, cmp=L.LEAP_CMP_LEXI, speedup=to_dev(sp, torch.float32),
                                       ntokens=to_dev(tok, torch.int32))
    orc = O.rank_advantages(pt.reshape(-1, G), nt.reshape(-1, G), M, 0, G, 0.8, cmp=O.CMP_LEXI,
                            speedup=sp.reshape(-1, G), ntokens=tok.reshape(-1, G))
    _compare(gpu, orc, M)


@pytest.mark.parametrize("M", [1, 3, 8])
def test_quad_pair_and_generic_kernels_agree_at_64(M):
    """G = 64 runs the quad kernel (two groups per warp, 16-byte stores) when
    the buffers allow it; outputs offset by 8 bytes send the call to the pair
    kernel, by 4 bytes to the generic one.  An odd group count leaves the last
    warp with one group.  All three equal the oracle and each other, bit for bit."""
    G = 64
    rng = np.random.default_rng(11 * M)
    groups = 37
    n = groups * G
    nt = rng.integers(1, M + 1, size=n).astype(np.int8)
    pt = np.minimum(np.where(rng.random(n) < 0.5, rng.integers(1, M + 1, size=n), 0), nt).astype(np.int8)
    pt[70] = M + 1                                  # one malformed outcome
    L = leap()
    dev = torch.device("cuda")
    pt_d, nt_d = torch.as_tensor(pt, device=dev), torch.as_tensor(nt, device=dev)
    tau = (16, 48)
    L.leap_get_device_status()
    quad = L.leap_group_rank_advantages(pt_d, nt_d, G=G, M=M, tau_min=tau[0], tau_max=tau[1], gamma=0.8)
    results = [quad]
    for shift4, shift1 in ((2, 2), (1, 1)):         # 8-byte / 2-byte offsets (pair); 4-byte / 1-byte (generic)
        off = lambda k, dt, sh: torch.empty(k + sh, dtype=dt, device=dev)[sh:]
        out = dict(gate=off(groups, torch.uint8, shift1), r=off(n, torch.uint8, shift1),
                   n_worse=off(n, torch.int32, shift4), n_better=off(n, torch.int32, shift4),
                   R=off(n, torch.float32, shift4), A=off(n, torch.float32, shift4),
                   turn_adv=off(n * M, torch.float32, shift4), T_eff=off(n, torch.uint8, shift1))
        results.append(L.leap_group_rank_advantages(pt_d, nt_d, G=G, M=M, tau_min=tau[0], tau_max=tau[1],
                                                    gamma=0.8, out=out))
    torch.cuda.synchronize()
    assert L.leap_get_device_status() & L.LEAP_DEV_BAD_OUTCOME
    for other in results[1:]:
        for k in quad:
            assert torch.equal(quad[k], other[k]), k
    orc = O.rank_advantages(pt.reshape(-1, G), nt.reshape(-1, G), M, tau[0], tau[1], 0.8)
    _compare(quad, orc, M)


@pytest.mark.parametrize("reward", [0, 1])
@pytest.mark.parametrize("M", [1, 3, 8])
def test_quad_pair_and_generic_counters_and_rewards_at_64(M, reward):
    """The quad kernel also serves the training counters (two groups' counts
    in one warp reduction) and the static-scalar reward (half-warp sums): on
    an odd group count, with one malformed outcome and a computed gate, the
    counters of the quad, pair and generic kernels all equal the oracle's, the
    integer outputs agree bit for bit, and the advantages match the oracle."""
    G = 64
    rng = np.random.default_rng(13 * M + reward)
    groups = 37
    n = groups * G
    nt = rng.integers(1, M + 1, size=n).astype(np.int8)
    pt = np.minimum(np.where(rng.random(n) < 0.5, rng.integers(1, M + 1, size=n), 0), nt).astype(np.int8)
    pt[70] = M + 1
    L = leap()
    dev = torch.device("cuda")
    pt_d, nt_d = torch.as_tensor(pt, device=dev), torch.as_tensor(nt, device=dev)
    tau = (16, 48)
    L.leap_get_device_status()                      # clears the sticky flags
    orc = O.rank_advantages(pt.reshape(-1, G), nt.reshape(-1, G), M, tau[0], tau[1], 0.8, reward=reward,
                            static_c=0.5)
    exp = O.rank_stats(orc, pt.reshape(-1, G), M)
    results = []
    for shift4, shift1 in ((0, 0), (2, 2), (1, 1)):   # quad; pair (8 / 2-byte offsets); generic (4 / 1-byte)
        off = lambda k, dt, sh: torch.empty(k + sh, dtype=dt, device=dev)[sh:]
        out = dict(gate=off(groups, torch.uint8, shift1), r=off(n, torch.uint8, shift1),
                   n_worse=off(n, torch.int32, shift4), n_better=off(n, torch.int32, shift4),
                   R=off(n, torch.float32, shift4), A=off(n, torch.float32, shift4),
                   turn_adv=off(n * M, torch.float32, shift4), T_eff=off(n, torch.uint8, shift1))
        st = L.rank_stats_tensor("cuda")
        res = L.leap_group_rank_advantages(pt_d, nt_d, G=G, M=M, tau_min=tau[0], tau_max=tau[1], gamma=0.8,
                                           out=out, stats=st, reward=reward, static_c=0.5)
        assert L.read_rank_stats(st) == exp
        results.append(res)
    torch.cuda.synchronize()
    assert L.leap_get_device_status() == L.LEAP_DEV_BAD_OUTCOME   # read (and cleared) here
    for other in results[1:]:
        for k in ("gate", "r", "T_eff", "n_worse", "n_better"):
            assert torch.equal(results[0][k], other[k]), k
    for res in results:
        if reward == 0:
            _compare(res, orc, M)
        else:
            np.testing.assert_allclose(res["R"].cpu().numpy(), orc["R"].reshape(-1), rtol=0, atol=1e-7)
            assert np.max(np.abs(res["A"].cpu().numpy() - orc["A"].reshape(-1))) <= TOL_ADV
            ta = res["turn_adv"].cpu().numpy().reshape(-1, M)
            assert np.max(np.abs(ta - orc["turn_adv"].reshape(-1, M))) <= TOL_ADV


@pytest.mark.parametrize("G,M,nan", [(64, 3, False), (16, 2, False), (64, 3, True), (2, 1, False)])
def test_lexi_pair_and_generic_kernels_agree(G, M, nan):
    """The tie-broken comparator on the pair layout (even G <= 64, 8-byte
    aligned speedups and token counts) and on the generic kernel (a 4-byte
    offset on the outputs) give the same bits and equal the oracle, with
    exact ties, -0 against +0, and (nan) groups holding a NaN speedup."""
    rng = np.random.default_rng(17 * G + M + nan)
    groups = 4096 // G + 3
    n = groups * G
    nt = rng.integers(1, M + 1, size=n).astype(np.int8)
    pt = np.minimum(np.where(rng.random(n) < 0.6, rng.integers(1, M + 1, size=n), 0), nt).astype(np.int8)
    sp = rng.choice(np.array([0.0, -0.0, 0.5, 1.0, 2.0, np.inf], dtype=np.float32), size=n)
    tok = rng.choice(np.array([128, 256, 512], dtype=np.int32), size=n)
    if nan:
        sp[G * 2 + 1] = np.nan
        sp[G * 5: G * 5 + G // 2] = np.nan
    L = leap()
    dev = torch.device("cuda")
    args = dict(G=G, M=M, tau_min=0, tau_max=G, gamma=0.8, cmp=L.LEAP_CMP_LEXI, speedup=to_dev(sp, torch.float32),
                ntokens=to_dev(tok, torch.int32))
    pt_d, nt_d = to_dev(pt, torch.int8), to_dev(nt, torch.int8)
    pair = L.leap_group_rank_advantages(pt_d, nt_d, **args)
    off = lambda k, dt: torch.empty(k + 1, dtype=dt, device=dev)[1:]
    out = dict(gate=off(groups, torch.uint8), r=off(n, torch.uint8), n_worse=off(n, torch.int32),
               n_better=off(n, torch.int32), R=off(n, torch.float32), A=off(n, torch.float32),
               turn_adv=off(n * M, torch.float32), T_eff=off(n, torch.uint8))
    generic = L.leap_group_rank_advantages(pt_d, nt_d, out=out, **args)
    torch.cuda.synchronize()
    for k in pair:
        assert torch.equal(pair[k], generic[k]), k
    orc = O.rank_advantages(pt.reshape(-1, G), nt.reshape(-1, G), M, 0, G, 0.8, cmp=O.CMP_LEXI,
                            speedup=sp.reshape(-1, G), ntokens=tok.reshape(-1, G))
    _compare(pair, orc, M)
