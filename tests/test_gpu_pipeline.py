"""End-to-end parity of the whole hot path (rank advantages -> token counts ->
scatter -> fused loss fwd+bwd) on the benchmark workloads, each side running
its own pipeline from the same raw outcomes, layout and logits."""
import numpy as np
import pytest
import torch

from harness import (O, TOL_ADV, TOL_LOGP, TOL_LOSS_REL, bf16_rows_to_f64, check_dlogits_rows, leap,
                     oracle_rank, oracle_tokens, rows_f64, to_dev, torch_logp)
from paper_2608_01804_gb300 import synth

pytestmark = pytest.mark.gpu


def _gpu_pipeline(L, b, z, ids, old, V, gamma, tau, use_gate_in, agg=0, grad_scale=1.0):
    dev = "cuda"
    pt, nt = to_dev(b.pass_turn, torch.int8), to_dev(b.num_turns, torch.int8)
    gi = to_dev(b.gate_in, torch.uint8) if (use_gate_in and b.gate_in is not None) else None
    rk = L.leap_group_rank_advantages(pt, nt, G=b.G, M=b.M, tau_min=tau[0], tau_max=tau[1], gamma=gamma,
                                      gate_in=gi)
    so, sr, st = to_dev(b.seg_offsets, torch.int32), to_dev(b.seg_rollout, torch.int32), to_dev(b.seg_turn, torch.int8)
    Lc, tot = L.leap_rollout_token_counts(b.N, so, sr, st, rk["T_eff"], M=b.M)
    adv, w = L.leap_scatter_turn_advantages(b.N, so, sr, st, rk["turn_adv"], rk["T_eff"], Lc, tot, M=b.M, agg=agg)
    out = L.leap_grpo_loss_fwd(z, ids, old, adv, w, V=V, grad_scale=grad_scale)
    return rk, adv, w, out


def _oracle_pipeline(b, gamma, tau, use_gate_in, agg=0):
    orc = oracle_rank(b, tau=tau, gamma=gamma, use_gate_in=use_gate_in)
    ta = orc["turn_adv"].reshape(-1)
    T_eff = orc["T_eff"].reshape(-1)
    _, _, _, adv, w = oracle_tokens(b, ta, T_eff, agg)
    return orc, adv, w


@pytest.mark.parametrize("use_gate_in,tau", [(True, (0, 8)), (False, (4, 7))])
def test_tiny_workload_all_rows(use_gate_in, tau):
    """4 prompts x 8 x 2 turns x 256, V = 1024: every row and every output."""
    L = leap()
    b = synth.tiny_batch()
    V = 1024
    z = synth.logits(b.N, V, 2.0, 100, "cuda")
    ids = synth.token_ids(b.N, V, 101, "cuda")
    old = torch_logp(z, ids, V) + synth.normal(b.N, 0.05, 102, "cuda")
    rk, adv, w, out = _gpu_pipeline(L, b, z, ids, old, V, 0.9, tau, use_gate_in, grad_scale=100.0)
    orc, adv_o, w_o = _oracle_pipeline(b, 0.9, tau, use_gate_in)
    np.testing.assert_array_equal(rk["n_worse"].cpu().numpy(), orc["n_worse"].reshape(-1))
    assert np.max(np.abs(adv.cpu().numpy() - adv_o)) <= TOL_ADV
    np.testing.assert_allclose(w.cpu().numpy(), w_o, rtol=2e-7)
    res = O.grpo_loss_rows(rows_f64(z, range(b.N), V), ids.cpu().numpy(), old.cpu().numpy().astype(np.float64),
                           adv_o, w_o, grad_scale=100.0)
    assert np.max(np.abs(out["logp"].cpu().numpy() - res["logp"])) <= TOL_LOGP
    assert abs(out["loss"].item() - res["loss"]) <= TOL_LOSS_REL * abs(res["loss"])
    check_dlogits_rows(bf16_rows_to_f64(out["dlogits"]), res, list(range(b.N)))


def test_single_turn_workload_full_size_sampled():
    """16 x 8 x 256 = 32,768 rows at V = 151,936 in the benchmark's launch
    configuration; sampled rows against the oracle, the loss against the fp64
    sum of the kernel's own per-row terms and against the oracle's terms on the
    sampled rows."""
    L = leap()
    b = synth.single_turn_batch()
    V = 151936
    z = synth.logits(b.N, V, 3.0, 200, "cuda", spike_frac=0.01)
    ids = synth.token_ids(b.N, V, 201, "cuda")
    old = torch_logp(z, ids, V) + synth.normal(b.N, 0.05, 202, "cuda")
    rk, adv, w, out = _gpu_pipeline(L, b, z, ids, old, V, 1.0, (0, b.G), False)
    orc, adv_o, w_o = _oracle_pipeline(b, 1.0, (0, b.G), False)
    assert np.max(np.abs(adv.cpu().numpy() - adv_o)) <= TOL_ADV
    rng = np.random.default_rng(0)
    rows = sorted(set([0, 1, b.N - 1, b.N - 2] + list(rng.choice(b.N, 96, replace=False))))
    sel = torch.as_tensor(rows, device="cuda")
    res = O.grpo_loss_rows(rows_f64(z, rows, V), ids[sel].cpu().numpy(), old[sel].cpu().numpy().astype(np.float64),
                           adv_o[rows], w_o[rows])
    logp = out["logp"][sel].cpu().numpy()
    assert np.max(np.abs(logp - res["logp"])) <= TOL_LOGP
    ell = out["ell"][sel].cpu().numpy().astype(np.float64)
    np.testing.assert_allclose(ell, res["ell"], rtol=1e-4, atol=1e-6)
    check_dlogits_rows(bf16_rows_to_f64(out["dlogits"][sel]), res, rows)
    # Reduction: the loss is the fp64 sum of w * ell over all rows.
    tot = float((w.double() * out["ell"].double()).sum().item())
    assert abs(out["loss"].item() - tot) <= 1e-6 * abs(tot) + 1e-12
    # Masked padding rows: zero dlogits.
    masked = (w == 0).nonzero().view(-1)[:64]
    assert torch.all(out["dlogits"][masked] == 0)


def test_single_turn_whole_batch_loss_against_oracle():
    """The benchmark's whole-batch loss (32,768 rows at V = 151,936, 21,662 of
    them valid) against the oracle's fp64 loss over every valid row, computed
    on the host 512 rows at a time (3.3 G fp64 log-softmax terms)."""
    L = leap()
    b = synth.single_turn_batch()
    V = 151936
    z = synth.logits(b.N, V, 3.0, 200, "cuda", spike_frac=0.01)
    ids = synth.token_ids(b.N, V, 201, "cuda")
    old = torch_logp(z, ids, V) + synth.normal(b.N, 0.05, 202, "cuda")
    _, _, _, out = _gpu_pipeline(L, b, z, ids, old, V, 1.0, (0, b.G), False)
    loss = out["loss"].item()
    del out
    _, adv_o, w_o = _oracle_pipeline(b, 1.0, (0, b.G), False)
    live = np.nonzero(w_o)[0]
    assert len(live) == 21662
    ids_h = ids.cpu().numpy().astype(np.int64)
    old_h = old.cpu().numpy().astype(np.float64)
    total = 0.0
    for a in range(0, len(live), 512):
        rows = live[a:a + 512]
        res = O.grpo_loss_rows(rows_f64(z, rows, V), ids_h[rows], old_h[rows], adv_o[rows], w_o[rows],
                               want_dlogits=False)
        total += res["loss"]
    assert abs(loss - total) <= TOL_LOSS_REL * abs(total), (loss, total)


def test_multiturn_dcp_workload_chunked():
    """The packed multi-turn batch (~1M tokens) streamed through one 65,536-row
    logits chunk buffer with loss accumulation; three chunks are checked against
    the oracle on sampled rows, the advantages and weights on every token."""
    L = leap()
    b = synth.multiturn_dcp_batch()
    V, CH = 151936, 65536
    pt, nt = to_dev(b.pass_turn, torch.int8), to_dev(b.num_turns, torch.int8)
    rk = L.leap_group_rank_advantages(pt, nt, G=b.G, M=b.M, tau_min=8, tau_max=15, gamma=0.9)
    np.testing.assert_array_equal(rk["gate"].cpu().numpy(), b.gate_in)   # the drawn zone matches Eq. 2
    so, sr, st = to_dev(b.seg_offsets, torch.int32), to_dev(b.seg_rollout, torch.int32), to_dev(b.seg_turn, torch.int8)
    Lc, tot = L.leap_rollout_token_counts(b.N, so, sr, st, rk["T_eff"], M=b.M)
    adv, w = L.leap_scatter_turn_advantages(b.N, so, sr, st, rk["turn_adv"], rk["T_eff"], Lc, tot, M=b.M)
    orc, adv_o, w_o = _oracle_pipeline(b, 0.9, (8, 15), False)
    assert np.max(np.abs(adv.cpu().numpy() - adv_o)) <= TOL_ADV
    np.testing.assert_allclose(w.cpu().numpy(), w_o, rtol=2e-7)
    z = synth.logits(CH, V, 3.0, 300, "cuda", spike_frac=0.01)
    ids_all = synth.token_ids(b.N, V, 301, "cuda")
    loss = torch.zeros(1, device="cuda")
    dl = torch.empty_like(z)
    ws = L.loss_workspace(CH, V, "cuda")
    nchunks = -(-b.N // CH)
    total_o = 0.0
    for c in range(nchunks):
        a0, a1 = c * CH, min(b.N, (c + 1) * CH)
        n = a1 - a0
        ids = ids_all[a0:a1].contiguous()
        old = torch_logp(z[:n], ids, V) + synth.normal(n, 0.05, 400 + c, "cuda")
        out = L.leap_grpo_loss_fwd(z[:n], ids, old, adv[a0:a1].contiguous(), w[a0:a1].contiguous(), V=V, loss=loss,
                                   accumulate=True, dlogits=dl[:n], workspace=ws)
        if c in (0, nchunks // 2, nchunks - 1):
            rng = np.random.default_rng(c)
            live = np.nonzero(w_o[a0:a1])[0]
            rows = sorted(set(rng.choice(live, min(24, len(live)), replace=False).tolist() + [0, n - 1]))
            sel = torch.as_tensor(rows, device="cuda")
            res = O.grpo_loss_rows(rows_f64(z, rows, V), ids[sel].cpu().numpy(),
                                   old[sel].cpu().numpy().astype(np.float64), adv_o[a0:a1][rows], w_o[a0:a1][rows])
            assert np.max(np.abs(out["logp"][sel].cpu().numpy() - res["logp"])) <= TOL_LOGP
            check_dlogits_rows(bf16_rows_to_f64(dl[sel]), res, rows)
        total_o += float((out["ell"].double() * w[a0:a1].double()).sum().item())
    assert abs(loss.item() - total_o) <= 1e-5 * abs(total_o) + 1e-9


def test_streamed_step_equals_resident_step():
    """GrpoStep.run_streamed (logits in pinned host memory, copied chunk by
    chunk on a second stream while the loss runs) gives the same dlogits, bit
    for bit, as GrpoStep.run on resident logits, and exactly the fp32 sum of
    the per-chunk losses (each the fixed-order fp64 sum rounded to fp32);
    ragged last chunk."""
    from paper_2608_01804_gb300.step import GrpoStep
    b = synth.single_turn_batch(num_prompts=2)
    V = 151936
    z = synth.logits(b.N, V, 3.0, 210, "cuda", spike_frac=0.01)
    ids = synth.token_ids(b.N, V, 211, "cuda")
    old = torch_logp(z, ids, V) + synth.normal(b.N, 0.05, 212, "cuda")
    step = GrpoStep(b, V, "cuda", gamma=1.0, tau=(0, b.G), use_gate_in=False)
    dl_res = torch.empty_like(z)
    loss_res = step.run(z, ids, old, dl_res).clone()
    host = z.cpu().pin_memory()
    dl_str = torch.full_like(z, 7)
    loss_str = step.run_streamed(host, ids, old, dl_str, chunk_rows=1500).clone()
    torch.cuda.synchronize()
    assert torch.equal(dl_str, dl_res)
    L = leap()
    expect = torch.zeros(1, device="cuda")
    scratch = torch.empty_like(z)
    for a in range(0, b.N, 1500):
        e = min(b.N, a + 1500)
        part = L.leap_grpo_loss_fwd(z[a:e], ids[a:e], old[a:e], step.adv[a:e], step.w[a:e], V=V,
                                    dlogits=scratch[a:e], want_outputs=False)["loss"]
        expect = expect + part
    assert loss_str.item() == expect.item()
    # The whole-batch loss differs from the chunked one only by the fp32 sum over chunks.
    assert abs(loss_str.item() - loss_res.item()) <= 4 * 2.0 ** -24 * float(step.w.abs().sum().item()) * 2.0
    # A step built for smaller chunks grows its workspace for the streamed chunk size.
    small = GrpoStep(b, V, "cuda", gamma=1.0, tau=(0, b.G), use_gate_in=False, chunk_rows=256)
    dl_small = torch.full_like(z, 7)
    loss_small = small.run_streamed(host, ids, old, dl_small, chunk_rows=1500).clone()
    torch.cuda.synchronize()
    assert loss_small.item() == loss_str.item()
    assert torch.equal(dl_small, dl_res)
    # Only rows that can carry weight crossed the link (the padding did not).
    live = sum(hi - lo for lo, hi in step.weighted_row_runs())
    assert step.h2d_logit_bytes == live * V * 2 < b.N * V * 2
    assert live == int((step.w != 0).sum().item())
    # Copying every row gives the same results.
    dl_all = torch.full_like(z, 7)
    loss_all = step.run_streamed(host, ids, old, dl_all, chunk_rows=1500, weighted_only=False).clone()
    torch.cuda.synchronize()
    assert step.h2d_logit_bytes == b.N * V * 2
    assert loss_all.item() == loss_str.item() and torch.equal(dl_all, dl_res)


def test_streamed_step_packed_multiturn_stream():
    """The streamed step on a packed multi-turn stream (masked prompts and
    environment feedback between generated turns, DCP-pruned groups): only
    the generated turns' rows are copied, and dlogits equal the resident
    step's bit for bit."""
    from paper_2608_01804_gb300.step import GrpoStep
    b = synth.multiturn_dcp_batch(seed=5, num_prompts=4, G=4, M=3, len_lo=64, len_hi=256, prompt_lo=64,
                                  prompt_hi=256, tau=(1, 3))
    V = 9000
    z = synth.logits(b.N, V, 3.0, 220, "cuda", spike_frac=0.01)
    ids = synth.token_ids(b.N, V, 221, "cuda")
    old = torch_logp(z, ids, V) + synth.normal(b.N, 0.05, 222, "cuda")
    step = GrpoStep(b, V, "cuda", gamma=0.9, tau=(1, 3))
    dl_res = torch.empty_like(z)
    loss_res = step.run(z, ids, old, dl_res).clone()
    host = z.cpu().pin_memory()
    dl_str = torch.full_like(z, 7)
    step.run_streamed(host, ids, old, dl_str, chunk_rows=700)
    torch.cuda.synchronize()
    assert torch.equal(dl_str, dl_res)
    runs = step.weighted_row_runs()
    live = sum(hi - lo for lo, hi in runs)
    assert step.h2d_logit_bytes == live * V * 2 < b.N * V * 2
    wmask = (step.w != 0).cpu().numpy()
    inside = np.zeros(b.N, dtype=bool)
    for lo, hi in runs:
        inside[lo:hi] = True
    assert not (wmask & ~inside).any()            # every weighted row was copied
    assert loss_res.item() != 0.0


def test_graph_replay_equals_eager_step():
    """GrpoStep.capture: one CUDA-graph replay of the whole pass gives the
    eager run's loss, dlogits, advantages and weights bit for bit, and a
    replay after the inputs are refilled in place matches an eager run on the
    new inputs (the graph reads the buffers, it does not freeze them)."""
    from paper_2608_01804_gb300.step import GrpoStep
    L = leap()
    b = synth.tiny_batch()
    V = 1024
    z = synth.logits(b.N, V, 2.0, 220, "cuda")
    ids = synth.token_ids(b.N, V, 221, "cuda")
    old = torch_logp(z, ids, V) + synth.normal(b.N, 0.05, 222, "cuda")
    eager = GrpoStep(b, V, "cuda", gamma=0.9, tau=(0, 8))
    dl_e = torch.empty_like(z)
    loss_e = eager.run(z, ids, old, dl_e).clone()
    graphed = GrpoStep(b, V, "cuda", gamma=0.9, tau=(0, 8))
    dl_g = torch.full_like(z, 7)
    g = graphed.capture(z, ids, old, dl_g)
    dl_g.fill_(7)
    graphed.loss.fill_(123.0)
    g.replay()
    torch.cuda.synchronize()
    assert L.leap_get_device_status() == 0
    assert graphed.loss.item() == loss_e.item()
    assert torch.equal(dl_g, dl_e)
    assert torch.equal(graphed.adv, eager.adv) and torch.equal(graphed.w, eager.w)
    # New logits and old log-probs in the same buffers.
    z2 = synth.logits(b.N, V, 2.0, 223, "cuda")
    z.copy_(z2)
    old.copy_(torch_logp(z2, ids, V) + synth.normal(b.N, 0.05, 224, "cuda"))
    g.replay()
    loss_e2 = eager.run(z, ids, old, dl_e).clone()
    torch.cuda.synchronize()
    assert graphed.loss.item() == loss_e2.item() and graphed.loss.item() != loss_e.item()
    assert torch.equal(dl_g, dl_e)
