"""Edge cases of the loss and rank kernels: canary guard bands around every
output (nothing is written outside the rows and columns a call owns), NaN
propagation, and empty / degenerate inputs."""
import numpy as np
import pytest
import torch

from harness import leap, torch_logp, to_dev
from paper_2608_01804_gb300 import synth

pytestmark = pytest.mark.gpu

SENT = 1232.0   # exact in bf16 and fp32


def _vec(n, pad=64):
    """A length-n view into a sentinel-filled buffer with `pad` guard elements each side."""
    buf = torch.full((n + 2 * pad,), SENT, dtype=torch.float32, device="cuda")
    return buf, buf[pad:pad + n]


@pytest.mark.parametrize("single_read", [False, True])
@pytest.mark.parametrize("V,ld", [(1024, 1032), (151936, 151944)])
def test_loss_outputs_have_intact_guard_bands(V, ld, single_read):
    L = leap()
    N = 40
    z = synth.logits(N, V, 3.0, 71, "cuda", spike_frac=0.01, ld=ld)
    ids = synth.token_ids(N, V, 72, "cuda")
    old = torch_logp(z, ids, V) + synth.normal(N, 0.3, 73, "cuda")
    adv = synth.normal(N, 1.0, 74, "cuda")
    w = torch.rand(N, device="cuda") * 0.1
    w[::5] = 0.0
    bufs = {k: _vec(N) for k in ("logp", "lse", "ell")}
    lossbuf, loss = _vec(1)
    dl_buf = torch.full((N + 4, ld), SENT, dtype=torch.bfloat16, device="cuda")
    dl = dl_buf[2:2 + N]
    L.leap_grpo_loss_fwd(z, ids, old, adv, w, V=V, loss=loss, logp=bufs["logp"][1], lse=bufs["lse"][1],
                         ell=bufs["ell"][1], dlogits=dl, single_read=single_read)
    torch.cuda.synchronize()
    for k, (buf, view) in bufs.items():
        assert torch.all(buf[:64] == SENT) and torch.all(buf[64 + N:] == SENT), k
        assert torch.all(torch.isfinite(view)), k
    assert torch.all(lossbuf[:64] == SENT) and torch.all(lossbuf[65:] == SENT)
    assert torch.all(dl_buf[:2] == SENT) and torch.all(dl_buf[2 + N:] == SENT)
    assert torch.all(dl[:, V:] == SENT)                    # padding columns untouched
    assert torch.all(torch.isfinite(dl[:, :V].float()))
    # split backward and log-probs respect the same bands
    dl_buf.fill_(SENT)
    L.leap_grpo_loss_bwd(z, ids, old, adv, w, bufs["lse"][1], V=V, dlogits=dl)
    torch.cuda.synchronize()
    assert torch.all(dl_buf[:2] == SENT) and torch.all(dl_buf[2 + N:] == SENT) and torch.all(dl[:, V:] == SENT)
    lp_buf, lp = _vec(N)
    L.leap_token_logprobs(z, ids, V=V, logp=lp, want_lse=False)
    torch.cuda.synchronize()
    assert torch.all(lp_buf[:64] == SENT) and torch.all(lp_buf[64 + N:] == SENT)


def test_rank_and_scatter_outputs_have_intact_guard_bands():
    L = leap()
    b = synth.tiny_batch()
    n, M = b.n, b.M
    pad = 64
    out = {}
    views = {}
    for k, (size, dt) in dict(gate=(b.num_groups, torch.uint8), r=(n, torch.uint8), n_worse=(n, torch.int32),
                              n_better=(n, torch.int32), R=(n, torch.float32), A=(n, torch.float32),
                              turn_adv=(n * M, torch.float32), T_eff=(n, torch.uint8)).items():
        buf = torch.full((size + 2 * pad,), 77, dtype=dt, device="cuda")
        out[k] = buf
        views[k] = buf[pad:pad + size]
    L.leap_group_rank_advantages(to_dev(b.pass_turn, torch.int8), to_dev(b.num_turns, torch.int8), G=b.G, M=M,
                                 tau_max=b.G, gamma=0.9, gate_in=to_dev(b.gate_in, torch.uint8), out=views)
    torch.cuda.synchronize()
    for k, buf in out.items():
        assert torch.all(buf[:pad] == 77) and torch.all(buf[-pad:] == 77), k
    so, sr, st = to_dev(b.seg_offsets, torch.int32), to_dev(b.seg_rollout, torch.int32), to_dev(b.seg_turn, torch.int8)
    Lb = torch.full((n + 2 * pad,), 55, dtype=torch.int32, device="cuda")
    Lc = Lb[pad:pad + n]
    Lc, tot = L.leap_rollout_token_counts(b.N, so, sr, st, views["T_eff"], M=M, L=Lc)
    ab, adv = _vec(b.N)
    wb, w = _vec(b.N)
    L.leap_scatter_turn_advantages(b.N, so, sr, st, views["turn_adv"], views["T_eff"], Lc, tot, M=M, adv=adv, w=w)
    torch.cuda.synchronize()
    assert torch.all(Lb[:pad] == 55) and torch.all(Lb[-pad:] == 55)
    for buf in (ab, wb):
        assert torch.all(buf[:64] == SENT) and torch.all(buf[-64:] == SENT)


@pytest.mark.parametrize("single_read", [False, True])
def test_nan_logit_propagates_to_its_row_and_the_loss_only(single_read):
    L = leap()
    N, V = 16, 151936
    z = synth.logits(N, V, 3.0, 81, "cuda")
    ids = synth.token_ids(N, V, 82, "cuda")
    old = torch_logp(z, ids, V)
    adv = synth.normal(N, 1.0, 83, "cuda")
    w = torch.full((N,), 0.05, device="cuda")
    z[3, 1000] = float("nan")
    out = L.leap_grpo_loss_fwd(z, ids, old, adv, w, V=V, single_read=single_read)
    torch.cuda.synchronize()
    logp = out["logp"].cpu()
    assert torch.isnan(logp[3]) and torch.isnan(out["lse"][3].cpu())
    others = torch.cat([logp[:3], logp[4:]])
    assert torch.all(torch.isfinite(others))
    assert torch.isnan(out["loss"]).item() and torch.isnan(out["ell"][3]).item()
    assert torch.all(torch.isnan(out["dlogits"][3].float()))
    assert torch.all(torch.isfinite(out["dlogits"][[0, 1, 2, 4]].float()))


def test_degenerate_group_sizes_rejected_on_host():
    L = leap()
    pt = torch.zeros(1025, dtype=torch.int8, device="cuda")
    with pytest.raises(L.LeapError) as e:
        L.leap_group_rank_advantages(pt, pt, G=1025, M=2, tau_max=1025)
    assert e.value.status == L.LEAP_ERR_INVALID_ARG
    pt2 = torch.zeros(4, dtype=torch.int8, device="cuda")
    with pytest.raises(L.LeapError):
        L.leap_group_rank_advantages(pt2, pt2, G=4, M=0, tau_max=4)
    with pytest.raises(L.LeapError):
        L.leap_group_rank_advantages(pt2, pt2, G=4, M=2, tau_min=3, tau_max=2)
