"""GPU parity: token log-probs, the clipped surrogate (fused fwd+bwd, forward
only, split backward) and its deterministic reduction, against the oracle on
identical inputs."""
import numpy as np
import pytest
import torch

from harness import (O, TOL_LOGP, TOL_LOSS_REL, bf16_rows_to_f64, check_dlogits_rows, leap, rows_f64,
                     torch_logp)
from paper_2608_01804_gb300 import synth

pytestmark = pytest.mark.gpu


def _inputs(N, V, seed, sigma=2.0, spikes=0.0, old_sigma=0.05, ld=None, mask_frac=0.25, adv_scale=1.0):
    dev = "cuda"
    z = synth.logits(N, V, sigma, seed, dev, spike_frac=spikes, ld=ld)
    ids = synth.token_ids(N, V, seed + 1, dev)
    old = torch_logp(z, ids, V) + synth.normal(N, old_sigma, seed + 2, dev)
    rng = np.random.default_rng(seed + 3)
    adv = torch.as_tensor(rng.normal(0, adv_scale, N).astype(np.float32), device=dev)
    w = rng.uniform(0.01, 0.1, N).astype(np.float32)
    w[rng.random(N) < mask_frac] = 0.0
    return z, ids, old, adv, torch.as_tensor(w, device=dev)


def _oracle_rows(z, ids, old, adv, w, rows, V, **kw):
    zz = rows_f64(z, rows, V)
    sel = torch.as_tensor(np.asarray(rows), device=z.device, dtype=torch.long)
    f = lambda t: t.index_select(0, sel).cpu().numpy().astype(np.float64)
    return O.grpo_loss_rows(zz, f(ids).astype(np.int64), f(old), f(adv), f(w), **kw)


def _check_rows(out, orc, rows, V, dl=None):
    live = orc["live"]
    sel = torch.as_tensor(np.asarray(rows), device="cuda", dtype=torch.long)
    logp = out["logp"].index_select(0, sel).cpu().numpy().astype(np.float64)
    assert np.max(np.abs(logp - orc["logp"])) <= TOL_LOGP
    assert np.all(logp[~live] == 0)
    lse = out["lse"].index_select(0, sel).cpu().numpy().astype(np.float64)
    np.testing.assert_allclose(lse[live], orc["lse"][live], rtol=1e-5)
    if dl is not None:
        check_dlogits_rows(bf16_rows_to_f64(dl.index_select(0, sel)[:, :V]), orc, rows)


@pytest.mark.parametrize("single_read", [False, True])
@pytest.mark.parametrize("V,ld", [(1024, 1024), (1000, 1008), (1027, 1032), (5000, 5000), (8192, 8192),
                                  (30001, 30008), (60000, 60000), (100000, 100000), (151936, 151936), (151936, 152000),
                                  (200000, 200000)])
def test_fused_loss_all_rows(V, ld, single_read):
    """Every fused kernel (the short-row kernel up to V = 32,768, the
    row-pipelined one above it, and with single_read every cluster
    configuration above it, 4 and 8 CTAs), ragged V and padded ld."""
    L = leap()
    L.leap_get_device_status()
    N = 64 if V > 50000 else 256
    z, ids, old, adv, w = _inputs(N, V, seed=V % 97, sigma=3.0, spikes=0.01, ld=ld, old_sigma=0.3)
    ids[:4] = torch.tensor([0, V - 1, min(7, V - 1), min(8, V - 1)], dtype=torch.int32, device="cuda")
    w[:4] = 0.1
    if ld > V:
        sentinel = torch.full((N, ld - V), 3.0, dtype=torch.bfloat16, device="cuda")
    out = L.leap_grpo_loss_fwd(z, ids, old, adv, w, V=V, dlogits=torch.full_like(z, 3.0) if ld > V else None,
                               single_read=single_read)
    if ld > V:
        assert torch.equal(out["dlogits"][:, V:], sentinel)   # columns >= V untouched
    assert L.leap_get_device_status() == 0              # no bounded wait gave up
    rows = list(range(N))
    orc = _oracle_rows(z, ids, old, adv, w, rows, V)
    _check_rows(out, orc, rows, V, dl=out["dlogits"])
    assert abs(out["loss"].item() - orc["loss"]) <= TOL_LOSS_REL * abs(orc["loss"])
    assert (~orc["active"] & orc["live"]).any()        # the clipped branch was exercised


@pytest.mark.parametrize("single_read", [False, True])
def test_slice_boundaries_at_vocab_151936(single_read):
    """Targets placed on every CTA-slice and vector boundary of the cluster split."""
    L = leap()
    V = 151936
    per = -(-(-(-V // 8)) // 8) * 8      # elements per CTA slice for an 8-CTA cluster
    targets = sorted({0, 1, 7, 8, V - 8, V - 1} | {c * per + d for c in range(1, 8) for d in (-1, 0, 1)})
    N = len(targets)
    z, ids, old, adv, w = _inputs(N, V, seed=11, sigma=3.0, spikes=0.01, mask_frac=0.0)
    ids.copy_(torch.tensor(targets, dtype=torch.int32))
    old.copy_(torch_logp(z, ids, V) + synth.normal(N, 0.05, 12, "cuda"))
    out = L.leap_grpo_loss_fwd(z, ids, old, adv, w, V=V, single_read=single_read)
    orc = _oracle_rows(z, ids, old, adv, w, list(range(N)), V)
    _check_rows(out, orc, list(range(N)), V, dl=out["dlogits"])


@pytest.mark.parametrize("V", [1024, 151936])
def test_forward_only_and_split_backward_match_fused(V):
    L = leap()
    N = 128
    z, ids, old, adv, w = _inputs(N, V, seed=3, sigma=3.0, spikes=0.01, old_sigma=0.3)
    fused = L.leap_grpo_loss_fwd(z, ids, old, adv, w, V=V)
    fwd = L.leap_grpo_loss_fwd(z, ids, old, adv, w, V=V, want_dlogits=False)
    assert fwd["dlogits"] is None
    rows = list(range(N))
    orc = _oracle_rows(z, ids, old, adv, w, rows, V)
    _check_rows(fwd, orc, rows, V)
    assert abs(fwd["loss"].item() - orc["loss"]) <= TOL_LOSS_REL * abs(orc["loss"])
    assert abs(fused["loss"].item() - fwd["loss"].item()) <= TOL_LOSS_REL * abs(orc["loss"])
    dl = L.leap_grpo_loss_bwd(z, ids, old, adv, w, fwd["lse"], V=V)
    check_dlogits_rows(bf16_rows_to_f64(dl[:, :V]), orc, rows)


def test_large_vocab_default_path_and_single_read_limit():
    """The default fused kernel streams any V; the cluster kernel refuses V > 262,144."""
    L = leap()
    V, N = 300000, 24
    z, ids, old, adv, w = _inputs(N, V, seed=13, sigma=3.0, spikes=0.01, old_sigma=0.3)
    out = L.leap_grpo_loss_fwd(z, ids, old, adv, w, V=V)
    orc = _oracle_rows(z, ids, old, adv, w, list(range(N)), V)
    _check_rows(out, orc, list(range(N)), V, dl=out["dlogits"])
    assert abs(out["loss"].item() - orc["loss"]) <= TOL_LOSS_REL * abs(orc["loss"])
    with pytest.raises(L.LeapError) as e:
        L.leap_grpo_loss_fwd(z, ids, old, adv, w, V=V, single_read=True)
    assert e.value.status == L.LEAP_ERR_UNSUPPORTED


@pytest.mark.parametrize("V", [1024, 1000, 151936])
def test_token_logprobs(V):
    L = leap()
    N = 300 if V < 5000 else 40
    z, ids, *_ = _inputs(N, V, seed=21, sigma=3.0, spikes=0.01)
    logp, lse = L.leap_token_logprobs(z, ids, V=V)
    for inv_temp in (1.0, 0.7):
        logp, lse = L.leap_token_logprobs(z, ids, V=V, inv_temp=inv_temp)
        zz = rows_f64(z, range(N), V)
        lse_o, logp_o = O.log_softmax_rows(zz, ids.cpu().numpy(), inv_temp)
        assert np.max(np.abs(logp.cpu().numpy() - logp_o)) <= TOL_LOGP
        np.testing.assert_allclose(lse.cpu().numpy(), lse_o, rtol=1e-5)


def test_masked_rows_and_bad_ids():
    L = leap()
    L.leap_get_device_status()
    V, N = 151936, 16
    z, ids, old, adv, w = _inputs(N, V, seed=5, mask_frac=0.0)
    w[3] = 0.0
    ids[5] = V          # bad id with nonzero weight
    ids[6] = -3
    ids[3] = V + 10     # bad id on a masked row: not an error
    dl = torch.full_like(z, 1.0)
    out = L.leap_grpo_loss_fwd(z, ids, old, adv, w, V=V, dlogits=dl)
    flags = L.leap_get_device_status()
    assert flags == L.LEAP_DEV_BAD_ID
    for r in (3, 5, 6):
        assert torch.all(dl[r] == 0)
        assert out["logp"][r].item() == 0 and out["ell"][r].item() == 0
    rows = [0, 1, 2, 4, 7]
    orc = _oracle_rows(z, ids, old, adv, w, list(range(N)), V)
    assert abs(out["loss"].item() - orc["loss"]) <= TOL_LOSS_REL * abs(orc["loss"])
    _check_rows(out, _oracle_rows(z, ids, old, adv, w, rows, V), rows, V, dl=dl)


def test_accumulate_stats_and_determinism():
    L = leap()
    V, N = 1024, 4096
    z, ids, old, adv, w = _inputs(N, V, seed=8, sigma=2.0, old_sigma=0.3)
    st = L.stats_tensor("cuda")
    full = L.leap_grpo_loss_fwd(z, ids, old, adv, w, V=V, stats=st)
    s = L.read_stats(st)
    orc = O.grpo_loss_rows(rows_f64(z, range(N), V), ids.cpu().numpy(), old.cpu().numpy(), adv.cpu().numpy(),
                           w.cpu().numpy(), want_dlogits=False)
    assert s["live_tokens"] == int(orc["live"].sum())
    assert s["clipped_tokens"] == int((orc["live"] & ~orc["active"]).sum())
    assert abs(s["loss_sum"] - orc["loss"]) <= TOL_LOSS_REL * abs(orc["loss"])
    np.testing.assert_allclose(s["rho_sum"], orc["rho"][orc["live"]].sum(), rtol=1e-5)
    # Chunked with accumulation equals the whole (to fp32 rounding of the partials).
    loss = torch.zeros(1, device="cuda")
    for a in range(0, N, 1000):
        b = min(N, a + 1000)
        L.leap_grpo_loss_fwd(z[a:b], ids[a:b], old[a:b], adv[a:b], w[a:b], V=V, loss=loss, accumulate=True)
    assert abs(loss.item() - full["loss"].item()) <= 1e-5 * abs(full["loss"].item()) + 1e-9
    # Bitwise reproducible.
    again = L.leap_grpo_loss_fwd(z, ids, old, adv, w, V=V)
    assert again["loss"].item() == full["loss"].item()
    assert torch.equal(again["dlogits"], full["dlogits"])


def test_empty_batch():
    L = leap()
    z = torch.empty((0, 1024), dtype=torch.bfloat16, device="cuda")
    e = torch.empty(0, device="cuda")
    ids = torch.empty(0, dtype=torch.int32, device="cuda")
    loss = torch.full((1,), 5.0, device="cuda")
    L.leap_grpo_loss_fwd(z, ids, e, e, e, loss=loss)
    assert loss.item() == 0.0


@pytest.mark.parametrize("V,ld,N", [(8193, 8200, 700), (12000, 12000, 333), (16384, 16384, 700),
                                    (16385, 16392, 400), (24583, 24584, 333), (32000, 32000, 400),
                                    (32768, 32768, 400)])
def test_short_row_kernel_mid_vocab(V, ld, N):
    """The short-row kernel's mid-size shapes: eight warps of 4 KB slices
    (8,192 < V <= 16,384, two row groups per SM) and sixteen (16,384 < V <=
    32,768, one per SM).  Whole slices (16,384; 32,768), a single logit past
    the last whole slice (8,193; 16,385), ragged last vectors, padded ld, more
    rows than resident row groups, masked rows, and targets on the 2,048-logit
    slice boundaries; every row against the oracle."""
    L = leap()
    L.leap_get_device_status()
    z, ids, old, adv, w = _inputs(N, V, seed=V % 59 + 3, sigma=3.0, spikes=0.01, ld=ld, old_sigma=0.3)
    edges = [0, V - 1, 2047, 2048, 4095 % V, 4096 % V, 14335 % V, 14336 % V, 30719 % V, 30720 % V]
    ids[:len(edges)] = torch.tensor(edges, dtype=torch.int32, device="cuda")
    w[:len(edges)] = 0.1
    dl = torch.full_like(z, 3.0)
    out = L.leap_grpo_loss_fwd(z, ids, old, adv, w, V=V, dlogits=dl)
    assert L.leap_get_device_status() == 0
    if ld > V:
        assert torch.all(dl[:, V:] == 3.0)        # columns >= V untouched
    rows = list(range(N))
    orc = _oracle_rows(z, ids, old, adv, w, rows, V)
    _check_rows(out, orc, rows, V, dl=dl)
    assert abs(out["loss"].item() - orc["loss"]) <= TOL_LOSS_REL * abs(orc["loss"])
    assert (~orc["live"]).any() and (~orc["active"] & orc["live"]).any()


@pytest.mark.parametrize("V", [1000, 16384, 32000])
@pytest.mark.parametrize("N", [1, 5])
def test_short_row_kernel_few_rows(V, N):
    """Fewer rows than row groups: one CTA with a single row group at work
    (N = 1), and a handful of rows with one masked, for each shape family."""
    L = leap()
    L.leap_get_device_status()
    ld = (V + 7) // 8 * 8
    z, ids, old, adv, w = _inputs(N, V, seed=N + V % 31, sigma=3.0, spikes=0.01, ld=ld, old_sigma=0.3, mask_frac=0.0)
    if N > 1:
        w[N // 2] = 0.0
    dl = torch.full_like(z, float("nan"))
    out = L.leap_grpo_loss_fwd(z, ids, old, adv, w, V=V, dlogits=dl)
    assert L.leap_get_device_status() == 0
    assert not torch.isnan(dl[:, :V]).any()
    rows = list(range(N))
    orc = _oracle_rows(z, ids, old, adv, w, rows, V)
    _check_rows(out, orc, rows, V, dl=dl)
    assert abs(out["loss"].item() - orc["loss"]) <= TOL_LOSS_REL * abs(orc["loss"]) + 1e-12


@pytest.mark.parametrize("V", [32769, 32776, 40960, 40968, 49159])
def test_default_fused_kernel_chunk_boundaries(V):
    """Vocabularies just past the short-row limit and around the pipelined
    kernel's 16 KB (8,192-logit) staging chunks: four whole chunks plus a
    partial vector (32,769), a 16-byte last chunk (32,776), exactly five
    chunks (40,960), five chunks and one vector (40,968), a ragged sixth chunk
    with a partial vector (49,159); every row against the oracle."""
    L = leap()
    L.leap_get_device_status()
    N = 300
    ld = (V + 7) // 8 * 8
    z, ids, old, adv, w = _inputs(N, V, seed=V % 61, sigma=3.0, spikes=0.01, ld=ld, old_sigma=0.3)
    ids[:6] = torch.tensor([0, V - 1, 8191, 8192, 32767, 32768], dtype=torch.int32, device="cuda")
    w[:6] = 0.1
    out = L.leap_grpo_loss_fwd(z, ids, old, adv, w, V=V)
    assert L.leap_get_device_status() == 0
    rows = list(range(N))
    orc = _oracle_rows(z, ids, old, adv, w, rows, V)
    _check_rows(out, orc, rows, V, dl=out["dlogits"])
    assert abs(out["loss"].item() - orc["loss"]) <= TOL_LOSS_REL * abs(orc["loss"])


@pytest.mark.parametrize("N,pattern", [(1, "live"), (151, "random"), (152, "masked"), (153, "runs"),
                                       (1000, "live"), (3001, "runs"), (3001, "random"), (5000, "head")])
@pytest.mark.parametrize("interleaved", [False, True])
def test_default_fused_kernel_row_partition(N, pattern, interleaved):
    """The default fused kernel's persistent CTAs share the rows out among
    themselves and pipeline them (pass 1 of a live row beside pass 2 of the
    previous one, masked rows in between), in stream order or with the live
    rows spread among the masked ones: every row is written, whatever the
    pattern of live and masked rows
    and whether N is below, at or above the CTA count, the loss equals the
    oracle's sum over all rows, and both orders give the same bits."""
    L = leap()
    L.leap_get_device_status()
    V = 33000                                  # above the short-row limit: the pipelined kernel
    z, ids, old, adv, w = _inputs(N, V, seed=N % 53 + 60, sigma=3.0, spikes=0.01, old_sigma=0.3, mask_frac=0.0)
    r = np.arange(N)
    keep = {"live": np.ones(N, bool), "masked": np.zeros(N, bool), "random": np.random.default_rng(N).random(N) < 0.6,
            "runs": (r // 97) % 3 != 1, "head": r < N // 7}[pattern]
    w.mul_(torch.as_tensor(keep.astype(np.float32), device="cuda"))
    dl = torch.full_like(z, float("nan"))
    out = L.leap_grpo_loss_fwd(z, ids, old, adv, w, V=V, dlogits=dl, interleaved_rows=interleaved)
    assert L.leap_get_device_status() == 0
    assert not torch.isnan(dl).any()          # every row written
    if interleaved:                           # the row order changes nothing, bit for bit
        ref = L.leap_grpo_loss_fwd(z, ids, old, adv, w, V=V)
        assert torch.equal(ref["dlogits"], dl) and ref["loss"].item() == out["loss"].item()
    assert torch.all(dl[torch.as_tensor(~keep, device="cuda")] == 0)
    rows = list(range(N))
    orc = _oracle_rows(z, ids, old, adv, w, rows, V)
    if keep.any():
        assert abs(out["loss"].item() - orc["loss"]) <= TOL_LOSS_REL * abs(orc["loss"])
    else:
        assert out["loss"].item() == 0.0
    sample = sorted(set(np.linspace(0, N - 1, min(N, 48)).astype(int).tolist()))
    _check_rows(out, _oracle_rows(z, ids, old, adv, w, sample, V), sample, V, dl=dl)
