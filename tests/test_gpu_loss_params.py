"""GPU parity of the clipped surrogate (Eq. 3) away from its defaults: a
sampling temperature (inv_temp = 0.7) and an asymmetric clip range
(eps_low = 0.2, eps_high = 0.28), on every kernel that evaluates the loss or
its gradient: the persistent row-pipelined fused kernel with more rows than CTAs,
the short-row kernel at mid-size rows, the single-read kernel at short and long
rows, the forward-only loss with the
split backward, and the fused lm-head with dhidden and dW.  Old log-probs are
drawn around the tempered policy's own log-probs with sigma 0.3, and four
planted tokens sit beyond each edge and between 1.2 and 1.28 (where only the
asymmetric range keeps the gradient), so that every branch is exercised."""
import numpy as np
import pytest
import torch

from harness import (O, TOL_LOGP, TOL_LOSS_REL, bf16_rows_to_f64, check_dlogits_rows, leap, rows_f64,
                     torch_logp)
from paper_2608_01804_gb300 import synth

pytestmark = pytest.mark.gpu

INV_TEMP = 0.7
EPS_LOW, EPS_HIGH = 0.2, 0.28
PARAMS = dict(inv_temp=INV_TEMP, eps_low=EPS_LOW, eps_high=EPS_HIGH)


# Planted ratios (rows 0-3): above the high edge, between 1.2 and 1.28 (only the
# asymmetric range leaves it unclipped), below the low edge, and inside.
PLANT_RHO = (1.35, 1.24, 0.75, 0.9)
PLANT_ADV = (0.8, 1.1, -0.7, -1.3)


def _inputs(N, V, seed, mask_frac=0.2):
    dev = "cuda"
    z = synth.logits(N, V, 3.0, seed, dev, spike_frac=0.01)
    ids = synth.token_ids(N, V, seed + 1, dev)
    cur = torch_logp(z, ids, V, inv_temp=INV_TEMP)
    old = cur + synth.normal(N, 0.3, seed + 2, dev)
    rng = np.random.default_rng(seed + 3)
    adv = rng.normal(0, 1, N).astype(np.float32)
    w = rng.uniform(0.01, 0.1, N).astype(np.float32)
    w[rng.random(N) < mask_frac] = 0.0
    k = len(PLANT_RHO)
    old[:k] = cur[:k] - torch.log(torch.tensor(PLANT_RHO, device=dev))
    adv[:k] = PLANT_ADV
    w[:k] = 0.05
    return z, ids, old, torch.as_tensor(adv, device=dev), torch.as_tensor(w, device=dev)


def _oracle(z, ids, old, adv, w, V, want_dlogits=True):
    h = lambda t: t.cpu().numpy().astype(np.float64)
    return O.grpo_loss_rows(rows_f64(z, range(z.shape[0]), V), ids.cpu().numpy().astype(np.int64), h(old), h(adv),
                            h(w), want_dlogits=want_dlogits, **PARAMS)


def _both_edges_crossed(orc, adv):
    a = adv.cpu().numpy()
    live = orc["live"]
    hi = live & (a >= 0) & (orc["rho"] > 1.0 + EPS_HIGH)
    lo = live & (a < 0) & (orc["rho"] < 1.0 - EPS_LOW)
    # Tokens that only the asymmetric range decides: above 1.2 but not above 1.28.
    mid = live & (a >= 0) & (orc["rho"] > 1.2) & (orc["rho"] <= 1.0 + EPS_HIGH)
    assert hi.any() and lo.any() and mid.any()


def _check(out, orc, V, dl=None):
    live = orc["live"]
    logp = out["logp"].cpu().numpy().astype(np.float64)
    assert np.max(np.abs(logp - orc["logp"])) <= TOL_LOGP
    np.testing.assert_allclose(out["lse"].cpu().numpy()[live], orc["lse"][live], rtol=1e-5)
    ell = out["ell"].cpu().numpy().astype(np.float64)
    band = (np.abs(orc["rho"] - (1 + EPS_HIGH)) < 1e-5) | (np.abs(orc["rho"] - (1 - EPS_LOW)) < 1e-5)
    np.testing.assert_allclose(ell[~band], orc["ell"][~band], rtol=1e-4, atol=1e-6)
    assert abs(out["loss"].item() - orc["loss"]) <= TOL_LOSS_REL * abs(orc["loss"])
    if dl is not None:
        check_dlogits_rows(bf16_rows_to_f64(dl[:, :V]), orc, list(range(dl.shape[0])), EPS_LOW, EPS_HIGH)


def test_default_fused_kernel_many_rows_per_cta():
    """V = 151,936 with 400 rows: each of the 152 persistent CTAs walks two or
    three rows, so the pass-1 / pass-2 pipeline of the default fused kernel
    hands rows over at both parameter sets' clip edges."""
    L = leap()
    L.leap_get_device_status()
    V, N = 151936, 400
    z, ids, old, adv, w = _inputs(N, V, seed=41)
    out = L.leap_grpo_loss_fwd(z, ids, old, adv, w, V=V, **PARAMS)
    assert L.leap_get_device_status() == 0
    orc = _oracle(z, ids, old, adv, w, V)
    _both_edges_crossed(orc, adv)
    _check(out, orc, V, dl=out["dlogits"])


@pytest.mark.parametrize("V,N", [(1024, 2048), (1000, 700), (8192, 512), (151936, 96)])
def test_single_read_kernel(V, N):
    L = leap()
    L.leap_get_device_status()
    z, ids, old, adv, w = _inputs(N, V, seed=V % 89 + 7)
    out = L.leap_grpo_loss_fwd(z, ids, old, adv, w, V=V, single_read=True, **PARAMS)
    assert L.leap_get_device_status() == 0
    orc = _oracle(z, ids, old, adv, w, V)
    _both_edges_crossed(orc, adv)
    _check(out, orc, V, dl=out["dlogits"])


@pytest.mark.parametrize("V,N", [(16384, 700), (32000, 400)])
def test_short_row_kernel_mid_vocab(V, N):
    """The short-row kernel's eight- and sixteen-warp row groups (4 KB slices)
    at both clip edges and the tempered softmax."""
    L = leap()
    L.leap_get_device_status()
    z, ids, old, adv, w = _inputs(N, V, seed=V % 83 + 5)
    out = L.leap_grpo_loss_fwd(z, ids, old, adv, w, V=V, **PARAMS)
    assert L.leap_get_device_status() == 0
    orc = _oracle(z, ids, old, adv, w, V)
    _both_edges_crossed(orc, adv)
    _check(out, orc, V, dl=out["dlogits"])


@pytest.mark.parametrize("V,N", [(1024, 1024), (151936, 160)])
def test_forward_only_then_split_backward(V, N):
    L = leap()
    z, ids, old, adv, w = _inputs(N, V, seed=V % 83 + 11)
    fwd = L.leap_grpo_loss_fwd(z, ids, old, adv, w, V=V, want_dlogits=False, **PARAMS)
    assert fwd["dlogits"] is None
    orc = _oracle(z, ids, old, adv, w, V)
    _both_edges_crossed(orc, adv)
    _check(fwd, orc, V)
    dl = L.leap_grpo_loss_bwd(z, ids, old, adv, w, fwd["lse"], V=V, grad_scale=1.0, **PARAMS)
    check_dlogits_rows(bf16_rows_to_f64(dl[:, :V]), orc, list(range(N)), EPS_LOW, EPS_HIGH)


def test_fused_lmhead_with_gradients():
    """logits = hidden . W^T on tcgen05, then Eq. 3 at the same temperature and
    clip range; dhidden row by row and dW element by element against fp64."""
    L = leap()
    L.leap_get_device_status()
    N, H, V = 300, 256, 1000
    g = torch.Generator(device="cuda")
    g.manual_seed(77)
    hidden = torch.randn((N, H), generator=g, device="cuda").to(torch.bfloat16)
    W = (torch.randn((V, H), generator=g, device="cuda") * 0.16).to(torch.bfloat16)
    ids = torch.randint(0, V, (N,), generator=g, device="cuda", dtype=torch.int32)
    z = hidden.float() @ W.float().T
    logp = torch.log_softmax(z * INV_TEMP, dim=1).gather(1, ids.long().view(-1, 1)).view(-1)
    old = logp + torch.randn(N, generator=g, device="cuda") * 0.3
    k = len(PLANT_RHO)
    old[:k] = logp[:k] - torch.log(torch.tensor(PLANT_RHO, device="cuda"))
    rng = np.random.default_rng(78)
    av = rng.normal(0, 1, N).astype(np.float32)
    av[:k] = PLANT_ADV
    adv = torch.as_tensor(av, device="cuda")
    wv = rng.uniform(0.01, 0.1, N).astype(np.float32)
    wv[rng.random(N) < 0.2] = 0.0
    wv[:k] = 0.05
    w = torch.as_tensor(wv, device="cuda")
    out = L.leap_fused_lmhead_logprobs(hidden, W, ids, old, adv, w, want_dW=True, **PARAMS)
    torch.cuda.synchronize()
    assert L.leap_get_device_status() == 0
    hf, Wf = bf16_rows_to_f64(hidden), bf16_rows_to_f64(W)
    h = lambda t: t.cpu().numpy().astype(np.float64)
    orc = O.lmhead_loss_rows(hf, Wf, ids.cpu().numpy(), h(old), h(adv), h(w), want_dW=True, **PARAMS)
    _both_edges_crossed(orc, adv)
    live = orc["live"]
    assert np.max(np.abs(h(out["logp"]) - orc["logp"])) <= TOL_LOGP
    np.testing.assert_allclose(out["lse"].cpu().numpy()[live], orc["lse"][live], rtol=1e-5)
    assert abs(out["loss"].item() - orc["loss"]) <= TOL_LOSS_REL * abs(orc["loss"])
    band = (np.abs(orc["rho"] - (1 + EPS_HIGH)) < 1e-5) | (np.abs(orc["rho"] - (1 - EPS_LOW)) < 1e-5)
    dh = bf16_rows_to_f64(out["dhidden"])
    for k in range(N):
        if band[k]:
            continue
        ref = orc["dhidden"][k]
        nrm = np.linalg.norm(ref)
        if nrm == 0:
            assert np.all(dh[k] == 0), k
        else:
            assert np.linalg.norm(dh[k] - ref) <= 1e-2 * nrm, k
    # dW: elementwise 2^-8 T with T = |dlogits|^T |hidden| (bf16 dlogits, fp32 sums).
    keep = ~band
    dl_o = orc["dlogits"][keep]
    ref = dl_o.T @ hf[keep]
    T = np.abs(dl_o).T @ np.abs(hf[keep])
    err = np.abs(out["dW"].cpu().numpy().astype(np.float64) - ref)
    if band.any():   # a token on a clip edge may have taken either branch: allow its whole term
        T = T + np.abs(orc["dlogits"][band]).T @ np.abs(hf[band]) * 2 ** 8
    assert np.all(err <= 2.0 ** -8 * T + 1e-30), float(np.max(err / (T + 1e-30)))
