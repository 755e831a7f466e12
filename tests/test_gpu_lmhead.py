"""GPU parity of the tcgen05 path: the plain GEMM against torch's fp32 matmul of
the same bf16 values, and the fused lm-head (log-probs, loss, dhidden)
against the fp64 oracle.

Tolerances: the GEMM output is bf16 of an fp32 sum, so |C - ref| <= one bf16
ulp of |ref| plus fp32 accumulation slack (1e-4 of the row's largest
|ref|).  dhidden is a sum over V of bf16-rounded dlogits (relative 2^-9 each)
rounded once more to bf16, so its normwise relative error per row is bounded
by about 2^-8: the test uses 1e-2.  Log-probs 2e-3 absolute, loss 1e-4
relative, as everywhere.

dW = sum over tokens of bf16-rounded dlogits (relative error <= 2^-9 each,
round to nearest) times exact bf16 hidden values, accumulated in fp32 and
kept in fp32.  So |dW - dW_ref| <= 2^-9 T + (fp32 accumulation) with
T = |dlogits|^T |hidden| (fp64, the oracle's dlogits): the test uses 2^-8 T.
The fp32 weight-gradient GEMM alone (exact bf16 products, fp32 sums) is held
to 2^-14 of sum_k |a b|."""
import numpy as np
import pytest
import torch

from harness import O, TOL_LOGP, TOL_LOSS_REL, bf16_rows_to_f64, leap

pytestmark = pytest.mark.gpu


def _bf16(shape, sigma, seed):
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    return (torch.randn(shape, generator=g, device="cuda") * sigma).to(torch.bfloat16)


@pytest.mark.parametrize("M,N,K", [(128, 256, 64), (256, 512, 320), (200, 300, 136), (1000, 1000, 1024),
                                   (130, 520, 5120)])
def test_gemm_bf16_nt(M, N, K):
    L = leap()
    A = _bf16((M, K), 1.0, M + K)
    B = _bf16((N, K), 0.5, N + 3 * K)
    C = L.leap_gemm_bf16_nt(A, B)
    ref = (A.double() @ B.double().T)
    got = C.double()
    bound = 2.0 ** -8 * ref.abs() + 1e-4 * ref.abs().amax(dim=1, keepdim=True) + 1e-30
    bad = (got - ref).abs() > bound
    assert not bad.any(), "max excess %r at %r" % (((got - ref).abs() - bound).max().item(),
                                                   torch.nonzero(bad)[:5].tolist())


def _tn_bound(A, B):
    return 2.0 ** -14 * (A.double().abs().T @ B.double().abs()) + 1e-30


@pytest.mark.parametrize("M,N,K", [(128, 256, 64), (256, 512, 320), (1000, 1000, 1024),
                                   (64, 40, 100), (2376, 520, 8192), (136, 5120, 72), (200, 296, 136)])
def test_gemm_bf16_tn_f32(M, N, K):
    """C = A^T B with both operands MN-major in shared memory (contraction over rows)."""
    L = leap()
    A = _bf16((K, M), 1.0, M + 7 * K)
    B = _bf16((K, N), 0.5, N + 5 * K)
    C = L.leap_gemm_bf16_tn_f32(A, B)
    ref = A.double().T @ B.double()
    bad = (C.double() - ref).abs() > _tn_bound(A, B)
    assert not bad.any(), torch.nonzero(bad)[:5].tolist()


def test_gemm_bf16_tn_f32_accumulate_and_empty():
    L = leap()
    A = _bf16((200, 136), 1.0, 1)
    B = _bf16((200, 264), 1.0, 2)
    C0 = _bf16((136, 264), 3.0, 3).float()
    C = C0.clone()
    L.leap_gemm_bf16_tn_f32(A, B, out=C, accumulate=True)
    ref = C0.double() + A.double().T @ B.double()
    assert not ((C.double() - ref).abs() > _tn_bound(A, B) + 2.0 ** -23 * C0.double().abs()).any()
    # K = 0: an empty sum.
    E = torch.full((136, 264), 5.0, device="cuda")
    L.leap_gemm_bf16_tn_f32(A[:0], B[:0], out=E, accumulate=True)
    assert torch.all(E == 5.0)
    L.leap_gemm_bf16_tn_f32(A[:0], B[:0], out=E)
    assert torch.all(E == 0.0)


def _check_dW(dW, orc, hf):
    """Elementwise 2^-8 T bound (T = |dlogits|^T |hidden|) on the rows given by the oracle."""
    ref = orc["dW"]
    T = np.abs(orc["dlogits_sel"]).T @ np.abs(hf)
    err = np.abs(dW - ref)
    assert np.all(err <= 2.0 ** -8 * T + 1e-30), float(np.max(err / (T + 1e-30)))


def _lmhead_inputs(N, H, V, seed, old_sigma=0.3):
    hidden = _bf16((N, H), 1.0, seed)
    W = _bf16((V, H), 0.02 * 8, seed + 1)     # wider logits than 0.02 so the softmax is not flat
    g = torch.Generator(device="cuda")
    g.manual_seed(seed + 2)
    ids = torch.randint(0, V, (N,), generator=g, device="cuda", dtype=torch.int32)
    z = hidden.float() @ W.float().T
    logp = torch.log_softmax(z, dim=1).gather(1, ids.long().view(-1, 1)).view(-1)
    old = logp + torch.randn(N, generator=g, device="cuda") * old_sigma
    rng = np.random.default_rng(seed)
    adv = torch.as_tensor(rng.normal(0, 1, N).astype(np.float32), device="cuda")
    w = rng.uniform(0.01, 0.1, N).astype(np.float32)
    w[rng.random(N) < 0.25] = 0.0
    return hidden, W, ids, old, adv, torch.as_tensor(w, device="cuda")


@pytest.mark.parametrize("N,H,V", [(128, 64, 256), (300, 256, 1000), (520, 512, 4100), (256, 1024, 32000)])
def test_fused_lmhead_all_rows(N, H, V):
    L = leap()
    L.leap_get_device_status()
    hidden, W, ids, old, adv, w = _lmhead_inputs(N, H, V, seed=N + V)
    out = L.leap_fused_lmhead_logprobs(hidden, W, ids, old, adv, w)
    torch.cuda.synchronize()
    assert L.leap_get_device_status() == 0
    hf = bf16_rows_to_f64(hidden)
    Wf = bf16_rows_to_f64(W)
    orc = O.lmhead_loss_rows(hf, Wf, ids.cpu().numpy(), old.cpu().numpy().astype(np.float64),
                             adv.cpu().numpy().astype(np.float64), w.cpu().numpy().astype(np.float64))
    live = orc["live"]
    logp = out["logp"].cpu().numpy().astype(np.float64)
    assert np.max(np.abs(logp - orc["logp"])) <= TOL_LOGP
    assert np.all(logp[~live] == 0)
    np.testing.assert_allclose(out["lse"].cpu().numpy()[live], orc["lse"][live], rtol=1e-5)
    assert abs(out["loss"].item() - orc["loss"]) <= TOL_LOSS_REL * abs(orc["loss"])
    dh = bf16_rows_to_f64(out["dhidden"])
    ref = orc["dhidden"]
    for k in range(N):
        nrm = np.linalg.norm(ref[k])
        if nrm == 0:
            assert np.all(dh[k] == 0)
        else:
            assert np.linalg.norm(dh[k] - ref[k]) <= 1e-2 * nrm, (k, np.linalg.norm(dh[k] - ref[k]) / nrm)


@pytest.mark.parametrize("N,H,V", [(128, 64, 256), (300, 256, 1000), (520, 512, 4100), (40000, 128, 1000)])
def test_fused_lmhead_dW(N, H, V):
    """dW over every row; N = 40,000 spans three 16,384-token chunks (the last ragged)."""
    L = leap()
    L.leap_get_device_status()
    hidden, W, ids, old, adv, w = _lmhead_inputs(N, H, V, seed=3 * N + V)
    out = L.leap_fused_lmhead_logprobs(hidden, W, ids, old, adv, w, want_dW=True)
    base = L.leap_fused_lmhead_logprobs(hidden, W, ids, old, adv, w)
    torch.cuda.synchronize()
    assert L.leap_get_device_status() == 0
    # Asking for dW changes nothing else.
    assert torch.equal(out["dhidden"], base["dhidden"]) and torch.equal(out["logp"], base["logp"])
    assert out["loss"].item() == base["loss"].item()
    hf = bf16_rows_to_f64(hidden)
    orc = O.lmhead_loss_rows(hf, bf16_rows_to_f64(W), ids.cpu().numpy(), old.cpu().numpy().astype(np.float64),
                             adv.cpu().numpy().astype(np.float64), w.cpu().numpy().astype(np.float64),
                             want_dhidden=False, want_dW=True)
    orc["dlogits_sel"] = orc["dlogits"]
    _check_dW(out["dW"].cpu().numpy().astype(np.float64), orc, hf)
    # dW alone (no dhidden) and accumulation into a preset dW.
    only = L.leap_fused_lmhead_logprobs(hidden, W, ids, old, adv, w, want_dhidden=False, want_dW=True)
    assert only["dhidden"] is None and torch.equal(only["dW"], out["dW"])
    D0 = _bf16((V, H), 0.01, 9).float()
    acc = L.leap_fused_lmhead_logprobs(hidden, W, ids, old, adv, w, want_dhidden=False, dW=D0.clone(),
                                       want_dW=True, accumulate=True, loss=torch.zeros(1, device="cuda"))
    diff = (acc["dW"] - D0 - out["dW"]).abs().double().cpu().numpy()
    T = np.abs(orc["dlogits"]).T @ np.abs(hf)
    assert np.all(diff <= 2.0 ** -8 * T + 2.0 ** -22 * np.abs(D0.double().cpu().numpy()) + 1e-30)


def test_fused_lmhead_dW_no_tokens():
    L = leap()
    H, V = 64, 256
    hidden = torch.empty((0, H), dtype=torch.bfloat16, device="cuda")
    W = _bf16((V, H), 0.1, 1)
    e32 = torch.empty(0, dtype=torch.float32, device="cuda")
    ids = torch.empty(0, dtype=torch.int32, device="cuda")
    dW = torch.full((V, H), 3.0, device="cuda")
    out = L.leap_fused_lmhead_logprobs(hidden, W, ids, e32, e32, e32, want_dhidden=False, want_dW=True, dW=dW)
    torch.cuda.synchronize()
    assert torch.all(out["dW"] == 0) and out["loss"].item() == 0.0


def test_fused_lmhead_forward_only():
    L = leap()
    hidden, W, ids, old, adv, w = _lmhead_inputs(256, 128, 3000, seed=5)
    out = L.leap_fused_lmhead_logprobs(hidden, W, ids, old, adv, w, want_dhidden=False)
    assert out["dhidden"] is None
    full = L.leap_fused_lmhead_logprobs(hidden, W, ids, old, adv, w)
    assert out["loss"].item() == full["loss"].item()
    assert torch.equal(out["logp"], full["logp"])


def test_fused_lmhead_full_size_sampled():
    """65,536 tokens x H = 5,120 x V = 151,936 (the benchmark's lm-head workload):
    sampled rows against the oracle; the loss against the fp64 sum of the
    kernel's own per-row terms."""
    from paper_2608_01804_gb300 import synth
    L = leap()
    N, H, V = 65536, 5120, 151936
    hidden = synth.normal((N, H), 1.0, 600, "cuda", dtype=torch.bfloat16)
    W = synth.normal((V, H), 0.02, 601, "cuda", dtype=torch.bfloat16)
    ids = synth.token_ids(N, V, 602, "cuda")
    rng = np.random.default_rng(603)
    rows = sorted(set([0, 1, 127, 128, N - 1] + rng.choice(N, 7, replace=False).tolist()))
    sel = torch.as_tensor(rows, device="cuda")
    z_sel = (hidden[sel].float() @ W.float().T)
    old = torch.full((N,), -12.0, device="cuda")
    old[sel] = torch.log_softmax(z_sel, 1).gather(1, ids[sel].long().view(-1, 1)).view(-1) + 0.3
    adv = torch.as_tensor(rng.normal(0, 1, N).astype(np.float32), device="cuda")
    w = torch.full((N,), 1.0 / N, device="cuda")
    w[rows[2]] = 0.0
    out = L.leap_fused_lmhead_logprobs(hidden, W, ids, old, adv, w)
    torch.cuda.synchronize()
    assert L.leap_get_device_status() == 0
    Wf = bf16_rows_to_f64(W)
    hf = bf16_rows_to_f64(hidden[sel])
    orc = O.lmhead_loss_rows(hf, Wf, ids[sel].cpu().numpy(), old[sel].cpu().numpy().astype(np.float64),
                             adv[sel].cpu().numpy().astype(np.float64), w[sel].cpu().numpy().astype(np.float64))
    logp = out["logp"][sel].cpu().numpy().astype(np.float64)
    assert np.max(np.abs(logp - orc["logp"])) <= TOL_LOGP
    np.testing.assert_allclose(out["ell"][sel].cpu().numpy(), orc["ell"], rtol=1e-4, atol=1e-7)
    dh = bf16_rows_to_f64(out["dhidden"][sel])
    for k in range(len(rows)):
        nrm = np.linalg.norm(orc["dhidden"][k])
        if nrm == 0:
            assert np.all(dh[k] == 0)
        else:
            assert np.linalg.norm(dh[k] - orc["dhidden"][k]) <= 1e-2 * nrm
    tot = float((w.double() * out["ell"].double()).sum().item())
    assert abs(out["loss"].item() - tot) <= 1e-6 * abs(tot) + 1e-12


def test_fused_lmhead_dW_full_size():
    """The benchmark's lm-head workload with dW: (1) with every row live, the
    identity <dW, W> = <dhidden, hidden> (both equal sum dlogits * z), whose
    gap is bounded by the bf16 rounding of dhidden; (2) with seven live rows
    spread over the four 16,384-token chunks' edges, sampled rows of dW
    against the oracle (masked rows add nothing to dW)."""
    from paper_2608_01804_gb300 import synth
    L = leap()
    N, H, V = 65536, 5120, 151936
    hidden = synth.normal((N, H), 1.0, 610, "cuda", dtype=torch.bfloat16)
    W = synth.normal((V, H), 0.02, 611, "cuda", dtype=torch.bfloat16)
    ids = synth.token_ids(N, V, 612, "cuda")
    rng = np.random.default_rng(613)
    adv = torch.as_tensor(rng.normal(0, 1, N).astype(np.float32), device="cuda")
    old = torch.full((N,), -12.0, device="cuda")
    ws = torch.empty(L.leap_fused_lmhead_workspace_size(N, H, V, True, True), dtype=torch.uint8, device="cuda")
    dW = torch.empty((V, H), dtype=torch.float32, device="cuda")
    w = torch.full((N,), 1.0 / N, device="cuda")
    out = L.leap_fused_lmhead_logprobs(hidden, W, ids, old, adv, w, want_dW=True, dW=dW, workspace=ws)
    torch.cuda.synchronize()
    assert L.leap_get_device_status() == 0
    lhs = rhs = s_w = s_h = 0.0
    for a in range(0, V, 16384):
        t = dW[a:a + 16384].double() * W[a:a + 16384].double()
        lhs += t.sum().item()
        s_w += t.abs().sum().item()
    for a in range(0, N, 8192):
        t = out["dhidden"][a:a + 8192].double() * hidden[a:a + 8192].double()
        rhs += t.sum().item()
        s_h += t.abs().sum().item()
    assert abs(lhs - rhs) <= 2.0 ** -8 * s_h + 1e-5 * s_w, (lhs, rhs, s_h, s_w)
    # Seven live rows: chunk edges and interiors.
    rows = [0, 16383, 16384, 30001, 49151, 49152, N - 1]
    sel = torch.as_tensor(rows, device="cuda")
    w = torch.zeros(N, device="cuda")
    w[sel] = 0.125
    z_sel = hidden[sel].float() @ W.float().T
    old[sel] = torch.log_softmax(z_sel, 1).gather(1, ids[sel].long().view(-1, 1)).view(-1) + 0.2
    out = L.leap_fused_lmhead_logprobs(hidden, W, ids, old, adv, w, want_dhidden=False, want_dW=True, dW=dW,
                                       workspace=ws)
    torch.cuda.synchronize()
    assert L.leap_get_device_status() == 0
    vs = sorted(set(ids[sel].tolist() + [0, 1, 127, 128, V - 1] + rng.choice(V, 40, replace=False).tolist()))
    hf = bf16_rows_to_f64(hidden[sel])
    orc = O.lmhead_loss_rows(hf, bf16_rows_to_f64(W), ids[sel].cpu().numpy(),
                             old[sel].cpu().numpy().astype(np.float64), adv[sel].cpu().numpy().astype(np.float64),
                             w[sel].cpu().numpy().astype(np.float64), want_dhidden=False, want_dW=True, dW_rows=vs)
    orc["dlogits_sel"] = orc["dlogits"][:, vs]
    _check_dW(dW[torch.as_tensor(vs, device="cuda")].double().cpu().numpy(), orc, hf)
