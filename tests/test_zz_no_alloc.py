"""leap_grpo_loss_fwd_noalloc: the loss entry point for callers that cannot
allocate device memory where they call it (a C caller with no allocator of
its own, or a process whose device memory is fixed up front by a pool).  Its
scratch is libleap's own device array; this checks, through the C ABI, that
two calls in a row give what the workspace entry point gives on the same
inputs (a small call then a larger one, then a small one again, so nothing a
larger call leaves in the array can leak into a smaller one), that a batch
split into two calls with accumulation and statistics equals one workspace
call over the whole batch, and that a batch beyond the array's limit is
refused.  This file is collected last so a failure here never hides the other
tests."""
import ctypes

import numpy as np
import pytest
import torch

from harness import TOL_LOGP, TOL_LOSS_REL, leap, torch_logp
from paper_2608_01804_gb300 import synth

pytestmark = pytest.mark.gpu


def _inputs(N, V, seed):
    z = synth.logits(N, V, 3.0, seed, "cuda", spike_frac=0.01)
    ids = synth.token_ids(N, V, seed + 1, "cuda")
    old = torch_logp(z, ids, V) + synth.normal(N, 0.3, seed + 2, "cuda")
    rng = np.random.default_rng(seed)
    adv = torch.as_tensor(rng.normal(0, 1, N).astype(np.float32), device="cuda")
    w = rng.uniform(0.01, 0.1, N).astype(np.float32)
    w[rng.random(N) < 0.3] = 0.0
    return z, ids, old, adv, torch.as_tensor(w, device="cuda")


def test_two_calls_match_the_workspace_entry_point():
    L = leap()
    L.leap_get_device_status()
    for call, (N, V, seed) in enumerate([(512, 151936, 31), (4096, 1024, 37), (512, 151936, 41)]):
        z, ids, old, adv, w = _inputs(N, V, seed)
        ref = L.leap_grpo_loss_fwd(z, ids, old, adv, w, V=V)
        got = L.leap_grpo_loss_fwd_noalloc(z, ids, old, adv, w, V=V)
        torch.cuda.synchronize()
        assert L.leap_get_device_status() == 0
        r, g = ref["loss"].item(), got["loss"].item()
        assert abs(g - r) <= TOL_LOSS_REL * abs(r), (call, g, r)
        assert torch.max(torch.abs(got["logp"] - ref["logp"])).item() <= TOL_LOGP
        assert torch.max(torch.abs(got["ell"] - ref["ell"])).item() <= 1e-6
        assert torch.equal(got["dlogits"], ref["dlogits"])


def test_chunked_calls_with_accumulation_and_stats():
    """Two no-workspace calls over the two halves of a batch, the second
    accumulating loss and statistics, against one workspace call over the
    whole batch (the chunking the header recommends above the row limit)."""
    L = leap()
    N, V = 6000, 4096
    z, ids, old, adv, w = _inputs(N, V, 43)
    st_ref = L.stats_tensor("cuda")
    ref = L.leap_grpo_loss_fwd(z, ids, old, adv, w, V=V, stats=st_ref)
    st = L.stats_tensor("cuda")
    loss = torch.zeros(1, device="cuda")
    h = 2500
    parts = [L.leap_grpo_loss_fwd_noalloc(z[a:b], ids[a:b], old[a:b], adv[a:b], w[a:b], V=V, loss=loss, stats=st,
                                          accumulate=a > 0)
             for a, b in ((0, h), (h, N))]
    torch.cuda.synchronize()
    assert L.leap_get_device_status() == 0
    r, s = L.read_stats(st_ref), L.read_stats(st)
    assert s["live_tokens"] == r["live_tokens"] and s["clipped_tokens"] == r["clipped_tokens"]
    assert abs(s["loss_sum"] - r["loss_sum"]) <= 1e-12 * max(1.0, abs(r["loss_sum"]))
    assert abs(s["rho_sum"] - r["rho_sum"]) <= 1e-9 * abs(r["rho_sum"])
    assert abs(loss.item() - ref["loss"].item()) <= TOL_LOSS_REL * abs(ref["loss"].item())
    for (a, b), got in zip(((0, h), (h, N)), parts):
        assert torch.equal(got["dlogits"], ref["dlogits"][a:b])
        assert torch.equal(got["ell"], ref["ell"][a:b])


def test_batch_beyond_the_limit_is_refused():
    L = leap()
    lib = L.lib()
    N, V = L.LEAP_NOALLOC_MAX_ROWS + 1, 8
    z = torch.zeros((N, V), dtype=torch.bfloat16, device="cuda")
    ids = torch.zeros(N, dtype=torch.int32, device="cuda")
    f = torch.zeros(N, dtype=torch.float32, device="cuda")
    loss = torch.zeros(1, device="cuda")
    p = L.LossParams(0.2, 0.2, 1.0, 1.0, 0)
    st = lib.leap_grpo_loss_fwd_noalloc(ctypes.byref(p), ctypes.c_void_p(z.data_ptr()), V,
                                        ctypes.c_void_p(ids.data_ptr()), ctypes.c_void_p(f.data_ptr()),
                                        ctypes.c_void_p(f.data_ptr()), ctypes.c_void_p(f.data_ptr()), N, V,
                                        ctypes.c_void_p(loss.data_ptr()), None, None, None, None, None,
                                        ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == L.LEAP_ERR_INVALID_ARG
