"""Failure paths on the GPU, in the forms that fault nothing: a bounded wait
that can never complete gives up after its limit and reports LEAP_DEV_TIMEOUT
through the status word, after which the context still computes correct
results; and a data error (an id outside the vocabulary) is masked and
reported, not read out of bounds."""
import numpy as np
import pytest
import torch

from harness import O, TOL_LOSS_REL, leap, rows_f64, torch_logp
from paper_2608_01804_gb300 import synth

pytestmark = pytest.mark.gpu


def _small_loss_matches_oracle(L, seed):
    V, N = 1024, 64
    z = synth.logits(N, V, 2.0, seed, "cuda")
    ids = synth.token_ids(N, V, seed + 1, "cuda")
    old = torch_logp(z, ids, V) + synth.normal(N, 0.2, seed + 2, "cuda")
    adv = synth.normal(N, 1.0, seed + 3, "cuda")
    w = torch.full((N,), 1.0 / N, device="cuda")
    out = L.leap_grpo_loss_fwd(z, ids, old, adv, w, V=V)
    h = lambda t: t.cpu().numpy().astype(np.float64)
    orc = O.grpo_loss_rows(rows_f64(z, range(N), V), ids.cpu().numpy(), h(old), h(adv), h(w), want_dlogits=False)
    assert abs(out["loss"].item() - orc["loss"]) <= TOL_LOSS_REL * abs(orc["loss"])


@pytest.mark.parametrize("limit_ns", [1_000_000, 20_000_000])
def test_bounded_wait_gives_up_and_reports_timeout(limit_ns):
    L = leap()
    L.leap_get_device_status()
    waited = torch.zeros(1, dtype=torch.int64, device="cuda")
    L.leap_selftest_bounded_wait(limit_ns, waited)
    flags = L.leap_get_device_status()          # synchronises: the kernel has returned
    assert flags == L.LEAP_DEV_TIMEOUT
    took = int(waited.item())
    assert limit_ns <= took < limit_ns + 500_000_000, took
    # The context is intact: the next calls compute the oracle's results and
    # raise no new status bit.
    _small_loss_matches_oracle(L, 900 + limit_ns % 7)
    assert L.leap_get_device_status() == 0


def test_selftest_limit_out_of_range_is_refused():
    L = leap()
    for bad in (0, 999, 10_000_000_001):
        with pytest.raises(L.LeapError) as e:
            L.leap_selftest_bounded_wait(bad)
        assert e.value.status == L.LEAP_ERR_INVALID_ARG
