"""Shared helpers for the parity tests: building inputs once and running the
same inputs through libleap (GPU) and through the fp64 oracle (CPU).

Tolerances (stated for the method's outputs):
  bit-exact     gate, tiers r, N_worse, N_better, T_eff, R (fp32 of an exact quotient),
                per-rollout token counts and totals
  1e-5 abs      A and the per-turn / per-token advantages
  2e-3 abs      per-token log-probs and dlogits (plus a per-element relative bound
                of one bf16 ulp on dlogits, which is the meaningful one when the
                weights make dlogits small)
  1e-4 rel      the loss
Tokens whose probability ratio lies within CLIP_BAND of a clip edge (1 - eps_low
or 1 + eps_high, the call's own clip range) may take either branch of the clip
decision (fp32 on the GPU, fp64 in the oracle); their dlogits row must equal the
oracle's unclipped row or be all zeros.
"""

from __future__ import annotations

import os
import sys

import numpy as np
import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from oracle import leap_oracle as O  # noqa: E402

TOL_ADV = 1e-5
TOL_LOGP = 2e-3
TOL_DLOGITS = 2e-3
TOL_LOSS_REL = 1e-4
CLIP_BAND = 1e-5

requires_gpu = pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")


def leap():
    """The binding, with the library built for this machine."""
    from paper_2608_01804_gb300 import build
    build.build()
    from paper_2608_01804_gb300 import leap as L
    L.lib()
    return L


def torch_logp(logits, ids, V, inv_temp=1.0, chunk=2048):
    """Current-policy log-probs of the sampled ids with torch's own fp32
    log_softmax.  Input generation only (old log-probs = these + noise); it is
    neither the oracle nor libleap."""
    out = torch.empty(logits.shape[0], dtype=torch.float32, device=logits.device)
    for a in range(0, logits.shape[0], chunk):
        b = min(logits.shape[0], a + chunk)
        x = logits[a:b, :V].float() * inv_temp
        out[a:b] = torch.log_softmax(x, dim=1).gather(1, ids[a:b].long().view(-1, 1)).view(-1)
    return out


def rows_f64(logits, rows, V):
    """Exact fp64 copies of the chosen bf16 logits rows."""
    idx = torch.as_tensor(np.asarray(rows), device=logits.device, dtype=torch.long)
    bits = logits.index_select(0, idx)[:, :V].contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
    return O.bf16_bits_to_f64(bits)


def bf16_rows_to_f64(t):
    return O.bf16_bits_to_f64(t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16))


def oracle_rank(batch, tau=None, gamma=0.9, eps_std=1e-6, norm=O.ADVNORM_GRPO_STD, std_unbiased=True,
                use_gate_in=True):
    G = batch.G
    pt = batch.pass_turn.reshape(-1, G)
    nt = batch.num_turns.reshape(-1, G)
    tau = tau or (0, G)
    gate_in = batch.gate_in if use_gate_in else None
    return O.rank_advantages(pt, nt, batch.M, tau[0], tau[1], gamma, eps_std, norm, std_unbiased, gate_in)


def oracle_tokens(batch, turn_adv_flat, T_eff_flat, agg=O.AGG_SEQ_MEAN_TOKEN_MEAN):
    L, nv, rv = O.rollout_token_counts(batch.seg_offsets, batch.seg_rollout, batch.seg_turn, T_eff_flat)
    adv, w = O.token_advantages(batch.N, batch.seg_offsets, batch.seg_rollout, batch.seg_turn, turn_adv_flat,
                                T_eff_flat, batch.M, agg, L, nv, rv)
    return L, nv, rv, adv, w


def to_dev(x, dtype, device="cuda"):
    return torch.as_tensor(np.ascontiguousarray(x)).to(dtype).to(device)


def check_dlogits_rows(d_gpu_f64, orc, rows_idx_local, eps_low=0.2, eps_high=0.2):
    """Compares GPU dlogits rows (bf16, as fp64) with the oracle's fp64 rows.

    Two bounds per element: |gpu - bf16(oracle)| <= TOL_DLOGITS, the oracle's
    fp64 value rounded once to the output type; and |gpu - oracle| within one
    bf16 ulp of the exact value (2^-8 relative) plus fp32 slack of 1e-6 of the
    row's largest magnitude.  eps_low / eps_high are the clip range the call
    used (the edges where either branch is accepted).  Returns the max
    absolute error over strictly compared rows.
    """
    exact = orc["dlogits"]
    exact_bf = O.bf16_bits_to_f64(O.f64_to_bf16_bits(exact))
    rho = orc["rho"]
    band = (np.abs(rho - (1.0 + eps_high)) < CLIP_BAND) | (np.abs(rho - (1.0 - eps_low)) < CLIP_BAND)
    worst = 0.0
    for k in range(exact.shape[0]):
        g, e = d_gpu_f64[k], exact[k]
        err = np.abs(g - e)
        bound = 2.0 ** -8 * np.abs(e) + 1e-6 * np.abs(e).max() + 1e-30
        ok_abs = bool(np.all(np.abs(g - exact_bf[k]) <= TOL_DLOGITS))
        ok_rel = bool(np.all(err <= bound))
        if band[k]:
            assert (ok_abs and ok_rel) or np.all(g == 0.0), "boundary row %d matches neither branch" % k
            continue
        if not ok_abs:
            j = int(np.argmax(np.abs(g - exact_bf[k])))
            raise AssertionError("dlogits row %d col %d: |gpu - bf16(oracle)| = %r (gpu %r, oracle %r)"
                                 % (k, j, abs(g[j] - exact_bf[k][j]), g[j], e[j]))
        if not ok_rel:
            j = int(np.argmax(err - bound))
            raise AssertionError("dlogits row %d col %d: gpu %r oracle %r beyond one bf16 ulp" % (k, j, g[j], e[j]))
        worst = max(worst, float(err.max()))
    return worst
