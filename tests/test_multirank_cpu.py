"""Data-parallel path on CPU (gloo, world size 2), with the oracle as compute.

Groups are sharded contiguously across ranks; each rank runs the rank /
token steps on its own groups, all-reduces the two loss normalisers (the one
exchange of the path), computes its partial loss, and the partial losses sum
to the single-rank loss.  A rank that leaves before the exchange ends the
other rank's collective with an error instead of a hang.
"""
import datetime
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from harness import O
from paper_2608_01804_gb300 import synth

V = 24


def _data():
    b = synth.multiturn_dcp_batch(seed=4, num_prompts=6, G=8, M=3, len_lo=8, len_hi=40, tau=(4, 7))
    rng = np.random.default_rng(5)
    z = rng.normal(0, 2, size=(b.N, V))
    ids = rng.integers(0, V, size=b.N)
    _, logp = O.log_softmax_rows(z, ids)
    old = logp + rng.normal(0, 0.3, size=b.N)
    return b, z, ids, old


def _partial_loss(b, z, ids, old, rank, world, agg, allreduce):
    part = synth.shard(b, rank, world)
    G = part.G
    if part.n:
        orc = O.rank_advantages(part.pass_turn.reshape(-1, G), part.num_turns.reshape(-1, G), part.M, 4, 7, 0.9,
                                gate_in=part.gate_in)
        ta, te = orc["turn_adv"].reshape(-1), orc["T_eff"].reshape(-1)
    else:
        ta, te = np.zeros(0), np.zeros(0, dtype=np.int64)
    L, nv, rv = O.rollout_token_counts(part.seg_offsets, part.seg_rollout, part.seg_turn, te)
    totals = allreduce(torch.tensor([nv, rv], dtype=torch.int64))
    adv, w = O.token_advantages(part.N, part.seg_offsets, part.seg_rollout, part.seg_turn, ta, te, part.M, agg, L,
                                int(totals[0]), int(totals[1]))
    t0, t1 = part.info["token_range"]
    return O.grpo_loss_rows(z[t0:t1], ids[t0:t1], old[t0:t1], adv, w, want_dlogits=False)["loss"]


def _worker(rank, world, port, agg, q, drop_rank):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world, timeout=datetime.timedelta(seconds=10))
    try:
        if rank == drop_rank:
            os._exit(3)        # leaves between steps, before the exchange
        b, z, ids, old = _data()

        def allreduce(t):
            dist.all_reduce(t)
            return t

        part = _partial_loss(b, z, ids, old, rank, world, agg, allreduce)
        total = allreduce(torch.tensor([part], dtype=torch.float64))
        q.put((rank, float(total.item())))
    except Exception as e:  # reported to the parent
        q.put((rank, "error: %s" % type(e).__name__))
        q.close()
        q.join_thread()
        os._exit(0)            # the group is broken: do not wait on it
    dist.destroy_process_group()


def _run(world, agg, drop_rank=-1):
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_worker, args=(r, world, port, agg, q, drop_rank)) for r in range(world)]
    for p in procs:
        p.start()
    out = {}
    for _ in range(world - (1 if drop_rank >= 0 else 0)):
        r, v = q.get(timeout=120)
        out[r] = v
    for r, p in enumerate(procs):
        p.join(timeout=60)
        if p.is_alive():
            p.kill()
        if r == drop_rank:
            out[r] = "left" if p.exitcode == 3 else "exit %r" % p.exitcode
    return out


@pytest.mark.parametrize("agg", [O.AGG_SEQ_MEAN_TOKEN_MEAN, O.AGG_TOKEN_MEAN])
def test_sharded_loss_equals_single_rank(agg):
    b, z, ids, old = _data()
    whole = _partial_loss(b, z, ids, old, 0, 1, agg, lambda t: t)
    out = _run(2, agg)
    for r in range(2):
        assert isinstance(out[r], float), out
        assert out[r] == pytest.approx(whole, rel=1e-12)
    # Without the exchange (local normalisers) the shards would not sum to the whole.
    local = sum(_partial_loss(b, z, ids, old, r, 2, agg, lambda t: t) for r in range(2))
    assert local != pytest.approx(whole, rel=1e-6)


def test_rank_leaving_before_the_exchange_is_an_error_not_a_hang():
    out = _run(2, O.AGG_SEQ_MEAN_TOKEN_MEAN, drop_rank=1)
    assert out[1] == "left"
    assert isinstance(out[0], str) and out[0].startswith("error"), out
