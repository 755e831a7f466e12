"""The product's data-parallel path (GrpoStep.run with a process group) on two
processes that share the one GPU, joined by a gloo process group.  Each rank
ranks, counts and scatters its own rollout groups (synth.shard: contiguous
groups with their tokens), the two loss normalisers are all-reduced (the one
exchange of the path: through host memory for gloo), and the fused loss runs
on the rank's own rows.  The per-rank losses must sum to the single-process
loss and every rank's dlogits rows must equal the single-process rows bit for
bit (same global weights, per-row kernels).  No kernel of one rank waits on
the other: the only rendezvous is the host all-reduce, bounded by the
process group's timeout."""
import multiprocessing as mp
import os
import socket

import pytest
import torch

from harness import ROOT, leap, torch_logp
from paper_2608_01804_gb300 import synth

pytestmark = pytest.mark.gpu

WORLD = 2


def _batch(kind):
    if kind == "tiny":
        return synth.tiny_batch(), 1024, (0, 8)
    return synth.multiturn_dcp_batch(seed=9, num_prompts=6, G=8, len_lo=64, len_hi=512, tau=(3, 6)), 2048, (3, 6)


def _inputs(b, V, seed):
    z = synth.logits(b.N, V, 2.0, seed, "cuda")
    ids = synth.token_ids(b.N, V, seed + 1, "cuda")
    old = torch_logp(z, ids, V) + synth.normal(b.N, 0.2, seed + 2, "cuda")
    return z, ids, old


def _rank_main(rank, port, kind, outdir):
    import datetime
    import sys
    sys.path.insert(0, ROOT)
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    torch.distributed.init_process_group("gloo", rank=rank, world_size=WORLD,
                                         timeout=datetime.timedelta(seconds=120))
    from paper_2608_01804_gb300.step import GrpoStep
    torch.cuda.set_device(0)
    b, V, tau = _batch(kind)
    z, ids, old = _inputs(b, V, 31)
    sh = synth.shard(b, rank, WORLD)
    t0, t1 = sh.info["token_range"]
    step = GrpoStep(sh, V, "cuda", gamma=0.9, tau=tau)
    dl = torch.empty_like(z[t0:t1])
    loss = step.run(z[t0:t1].contiguous(), ids[t0:t1].contiguous(), old[t0:t1].contiguous(), dl,
                    pg=torch.distributed.group.WORLD)
    torch.cuda.synchronize()
    torch.save(dict(loss=loss.item(), dlogits=dl.cpu(), totals=step.totals.cpu(), rows=(t0, t1)),
               os.path.join(outdir, "rank%d.pt" % rank))
    torch.distributed.destroy_process_group()


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


@pytest.mark.parametrize("kind", ["tiny", "multiturn"])
def test_two_ranks_sum_to_the_single_process_step(kind, tmp_path):
    from paper_2608_01804_gb300.step import GrpoStep
    L = leap()
    b, V, tau = _batch(kind)
    z, ids, old = _inputs(b, V, 31)
    ref = GrpoStep(b, V, "cuda", gamma=0.9, tau=tau)
    dl_ref = torch.empty_like(z)
    loss_ref = ref.run(z, ids, old, dl_ref).item()
    assert L.leap_get_device_status() == 0

    ctx = mp.get_context("spawn")
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, port, kind, str(tmp_path))) for r in range(WORLD)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=300)
    for p in procs:
        if p.is_alive():
            p.kill()
            p.join()
    assert [p.exitcode for p in procs] == [0] * WORLD

    total = 0.0
    covered = 0
    for r in range(WORLD):
        res = torch.load(os.path.join(tmp_path, "rank%d.pt" % r))
        t0, t1 = res["rows"]
        assert torch.equal(res["totals"], ref.totals.cpu())       # global normalisers on every rank
        assert torch.equal(res["dlogits"], dl_ref[t0:t1].cpu())
        total += res["loss"]
        covered += t1 - t0
    assert covered == b.N
    assert abs(total - loss_ref) <= 1e-4 * abs(loss_ref), (total, loss_ref)
