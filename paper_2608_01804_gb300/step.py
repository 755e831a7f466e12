"""One pass of the LEAP loss hot path over a resident batch, through libleap.

GrpoStep owns the device buffers of one batch shape and runs, on the current
stream:
  1. leap_group_rank_advantages    DCP gate, tiers, tournament, R, A, A_hat (Sec. 3.1-3.3)
  2. leap_rollout_token_counts     per-rollout optimised-token counts, local totals
  3. (data parallel) all_reduce(totals)  the one exchange: global loss normalisers
  4. leap_scatter_turn_advantages  per-token advantage and aggregation weight
     (one process: steps 2 and 4 as one call, leap_token_advantages)
  5. leap_grpo_loss_fwd            clipped surrogate + fused dlogits (Eq. 3)
Only step 3 leaves libleap, and only when a process group with more than one
rank is passed in.  run() takes resident logits, run_chunked() a stream that
exists chunk by chunk, run_streamed() logits in pinned host memory.  capture() records steps 1-5 as one CUDA graph for
batches small enough that launching six kernels one by one costs more than
running them.
"""

from __future__ import annotations

import torch

from . import leap as L


class GrpoStep:
    def __init__(self, batch, V, device, *, gamma=0.9, tau=None, use_gate_in=True, eps_std=1e-6,
                 eps_low=0.2, eps_high=0.2, inv_temp=1.0, grad_scale=1.0, agg=L.LEAP_AGG_SEQ_MEAN_TOKEN_MEAN,
                 chunk_rows=None):
        self.b = batch
        self.V = int(V)
        self.dev = torch.device(device)
        self.gamma, self.eps_std = gamma, eps_std
        self.tau = tau if tau is not None else (0, batch.G)
        self.use_gate_in = use_gate_in and batch.gate_in is not None
        self.loss_kw = dict(eps_low=eps_low, eps_high=eps_high, inv_temp=inv_temp, grad_scale=grad_scale)
        self.agg = agg
        n, N, M = batch.n, batch.N, batch.M
        d = self.dev
        as_dev = lambda x, dt: torch.as_tensor(x).to(dt).to(d)
        # Per-batch structure (inputs).
        self.pass_turn = as_dev(batch.pass_turn, torch.int8)
        self.num_turns = as_dev(batch.num_turns, torch.int8)
        self.gate_in = as_dev(batch.gate_in, torch.uint8) if self.use_gate_in else None
        self.seg_offsets = as_dev(batch.seg_offsets, torch.int32)
        self.seg_rollout = as_dev(batch.seg_rollout, torch.int32)
        self.seg_turn = as_dev(batch.seg_turn, torch.int8)
        # Intermediates and outputs.
        e = lambda shape, dt: torch.empty(shape, dtype=dt, device=d)
        self.rank_out = dict(gate=e(batch.num_groups, torch.uint8), r=e(n, torch.uint8),
                             n_worse=e(n, torch.int32), n_better=e(n, torch.int32), R=e(n, torch.float32),
                             A=e(n, torch.float32), turn_adv=e(n * M, torch.float32), T_eff=e(n, torch.uint8))
        self.L = e(n, torch.int32)
        self.totals = e(2, torch.int64)
        self.adv = e(N, torch.float32)
        self.w = e(N, torch.float32)
        self.loss = e(1, torch.float32)
        self.chunk_rows = int(chunk_rows) if chunk_rows else N
        self.workspace = L.loss_workspace(min(N, self.chunk_rows), self.V, d)

    def advantages(self, pg=None):
        """Steps 1-4: per-token advantages and weights."""
        b = self.b
        L.leap_group_rank_advantages(self.pass_turn, self.num_turns, G=b.G, M=b.M, tau_min=self.tau[0],
                                     tau_max=self.tau[1], gamma=self.gamma, eps_std=self.eps_std,
                                     gate_in=self.gate_in, out=self.rank_out)
        if pg is None or torch.distributed.get_world_size(pg) == 1:   # counts + scatter in one launch
            L.leap_token_advantages(b.N, self.seg_offsets, self.seg_rollout, self.seg_turn, self.rank_out["turn_adv"],
                                    self.rank_out["T_eff"], M=b.M, agg=self.agg, L=self.L, totals=self.totals,
                                    adv=self.adv, w=self.w)
            return
        L.leap_rollout_token_counts(b.N, self.seg_offsets, self.seg_rollout, self.seg_turn,
                                    self.rank_out["T_eff"], M=b.M, L=self.L, totals=self.totals)
        if torch.distributed.get_backend(pg) == "nccl":
            torch.distributed.all_reduce(self.totals, group=pg)
        else:   # a host backend (gloo): the two counters travel through host memory
            host = self.totals.cpu()
            torch.distributed.all_reduce(host, group=pg)
            self.totals.copy_(host)
        L.leap_scatter_turn_advantages(b.N, self.seg_offsets, self.seg_rollout, self.seg_turn,
                                       self.rank_out["turn_adv"], self.rank_out["T_eff"], self.L, self.totals,
                                       M=b.M, agg=self.agg, adv=self.adv, w=self.w)

    def loss_pass(self, logits, ids, old_logp, dlogits, row0=0, accumulate=False, stats=None,
                  interleaved_rows=False):
        """Step 5 over rows [row0, row0 + logits.shape[0]) of the packed stream."""
        n = logits.shape[0]
        return L.leap_grpo_loss_fwd(logits, ids, old_logp, self.adv[row0:row0 + n], self.w[row0:row0 + n],
                                    V=self.V, loss=self.loss, dlogits=dlogits, want_outputs=False,
                                    workspace=self.workspace, accumulate=accumulate, stats=stats,
                                    interleaved_rows=interleaved_rows, **self.loss_kw)

    def run(self, logits, ids, old_logp, dlogits, pg=None):
        """The whole pass for a batch whose logits are all resident."""
        self.advantages(pg)
        self.loss_pass(logits, ids, old_logp, dlogits)
        return self.loss

    def run_chunked(self, chunks, ids, old_logp, pg=None):
        """The whole pass for a packed stream whose logits exist one chunk at a
        time (a stream longer than HBM holds, e.g. the forward pass producing
        the logits chunk by chunk).  `chunks` yields (row0, logits, dlogits):
        consecutive row ranges [row0, row0 + logits.shape[0]) that cover the
        stream in order; ids and old_logp are device tensors of all rows.  The
        advantages and weights are computed once for the whole stream, then
        the fused loss runs chunk by chunk, accumulating the loss.  A packed
        stream holds long runs of masked rows (prompts, environment feedback),
        so the loss spreads each SM's live rows evenly among its masked ones
        (LEAP_LOSS_INTERLEAVED_ROWS)."""
        self.advantages(pg)
        for c, (row0, z, dl) in enumerate(chunks):
            n = z.shape[0]
            self._ensure_workspace(n)
            self.loss_pass(z, ids[row0:row0 + n], old_logp[row0:row0 + n], dl, row0=row0, accumulate=c > 0,
                           interleaved_rows=True)
        return self.loss

    def capture(self, logits, ids, old_logp, dlogits, warmup=2):
        """A CUDA graph of run() on these buffers.

        One g.replay() is the whole pass (rank, counts, scatter, loss and its
        two reduction launches) with a single host call instead of one per
        kernel, which is what bounds the step on small batches.  The graph
        reads whatever the buffers hold when it replays (refill them in place
        between replays) and leaves the loss in self.loss.  Single process
        only: the all-reduce of the normalisers stays outside graphs.  The
        warm-up calls run the library's one-time setup (device attributes,
        kernel attributes) before capture.
        """
        cur = torch.cuda.current_stream(self.dev)
        side = torch.cuda.Stream(self.dev)
        side.wait_stream(cur)
        with torch.cuda.stream(side):
            for _ in range(warmup):
                self.run(logits, ids, old_logp, dlogits)
        cur.wait_stream(side)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            self.run(logits, ids, old_logp, dlogits)
        return g

    def weighted_row_runs(self):
        """Row ranges [a, b) of the packed stream that can carry loss weight:
        the tokens of generated turns (segments with a turn index).  Every
        other row (prompt, environment feedback, padding) has w = 0, so the
        loss never reads its logits; a turn pruned by DCP may still be in a
        range (its rows are read only if weighted, which they are not)."""
        if getattr(self, "_runs", None) is None:
            b = self.b
            runs = []
            for s in range(len(b.seg_rollout)):
                if b.seg_turn[s] < 0:
                    continue
                lo, hi = int(b.seg_offsets[s]), int(b.seg_offsets[s + 1])
                if hi <= lo:
                    continue
                if runs and runs[-1][1] == lo:
                    runs[-1][1] = hi
                else:
                    runs.append([lo, hi])
            self._runs = [tuple(r) for r in runs]
        return self._runs

    def run_streamed(self, host_logits, ids, old_logp, dlogits, chunk_rows=4096, pg=None, weighted_only=True):
        """The whole pass for a batch whose logits are in pinned host memory.

        Chunks of `chunk_rows` rows go to two device staging buffers on a copy
        stream while the loss runs on the previous chunk on the current stream
        (the loss accumulates over chunks with LEAP_LOSS_ACCUMULATE; dlogits
        rows are written in place), so the host-to-device copy of the logits
        hides the compute.  ids and old_logp are device tensors of all rows.
        With weighted_only (the default) only the rows that can carry loss
        weight (weighted_row_runs) cross the link: the loss never reads the
        logits of a row of weight 0, and writes its dlogits row as zeros.
        self.h2d_logit_bytes holds the logit bytes the call copied.
        """
        if not host_logits.is_pinned():
            raise ValueError("host_logits must be in pinned host memory")
        N, ld = host_logits.shape
        runs = self.weighted_row_runs() if weighted_only else [(0, N)]
        row_bytes = ld * host_logits.element_size()
        self.h2d_logit_bytes = 0
        self._ensure_workspace(min(N, chunk_rows))
        comp = torch.cuda.current_stream(self.dev)
        cs = self._copy_stream()
        staging = self._staging(chunk_rows, ld, host_logits.dtype)
        start = torch.cuda.Event()        # after every earlier use of the staging buffers
        start.record(comp)
        cs.wait_event(start)
        self.advantages(pg)                # overlaps the first chunk's copy
        free = [None, None]
        for c, a in enumerate(range(0, N, chunk_rows)):
            b = min(N, a + chunk_rows)
            buf = staging[c % 2][:b - a]
            if free[c % 2] is not None:
                cs.wait_event(free[c % 2])          # the loss that read this buffer is done
            with torch.cuda.stream(cs):
                for lo, hi in runs:
                    lo, hi = max(lo, a), min(hi, b)
                    if lo < hi:
                        buf[lo - a:hi - a].copy_(host_logits[lo:hi], non_blocking=True)
                        self.h2d_logit_bytes += (hi - lo) * row_bytes
            copied = torch.cuda.Event()
            copied.record(cs)
            comp.wait_event(copied)
            self.loss_pass(buf, ids[a:b], old_logp[a:b], dlogits[a:b], row0=a, accumulate=c > 0)
            done = torch.cuda.Event()
            done.record(comp)
            free[c % 2] = done
        return self.loss

    def _ensure_workspace(self, rows):
        """Grows the loss workspace to cover `rows` rows per loss call."""
        need = L.leap_grpo_loss_workspace_size(rows, self.V)
        if self.workspace.numel() < need:
            self.workspace = L.loss_workspace(rows, self.V, self.dev)

    def _copy_stream(self):
        if getattr(self, "_cs", None) is None:
            self._cs = torch.cuda.Stream(self.dev)
        return self._cs

    def _staging(self, rows, ld, dtype):
        key = (rows, ld, dtype)
        if getattr(self, "_stage_key", None) != key:
            self._stage = [torch.empty((rows, ld), dtype=dtype, device=self.dev) for _ in range(2)]
            self._stage_key = key
        return self._stage

    # libleap counts tokens in one launch up to this many rollouts, three above it;
    # counts and scatter share one launch for tables of up to 768 segments.
    ONE_BLOCK_COUNT_ROLLOUTS = 12000
    ONE_LAUNCH_TOKEN_SEGMENTS = 768

    def token_launches(self, pg=None):
        """Launches of steps 2-4: 1 when counts and scatter share a launch."""
        b = self.b
        single = pg is None or torch.distributed.get_world_size(pg) == 1
        S = len(b.seg_rollout)
        if single and S <= self.ONE_LAUNCH_TOKEN_SEGMENTS and 5 * b.n + 4 * (S + 1) + 17 * S + 16 <= 48 * 1024:
            return 1
        return (1 if b.n <= self.ONE_BLOCK_COUNT_ROLLOUTS else 3) + 1

    def launches_per_run(self, pg=None):
        """Kernel launches one run() makes: rank 1, tokens 1-4, loss 1 + reduce 2."""
        return 1 + self.token_launches(pg) + 1 + 2
