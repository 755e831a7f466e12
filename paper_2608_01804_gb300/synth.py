"""Seeded synthetic rollout batches shaped like LEAP's training workloads.

The paper trains on CUDA-generation RL rollouts (CUDA-Agent data, KernelBench
evaluation) and on KodCode; none of that data or any model is available, so
these generators stand in for it with the batch shapes of the benchmark
configurations: groups of G rollouts per prompt, up to M turns, per-turn
pass flags, response lengths, environment-feedback segments, bf16 logits.

This module draws inputs only.  It computes nothing the method defines (no
gate, tier, tournament, advantage, log-prob or loss): where a workload needs
a DCP decision (which prompts were expanded to multi-turn), the generator
draws the first-turn failure count inside or outside the stated [tau_min,
tau_max] zone and records the expansion flag as `gate_in`, as a rollout
system would.

Host-side structures are numpy arrays; dense tensors (logits, hidden states)
are torch tensors drawn on the requested device from a seeded torch.Generator.
"""

from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np
import torch


@dataclass
class RolloutBatch:
    """Outcomes and packed token layout of one batch of rollout groups."""
    num_groups: int
    G: int
    M: int
    pass_turn: np.ndarray        # int8 [n]: 0 = never passed, m = first pass at turn m
    num_turns: np.ndarray        # int8 [n]: generated turns
    speedup: np.ndarray          # f32 [n]
    ntokens: np.ndarray          # int32 [n]: generated tokens of the rollout
    gate_in: np.ndarray | None   # u8 [num_groups] recorded expansion flag, or None
    N: int                       # tokens in the packed stream
    seg_offsets: np.ndarray      # int32 [S+1]
    seg_rollout: np.ndarray      # int32 [S]
    seg_turn: np.ndarray         # int8 [S]: turn index, -1 = feedback / padding
    info: dict = field(default_factory=dict)

    @property
    def n(self) -> int:
        return self.num_groups * self.G


def _segments_to_arrays(segs):
    offs = [0]
    roll, turn = [], []
    for length, i, t in segs:
        offs.append(offs[-1] + int(length))
        roll.append(i)
        turn.append(t)
    return (np.asarray(offs, dtype=np.int32), np.asarray(roll, dtype=np.int32),
            np.asarray(turn, dtype=np.int8))


def padded_batch(num_prompts, G, M, slot_len, pass_prob, len_lo, len_hi, seed, gate_in=None,
                 speedup_sigma=0.5):
    """Padded layout [rollout, turn slot, slot_len] (the tiny and single-turn workloads).

    Per rollout and turn: pass flag ~ Bernoulli(pass_prob), response length ~
    U{len_lo..len_hi}, speedup ~ LogNormal(0, speedup_sigma).  A rollout stops
    at its first pass; otherwise it runs all M turns.  Each turn slot holds the
    turn's tokens followed by padding; unused slots are all padding.
    """
    rng = np.random.default_rng(seed)
    n = num_prompts * G
    flags = rng.random((n, M)) < pass_prob
    lens = rng.integers(len_lo, len_hi + 1, size=(n, M))
    speed = rng.lognormal(0.0, speedup_sigma, size=n).astype(np.float32)
    pass_turn = np.zeros(n, dtype=np.int8)
    num_turns = np.full(n, M, dtype=np.int8)
    for i in range(n):
        hit = np.nonzero(flags[i])[0]
        if len(hit):
            pass_turn[i] = hit[0] + 1
            num_turns[i] = hit[0] + 1
    segs = []
    ntok = np.zeros(n, dtype=np.int32)
    starts = np.arange(n + 1, dtype=np.int64) * (M * slot_len)
    for i in range(n):
        for t in range(M):
            if t < num_turns[i]:
                segs.append((lens[i, t], i, t))
                ntok[i] += lens[i, t]
                if slot_len - lens[i, t] > 0:
                    segs.append((slot_len - lens[i, t], -1, -1))
            else:
                segs.append((slot_len, -1, -1))
    so, sr, st = _segments_to_arrays(segs)
    gi = None if gate_in is None else np.asarray(gate_in, dtype=np.uint8)
    return RolloutBatch(num_prompts, G, M, pass_turn, num_turns, speed, ntok, gi, int(so[-1]), so, sr, st,
                        info=dict(layout="padded", slot_len=slot_len, rollout_starts=starts))


def tiny_batch(seed=0):
    """4 prompts x G=8 x 2 turn slots x 256 tokens (16,384 rows); turn 2 pruned for prompts 0 and 1."""
    return padded_batch(4, 8, 2, 256, 0.4, 64, 256, seed, gate_in=[0, 0, 1, 1])


def single_turn_batch(seed=1, num_prompts=16):
    """16 prompts x G=8 x 256 tokens (32,768 rows), one turn, pass ~ Bernoulli(0.3)."""
    return padded_batch(num_prompts, 8, 1, 256, 0.3, 64, 256, seed, gate_in=None)


def multiturn_dcp_batch(seed=2, num_prompts=32, G=16, M=3, len_lo=256, len_hi=2048, frac_expanded=0.4,
                        tau=(8, 15), later_pass_prob=0.35, prompt_lo=256, prompt_hi=1024):
    """Packed ragged multi-turn batch (the DCP workload).

    A fraction `frac_expanded` of prompts is drawn as multi-turn: their
    first-turn failure count is uniform in [tau[0], tau[1]]; the others draw it
    outside that zone.  In expanded groups each first-turn failure receives an
    environment-feedback segment and another turn, up to M, passing each later
    turn with probability `later_pass_prob`.  Each rollout's packed sequence
    starts with its prompt (U{prompt_lo..prompt_hi} tokens, one length per
    prompt, shared by its G rollouts; prompt_hi = 0 leaves prompts out), then
    its turns; generated turns and feedback segments are U{len_lo..len_hi}
    tokens.  Prompt and feedback tokens are masked segments (turn -1).
    """
    rng = np.random.default_rng(seed)
    n = num_prompts * G
    n_exp = int(round(frac_expanded * num_prompts))
    expanded = np.zeros(num_prompts, dtype=np.uint8)
    expanded[rng.permutation(num_prompts)[:n_exp]] = 1
    outside = [k for k in range(G + 1) if not (tau[0] <= k <= tau[1])]
    pass_turn = np.zeros(n, dtype=np.int8)
    num_turns = np.ones(n, dtype=np.int8)
    for g in range(num_prompts):
        n_fail = int(rng.integers(tau[0], tau[1] + 1)) if expanded[g] else int(rng.choice(outside))
        fails = np.zeros(G, dtype=bool)
        fails[rng.permutation(G)[:n_fail]] = True
        for j in range(G):
            i = g * G + j
            if not fails[j]:
                pass_turn[i], num_turns[i] = 1, 1
            elif not expanded[g]:
                pass_turn[i], num_turns[i] = 0, 1
            else:
                t = 2
                while True:
                    if rng.random() < later_pass_prob:
                        pass_turn[i], num_turns[i] = t, t
                        break
                    if t == M:
                        pass_turn[i], num_turns[i] = 0, M
                        break
                    t += 1
    speed = rng.lognormal(0.0, 0.5, size=n).astype(np.float32)
    prompt_len = (rng.integers(prompt_lo, prompt_hi + 1, size=num_prompts) if prompt_hi > 0
                  else np.zeros(num_prompts, dtype=np.int64))
    segs = []
    ntok = np.zeros(n, dtype=np.int32)
    starts = np.zeros(n + 1, dtype=np.int64)
    cur = 0
    for i in range(n):
        starts[i] = cur
        pl = int(prompt_len[i // G])
        if pl > 0:
            segs.append((pl, -1, -1))
            cur += pl
        for t in range(int(num_turns[i])):
            if t > 0:
                fb = int(rng.integers(len_lo, len_hi + 1))
                segs.append((fb, -1, -1))
                cur += fb
            ln = int(rng.integers(len_lo, len_hi + 1))
            segs.append((ln, i, t))
            ntok[i] += ln
            cur += ln
    starts[n] = cur
    so, sr, st = _segments_to_arrays(segs)
    return RolloutBatch(num_prompts, G, M, pass_turn, num_turns, speed, ntok, expanded, int(so[-1]), so, sr, st,
                        info=dict(layout="packed", expanded_prompts=int(n_exp), tau=tau, rollout_starts=starts))


def shard(batch, rank, world):
    """The rollout groups [g0, g1) of this rank (contiguous split) with their
    tokens: segment offsets re-based to the shard, rollout indices local."""
    per = -(-batch.num_groups // world)
    g0, g1 = min(batch.num_groups, rank * per), min(batch.num_groups, (rank + 1) * per)
    i0, i1 = g0 * batch.G, g1 * batch.G
    starts = batch.info["rollout_starts"]
    t0, t1 = int(starts[i0]), int(starts[i1])
    so = batch.seg_offsets
    s0 = int(np.searchsorted(so, t0, side="left"))
    s1 = int(np.searchsorted(so, t1, side="left"))
    seg_offsets = (so[s0:s1 + 1] - t0).astype(np.int32)
    sr = batch.seg_rollout[s0:s1].copy()
    sr[sr >= 0] -= i0
    info = dict(batch.info, rollout_starts=starts[i0:i1 + 1] - t0, shard=(g0, g1), token_range=(t0, t1))
    return RolloutBatch(g1 - g0, batch.G, batch.M, batch.pass_turn[i0:i1], batch.num_turns[i0:i1],
                        batch.speedup[i0:i1], batch.ntokens[i0:i1],
                        None if batch.gate_in is None else batch.gate_in[g0:g1], t1 - t0, seg_offsets, sr,
                        batch.seg_turn[s0:s1].copy(), info=info)


def lmhead_batch(seed=4, n_rollouts=8, tokens=8192):
    """One group of `n_rollouts` single-turn rollouts of `tokens` response tokens
    each, every token valid (the fused lm-head workload: 8 x 8,192 = 65,536
    tokens), pass ~ Bernoulli(0.5)."""
    return padded_batch(1, n_rollouts, 1, tokens, 0.5, tokens, tokens, seed, gate_in=None)


def tournament_outcomes(seed=3, num_groups=65536, G=64, M=3, dup_frac=0.1):
    """Outcome tuples only (no tokens): pass ~ Bernoulli(0.5), turn index ~ U{1..M},
    speedup ~ LogNormal(0, 1), tokens ~ U{128..8192}; about `dup_frac` of the
    rollouts copy the whole tuple of another rollout of the same group."""
    rng = np.random.default_rng(seed)
    n = num_groups * G
    passed = rng.random(n) < 0.5
    turn = rng.integers(1, M + 1, size=n)
    speed = rng.lognormal(0.0, 1.0, size=n).astype(np.float32)
    tok = rng.integers(128, 8193, size=n).astype(np.int32)
    dup = rng.random(n) < dup_frac
    src_local = rng.integers(0, G, size=n)
    idx = np.nonzero(dup)[0]
    src = (idx // G) * G + src_local[idx]
    passed[idx], turn[idx], speed[idx], tok[idx] = passed[src], turn[src], speed[src], tok[src]
    pass_turn = np.where(passed, turn, 0).astype(np.int8)
    num_turns = turn.astype(np.int8)
    return pass_turn, num_turns, speed, tok


# ---------------------------------------------------------------------------
# Dense tensors.
# ---------------------------------------------------------------------------
def _gen(seed, device):
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def logits(N, V, sigma, seed, device, spike_frac=0.0, spike=15.0, ld=None, chunk_rows=4096):
    """bf16 logits [N, ld] (columns >= V are left as zeros) ~ N(0, sigma^2), with a
    fraction `spike_frac` of entries raised by `spike`."""
    ld = V if ld is None else ld
    out = torch.zeros((N, ld), dtype=torch.bfloat16, device=device)
    g = _gen(seed, device)
    for a in range(0, N, chunk_rows):
        b = min(N, a + chunk_rows)
        x = torch.randn((b - a, V), generator=g, device=device, dtype=torch.float32).mul_(sigma)
        if spike_frac > 0:
            x.add_((torch.rand((b - a, V), generator=g, device=device) < spike_frac).float().mul_(spike))
        out[a:b, :V] = x.to(torch.bfloat16)
        del x
    return out


def token_ids(N, V, seed, device):
    g = _gen(seed, device)
    return torch.randint(0, V, (N,), generator=g, device=device, dtype=torch.int32)


def normal(shape, sigma, seed, device, dtype=torch.float32):
    g = _gen(seed, device)
    return torch.randn(shape, generator=g, device=device, dtype=torch.float32).mul_(sigma).to(dtype)
