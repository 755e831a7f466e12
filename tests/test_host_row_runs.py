"""Host logic of the streamed step: the row ranges that
GrpoStep.weighted_row_runs hands to the host-to-device copy (only these rows'
logits cross the link).  Checked against the oracle's token weights (Sec. 3.3,
Sec. 4.1 aggregation): every row that can carry loss weight lies in a run,
under the recorded DCP gate and with every group expanded; the runs are
sorted, disjoint and maximal (no two touch), and they hold exactly the rows of
generated-turn segments."""
import types

import numpy as np
import pytest

from oracle import leap_oracle as O
from paper_2608_01804_gb300 import synth
from paper_2608_01804_gb300.step import GrpoStep


def _runs(batch):
    # The method reads only the batch layout and its own cache.
    return GrpoStep.weighted_row_runs(types.SimpleNamespace(b=batch, _runs=None))


def _oracle_weights(batch, gate_in):
    G, M = batch.G, batch.M
    out = O.rank_advantages(batch.pass_turn.reshape(-1, G), batch.num_turns.reshape(-1, G), M, 0, G, 0.9,
                            gate_in=gate_in)
    T_eff = out["T_eff"].reshape(-1)
    L, n_tok, n_roll = O.rollout_token_counts(batch.seg_offsets, batch.seg_rollout, batch.seg_turn, T_eff)
    _, w = O.token_advantages(batch.N, batch.seg_offsets, batch.seg_rollout, batch.seg_turn,
                              out["turn_adv"].reshape(-1), T_eff, M, O.AGG_SEQ_MEAN_TOKEN_MEAN, L, n_tok, n_roll)
    return w


@pytest.mark.parametrize("maker", ["tiny", "single_turn", "multiturn"])
def test_weighted_row_runs_cover_every_weighted_row(maker):
    batch = {"tiny": synth.tiny_batch, "single_turn": synth.single_turn_batch,
             "multiturn": synth.multiturn_dcp_batch}[maker]()
    runs = _runs(batch)
    assert runs, "a batch with generated tokens has at least one run"
    in_run = np.zeros(batch.N, dtype=bool)
    prev_hi = -1
    for lo, hi in runs:
        assert 0 <= lo < hi <= batch.N
        assert lo > prev_hi                 # sorted, disjoint, and adjacent runs merged
        in_run[lo:hi] = True
        prev_hi = hi
    # Exactly the rows of segments with a turn index.
    turn_rows = np.zeros(batch.N, dtype=bool)
    for s in range(len(batch.seg_turn)):
        if batch.seg_turn[s] >= 0:
            turn_rows[int(batch.seg_offsets[s]):int(batch.seg_offsets[s + 1])] = True
    assert np.array_equal(in_run, turn_rows)
    gates = [None] + ([batch.gate_in] if batch.gate_in is not None else [])
    for gate_in in gates:
        w = _oracle_weights(batch, gate_in)
        assert np.all(in_run[w != 0])       # no weighted row is left on the host
        assert (w != 0).any()
    if maker != "single_turn":
        assert in_run.sum() < batch.N       # prompts, feedback or padding stay behind


def test_weighted_row_runs_are_cached_and_stable():
    batch = synth.tiny_batch()
    ns = types.SimpleNamespace(b=batch, _runs=None)
    first = GrpoStep.weighted_row_runs(ns)
    assert GrpoStep.weighted_row_runs(ns) is first
    assert first == _runs(synth.tiny_batch())
