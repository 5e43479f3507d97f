"""Parity at the interface's limits and on ragged shapes: the largest
vocabulary, hidden size, LM order and phrase length, many labels per frame,
long chunks, and row counts that leave a partial 128-row tile."""
from __future__ import annotations

import numpy as np
import pytest

import synth
from tests import parity_util as pu

pytestmark = pytest.mark.gpu


def _check(inp, chunks=1, T=None, streams=None, max_chain=None):
    run = pu.GpuRun(inp, streams if streams is not None else range(inp.w.B), chunks, T=T)
    pu.assert_reports(pu.replay(inp, run, range(len(run.streams))))
    return run


def test_largest_vocabulary():
    """V = 16384 labels (the ceiling), a 3-gram LM and a phrase list."""
    w = synth.scaled(synth.WORKLOADS[0], V=16384, H=64, B=3, T=8, lm_total=40000, n_phr=40, phr_len=(2, 5))
    _check(pu.Inputs(w))


def test_largest_hidden_size():
    """H = 8192 (the ceiling): 128 k-blocks in the tensor-core mainloop."""
    w = synth.scaled(synth.WORKLOADS[0], V=256, H=8192, B=2, T=6)
    _check(pu.Inputs(w))


def test_order_16_lm_and_32_label_phrases_fill_the_chains():
    """A 16-gram LM over 8 labels and phrases of up to 32 labels with a large
    boost weight: the decoded histories match long contexts and long phrase
    prefixes, so the LM and trie suffix chains run up to their capacities."""
    w = synth.scaled(synth.WORKLOADS[0], V=8, H=64, B=4, T=60, lm_order=16, lm_total=60000, n_phr=12,
                     phr_len=(16, 32), beta=4.0, lam=0.3)
    lmA = synth.ngram_lm(w.lm_seed, w.V, 16, w.lm_total, 1.05)
    ph = synth.phrases(w.boost_seed, w.V, 12, 16, 32, 0.0)
    inp = pu.Inputs(w, lmA=lmA, ph=ph)
    steps = w.T * w.max_sym
    run = pu.GpuRun(inp, range(w.B), 2, capture_steps=steps)
    pu.assert_reports(pu.replay(inp, run, range(w.B)))
    rows = run.cap_rows.cpu().numpy()  # per step of the last chunk: (t, last, LM state, trie node)
    live = rows[rows[:, :, 0] >= 0]
    lm_depth = max(len(run.lm.state_tuple(int(s))) for s in live[:, 2])
    tr_depth = max(len(run.bo.node_tuple(int(q))) for q in live[:, 3])
    assert lm_depth >= 6, lm_depth
    assert tr_depth >= 12, tr_depth


def test_many_labels_per_frame():
    """max_symbols = 64 (the ceiling): 256 label steps for a 4-frame chunk."""
    w = synth.scaled(synth.WORKLOADS[0], B=3, T=4, max_sym=64)
    _check(pu.Inputs(w), chunks=2)


def test_long_chunk_single_stream():
    """One stream, 1024 frames in one chunk, one label per frame at most."""
    w = synth.scaled(synth.WORKLOADS[0], V=64, H=64, B=1, T=1024, max_sym=1, lm_total=900, n_phr=8, phr_len=(2, 4))
    _check(pu.Inputs(w))


@pytest.mark.parametrize("B", [1, 127, 129])
def test_partial_row_tiles(B):
    """Row counts around the 128-row tile: the last tile is partial."""
    w = synth.scaled(synth.WORKLOADS[1], V=512, H=128, B=B, T=3, lm_total=20000)
    run = pu.GpuRun(pu.Inputs(w), range(B), 1)
    sample = sorted(set([0, B // 2, B - 1]))
    pu.assert_reports(pu.replay(pu.Inputs(w), run, sample))
