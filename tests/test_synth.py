"""The seeded input generator: Philox known answers, distributions, and the
structural properties the LM and phrase list are drawn with."""
import numpy as np
import pytest

import synth


def test_philox4x32_10_known_answers():
    # Published known-answer vectors of Philox4x32-10 (Salmon et al., SC'11).
    assert synth.philox4x32_10([0, 0, 0, 0], [0, 0]) == [0x6627E8D5, 0xE169C58D, 0xBC57AC4C, 0x9B00DBD8]
    assert synth.philox4x32_10([0xFFFFFFFF] * 4, [0xFFFFFFFF] * 2) == [0x408F276D, 0x41C83B0E, 0xA20BC7C6,
                                                                       0x6D5451FD]
    assert synth.philox4x32_10([0x243F6A88, 0x85A308D3, 0x13198A2E, 0x03707344], [0xA4093822, 0x299F31D0]) == [
        0xD16CFE09, 0x94FDCCEB, 0x5001E420, 0x24126EA1]


def test_normal_moments_and_addressing():
    a = synth.bf16_to_f32(synth.normal_bf16(7, 1, 3, 0, 400_000, 2.0)).astype(np.float64)
    assert abs(a.mean()) < 0.02 and abs(a.std() - 2.0) < 0.02
    # any window of the stream is the same data
    b = synth.normal_bf16(7, 1, 3, 1001, 5000, 2.0)
    assert np.array_equal(b, synth.normal_bf16(7, 1, 3, 0, 6001, 2.0)[1001:])
    # a subset of streams sees what it sees inside a larger batch
    w = synth.scaled(synth.WORKLOADS[1], H=64)
    full = synth.enc_chunk(w, range(6), 2)
    sub = synth.enc_chunk(w, [4, 1], 2)
    assert np.array_equal(sub[0], full[4]) and np.array_equal(sub[1], full[1])


def test_lm_closure_and_budget():
    lm = synth.ngram_lm(5, 64, 4, 6000, 1.1)
    assert len(lm.logp[0]) == 64
    assert abs(lm.total - 6000) < 0.05 * 6000
    sets = [set(map(tuple, t.tolist())) for t in lm.tokens]
    for k in range(1, lm.order):
        for g in sets[k]:
            assert g[:-1] in sets[k - 1], "prefix closure"
            assert g[1:] in sets[k - 1], "suffix closure"
    # sorted, no duplicates
    for t in lm.tokens:
        rows = list(map(tuple, t.tolist()))
        assert rows == sorted(set(rows))
    # top order carries no backoff weight
    assert np.all(lm.bow[-1] == 0)


def test_phrases_constraints():
    p = synth.phrases(11, 8, 40, 2, 5, 0.3)
    assert p.n == 40
    ph = [tuple(p.phrase(i)) for i in range(p.n)]
    assert len(set(ph)) == len(ph)
    for a in ph:
        assert 2 <= len(a) <= 5 and all(0 <= x < 8 for x in a)
        for b in ph:
            if a != b:
                assert b[: len(a)] != a, "no phrase is a prefix of another"
