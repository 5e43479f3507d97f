"""The library's ARPA reader (host parser, and LM tables built from a file)
against the oracle's independent reader."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import paper_2609_14991_gb300 as tsd
import synth
from tests.arpa_util import write_arpa


def _same(prod, ora):
    toks, lps, bws, skipped = prod
    assert skipped == ora.skipped
    assert len(toks) == ora.order
    for k in range(ora.order):
        assert np.array_equal(toks[k], ora.tokens[k])
        assert np.array_equal(lps[k], ora.logp[k])
        assert np.array_equal(bws[k], ora.bow[k])


def test_parse_numeric_ids_matches_oracle():
    a = synth.ngram_lm(31, 50, 4, 1500, 1.1)
    text = write_arpa(a)
    _same(tsd.parse_arpa(text, a.V), oracle.read_arpa(text, a.V))


def test_parse_vocab_and_markers_matches_oracle():
    a = synth.ngram_lm(32, 20, 3, 300, 1.05)
    vocab = ["\u2581tok%d" % i for i in range(a.V)]
    extra = {1: [(-1.25, "</s>", None), (-99, "<s>", -0.5), (-2.0, "<unk>", None)],
             2: [(-0.3, "<s> %s" % vocab[2], -0.1), (-0.6, "%s </s>" % vocab[4], None)],
             3: [(-0.2, "<s> %s %s" % (vocab[2], vocab[3]), None)]}
    text = write_arpa(a, vocab=vocab, extra=extra)
    prod = tsd.parse_arpa(text, a.V, vocab=vocab)
    _same(prod, oracle.read_arpa(text, a.V, vocab=vocab))
    assert prod[3] == 6
    for k in range(a.order):  # the kept lines are exactly the model's n-grams
        assert np.array_equal(prod[0][k], a.tokens[k])


def test_parse_crlf_and_spaces():
    text = "\\data\\\r\nngram 1=2\r\nngram 2=1\r\n\r\n\\1-grams:\r\n-0.5 0 -0.25\r\n-0.5   1\r\n\r\n" \
           "\\2-grams:\r\n-0.1  0 1\r\n\r\n\\end\\\r\n"
    toks, lps, bws, skipped = tsd.parse_arpa(text, 2)
    assert skipped == 0
    assert toks[0].tolist() == [[0], [1]] and toks[1].tolist() == [[0, 1]]
    assert lps[1][0] == pytest.approx(-0.1 * np.log(10.0), rel=1e-7)
    assert bws[0][0] == pytest.approx(-0.25 * np.log(10.0), rel=1e-7) and bws[0][1] == 0.0


@pytest.mark.parametrize("text,what", [
    ("ngram 1=1\n\\1-grams:\n-1 0\n", "no header"),
    ("\\data\\\nngram 1=2\n\n\\1-grams:\n-1 0\n\n\\end\\\n", "count mismatch"),
    ("\\data\\\nngram 1=1\n\n\\1-grams:\n-x 0\n\n\\end\\\n", "bad number"),
    ("\\data\\\nngram 1=1\nngram 2=1\n\n\\1-grams:\n-1 0\n\n\\end\\\n", "section missing"),
    ("\\data\\\nngram 1=1\n\n\\1-grams:\n-1 0 1 2 3\n\n\\end\\\n", "field count"),
])
def test_parse_rejects(text, what):
    with pytest.raises(tsd.TsdError):
        tsd.parse_arpa(text, 4)


def test_parse_rejects_repeated_word():
    with pytest.raises(tsd.TsdError):
        tsd.parse_arpa("\\data\\\nngram 1=1\n\n\\1-grams:\n-1 a\n\n\\end\\\n", 2, vocab=["a", "a"])


@pytest.mark.gpu
def test_decoder_from_arpa_matches_oracle_from_arpa():
    """A decoder whose LM is built from an ARPA file decodes like the oracle
    reading the same file (follow mode: states bit-exact, labels where the
    oracle's top-2 gap exceeds 1e-3, fused scores within 1e-4)."""
    import torch

    from tests import parity_util as pu

    w = synth.scaled(synth.WORKLOADS[0], V=64, H=128, B=3, T=30, lm_total=2500, n_phr=8, phr_len=(2, 4))
    a = synth.ngram_lm(w.lm_seed, w.V, 3, w.lm_total, w.zipf)
    vocab = ["w%d" % i for i in range(w.V)]
    text = write_arpa(a, vocab=vocab, extra={1: [(-1.0, "</s>", None), (-99, "<s>", -0.3)],
                                             2: [(-0.5, "<s> w1", None)]})
    ora = oracle.read_arpa(text, w.V, vocab=vocab)
    ph = synth.phrases(w.boost_seed, w.V, w.n_phr, 2, 4, 0.0)
    E, W = synth.joint_weights(w)
    dev = torch.device("cuda", 0)
    lm_gpu = tsd.NGram.from_arpa(text, w.V, vocab=vocab)
    dec = tsd.Decoder(w.V, w.H, torch.from_numpy(W.view(np.int16)).to(dev), torch.from_numpy(E.view(np.int16)).to(dev),
                      lm=lm_gpu, boost=tsd.Boost.from_phrases(w.V, ph, w.bonus),
                      max_symbols=w.max_sym, max_streams=w.B, max_T=w.T)
    slots = [dec.open() for _ in range(w.B)]
    olm = oracle.LM(ora.V, ora.tokens, ora.logp, ora.bow)
    obo = oracle.Boost.from_phrases(w.V, ph, w.bonus)
    model = oracle.Model(w.V, w.H, E, W)
    enc = synth.enc_chunk(w, range(w.B), 0)
    out = dec.decode_chunk(slots, torch.from_numpy(enc.view(np.int16)).to(dev), w.lam, w.beta)
    torch.cuda.synchronize()
    toks, frames, scores, counts = (x.cpu().numpy() for x in (out.tokens, out.frames, out.scores, out.counts))
    for i in range(w.B):
        n = int(counts[i])
        st = oracle.Stream(w.V)
        _, _, _, rep = oracle.decode_chunk(st, model, olm, obo, enc[i], w.lam, w.beta, w.max_sym,
                                           follow=(toks[i, :n], frames[i, :n], scores[i, :n]))
        assert rep[oracle.REP_INCONSISTENT] == 0 and rep[oracle.REP_MISMATCH] == 0, rep
        assert rep[oracle.REP_MAX_SCORE_DIFF] <= pu.SCORE_TOL, rep
        lm_state, _, last = dec.state(slots[i])
        hist = st.history()
        assert lm_gpu.state_tuple(lm_state) == olm.state(hist)  # the longest suffix of the history that is a state
        assert last == (hist[-1] if hist else w.V)
