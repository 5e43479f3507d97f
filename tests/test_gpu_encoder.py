"""The cache-aware encoder chunk step on the GPU against the oracle.

Tolerance.  Both sides round to bf16 at the same points but reach them
through different sums (tensor-core fp32 vs float64), so a rounding point can
land on either side of a bf16 boundary, and the flip travels on.  Measured
on the oracle itself: perturbing its weights by 3e-7 (relative, the size of
fp32 rounding) moves the bf16 outputs of a 2-block encoder by 0.0024 on
average and at most one output ulp (0.016), and of the 24-block 0.6B-shaped
encoder by 0.0054 on average and at most 0.033.  The GPU is held to four times
the average and twice the maximum; outputs have unit scale.  Where results
must be exact, they are: a stream's output does not depend on the other
streams of the call or on its slot."""
from __future__ import annotations

import numpy as np
import pytest

import synth
from oracle import encoder as oe

pytestmark = pytest.mark.gpu

SMALL = synth.EncoderCfg("small", d=256, layers=2, heads=4, ff=512, kernel=5, left=12, chunk=5, feat=16, stack=4)


def _gpu(w, max_streams, max_chunk=None):
    import paper_2609_14991_gb300 as tsd

    return tsd.Encoder(w, max_streams=max_streams, max_chunk=max_chunk)


def _feats(cfg, streams, first, C):
    import torch

    return torch.from_numpy(synth.features(cfg, streams, first, C).view(np.int16)).cuda()


def _oracle_stream(w, stream, chunks, C):
    cfg = w.cfg
    E, st = oe.Encoder(w), oe.EncoderStream(cfg)
    out = []
    for c in range(chunks):
        out.append(oe.bits_to_f64(oe.encode_chunk(E, st, synth.features(cfg, [stream], c * C, C)[0])))
    return np.stack(out)


def _close(got_bits, want, mean_tol, max_tol):
    got = oe.bits_to_f64(got_bits)
    err = np.abs(got - want)
    assert err.mean() <= mean_tol and err.max() <= max_tol, (err.mean(), err.max())
    return err


@pytest.mark.parametrize("dh", [64, 128])
def test_small_encoder_matches_oracle(dh):
    """Three streams, seven chunks: the attention cache fills (12 frames =
    2.4 chunks), then its ring wraps; the convolution cache carries 4 frames."""
    cfg = synth.EncoderCfg("small", d=256, layers=2, heads=256 // dh, ff=512, kernel=5, left=12, chunk=5, feat=16,
                           stack=4)
    w = synth.encoder_weights(cfg)
    enc = _gpu(w, max_streams=4)
    slots = [enc.open() for _ in range(3)]
    streams = [0, 7, 2]
    got = []
    for c in range(7):
        got.append(enc.encode_chunk(slots, _feats(cfg, streams, c * cfg.chunk, cfg.chunk)).cpu().numpy())
    enc.check()
    got = np.stack(got, axis=1)  # [stream][chunk][C][d]
    for i, s in enumerate(streams):
        _close(got[i].view(np.uint16), _oracle_stream(w, s, 7, cfg.chunk), 0.0095, 0.032)


def test_ragged_chunks_and_zero_left_context():
    """Chunk sizes that change from call to call (one graph per size), a
    chunk of one frame, and an encoder without attention history."""
    for left in (12, 0):
        cfg = synth.EncoderCfg("ragged", d=128, layers=2, heads=2, ff=256, kernel=3, left=left, chunk=4, feat=16,
                               stack=4)
        w = synth.encoder_weights(cfg)
        enc = _gpu(w, max_streams=2, max_chunk=6)
        slot = enc.open()
        E, st = oe.Encoder(w), oe.EncoderStream(cfg)
        first = 0
        for C in (4, 1, 6, 3, 6, 2):
            g = enc.encode_chunk([slot], _feats(cfg, [5], first, C)).cpu().numpy()[0]
            want = oe.bits_to_f64(oe.encode_chunk(E, st, synth.features(cfg, [5], first, C)[0]))
            _close(g.view(np.uint16), want, 0.0095, 0.032)
            first += C


def test_chunk_longer_than_the_left_context():
    """C > left: only the chunk's last `left` frames go into the cache ring."""
    cfg = synth.EncoderCfg("short-left", d=128, layers=2, heads=2, ff=256, kernel=4, left=3, chunk=5, feat=16,
                           stack=4)
    w = synth.encoder_weights(cfg)
    enc = _gpu(w, max_streams=2)
    slots = [enc.open() for _ in range(2)]
    got = np.stack([enc.encode_chunk(slots, _feats(cfg, [4, 9], c * 5, 5)).cpu().numpy() for c in range(4)], axis=1)
    for i, s in enumerate((4, 9)):
        _close(got[i].view(np.uint16), _oracle_stream(w, s, 4, 5), 0.0095, 0.032)


def test_interface_limits():
    """The largest left context (128 frames), chunks of 32 frames and 128-wide
    heads: the attention window and its shared memory at their maximum."""
    cfg = synth.EncoderCfg("limits", d=256, layers=1, heads=2, ff=256, kernel=32, left=128, chunk=32, feat=16,
                           stack=4)
    w = synth.encoder_weights(cfg)
    enc = _gpu(w, max_streams=2)
    slots = [enc.open() for _ in range(2)]
    got = np.stack([enc.encode_chunk(slots, _feats(cfg, [1, 2], c * 32, 32)).cpu().numpy() for c in range(6)],
                   axis=1)
    enc.check()
    for i, s in enumerate((1, 2)):
        _close(got[i].view(np.uint16), _oracle_stream(w, s, 6, 32), 0.0095, 0.032)


def test_0p6b_shape_sampled_streams():
    """The 0.6B-shaped encoder (d 1024, 24 blocks, 8 heads, ff 4096, left 70,
    13-frame chunks) at the bench's launch configuration (256 streams per
    call), two chunks; three streams checked against the oracle."""
    cfg = synth.ENCODERS["0.6b"]
    w = synth.encoder_weights(cfg)
    B = 256
    enc = _gpu(w, max_streams=B)
    slots = [enc.open() for _ in range(B)]
    got = []
    for c in range(2):
        got.append(enc.encode_chunk(slots, _feats(cfg, range(B), c * cfg.chunk, cfg.chunk)).cpu().numpy())
    enc.check()
    got = np.stack(got, axis=1)
    for s in (0, 131, 255):
        _close(got[s].view(np.uint16), _oracle_stream(w, s, 2, cfg.chunk), 0.022, 0.07)


def test_streams_do_not_interact():
    """A stream's output is bit-identical whatever else the call holds and
    whichever slot it sits in."""
    cfg = SMALL
    w = synth.encoder_weights(cfg)
    a_enc, b_enc = _gpu(w, max_streams=6), _gpu(w, max_streams=6)
    a_slots = [a_enc.open() for _ in range(5)]
    b_enc.open()
    b_enc.open()
    b_slot = b_enc.open()  # slot 2, alone in its calls
    for c in range(4):
        a = a_enc.encode_chunk(a_slots, _feats(cfg, [9, 3, 4, 1, 8], c * cfg.chunk, cfg.chunk)).cpu().numpy()
        b = b_enc.encode_chunk([b_slot], _feats(cfg, [4], c * cfg.chunk, cfg.chunk)).cpu().numpy()
        assert np.array_equal(a[2], b[0])


def test_two_branch_split_inside_a_tile():
    """A call of 40 streams x 13 frames (520 rows) runs as two parallel
    halves of 20 streams whose boundary, row 260, falls inside a 128-row
    tile: every stream's output is bit-identical to the same stream encoded
    alone (a single-branch call), and two streams match the oracle."""
    cfg = synth.EncoderCfg("split", d=256, layers=2, heads=4, ff=512, kernel=5, left=12, chunk=13, feat=16, stack=4)
    w = synth.encoder_weights(cfg)
    n = 40
    many, one = _gpu(w, max_streams=n), _gpu(w, max_streams=n)
    m_slots = [many.open() for _ in range(n)]
    o_slots = [one.open() for _ in range(n)]
    got = []
    for c in range(3):
        a = many.encode_chunk(m_slots, _feats(cfg, range(n), c * 13, 13)).cpu().numpy()
        for i in (0, 19, 20, 21, 39):
            b = one.encode_chunk([o_slots[i]], _feats(cfg, [i], c * 13, 13)).cpu().numpy()
            assert np.array_equal(a[i], b[0]), (c, i)
        got.append(a)
    many.check()
    # two branches of (subsampling, the first layer norm, 14 kernels per block), then the frame counts
    assert many.launches_per_chunk(n, 13) == 2 * (2 + 14 * 2) + 1
    assert one.launches_per_chunk(1, 13) == 2 + 14 * 2 + 1
    got = np.stack(got, axis=1)
    for s in (19, 20):
        _close(got[s].view(np.uint16), _oracle_stream(w, s, 3, 13), 0.0095, 0.032)


def test_reopened_slot_starts_fresh():
    cfg = SMALL
    w = synth.encoder_weights(cfg)
    enc = _gpu(w, max_streams=2)
    s = enc.open()
    first = enc.encode_chunk([s], _feats(cfg, [1], 0, cfg.chunk)).cpu().numpy()
    enc.encode_chunk([s], _feats(cfg, [1], cfg.chunk, cfg.chunk))
    enc.close(s)
    s2 = enc.open()
    again = enc.encode_chunk([s2], _feats(cfg, [1], 0, cfg.chunk)).cpu().numpy()
    assert np.array_equal(first, again)


def test_rejections():
    import paper_2609_14991_gb300 as tsd

    w = synth.encoder_weights(SMALL)
    enc = _gpu(w, max_streams=2)
    s = enc.open()
    with pytest.raises(tsd.TsdError):
        enc.encode_chunk([s], _feats(SMALL, [0], 0, SMALL.chunk + 1))  # C > max_chunk
    with pytest.raises(tsd.TsdError):
        enc.encode_chunk([s + 1], _feats(SMALL, [0], 0, SMALL.chunk))  # slot not open
    bad = synth.EncoderCfg("bad", d=192, layers=1, heads=3, ff=256, feat=16, stack=4)
    with pytest.raises(tsd.TsdError):
        _gpu(synth.encoder_weights(bad), max_streams=1)


def test_encoder_output_feeds_the_decoder():
    """The encoder's frames are the decoder's enc input (d = H): one chunk
    through both, decoded labels checked against the oracle decode of the
    same frames."""
    import torch

    import paper_2609_14991_gb300 as tsd
    import oracle

    cfg = synth.EncoderCfg("pipe", d=256, layers=2, heads=4, ff=512, kernel=5, left=12, chunk=13, feat=16, stack=4)
    w = synth.encoder_weights(cfg)
    wl = synth.scaled(synth.WORKLOADS[0], V=256, H=256, B=3, T=13)
    enc = _gpu(w, max_streams=3)
    es = [enc.open() for _ in range(3)]
    frames = enc.encode_chunk(es, _feats(cfg, [0, 1, 2], 0, 13))
    E, W = synth.joint_weights(wl)
    lmA = synth.ngram_lm(wl.lm_seed, wl.V, 3, 5000, wl.zipf)
    dec = tsd.Decoder(wl.V, wl.H, torch.from_numpy(W.view(np.int16)).cuda(), torch.from_numpy(E.view(np.int16)).cuda(),
                      lm=tsd.NGram.from_arrays(lmA), max_streams=3, max_T=13)
    ds = [dec.open() for _ in range(3)]
    out = dec.decode_chunk(ds, frames, wl.lam, 0.0)
    torch.cuda.synchronize()
    t, f, sc, n = (x.cpu().numpy() for x in (out.tokens, out.frames, out.scores, out.counts))
    fr = frames.cpu().numpy().view(np.uint16)
    model, olm = oracle.Model(wl.V, wl.H, E, W), oracle.LM.from_arrays(lmA)
    for i in range(3):
        _, _, _, rep = oracle.decode_chunk(oracle.Stream(wl.V), model, olm, None, fr[i], wl.lam, 0.0, wl.max_sym,
                                           follow=(t[i, :n[i]], f[i, :n[i]], sc[i, :n[i]]))
        assert rep[oracle.REP_INCONSISTENT] == 0 and rep[oracle.REP_MISMATCH] == 0, (i, rep)
        assert rep[oracle.REP_MAX_SCORE_DIFF] <= 1e-4
