"""The pins must catch plausible mistakes in the oracle.

Each case plants one mistake in a copy of oracle.cpp (on the CPU, in a
temporary directory), builds it, and runs the pin suite against that build in
a subprocess; the suite must fail.
"""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

MUTATIONS = {
    "backoff weight dropped": ("double b = (j >= 0) ? bow[len - 1][(size_t)j] : 0.0;", "double b = 0.0;"),
    "backoff to the wrong suffix": ("return b + score_ctx(h + 1, len - 1, v);",
                                    "return b + score_ctx(h, len - 1, v);"),
    "W_out read transposed": (
        "const uint16_t* wk = m.W + (size_t)k * N;\n"
        "    for (int32_t v = 0; v < N; ++v) logits[(size_t)v] += xk * (double)bf16_bits_to_float(wk[v]);",
        "for (int32_t v = 0; v < N; ++v) logits[(size_t)v] += "
        "xk * (double)bf16_bits_to_float(m.W[((size_t)v * H + k) % ((size_t)H * N)]);"),
    "blank gets an LM score": ("fused[(size_t)V] = logits[(size_t)V] - lse;\n}",
                               "fused[(size_t)V] = logits[(size_t)V] - lse + "
                               "(lms.n ? lms.score(y, ylen, 0) : 0.0);\n}"),
    "ReLU missing": ("if (s < 0.0f) s = 0.0f;", ""),
    "no restart after a phrase": (
        "if (l > 0 && b->is_phrase(g + (len - l), l)) h.rho = (int64_t)h.y.size();", "(void)l;"),
    "log-softmax sign": ("double f = logits[(size_t)v] - lse;", "double f = logits[(size_t)v] + lse;"),
    "beam without merging": ("if (o.y == h.y) {", "if (false) {"),
    "LM state takes the shortest suffix": ("for (int64_t l = n; l >= 1; --l) {\n      if (find(hist",
                                           "for (int64_t l = 1; l <= n; ++l) {\n      if (find(hist"),
    "only the first LM of several": ("for (int i = 1; i < n; ++i) t += alpha[i] * lm[i]->score(y, len, v);",
                                     "(void)0;"),
    "LM weight ignored": ("double t = alpha[0] * lm[0]->score(y, len, v);", "double t = lm[0]->score(y, len, v);"),
    "pruned set not ranked by the acoustic model": (
        "[&](int32_t a, int32_t b) { return logits[(size_t)a] > logits[(size_t)b]; });",
        "[&](int32_t a, int32_t b) { return fused_rank_bug(a, b); });"),
    "LSTM input and forget gates swapped": (
        "const double i = sigmoid(g[(size_t)4 * u]), f = sigmoid(g[(size_t)4 * u + 1]);",
        "const double f = sigmoid(g[(size_t)4 * u]), i = sigmoid(g[(size_t)4 * u + 1]);"),
    "prediction network advances on blank": (
        "      rep[REP_STEPS] += 1;\n      if (y == V) break;",
        "      rep[REP_STEPS] += 1;\n      if (y == V && pn) lstm_step(*pn, V, s->pred);\n      if (y == V) break;"),
    "S-th label of a frame stays in the frame": ("merge_into((c.tok == V || e == S - 1) ? F : A2, std::move(h));",
                                                  "merge_into((c.tok == V) ? F : A2, std::move(h));"),
    "frame-exit set re-sorted by score": ("    for (size_t i = 0; i < F.size(); ++i)\n      if (keep[i]) F2.push_back(std::move(F[i]));",
                                          "    for (size_t r = 0; r < (size_t)K; ++r) F2.push_back(std::move(F[order[r]]));"),
    "failed match not cancelled": (
        "return bonus * (double)(match(gv.data(), len + 1) - match(g, len));",
        "return bonus * (double)std::max(0, match(gv.data(), len + 1) - match(g, len));"),
}


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_planted_mistake(name, tmp_path):
    src = open(os.path.join(ROOT, "oracle", "oracle.cpp")).read()
    a, b = MUTATIONS[name]
    assert a in src, "mutation anchor not found; update the mutation list"
    cpp = tmp_path / "mutant.cpp"
    cpp.write_text(src.replace(a, b).replace("fused_rank_bug(a, b)", "a < b"))
    so = tmp_path / "mutant.so"
    subprocess.check_call(["g++", "-O1", "-std=c++17", "-ffp-contract=off", "-shared", "-fPIC", str(cpp), "-o",
                           str(so)])
    r = subprocess.run([sys.executable, "-m", "pytest", os.path.join(ROOT, "tests", "test_oracle_pins.py"),
                        os.path.join(ROOT, "tests", "test_oracle_multilm.py"),
                        os.path.join(ROOT, "tests", "test_oracle_pruned.py"),
                        os.path.join(ROOT, "tests", "test_oracle_pred.py"),
                        os.path.join(ROOT, "tests", "test_oracle_beam_multi.py"), "-q", "-x", "-p", "no:cacheprovider"],
                       cwd=ROOT, capture_output=True, text=True,
                       env=dict(os.environ, TSD_ORACLE_LIB=str(so)), timeout=600)
    assert r.returncode != 0, f"pins did not catch: {name}\n{r.stdout[-2000:]}"


# Planted mistakes in copies of the encoder oracle (oracle/encoder.py).
ENCODER_MUTATIONS = {
    "content bias u dropped": ('qu = rnd(q[:, c] + P["pos_u"][c])', 'qu = rnd(q[:, c])'),
    "relative offset sign flipped": ("delta = pos_q[:, None] - pos_k[None, :]",
                                     "delta = pos_k[None, :] - pos_q[:, None]"),
    "sin and cos swapped in the position code": ("r[:, 0::2] = np.sin(ang)\n    r[:, 1::2] = np.cos(ang)",
                                                 "r[:, 0::2] = np.cos(ang)\n    r[:, 1::2] = np.sin(ang)"),
    "attention cache ignored": ("K = np.concatenate([st.k[l], k])", "K = np.concatenate([st.k[l][:0], k])"),
    "attention cache keeps the oldest frames": ("st.k[l] = K[-cfg.left:] if cfg.left > 0 else K[:0]",
                                                "st.k[l] = K[:cfg.left]"),
    "convolution cache not carried": ("st.conv[l] = seq[seq.shape[0] - (K - 1):]", "pass"),
    "convolution taps reversed": ("dw[t] = (P[\"dw_w\"] * seq[t:t + K].T).sum(axis=1) + P[\"dw_b\"]",
                                  "dw[t] = (P[\"dw_w\"][:, ::-1] * seq[t:t + K].T).sum(axis=1) + P[\"dw_b\"]"),
    "GLU halves swapped": ("glu = rnd(y[:, :d] * sigmoid(y[:, d:]))", "glu = rnd(y[:, d:] * sigmoid(y[:, :d]))"),
    "feed-forward half step dropped": ("x = x + 0.5 * _feed_forward(x, *P[\"ln_ff1\"]",
                                       "x = x + 1.0 * _feed_forward(x, *P[\"ln_ff1\"]"),
    "softmax over the head dimension": ("a = rnd(a / a.sum(axis=1, keepdims=True))",
                                        "a = rnd(a / a.sum(axis=0, keepdims=True))"),
    "batch norm shift dropped": ('z = rnd(swish(dw * P["bn_scale"] + P["bn_shift"]))',
                                 'z = rnd(swish(dw * P["bn_scale"]))'),
    "rounding to nearest truncates": ("return np.ldexp(np.rint(np.ldexp(m, 8)), e - 8)",
                                      "return np.ldexp(np.trunc(np.ldexp(m, 8)), e - 8)"),
}


@pytest.mark.parametrize("name", sorted(ENCODER_MUTATIONS))
def test_encoder_pins_catch_planted_mistake(name, tmp_path):
    src = open(os.path.join(ROOT, "oracle", "encoder.py")).read()
    a, b = ENCODER_MUTATIONS[name]
    assert a in src, "mutation anchor not found; update the mutation list"
    mod = tmp_path / "encoder_mutant.py"
    mod.write_text(src.replace(a, b))
    r = subprocess.run([sys.executable, "-m", "pytest", os.path.join(ROOT, "tests", "test_oracle_encoder.py"), "-q",
                        "-x", "-p", "no:cacheprovider"], cwd=ROOT, capture_output=True, text=True,
                       env=dict(os.environ, TSD_ORACLE_ENCODER=str(mod)), timeout=600)
    assert r.returncode != 0, f"pins did not catch: {name}\n{r.stdout[-2000:]}"
