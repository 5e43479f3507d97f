"""Writes ARPA text from per-order n-gram arrays (test helper: both the
oracle's reader and the library's reader are checked against files it
writes)."""
from __future__ import annotations

import math


def write_arpa(a, vocab=None, extra=None, digits: int = 9) -> str:
    """ARPA text of arrays a (natural log, as synth.ngram_lm returns), with
    log10 values printed to `digits` significant digits.  extra: optional
    {order: [(log10 p, "w1 w2 ...", log10 bow or None)]} lines appended to
    their sections (and counted in the header), e.g. sentence markers."""
    extra = extra or {}
    name = (lambda t: vocab[t]) if vocab is not None else (lambda t: str(int(t)))
    ln10 = math.log(10.0)
    out = ["\\data\\"]
    for k in range(1, a.order + 1):
        out.append("ngram %d=%d" % (k, len(a.logp[k - 1]) + len(extra.get(k, []))))
    out.append("")
    for k in range(1, a.order + 1):
        out.append("\\%d-grams:" % k)
        toks, lp, bw = a.tokens[k - 1], a.logp[k - 1], a.bow[k - 1]
        for i in range(len(lp)):
            words = " ".join(name(t) for t in toks[i])
            line = "%.*g\t%s" % (digits, float(lp[i]) / ln10, words)
            if k < a.order and float(bw[i]) != 0.0:
                line += "\t%.*g" % (digits, float(bw[i]) / ln10)
            out.append(line)
        for p10, words, b10 in extra.get(k, []):
            out.append("%.*g\t%s" % (digits, p10, words) + ("" if b10 is None else "\t%.*g" % (digits, b10)))
        out.append("")
    out.append("\\end\\")
    return "\n".join(out) + "\n"
