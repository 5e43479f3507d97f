"""The range-checked build (TSD_CHECKS): the fused row pass checks every
slot, state, arc, label, trie node and dense-row index it follows and
records the first violation in the decoder's status word instead of
following it.  On the tiny workload (config 0, all of its label steps
captured) it must decode with parity and leave the status word clean."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r"""
import os, sys
sys.path.insert(0, os.environ["TSD_ROOT"])
import paper_2609_14991_gb300 as tsd
assert tsd.LIB_PATH.endswith("libtsd_checks.so"), tsd.LIB_PATH
import synth
from tests import parity_util as pu
w = synth.WORKLOADS[0]
inp = pu.Inputs(w)
run = pu.GpuRun(inp, range(w.B), 1, capture_steps=w.T * w.max_sym)  # checks the status word at the end
pu.assert_reports(pu.replay(inp, run, range(w.B)))
print("checked build ok", sum(int(run.chunks[0]["count"][i]) for i in range(w.B)), "labels")
"""


def test_checked_build_decodes_config0_with_parity():
    from paper_2609_14991_gb300 import _build

    lib = _build.build(checks=True)
    env = dict(os.environ, TSD_LIBRARY=lib, TSD_ROOT=ROOT)
    r = subprocess.run([sys.executable, "-c", CHILD], cwd=ROOT, env=env, capture_output=True, text=True,
                       timeout=900)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-4000:]
    assert "checked build ok" in r.stdout
