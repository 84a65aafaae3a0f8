"""The debug build (device-side index checks on, -DVMLA_DEBUG_CHECKS=1): it
compiles, raises no false alarm on valid inputs, computes bit-for-bit what the
release build computes, and counts the online softmax's output rescales,
which inputs with a dominant key in the last key block must trigger. Each
build runs in a process of its own."""

import os
import subprocess
import sys

import pytest
import torch

pytestmark = pytest.mark.gpu
HERE = os.path.dirname(os.path.abspath(__file__))


def test_debug_build_matches_release_without_false_alarms(tmp_path):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    sys.path.insert(0, os.path.dirname(HERE))
    from paper_2605_30351_gb300 import build

    release = build.build()
    debug = build.build(debug=True)
    outs = {}
    for name, lib in (("release", release), ("debug", debug)):
        path = str(tmp_path / f"{name}.pt")
        r = subprocess.run([sys.executable, os.path.join(HERE, "debug_build_case.py"), lib, path],
                           capture_output=True, text=True, timeout=600)
        assert r.returncode == 0, r.stderr[-3000:]
        outs[name] = torch.load(path)
    assert outs["debug"]["status"] == 0 and outs["release"]["status"] == 0
    # the planted late key makes a third of the rows rescale their output at
    # the last key block: 2 x 160 absorbed rows and 2 x 100 x 12 dense rows
    # (at least; earlier blocks may rescale some rows too)
    assert outs["release"]["rescales"] == -1
    assert outs["debug"]["rescales"] >= 2 * 160 + 2 * 100 * 12, outs["debug"]["rescales"]
    for key, t in outs["release"].items():
        if key not in ("status", "rescales"):
            assert torch.equal(t, outs["debug"][key]), key
