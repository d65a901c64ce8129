"""The debug build of the library (STATEKV_DEBUG_CHECKS=1): bounds checks that
record a fault in the status word instead of trapping, and guard bands after
every arena region that statekv_debug_check compares with their fill.

The debug library runs in a child process (STATEKV_DEBUG=1 selects it when the
binding loads), so this process keeps the release build.  The child checks
that the debug build gives the oracle's results on small cases with no check
firing, then overwrites one guard byte from the host (the arena is caller
memory) and expects the canary fault: no GPU fault is involved.
"""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r'''
import sys
sys.path.insert(0, ROOT)
from paper_2605_31598_gb300 import build_ext
build_ext.build(debug=True)
import torch
from paper_2605_31598_gb300 import statekv
from paper_2605_31598_gb300.inputs import WORKLOADS, Shape
assert statekv.LIB_PATH.endswith("libstatekv_debug.so")
from tests.parity import run_parity

# clean runs: results equal the oracle's, every guard band intact
for shape, n, kind in [(WORKLOADS["toy"], 8, None), (Shape(7, 1, 128, 196, 50, 4), 4, "peaked")]:
    eng = run_parity(shape, n, kind=kind)
    assert eng.debug_check() == 0
    assert eng.sync() == 0, "a debug check fired on a clean run"
    eng.close()

# a guard byte overwritten by the host: the check reports a canary fault
eng = statekv.StateKV(statekv.make_config(WORKLOADS["toy"]))
last = eng.nbytes - 1  # the band after the last region ends the arena
eng.arena[last] = 0
torch.cuda.synchronize()
assert eng.debug_check() == 0
rc = eng.sync()
word = eng.device_error()
assert rc == 7 and (word & 0xFF) == 6, (rc, hex(word))
print("debug build ok: clean runs match the oracle, canary fault reported", hex(word))
'''


@pytest.mark.gpu
def test_debug_build_checks_and_guard_bands():
    import torch

    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    env = dict(os.environ, STATEKV_DEBUG="1")
    r = subprocess.run([sys.executable, "-c", "ROOT = %r\n" % ROOT + CHILD], env=env, cwd=ROOT,
                       capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-3000:]
    assert "debug build ok" in r.stdout
    print(r.stdout.strip().splitlines()[-1])
    # this process runs the release build, which refuses the check
    from paper_2605_31598_gb300 import StateKV, make_config
    from paper_2605_31598_gb300.inputs import WORKLOADS

    eng = StateKV(make_config(WORKLOADS["toy"]))
    assert eng.debug_check() == 2  # STATEKV_ERR_UNSUPPORTED
    assert eng.sync() == 0


def test_release_build_exports_the_check():
    """The release library exports statekv_debug_check (a null handle is refused)."""
    from paper_2605_31598_gb300 import build_ext, statekv

    build_ext.build()
    assert statekv.lib().statekv_debug_check(None, None) == 1  # STATEKV_ERR_INVALID_ARG


def test_debug_build_compiles():
    """nvcc builds the debug library (no GPU needed)."""
    from paper_2605_31598_gb300 import build_ext

    path = build_ext.build(debug=True)
    assert os.path.exists(path) and path.endswith("libstatekv_debug.so")
