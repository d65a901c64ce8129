"""Failure detection on the GPU with a wait that runs out, not a fault.

The watchdog self-test makes the attention kernel's producer wait on a
barrier that nothing completes.  The wait is bounded by the handle's
watchdog: it expires, the kernel records DEVICE_TIMEOUT with the waiting site
in the mapped status word, every warp leaves through its own bounded wait,
and the launch completes.  The handle then reports the error on every call
(sticky), while the CUDA context stays usable for other handles.
"""
import time

import pytest
import torch

from paper_2605_31598_gb300 import StateKV, make_config
from paper_2605_31598_gb300.inputs import WORKLOADS, batch_qkv

pytestmark = pytest.mark.gpu

DEVICE_TIMEOUT = 5  # STATEKV_ERR_DEVICE_TIMEOUT


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__ as g

    g.build()
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def test_expired_wait_is_reported_and_the_context_survives():
    shape = WORKLOADS["toy"]
    eng = StateKV(make_config(shape, watchdog_ms=100))
    t0 = time.monotonic()
    assert eng.watchdog_selftest() == 0
    assert eng.sync() == DEVICE_TIMEOUT
    elapsed = time.monotonic() - t0
    code = eng.device_error()
    assert code & 0xFF == 1, hex(code)  # an attention-kernel wait expired
    assert (code >> 8) & 0xFF == 1, hex(code)  # the self-test's barrier was the first
    assert elapsed < 10.0  # a 100 ms watchdog: the launch ends by itself
    # sticky: the handle refuses further work
    q, k, v = batch_qkv(shape, 1, streams=[0], layers=[0], device="cuda")
    assert eng.prefill_frame(q, k, v, torch.empty_like(q)) == DEVICE_TIMEOUT
    # the context is still usable: a fresh handle runs a frame
    fresh = StateKV(make_config(shape))
    out = torch.full_like(q, float("nan"))
    assert fresh.prefill_frame(q, k, v, out) == 0
    assert fresh.sync() == 0
    assert torch.isfinite(out.float()).all()
