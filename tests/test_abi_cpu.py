"""The C-ABI library builds for sm_103a, loads without a GPU, exports every
entry point declared in include/statekv.h, and validates configurations on
the host (no device call is made here)."""
import ctypes
import os
import re

import pytest

from paper_2605_31598_gb300 import build_ext, statekv
from paper_2605_31598_gb300.inputs import WORKLOADS

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    build_ext.build()
    return statekv.lib()


def declared_functions():
    names = set()
    for f in os.listdir(os.path.join(ROOT, "include")):
        if f.endswith(".h"):
            src = open(os.path.join(ROOT, "include", f)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names |= set(re.findall(r"\b(statekv_[a-z_]+)\s*\(", src))
    return sorted(names)


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("statekv_init", "statekv_prefill_frame", "statekv_state_view",
                     "statekv_cache_view"):
        assert required in names


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), f"{name} missing from libstatekv.so"
    assert set(statekv.EXPORTED) <= set(declared_functions())


def test_status_strings(lib):
    for code in range(8):
        assert statekv.statekv_status_string(code)
    assert "unknown" in statekv.statekv_status_string(99)


def _cfg(**kw):
    base = dict(num_streams=1, num_layers=1, num_q_heads=28, num_kv_heads=4, head_dim=128,
                tokens_per_frame=196, state_capacity=1568, max_frames=64, causal_in_frame=1,
                host_staging=0, softmax_scale=0.0, watchdog_ms=0)
    base.update(kw)
    return statekv.statekv_config(**base)


@pytest.mark.parametrize("kw,status", [
    (dict(num_q_heads=30), 1),            # Hq % Hkv != 0
    (dict(head_dim=96), 2),               # not built
    (dict(head_dim=0), 1),
    (dict(tokens_per_frame=0), 1),
    (dict(state_capacity=-1), 1),
    (dict(max_frames=0), 1),
    (dict(causal_in_frame=2), 1),
    (dict(selection=3), 1),               # no such selection policy
    (dict(selection=-1), 1),
    (dict(softmax_scale=-1.0), 1),
    (dict(state_capacity=30000), 2),      # pool beyond the select kernel's limit
    (dict(tokens_per_frame=5000), 2),
    (dict(max_frames=20_000_000, tokens_per_frame=196), 1),  # positions overflow int32
])
def test_bad_configs_rejected_on_host(lib, kw, status):
    n = ctypes.c_size_t(0)
    assert lib.statekv_arena_bytes(ctypes.byref(_cfg(**kw)), ctypes.byref(n)) == status


def test_arena_sizes_cover_states_and_caches(lib):
    for name, shape in WORKLOADS.items():
        cfg = statekv.make_config(shape)
        n = statekv.statekv_arena_bytes(cfg)
        units = shape.num_streams * shape.num_layers * shape.num_kv_heads
        cache = 2 * units * shape.max_frames * shape.tokens_per_frame * shape.head_dim * 2
        state = 2 * units * shape.state_capacity * shape.head_dim * 2
        assert n >= cache + state, name
        assert n % 256 == 0
        staged = statekv.statekv_arena_bytes(statekv.make_config(shape, host_staging=True))
        assert staged > n
    # the 8-stream, 1024-frame decode cache (~92 GB) fits one GB300
    assert statekv.statekv_arena_bytes(statekv.make_config(WORKLOADS["qwen7b_8streams"])) < 200e9


def test_null_arguments_rejected(lib):
    n = ctypes.c_size_t(0)
    assert lib.statekv_arena_bytes(None, ctypes.byref(n)) == 1
    assert lib.statekv_arena_bytes(ctypes.byref(_cfg()), None) == 1
    h = ctypes.c_void_p(0)
    assert lib.statekv_init(ctypes.byref(_cfg()), None, 1 << 30, ctypes.byref(h)) == 1
    assert lib.statekv_prefill_frame(None, None, None) == 1
    assert lib.statekv_prefill_frames_host(None, None, 0, None) == 1
    assert lib.statekv_watchdog_selftest(None, None) == 1
    assert lib.statekv_state_view(None, 0, 0, None) == 1
    assert lib.statekv_cache_view(None, 0, 0, None) == 1
    lib.statekv_destroy(None)


def test_diagnostics_arguments_rejected_on_host(lib):
    """Bad pointers or sizes come back as INVALID_ARG before any launch (the
    dummy addresses below are never dereferenced)."""
    fake = 1 << 20  # 16-byte aligned, never touched
    assert statekv.statekv_topb_mask(0, 1, 10, 16, 4, fake, 0) == 1        # null scores
    assert statekv.statekv_topb_mask(fake, 1, 10, 16, 4, 0, 0) == 1        # null mask
    assert statekv.statekv_topb_mask(fake, 1, 20, 16, 4, fake, 0) == 1     # n > row_stride
    assert statekv.statekv_topb_mask(fake, 1, 10, 16, -1, fake, 0) == 1    # B < 0
    assert statekv.statekv_topb_mask(fake + 2, 1, 10, 16, 4, fake, 0) == 1  # misaligned
    assert statekv.statekv_concentration_sums(fake, fake, 1, 20, 16, fake, 0) == 1
    assert statekv.statekv_concentration_sums(fake, fake, 1, 10, 16, fake + 4, 0) == 1
    assert statekv.statekv_state_metrics(fake, fake, fake, 1, 10, 7, 16, fake, 0) == 1
    assert statekv.statekv_state_metrics(fake, 0, fake, 1, 4, 4, 16, fake, 0) == 1
    assert lib.statekv_full_attention_scores(None, None, None, None, 0, None) == 1
    n = ctypes.c_size_t(0)
    assert lib.statekv_scores_workspace_bytes(None, 1, 1, ctypes.byref(n)) == 1
