"""statekv_full_attention_frame: the exact full self-attention baseline.

The call attends every query of the frame to all earlier tokens (read from
the decode cache) and to the frame's own tokens, and must equal the oracle's
exact attention (``oracle.full_attention``), whose earlier tokens come from
the input generator rather than from the GPU's cache.  It must not change any
state: the StateKV steps that follow still match their own results.
"""
import dataclasses

import numpy as np
import pytest
import torch

import oracle
from paper_2605_31598_gb300 import StateKV, make_config
from paper_2605_31598_gb300.inputs import WORKLOADS, batch_qkv

from .parity import OUT_ATOL


@pytest.mark.gpu
@pytest.mark.parametrize("name,nframes,check,causal,units", [
    ("toy", 8, (1, 2, 5, 8), True, [(0, 0)]),
    ("toy", 5, (3, 5), False, [(0, 0)]),
    # frame 10: 1764 earlier tokens, more than the state's 1568
    ("qwen7b_layer", 10, (1, 10), True, [(0, 0)]),
    # frame 12 of the 28-layer stack: 2156 earlier tokens > B = 2048
    ("qwen7b_stack", 12, (12,), True, [(0, 0), (0, 27)]),
])
def test_full_attention_matches_exact_oracle(name, nframes, check, causal, units):
    import __graft_entry__ as g

    g.build()
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    base = WORKLOADS[name]
    shape = dataclasses.replace(base, max_frames=max(base.max_frames, nframes))
    S, L, T = shape.num_streams, shape.num_layers, shape.tokens_per_frame
    eng = StateKV(make_config(shape, causal=causal))
    hist = {u: ([], []) for u in units}
    for n in range(1, nframes + 1):
        q, k, v = batch_qkv(shape, n, streams=range(S), layers=range(L), device="cuda")
        for u in units:
            hist[u][0].append(oracle.as_bf16_bits(k[u]))
            hist[u][1].append(oracle.as_bf16_bits(v[u]))
        if n in check:
            out = torch.full_like(q, float("nan"))
            assert eng.full_attention_frame(q, k, v, out) == 0
            torch.cuda.synchronize()
            for u in units:
                ref = oracle.full_attention(oracle.as_bf16_bits(q[u]), np.concatenate(hist[u][0]),
                                            np.concatenate(hist[u][1]), (n - 1) * T, causal=causal)
                got = out[u].float().cpu().numpy()
                assert np.isfinite(got).all()
                err = float(np.abs(got - ref).max())
                assert err <= OUT_ATOL, f"frame {n} unit {u}: max |O - O_exact| = {err}"
        assert eng.prefill_frame(q, k, v, torch.empty_like(q)) == 0
    assert eng.sync() == 0


@pytest.mark.gpu
def test_full_attention_changes_no_state_and_refuses_importance():
    import __graft_entry__ as g

    g.build()
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    shape = WORKLOADS["toy"]
    S, L, T, Hkv, B = (shape.num_streams, shape.num_layers, shape.tokens_per_frame,
                       shape.num_kv_heads, shape.state_capacity)
    eng = StateKV(make_config(shape))
    for n in range(1, 4):
        q, k, v = batch_qkv(shape, n, streams=range(S), layers=range(L), device="cuda")
        assert eng.prefill_frame(q, k, v, torch.empty_like(q)) == 0
    torch.cuda.synchronize()
    before = [x.clone() for x in eng.state(0, 0)[:3]] + [eng.cache(0, 0)[0].clone()]
    info_before = eng.state(0, 0)[3]
    q, k, v = batch_qkv(shape, 4, streams=range(S), layers=range(L), device="cuda")
    imp = torch.empty((S, L, Hkv, B + T), device="cuda")
    assert eng.full_attention_frame(q, k, v, torch.empty_like(q)) == 0
    from paper_2605_31598_gb300 import statekv

    args = eng._args(q, k, v, torch.empty_like(q), imp, 0, S, 0, L)
    assert statekv.statekv_full_attention_frame(eng.handle, args, 0) == 1  # INVALID_ARG
    torch.cuda.synchronize()
    after = [x.clone() for x in eng.state(0, 0)[:3]] + [eng.cache(0, 0)[0].clone()]
    info_after = eng.state(0, 0)[3]
    for a, b in zip(before, after):
        assert torch.equal(a, b)
    assert (info_before.count, info_before.virtual_len) == (info_after.count, info_after.virtual_len)
    assert eng.sync() == 0


@pytest.mark.gpu
@pytest.mark.parametrize("name", ["toy", "qwen7b_layer"])
def test_arena_prefilled_with_nan_changes_nothing(name):
    """The arena's prior contents do not matter: every byte 0xFF (bf16 NaN)
    before statekv_init.  Key tiles that run past the valid cache or state
    rows read them, so init must leave them finite; full attention and the
    method's step must match the oracle as on fresh memory."""
    import __graft_entry__ as g

    g.build()
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    shape = dataclasses.replace(WORKLOADS[name], max_frames=5)
    S, L, T = shape.num_streams, shape.num_layers, shape.tokens_per_frame
    cfg = make_config(shape)
    from paper_2605_31598_gb300 import statekv

    arena = torch.full((statekv.statekv_arena_bytes(cfg),), 0xFF, dtype=torch.uint8, device="cuda")
    eng = StateKV(cfg, arena=arena)
    hk, hv = [], []
    for n in range(1, 5):
        q, k, v = batch_qkv(shape, n, streams=range(S), layers=range(L), device="cuda")
        hk.append(oracle.as_bf16_bits(k[0, 0]))
        hv.append(oracle.as_bf16_bits(v[0, 0]))
        out = torch.full_like(q, float("nan"))
        assert eng.full_attention_frame(q, k, v, out) == 0
        torch.cuda.synchronize()
        ref = oracle.full_attention(oracle.as_bf16_bits(q[0, 0]), np.concatenate(hk),
                                    np.concatenate(hv), (n - 1) * T)
        got = out[0, 0].float().cpu().numpy()
        assert np.isfinite(got).all(), f"frame {n}: non-finite output"
        assert float(np.abs(got - ref).max()) <= OUT_ATOL
        step_out = torch.full_like(q, float("nan"))
        assert eng.prefill_frame(q, k, v, step_out) == 0
        torch.cuda.synchronize()
        assert torch.isfinite(step_out.float()).all(), f"frame {n}: non-finite step output"
    assert eng.sync() == 0
