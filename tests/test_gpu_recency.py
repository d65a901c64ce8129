"""The recency-window baseline (selection = 1): the state keeps the B most
recent tokens (the ReKV-style sliding window the paper compares StateKV with).

Checked against the oracle's recency policy on the toy stream (every frame,
untethered: the window is deterministic), and on the 7B layer shape against
exact attention over the window built from the input generator.  The state's
positions and rows must be the window's, bit for bit.
"""
import dataclasses

import numpy as np
import pytest
import torch

import oracle
from paper_2605_31598_gb300 import StateKV, make_config
from paper_2605_31598_gb300.inputs import WORKLOADS, batch_qkv

from .parity import OUT_ATOL


def _check_state(eng, shape, n, hist_k, hist_v, unit=(0, 0)):
    T, B = shape.tokens_per_frame, shape.state_capacity
    kk, vv, pp, info = eng.state(*unit)
    total = n * T
    want = list(range(max(0, total - B), total))
    assert info.count == len(want)
    allk = np.concatenate(hist_k)  # [tokens][Hkv][d]
    allv = np.concatenate(hist_v)
    kb, vb = oracle.as_bf16_bits(kk), oracle.as_bf16_bits(vv)
    pos = pp.cpu().numpy()
    for h in range(shape.num_kv_heads):
        got = pos[h, : info.count]
        assert sorted(got.tolist()) == want
        for slot, ps in enumerate(got):
            assert np.array_equal(kb[h, slot], allk[ps, h])
            assert np.array_equal(vb[h, slot], allv[ps, h])


@pytest.mark.gpu
@pytest.mark.parametrize("B", [32, 40])  # a multiple of T = 16 and not
def test_recency_toy_matches_oracle_every_frame(B):
    import __graft_entry__ as g

    g.build()
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    shape = dataclasses.replace(WORKLOADS["toy"], state_capacity=B)
    T, Hq, Hkv, d = shape.tokens_per_frame, shape.num_q_heads, shape.num_kv_heads, shape.head_dim
    eng = StateKV(make_config(shape, selection=1))
    lay = oracle.OracleLayer(Hq, Hkv, d, T, B, shape.max_frames, policy=1)
    hist_k, hist_v = [], []
    for n in range(1, shape.max_frames + 1):
        q, k, v = batch_qkv(shape, n, streams=[0], layers=[0], device="cuda")
        out = torch.full_like(q, float("nan"))
        assert eng.prefill_frame(q, k, v, out) == 0
        torch.cuda.synchronize()
        qb, kb, vb = (oracle.as_bf16_bits(x[0, 0]) for x in (q, k, v))
        ref, _, _ = lay.prefill_frame(qb, kb, vb)
        err = float(np.abs(out[0, 0].float().cpu().numpy() - ref).max())
        assert err <= OUT_ATOL, f"frame {n}: max |O - O_oracle| = {err}"
        hist_k.append(kb)
        hist_v.append(vb)
        _check_state(eng, shape, n, hist_k, hist_v)
    assert eng.sync() == 0


@pytest.mark.gpu
def test_recency_7b_layer_against_exact_window_attention():
    import __graft_entry__ as g

    g.build()
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    shape = WORKLOADS["qwen7b_layer"]
    T, B = shape.tokens_per_frame, shape.state_capacity
    eng = StateKV(make_config(shape, selection=1))
    hist_k, hist_v = [], []
    for n in range(1, 13):
        q, k, v = batch_qkv(shape, n, streams=[0], layers=[0], device="cuda")
        out = torch.full_like(q, float("nan"))
        assert eng.prefill_frame(q, k, v, out) == 0
        kb, vb = oracle.as_bf16_bits(k[0, 0]), oracle.as_bf16_bits(v[0, 0])
        if n in (1, 9, 12):
            torch.cuda.synchronize()
            w = min(B, (n - 1) * T)
            pk = np.concatenate(hist_k)[(n - 1) * T - w:] if hist_k else kb[:0]
            pv = np.concatenate(hist_v)[(n - 1) * T - w:] if hist_v else vb[:0]
            ref = oracle.full_attention(oracle.as_bf16_bits(q[0, 0]), np.concatenate([pk, kb]),
                                        np.concatenate([pv, vb]), w)
            err = float(np.abs(out[0, 0].float().cpu().numpy() - ref).max())
            assert err <= OUT_ATOL, f"frame {n}: max |O - O_exact| = {err}"
        hist_k.append(kb)
        hist_v.append(vb)
    torch.cuda.synchronize()
    _check_state(eng, shape, 12, hist_k, hist_v)
    # importance is not computed in this mode
    imp = torch.empty((1, 1, shape.num_kv_heads, B + T), device="cuda")
    q, k, v = batch_qkv(shape, 13, streams=[0], layers=[0], device="cuda")
    assert eng.prefill_frame(q, k, v, torch.empty_like(q), imp) == 1
    assert eng.sync() == 0
