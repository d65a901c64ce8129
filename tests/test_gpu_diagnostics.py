"""App. A diagnostics on the GPU against the oracle.

* full-attention layer-level scores: per key within 1e-3 relative (the
  importance tolerance) plus an absolute floor per KV head, the attention
  output within 2e-2, zero past the frame, and the row sum Hq * T;
* top-B masks: bit-exact against the oracle's (score desc, position asc)
  ranking on scores with many ties, including the degenerate budgets;
* concentration and state-metric sums: against the oracle's functions on the
  same (GPU-computed) scores, so that no decision sits in a tolerance band;
* end to end on the toy stream: concentration from GPU scores against the
  oracle's concentration on oracle scores.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2605_31598_gb300 import StateKV, make_config
from paper_2605_31598_gb300 import diagnostics
from paper_2605_31598_gb300.inputs import WORKLOADS, batch_qkv

from .parity import IMP_ATOL, IMP_RTOL, OUT_ATOL


def _need_gpu():
    import __graft_entry__ as g

    g.build()
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _stream_scores(shape, frames, kind=None):
    """Runs the stream through the method (so the decode cache fills) and, at
    each frame in ``frames``, the full-attention scores pass first.  Returns
    {frame: (scores [S][L][cap] fp32 cuda, out, q, k, v)} and the history."""
    eng = StateKV(make_config(shape))
    S, L = shape.num_streams, shape.num_layers
    cap = shape.max_frames * shape.tokens_per_frame
    ws = torch.empty(eng.scores_workspace_bytes(), dtype=torch.uint8, device="cuda")
    got = {}
    hist = []
    for n in range(1, max(frames) + 1):
        q, k, v = batch_qkv(shape, n, streams=range(S), layers=range(L), device="cuda", kind=kind)
        if n in frames:
            scores = torch.full((S, L, cap), float("nan"), device="cuda")
            out = torch.full_like(q, float("nan"))
            assert eng.full_attention_scores(q, k, v, out, scores, ws) == 0
            got[n] = (scores, out, q, k, v)
        assert eng.prefill_frame(q, k, v, torch.empty_like(q)) == 0
        hist.append((k, v))
    torch.cuda.synchronize()
    assert eng.sync() == 0
    return got, hist


def _oracle_scores(shape, got, hist, n, s=0, l=0):
    T = shape.tokens_per_frame
    _, _, q, k, v = got[n]
    kb = np.concatenate([oracle.as_bf16_bits(hk[s, l]) for hk, _ in hist[:n]])
    vb = np.concatenate([oracle.as_bf16_bits(hv[s, l]) for _, hv in hist[:n]])
    return oracle.full_attention(oracle.as_bf16_bits(q[s, l]), kb, vb, (n - 1) * T,
                                 return_scores=True)


@pytest.mark.gpu
@pytest.mark.parametrize("name,frames", [("toy", [1, 2, 5, 8]), ("qwen7b_layer", [1, 9, 12])])
def test_full_attention_scores_match_oracle(name, frames):
    _need_gpu()
    shape = WORKLOADS[name]
    T, Hq, Hkv = shape.tokens_per_frame, shape.num_q_heads, shape.num_kv_heads
    got, hist = _stream_scores(shape, frames)
    for n in frames:
        scores, out, _, _, _ = got[n]
        o_ref, s_ref = _oracle_scores(shape, got, hist, n)
        g = scores[0, 0].double().cpu().numpy()
        keys = n * T
        err = np.abs(g[:keys] - s_ref)
        assert np.all(err <= IMP_RTOL * s_ref + IMP_ATOL * Hkv), f"frame {n}: worst {err.max()}"
        assert np.all(g[keys:] == 0), f"frame {n}: columns past the frame not zero"
        assert abs(g.sum() - Hq * T) <= 1e-4 * Hq * T
        o_err = float(np.abs(out[0, 0].float().cpu().numpy() - o_ref).max())
        assert o_err <= OUT_ATOL, f"frame {n}: max |dO| = {o_err}"


@pytest.mark.gpu
def test_topb_mask_is_the_oracle_ranking_bit_exact():
    _need_gpu()
    rng = np.random.default_rng(3)
    rows, stride, n = 3, 1100, 1000
    # few distinct values: ties everywhere, plus zeros and exact duplicates
    vals = rng.integers(0, 37, size=(rows, stride)).astype(np.float32) / 8.0
    vals[1, ::7] = 0.0
    scores = torch.as_tensor(vals, device="cuda")
    for B in [0, 1, 17, 250, 999, 1000, 2000]:
        mask = diagnostics.topb_mask(scores, n, B).cpu().numpy()
        assert np.all(mask[:, n:] == 0)
        for r in range(rows):
            want = np.zeros(stride, np.uint8)
            if B > 0:
                want[oracle.top_b(vals[r, :n].astype(np.float64), B)] = 1
            assert np.array_equal(mask[r], want), f"row {r} B {B}"
    # an empty row keeps nothing
    assert diagnostics.topb_mask(scores, 0, 5).sum().item() == 0


@pytest.mark.gpu
def test_concentration_and_state_metric_kernels_match_oracle_functions():
    _need_gpu()
    rng = np.random.default_rng(4)
    rows, stride, n_seen, T = 2, 700, 500, 60
    s_n = (rng.random((rows, stride)) ** 3).astype(np.float32)
    s_next = (rng.random((rows, stride)) ** 3).astype(np.float32)
    g_n, g_next = torch.as_tensor(s_n, device="cuda"), torch.as_tensor(s_next, device="cuda")
    budgets = [1, 16, 64, 256, 500, 4096]
    c = diagnostics.concentration(g_n, n_seen, budgets)
    for r in range(rows):
        want = oracle.concentration(s_n[r, :n_seen].astype(np.float64), budgets)
        np.testing.assert_allclose(c[r], want, rtol=1e-12)
    for B in [1, 37, 256, 500, 560, 1000]:
        m = diagnostics.state_metrics(g_n, g_next, n_seen, T, B)
        for r in range(rows):
            want = oracle.state_metrics(s_n[r, :n_seen].astype(np.float64),
                                        s_next[r, :n_seen + T].astype(np.float64), B)
            for key in want:
                assert m[key][r] == pytest.approx(want[key], rel=1e-12), (key, r, B)


@pytest.mark.gpu
def test_concentration_end_to_end_on_the_toy_stream():
    """GPU scores -> GPU concentration, against the oracle's concentration of
    the oracle's scores; the concentration is a continuous function of the
    scores (a swap inside the top-B boundary moves it by the swapped gap), so
    it agrees within the score tolerance."""
    _need_gpu()
    shape = WORKLOADS["toy"]
    T = shape.tokens_per_frame
    frames = [3, 6, 8]
    got, hist = _stream_scores(shape, frames, kind="peaked")
    budgets = [1, 4, 16, 32, 64]
    for n in frames:
        scores = got[n][0][0]  # [L][cap] of stream 0
        c = diagnostics.concentration(scores, (n - 1) * T, budgets)[0]
        _, s_ref = _oracle_scores(shape, got, hist, n)
        want = oracle.concentration(s_ref[: (n - 1) * T], budgets)
        np.testing.assert_allclose(c, want, rtol=2e-3, atol=1e-6)
