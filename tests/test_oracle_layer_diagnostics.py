"""Pins of the oracle's layer-level selection (policy 2) and of the App. A
assumption diagnostics (concentration, candidate-pool recall, weighted
recall, retention, churn).

References are independent of the oracle's code: attention weights read back
from the library's scaled_dot_product_attention (fp64, identity values),
closed forms at Q = 0 and hand-computed sets.
"""
import numpy as np
import pytest
import torch

import oracle
from oracle import OracleLayer, bf16_bits_to_f64


def bits(x):
    t = torch.as_tensor(np.asarray(x, np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16).copy()


def sdpa_layer_scores(q_bits, k_bits, n_prefix, causal, scale):
    """App. A's layer-level score through the library routine: per query head,
    the attention weights summed over the frame's queries; then summed over
    all heads.  q [T][n_q][d], k [n_prefix + T][n_kv][d] bf16 bits."""
    F = torch.nn.functional
    q = bf16_bits_to_f64(q_bits)
    k = bf16_bits_to_f64(k_bits)
    T, n_q, d = q.shape
    n_keys, n_kv = k.shape[0], k.shape[1]
    G = n_q // n_kv
    mask = np.ones((T, n_keys), bool)
    if causal:
        mask[:, n_prefix:] = np.tril(np.ones((T, T), bool))
    m = torch.as_tensor(mask)[None, None]
    eye = torch.eye(n_keys, dtype=torch.float64)[None, None]
    total = np.zeros(n_keys)
    for h in range(n_q):
        qt = torch.as_tensor(q[:, h, :])[None, None]
        kt = torch.as_tensor(k[:, h // G, :])[None, None]
        A = F.scaled_dot_product_attention(qt, kt, eye, attn_mask=m, scale=scale)[0, 0]
        total += A.numpy().sum(axis=0)
    return total


@pytest.mark.parametrize("causal", [True, False])
def test_layer_scores_match_library_attention(causal):
    rng = np.random.default_rng(11)
    T, n_q, n_kv, d, n_prefix = 5, 6, 2, 16, 9
    q = bits(rng.standard_normal((T, n_q, d)))
    k = bits(rng.standard_normal((n_prefix + T, n_kv, d)))
    v = bits(rng.standard_normal((n_prefix + T, n_kv, d)))
    scale = 1.0 / np.sqrt(d)
    _, scores = oracle.full_attention(q, k, v, n_prefix, causal=causal, scale=scale,
                                      return_scores=True)
    ref = sdpa_layer_scores(q, k, n_prefix, causal, scale)
    np.testing.assert_allclose(scores, ref, rtol=1e-12, atol=1e-13)
    # every query row of every head sums to one
    assert abs(scores.sum() - n_q * T) < 1e-10


def test_layer_level_selection_is_the_top_b_of_the_layer_score():
    """Two frames with B = T + 2: the first frame is kept whole, so at the
    second frame the state is the whole history and the method's attention is
    the full attention.  The layer-level policy keeps the top B of the
    library-computed layer score over all 2T tokens, for every KV head, while
    the per-head policy is free to differ between heads."""
    rng = np.random.default_rng(5)
    T, n_q, n_kv, d = 6, 4, 2, 16
    B = T + 2
    scale = 1.0 / np.sqrt(d)
    frames = [(bits(rng.standard_normal((T, n_q, d)) * 2.0),
               bits(rng.standard_normal((T, n_kv, d)) * 2.0),
               bits(rng.standard_normal((T, n_kv, d)))) for _ in range(2)]
    shared = OracleLayer(n_q, n_kv, d, T, B, max_frames=4, scale=scale, policy=2)
    per_head = OracleLayer(n_q, n_kv, d, T, B, max_frames=4, scale=scale, policy=0)
    for q, k, v in frames:
        shared.prefill_frame(q, k, v)
        per_head.prefill_frame(q, k, v)
    k_all = np.concatenate([frames[0][1], frames[1][1]])
    ref = sdpa_layer_scores(frames[1][0], k_all, T, True, scale)
    order = np.lexsort((np.arange(2 * T), -ref))
    expect = np.sort(order[:B])
    for h in range(n_kv):
        np.testing.assert_array_equal(shared.state_positions(h), expect)
    # the inputs are chosen so that the per-head rankings disagree with it
    assert any(not np.array_equal(per_head.state_positions(h), expect) for h in range(n_kv))


def test_layer_level_selection_requires_agreeing_heads():
    T, n_q, n_kv, d, B = 2, 2, 2, 4, 2
    layer = OracleLayer(n_q, n_kv, d, T, B, max_frames=4, policy=2)
    count = np.array([2, 2], np.int32)
    pos = np.array([[0, 1], [0, 2]], np.int64)
    z = np.zeros((n_kv, B, d), np.uint16)
    layer.set_state(count, pos, z, z, 4)
    with pytest.raises(RuntimeError):
        layer.prefill_frame(np.zeros((T, n_q, d), np.uint16), np.zeros((T, n_kv, d), np.uint16),
                            np.zeros((T, n_kv, d), np.uint16))


def test_concentration_at_zero_queries_is_budget_over_history():
    """Q = 0: every visible key gets the same weight in each query row, so all
    historical keys score alike and C_{n,B} = min(B, |H|) / |H| (App. A.1)."""
    T, n_q, n_kv, d, n_prefix = 4, 2, 1, 8, 12
    rng = np.random.default_rng(2)
    q = np.zeros((T, n_q, d), np.uint16)
    k = bits(rng.standard_normal((n_prefix + T, n_kv, d)))
    v = bits(rng.standard_normal((n_prefix + T, n_kv, d)))
    _, scores = oracle.full_attention(q, k, v, n_prefix, return_scores=True)
    # closed form of one historical key: sum over heads and queries of 1 / visible
    per_key = n_q * sum(1.0 / (n_prefix + i + 1) for i in range(T))
    np.testing.assert_allclose(scores[:n_prefix], per_key, rtol=1e-12)
    budgets = [1, 3, 12, 20]
    c = oracle.concentration(scores[:n_prefix], budgets)
    np.testing.assert_allclose(c, [1 / 12, 3 / 12, 1.0, 1.0], rtol=1e-12)


def test_concentration_hand_example():
    s = np.array([0.1, 0.5, 0.2, 0.2])
    # top-1 {1}: 0.5 / 1.0; top-2 {1, 2} (0.2 tie, lower position): 0.7; top-3: 0.9
    np.testing.assert_allclose(oracle.concentration(s, [1, 2, 3, 4]), [0.5, 0.7, 0.9, 1.0])
    np.testing.assert_array_equal(oracle.top_b(s, 2), [1, 2])


def test_state_metrics_hand_example():
    """Frame n has seen 6 tokens, frame n + 1 adds positions 6..8 (App. A.2).
    S_n = top-3 of scores_n = {0, 2, 5}; S_{n+1} = top-3 of scores_next =
    {2, 4, 7}; pool P = S_n + {6, 7, 8} = {0, 2, 5, 6, 7, 8}.
      recall   |{2, 7}| / 3 = 2/3
      weighted (0.3 + 0.25) / (0.3 + 0.35 + 0.25) = 0.55 / 0.9
      retention |{2}| / 3 = 1/3;  churn |{4, 7}| / 3 = 2/3."""
    scores_n = np.array([0.9, 0.1, 0.8, 0.05, 0.2, 0.7])
    scores_next = np.array([0.01, 0.02, 0.3, 0.03, 0.35, 0.04, 0.0, 0.25, 0.0])
    m = oracle.state_metrics(scores_n, scores_next, 3)
    assert m["recall"] == pytest.approx(2 / 3)
    assert m["weighted_recall"] == pytest.approx(0.55 / 0.9)
    assert m["retention"] == pytest.approx(1 / 3)
    assert m["churn"] == pytest.approx(2 / 3)


def test_state_metrics_identities_on_generated_scores():
    """With both states full (B <= tokens seen): retention + churn = 1.  A
    budget covering every token keeps everything: recall 1, retention 1, and
    the churn is the new frame's share."""
    rng = np.random.default_rng(9)
    for _ in range(20):
        n_seen, T = int(rng.integers(5, 40)), int(rng.integers(1, 8))
        s_n = rng.random(n_seen)
        s_next = rng.random(n_seen + T)
        B = int(rng.integers(1, n_seen + 1))
        m = oracle.state_metrics(s_n, s_next, B)
        assert m["retention"] + m["churn"] == pytest.approx(1.0)
        assert 0.0 <= m["recall"] <= 1.0 and 0.0 <= m["weighted_recall"] <= 1.0 + 1e-12
        full = oracle.state_metrics(s_n, s_next, n_seen + T)
        assert full["recall"] == 1.0 and full["weighted_recall"] == pytest.approx(1.0)
        assert full["retention"] == 1.0 and full["churn"] == pytest.approx(T / (n_seen + T))
