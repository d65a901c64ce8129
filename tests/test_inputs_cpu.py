"""The synthetic input recipe, checked on CPU.

The recipe stands in for the paper's videos (Sec. 4): seeded N(0, 1) draws,
per-frame salient or boosted key tokens, and rotary embeddings applied at the
virtual positions of Sec. 3.3.  These tests re-draw the raw generators and
check each stated property of what the generator returns: the boost count
and factor, the rotation angle of every rotary pair, the variance, the
per-(stream, layer, frame) seeding and the call layout.
"""
import math

import numpy as np
import pytest
import torch

from paper_2605_31598_gb300 import inputs
from paper_2605_31598_gb300.inputs import ROPE_THETA, WORKLOADS, batch_qkv, frame_qkv


def raw(shape, frame, tag, n_heads, *, layer=0, stream=0, seed=0):
    """The unscaled N(0, 1) draw behind one tensor (same generator as the recipe)."""
    g = inputs._gen("cpu", seed, stream, layer, frame, tag)
    T, d = shape.tokens_per_frame, shape.head_dim
    return torch.randn((T, n_heads, d), generator=g, dtype=torch.float32)


def test_toy_salient_keys_and_no_rotation():
    shape = WORKLOADS["toy"]
    T = shape.tokens_per_frame
    for frame in (1, 3):
        q, k, v = frame_qkv(shape, frame)
        rq, rk, rv = (raw(shape, frame, t, h) for t, h in
                      (("q", shape.num_q_heads), ("k", shape.num_kv_heads), ("v", shape.num_kv_heads)))
        # no rotary embedding: Q and V are the raw draws rounded to bf16
        assert torch.equal(q, rq.to(torch.bfloat16))
        assert torch.equal(v, rv.to(torch.bfloat16))
        scale = torch.ones(T)
        scale[[0, T // 2]] = 4.0  # tokens 0 and T/2 of every frame
        assert torch.equal(k, (rk * scale[:, None, None]).to(torch.bfloat16))


@pytest.mark.parametrize("kind", ["qwen", "peaked"])
def test_boosted_keys_count_factor_and_rotation(kind):
    shape = WORKLOADS["qwen7b_layer"]
    T, Hkv, d = shape.tokens_per_frame, shape.num_kv_heads, shape.head_dim
    frame = 5
    sigma = d ** -0.5 if kind == "qwen" else 1.0
    q, k, v = frame_qkv(shape, frame, layer=2, kind=kind)
    rk = raw(shape, frame, "k", Hkv, layer=2) * sigma
    half = d // 2
    # Rotation preserves the norm of every pair (i, i + d/2), so the per-token
    # ratio of norms reads the boost factor back: round(0.05 T) tokens x3 per KV head.
    kk = k.float()
    pair_norm = torch.sqrt(kk[..., :half] ** 2 + kk[..., half:] ** 2)
    raw_norm = torch.sqrt(rk[..., :half] ** 2 + rk[..., half:] ** 2)
    ratio = (pair_norm.norm(dim=-1) / raw_norm.norm(dim=-1)).t()  # [Hkv][T]
    boosted = ratio > 2.0
    assert torch.all(boosted.sum(dim=1) == round(0.05 * T))
    assert torch.allclose(ratio[boosted], torch.full_like(ratio[boosted], 3.0), rtol=1e-2)
    assert torch.allclose(ratio[~boosted], torch.ones_like(ratio[~boosted]), rtol=1e-2)
    # different KV heads draw different token sets
    assert len({tuple(torch.nonzero(boosted[h]).flatten().tolist()) for h in range(Hkv)}) > 1
    # every pair of Q is rotated by (virtual position) * theta^(-2i/d)
    rq = raw(shape, frame, "q", shape.num_q_heads, layer=2) * sigma
    qq = q.float()
    pos = (frame - 1) * T + torch.arange(T, dtype=torch.float64)
    inv = ROPE_THETA ** (-2.0 * torch.arange(half, dtype=torch.float64) / d)
    want = torch.remainder(pos[:, None] * inv[None, :], 2 * math.pi)  # [T][half]
    got = torch.atan2(qq[..., half:], qq[..., :half]) - torch.atan2(rq[..., half:], rq[..., :half])
    diff = torch.remainder(got.double() - want[:, None, :] + math.pi, 2 * math.pi) - math.pi
    big = torch.sqrt(rq[..., :half] ** 2 + rq[..., half:] ** 2) > 0.3 * sigma  # angle well defined
    assert diff[big].abs().max() < 0.05
    # V is not rotated or boosted
    rv = raw(shape, frame, "v", Hkv, layer=2) * sigma
    assert torch.equal(v, rv.to(torch.bfloat16))


def test_qwen_scale_is_one_over_sqrt_head_dim():
    shape = WORKLOADS["qwen7b_layer"]
    q, _, v = frame_qkv(shape, 2)
    target = shape.head_dim ** -0.5
    assert abs(q.float().std().item() / target - 1.0) < 0.02
    assert abs(v.float().std().item() / target - 1.0) < 0.02


def test_seeding_per_stream_layer_frame():
    shape = WORKLOADS["qwen7b_layer"]
    a = frame_qkv(shape, 3, layer=1, stream=0)
    assert all(torch.equal(x, y) for x, y in zip(a, frame_qkv(shape, 3, layer=1, stream=0)))
    for other in (dict(layer=2, stream=0), dict(layer=1, stream=1)):
        b = frame_qkv(shape, 3, **other)
        assert not torch.equal(a[0], b[0])
    assert not torch.equal(a[1], frame_qkv(shape, 4, layer=1)[1])
    assert not torch.equal(a[2], frame_qkv(shape, 3, layer=1, seed=1)[2])


def test_batch_layout_matches_single_frames():
    shape = WORKLOADS["toy"]
    q, k, v = batch_qkv(shape, [2, 5], streams=[0, 3], layers=[1, 4])
    assert q.shape == (2, 2, shape.tokens_per_frame, shape.num_q_heads, shape.head_dim)
    assert k.shape == (2, 2, shape.tokens_per_frame, shape.num_kv_heads, shape.head_dim)
    for si, (s, f) in enumerate(zip([0, 3], [2, 5])):
        for li, l in enumerate([1, 4]):
            q1, k1, v1 = frame_qkv(shape, f, layer=l, stream=s)
            assert torch.equal(q[si, li], q1) and torch.equal(k[si, li], k1) and torch.equal(v[si, li], v1)


def test_workload_shapes_follow_the_configs():
    w = WORKLOADS
    assert (w["toy"].num_q_heads, w["toy"].num_kv_heads, w["toy"].head_dim,
            w["toy"].tokens_per_frame, w["toy"].state_capacity, w["toy"].max_frames) == (4, 1, 64, 16, 32, 8)
    for name in ("qwen7b_layer", "qwen7b_stack", "qwen7b_8streams"):
        s = w[name]
        assert (s.num_q_heads, s.num_kv_heads, s.head_dim, s.tokens_per_frame) == (28, 4, 128, 196)
    assert (w["qwen7b_layer"].state_capacity, w["qwen7b_layer"].max_frames) == (1568, 64)
    assert (w["qwen7b_stack"].num_layers, w["qwen7b_stack"].state_capacity,
            w["qwen7b_stack"].max_frames) == (28, 2048, 256)
    s = w["qwen72b_stack"]
    assert (s.num_layers, s.num_q_heads, s.num_kv_heads, s.state_capacity, s.max_frames) == (80, 64, 8, 4096, 512)
    s = w["qwen7b_8streams"]
    assert (s.num_streams, s.num_layers, s.state_capacity, s.max_frames) == (8, 28, 2048, 1024)
