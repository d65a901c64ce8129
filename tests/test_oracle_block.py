"""Pins of the full-block oracle (``oracle/block.py``) against the library's
own routines (torch bf16 rounding, rms_norm, silu, scaled_dot_product_attention
in fp64), closed forms and the algebraic properties of rotary embeddings.
"""
import numpy as np
import pytest
import torch

from oracle import block as ob
from oracle import bf16_bits_to_f64


def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.standard_normal(10000) * s for s in (1e-3, 1.0, 300.0)])
    x = x.astype(np.float32).astype(np.float64)  # fp32 values: one rounding step only
    want = torch.as_tensor(x, dtype=torch.float32).to(torch.bfloat16).double().numpy()
    np.testing.assert_array_equal(ob.round_bf16(x), want)
    np.testing.assert_array_equal(bf16_bits_to_f64(ob.to_bits(want)), want)


def test_rms_norm_closed_form_and_library():
    g = np.array([1.0, 2.0, -0.5, 0.25])
    x = np.full((1, 4), 3.0)
    np.testing.assert_allclose(ob.rms_norm(x, g, 0.0), g[None, :])  # constant row -> g
    rng = np.random.default_rng(1)
    x = rng.standard_normal((5, 64))
    gw = rng.standard_normal(64)
    want = torch.nn.functional.rms_norm(torch.as_tensor(x), (64,), torch.as_tensor(gw), eps=1e-6)
    np.testing.assert_allclose(ob.rms_norm(x, gw, 1e-6), want.numpy(), rtol=1e-12)
    # invariant under positive rescaling of the row (eps -> 0)
    np.testing.assert_allclose(ob.rms_norm(7.0 * x, gw, 0.0), ob.rms_norm(x, gw, 0.0), rtol=1e-12)


def test_silu_library_and_identity():
    x = np.linspace(-20, 20, 401)
    np.testing.assert_allclose(ob.silu(x), torch.nn.functional.silu(torch.as_tensor(x)).numpy(),
                               rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(ob.silu(x) - ob.silu(-x), x, atol=1e-12)


def test_rope_properties():
    rng = np.random.default_rng(2)
    d = 16
    freq, scale = ob.rope_frequencies(d, 1e6)
    assert scale == 1.0
    x = rng.standard_normal((3, 2, d))
    # position 0 is the identity
    np.testing.assert_allclose(ob.rope(x, np.zeros(3, int), freq, 1.0), x)
    # a rotation in each (k, k + d/2) plane: pair norms are kept
    y = ob.rope(x, np.array([5, 1000, 123456]), freq, 1.0)
    h = d // 2
    np.testing.assert_allclose(x[..., :h] ** 2 + x[..., h:] ** 2, y[..., :h] ** 2 + y[..., h:] ** 2)
    # scores depend on the relative position only
    q, k = rng.standard_normal((1, 1, d)), rng.standard_normal((1, 1, d))
    for m, n, s in [(7, 3, 100), (0, 50, 999), (12345, 10, 77)]:
        a = np.sum(ob.rope(q, np.array([m]), freq, 1.0) * ob.rope(k, np.array([n]), freq, 1.0))
        b = np.sum(ob.rope(q, np.array([m + s]), freq, 1.0) *
                   ob.rope(k, np.array([n + s]), freq, 1.0))
        assert a == pytest.approx(b, rel=1e-9)
    # hand case d = 2, theta irrelevant (one pair, frequency 1): angle = position
    x2 = np.array([[[1.0, 0.0]]])
    f1, _ = ob.rope_frequencies(2, 10.0)
    np.testing.assert_allclose(ob.rope(x2, np.array([1]), f1, 1.0),
                               [[[np.cos(1.0), np.sin(1.0)]]])


def test_yarn_frequencies():
    d, theta, L, s = 128, 1e6, 32768, 4.0
    plain, _ = ob.rope_frequencies(d, theta)
    f1, m1 = ob.rope_frequencies(d, theta, 1.0, L)
    np.testing.assert_array_equal(f1, plain)  # factor 1: plain RoPE
    assert m1 == 1.0
    f, m = ob.rope_frequencies(d, theta, s, L)
    r = L * plain / (2 * np.pi)  # trained context over wavelength
    np.testing.assert_allclose(f[r < 1.0], plain[r < 1.0] / s)   # long wavelengths: interpolated
    np.testing.assert_allclose(f[r > 32.0], plain[r > 32.0])     # short ones: kept
    assert ((r > 1.0) & (r < 32.0)).any()


def test_yarn_mid_ramp_frequency_hand_value():
    """YaRN's blend at a hand-chosen ramp point (d 4, theta 1e4, s 4).

    Pair 0 has frequency 1 (wavelength 2 pi) and pair 1 frequency
    1e4^(-1/2) = 0.01 (wavelength 200 pi).  With a trained context of
    L = 1750 pi, pair 1 sees r = L / (200 pi) = 8.75, a quarter of the way up
    the ramp from r = 1 to r = 32: gamma = (8.75 - 1) / 31 = 0.25, so its
    frequency is 0.75 * 0.01 / 4 + 0.25 * 0.01 = 0.004375 (the blend's weights
    swapped would give 0.008125).  Pair 0 sees r = 875 > 32 and keeps
    frequency 1.  The q/k factor is 0.1 ln 4 + 1 = 1.138629436111989.
    """
    f, m = ob.rope_frequencies(4, 1e4, 4.0, 1750 * np.pi)
    np.testing.assert_allclose(f, [1.0, 0.004375], rtol=1e-12)
    assert m == pytest.approx(1.138629436111989, rel=1e-14)
    # just below the ramp (r = 0.5 for pair 1): fully interpolated, 0.01 / 4
    f, _ = ob.rope_frequencies(4, 1e4, 4.0, 100 * np.pi)
    np.testing.assert_allclose(f, [1.0, 0.0025], rtol=1e-12)


def test_yarn_factor_scales_both_q_and_k():
    """The attention factor multiplies q and k alike, so the scale of a q.k
    logit grows by (0.1 ln s + 1)^2 = 1.2964769927807063 at s = 4 (a factor
    applied to one of them only would give 1.1386); and the attention of the
    step consumes the scaled q and k.  Checked at position 0, where the rotation is the
    identity for every frequency, against the same layer without scaling."""
    rng = np.random.default_rng(11)
    hidden, inter, n_q, n_kv, d, T = 64, 32, 1, 1, 64, 2
    w = _weights(rng, hidden, inter, n_q, n_kv, d)
    x = ob.round_bf16(rng.standard_normal((T, hidden)))
    plain = ob.OracleBlock(n_q, n_kv, d, T, 8, 2, [w], theta=1e4)
    yarn = ob.OracleBlock(n_q, n_kv, d, T, 8, 2, [w], theta=1e4, yarn_factor=4.0,
                          original_max=64)
    _, a = plain.layer_frame(0, x)
    _, b = yarn.layer_frame(0, x)
    q0a, k0a, q0b, k0b = a["q"][0, 0], a["k"][0, 0], b["q"][0, 0], b["k"][0, 0]
    # each side carries the factor once (bf16 rounding: a few parts in 1e3)
    np.testing.assert_allclose(np.dot(q0b, q0a) / np.dot(q0a, q0a), 1.138629436111989, rtol=8e-3)
    np.testing.assert_allclose(np.dot(k0b, k0a) / np.dot(k0a, k0a), 1.138629436111989, rtol=8e-3)
    # so the logit scale, |q| |k|, grows by the square
    np.testing.assert_allclose(np.linalg.norm(q0b) * np.linalg.norm(k0b) /
                               (np.linalg.norm(q0a) * np.linalg.norm(k0a)), 1.2964769927807063,
                               rtol=8e-3)
    # the step attends with them: key 0's importance is 1 (query 0 sees only
    # it) plus its softmax weight for query 1
    q1, k0, k1 = b["q"][1, 0], b["k"][0, 0], b["k"][1, 0]
    z = np.array([np.dot(q1, k0), np.dot(q1, k1)]) / np.sqrt(d)
    w0 = 1.0 / (1.0 + np.exp(z[1] - z[0]))
    np.testing.assert_allclose(b["imp"][0, 8], 1.0 + w0, rtol=1e-12)
    np.testing.assert_allclose(b["imp"][0, 9], 1.0 - w0, rtol=1e-12)


def _weights(rng, hidden, inter, n_q, n_kv, d, zero_out=False):
    r = lambda *s: ob.round_bf16(rng.standard_normal(s) * 0.08)
    w_o = np.zeros((hidden, n_q * d)) if zero_out else r(hidden, n_q * d)
    w_down = np.zeros((hidden, inter)) if zero_out else r(hidden, inter)
    return ob.BlockWeights(ob.round_bf16(1.0 + 0.1 * rng.standard_normal(hidden)),
                           r((n_q + 2 * n_kv) * d, hidden), r((n_q + 2 * n_kv) * d), w_o,
                           ob.round_bf16(1.0 + 0.1 * rng.standard_normal(hidden)),
                           r(2 * inter, hidden), w_down)


def test_block_with_zero_output_projections_is_the_identity():
    rng = np.random.default_rng(3)
    hidden, inter, n_q, n_kv, d, T = 32, 48, 2, 1, 64, 4
    w = _weights(rng, hidden, inter, n_q, n_kv, d, zero_out=True)
    blk = ob.OracleBlock(n_q, n_kv, d, T, 8, 4, [w, w])
    x = ob.round_bf16(rng.standard_normal((T, hidden)))
    np.testing.assert_array_equal(blk.frame(x), x)


def _torch_layer_frame1(x, w, n_q, n_kv, d, eps, theta):
    """The first frame (empty state: in-frame causal attention) through the
    library's fp64 routines, with bf16 rounding where the GPU stores bf16."""
    F = torch.nn.functional
    bf = lambda t: t.float().to(torch.bfloat16).double()
    T, hidden = x.shape
    X = torch.as_tensor(x)
    h = bf(F.rms_norm(X, (hidden,), torch.as_tensor(w.norm_attn), eps=eps))
    qkv = bf(F.linear(h, torch.as_tensor(w.w_qkv), torch.as_tensor(w.b_qkv)))
    q = qkv[:, : n_q * d].view(T, n_q, d)
    k = qkv[:, n_q * d: (n_q + n_kv) * d].view(T, n_kv, d)
    v = qkv[:, (n_q + n_kv) * d:].view(T, n_kv, d)
    half = d // 2
    inv = theta ** (-torch.arange(half, dtype=torch.float64) * 2.0 / d)
    ang = torch.arange(T, dtype=torch.float64)[:, None] * inv[None, :]
    c, s = torch.cos(ang)[:, None, :], torch.sin(ang)[:, None, :]
    rot = lambda t: torch.cat([t[..., :half] * c - t[..., half:] * s,
                               t[..., half:] * c + t[..., :half] * s], dim=-1)
    q, k = bf(rot(q)), bf(rot(k))
    G = n_q // n_kv
    kk = k.repeat_interleave(G, dim=1).transpose(0, 1)  # [n_q][T][d]
    vv = v.repeat_interleave(G, dim=1).transpose(0, 1)
    o = F.scaled_dot_product_attention(q.transpose(0, 1), kk, vv, is_causal=True)
    o = bf(o.transpose(0, 1).reshape(T, n_q * d))
    x1 = bf(X + F.linear(o, torch.as_tensor(w.w_o)))
    h2 = bf(F.rms_norm(x1, (hidden,), torch.as_tensor(w.norm_mlp), eps=eps))
    gu = bf(F.linear(h2, torch.as_tensor(w.w_gate_up)))
    inter = gu.shape[1] // 2
    a = bf(F.silu(gu[:, :inter]) * gu[:, inter:])
    return bf(x1 + F.linear(a, torch.as_tensor(w.w_down))).numpy()


def test_first_frame_layer_matches_library_composition():
    rng = np.random.default_rng(4)
    hidden, inter, n_q, n_kv, d, T = 64, 96, 4, 2, 64, 6
    w = _weights(rng, hidden, inter, n_q, n_kv, d)
    blk = ob.OracleBlock(n_q, n_kv, d, T, 16, 4, [w], eps=1e-6, theta=1e4)
    x = ob.round_bf16(rng.standard_normal((T, hidden)))
    got, _ = blk.layer_frame(0, x)
    want = _torch_layer_frame1(x, w, n_q, n_kv, d, 1e-6, 1e4)
    # both round at the same points; a rounding tie decided differently moves a
    # value by one bf16 ulp (2^-8 relative), so compare at a few ulps
    np.testing.assert_allclose(got, want, rtol=2 ** -6, atol=2 ** -10)
    assert np.mean(got == want) > 0.95
