"""Plain CPU oracle of one full per-frame transformer block (numpy, fp64).

TEST INFRASTRUCTURE ONLY (same rule as the rest of ``oracle/``): only
``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import it; it shares no code with the CUDA library.

One decoder layer of a Qwen2-style model processes one frame of T tokens per
stream, with the StateKV attention step of Sec. 3.3 in the middle:

    h  = RMSNorm(x) * g_attn
    qkv = h W_qkv^T + b_qkv
    q, k = RoPE(q, p), RoPE(k, p)     p = L_n + t, the virtual position (Sec. 3.3)
    o  = StateKV attention of (q, k, v)        (the per-layer oracle, Eq. 5 / 6)
    x1 = x + o W_o^T
    h2 = RMSNorm(x1) * g_mlp
    x2 = x1 + (SiLU(h2 W_gate^T) * (h2 W_up^T)) W_down^T

RoPE uses the rotate-half pairing (k, k + d/2) with inverse frequencies
theta^(-2k/d).  The "RoPE scaling" paragraph of Sec. 3.3 fixes one scaling
alpha for cache building and decoding alike; with YaRN (factor s > 1 over a
trained context L) each frequency is blended between interpolation (theta_k / s)
and extrapolation (theta_k) by a ramp over r_k = L / wavelength_k between
r = 1 and r = 32, and q and k are both scaled by 0.1 ln(s) + 1.

Rounding points (where the GPU stores bf16 between kernels) are mirrored:
every quantity written to memory as bf16 on the GPU is rounded to bf16 here
(round to nearest even); the arithmetic between those points is fp64.
Reading: RMSNorm applies its weight before the single bf16 rounding.
"""
from __future__ import annotations

import numpy as np

from . import OracleLayer, bf16_bits_to_f64


def round_bf16(x: np.ndarray) -> np.ndarray:
    """fp64 -> nearest bf16 value (via fp32, ties to even), returned as fp64."""
    f = np.asarray(x, np.float64).astype(np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return bf16_bits_to_f64(u.astype(np.uint16))


def to_bits(x: np.ndarray) -> np.ndarray:
    """fp64 values that are exact in bf16 -> their bf16 bit patterns."""
    f = np.asarray(x, np.float64).astype(np.float32)
    return (f.view(np.uint32) >> 16).astype(np.uint16)


def rms_norm(x: np.ndarray, g: np.ndarray, eps: float) -> np.ndarray:
    """x / sqrt(mean(x^2) + eps) * g over the last axis (fp64)."""
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * g


def silu(x: np.ndarray) -> np.ndarray:
    return x / (1.0 + np.exp(-x))


def rope_frequencies(d: int, theta: float, yarn_factor: float = 1.0,
                     original_max: int = 0) -> tuple[np.ndarray, float]:
    """Per-pair angular frequencies [d/2] and the q/k scale (YaRN's
    0.1 ln(s) + 1; 1 without scaling)."""
    k = np.arange(d // 2, dtype=np.float64)
    freq = theta ** (-2.0 * k / d)
    if yarn_factor <= 1.0:
        return freq, 1.0
    wavelength = 2.0 * np.pi / freq
    r = original_max / wavelength
    alpha, beta = 1.0, 32.0
    ramp = np.clip((r - alpha) / (beta - alpha), 0.0, 1.0)  # 0: interpolate, 1: keep
    freq = (1.0 - ramp) * freq / yarn_factor + ramp * freq
    return freq, 0.1 * np.log(yarn_factor) + 1.0


def rope(x: np.ndarray, positions: np.ndarray, freq: np.ndarray, scale: float) -> np.ndarray:
    """Rotate-half rotary embedding of x [T][H][d] at integer positions [T]."""
    half = x.shape[-1] // 2
    ang = positions.astype(np.float64)[:, None] * freq[None, :]
    cos = np.cos(ang)[:, None, :] * scale
    sin = np.sin(ang)[:, None, :] * scale
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * cos - x2 * sin, x2 * cos + x1 * sin], axis=-1)


class BlockWeights:
    """One layer's weights as fp64 arrays holding bf16 values."""

    def __init__(self, norm_attn, w_qkv, b_qkv, w_o, norm_mlp, w_gate_up, w_down):
        self.norm_attn, self.w_qkv, self.b_qkv, self.w_o = norm_attn, w_qkv, b_qkv, w_o
        self.norm_mlp, self.w_gate_up, self.w_down = norm_mlp, w_gate_up, w_down


class OracleBlock:
    """A stack of layers for one stream: per layer the StateKV oracle state."""

    def __init__(self, n_q, n_kv, d, T, B, max_frames, weights, *, eps=1e-6, theta=1e6,
                 yarn_factor=1.0, original_max=0, policy=0):
        self.n_q, self.n_kv, self.d, self.T = n_q, n_kv, d, T
        self.weights = weights
        self.eps = eps
        self.freq, self.qk_scale = rope_frequencies(d, theta, yarn_factor, original_max)
        self.layers = [OracleLayer(n_q, n_kv, d, T, B, max_frames, policy=policy)
                       for _ in weights]

    def layer_frame(self, l: int, x: np.ndarray) -> tuple[np.ndarray, dict]:
        """One frame through layer l: x [T][hidden] (bf16 values, fp64) -> the
        layer's output (bf16 values) and its intermediates."""
        w = self.weights[l]
        lay = self.layers[l]
        T, n_q, n_kv, d = self.T, self.n_q, self.n_kv, self.d
        pos = lay.virtual_len + np.arange(T)
        h = round_bf16(rms_norm(x, w.norm_attn, self.eps))
        qkv = h @ w.w_qkv.T
        if w.b_qkv is not None:
            qkv = qkv + w.b_qkv
        qkv = round_bf16(qkv)
        q = qkv[:, : n_q * d].reshape(T, n_q, d)
        k = qkv[:, n_q * d: (n_q + n_kv) * d].reshape(T, n_kv, d)
        v = qkv[:, (n_q + n_kv) * d:].reshape(T, n_kv, d)
        q = round_bf16(rope(q, pos, self.freq, self.qk_scale))
        k = round_bf16(rope(k, pos, self.freq, self.qk_scale))
        o, imp, kept = lay.prefill_frame(to_bits(q), to_bits(k), to_bits(v))
        o = round_bf16(o.reshape(T, n_q * d))
        x1 = round_bf16(x + o @ w.w_o.T)
        h2 = round_bf16(rms_norm(x1, w.norm_mlp, self.eps))
        gu = round_bf16(h2 @ w.w_gate_up.T)
        inter = gu.shape[1] // 2
        a = round_bf16(silu(gu[:, :inter]) * gu[:, inter:])
        x2 = round_bf16(x1 + a @ w.w_down.T)
        return x2, {"q": q, "k": k, "v": v, "attn": o, "x1": x1, "act": a, "imp": imp,
                    "kept": kept}

    def frame(self, x: np.ndarray) -> np.ndarray:
        for l in range(len(self.weights)):
            x, _ = self.layer_frame(l, x)
        return x
