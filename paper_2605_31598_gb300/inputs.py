"""Seeded synthetic video-token inputs for the per-frame prefill step.

This module only draws inputs; it holds none of the method's arithmetic and is
the one module that both the CUDA path's tests and the CPU oracle consume.
The paper's workloads are real videos through InternVL3 / Qwen / Eagle
backbones (Sec. 4); no dataset or weights are used here.  Synthetic Q/K/V of
the same shapes stand in for them:

* ``toy``    Q/K/V ~ N(0, 1) drawn in fp32, two fixed salient key tokens per
             frame (tokens 0 and T/2) scaled x4, no rotary embedding; cast to
             bf16 for both sides.
* ``qwen``   Q/K/V ~ N(0, 1) / sqrt(head_dim); round(0.05 T) key tokens per
             (stream, layer, frame, KV head), drawn without replacement, scaled
             x3; then rotary embedding (rotate-half pairs (i, i + d/2),
             inv_freq_i = theta^(-2i/d), theta = 1e6) at the virtual position
             (frame - 1) * T + t of each token; bf16.
* ``peaked`` as ``qwen`` with unit-variance Q/K/V (attention far from
             uniform, so many frame tokens win a state slot every frame).

Every tensor is drawn from its own generator seeded by
(seed, stream, layer, frame, tag), so a frame's inputs do not depend on how
many layers or streams are generated together.
"""
from __future__ import annotations

import hashlib
from dataclasses import dataclass

import torch

ROPE_THETA = 1.0e6


@dataclass(frozen=True)
class Shape:
    """Per-layer shapes of the cache-builder step."""

    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    tokens_per_frame: int
    state_capacity: int
    max_frames: int
    num_layers: int = 1
    num_streams: int = 1
    kind: str = "qwen"

    @property
    def group(self) -> int:
        return self.num_q_heads // self.num_kv_heads


# The five workloads: toy, one Qwen2-7B layer, the 28-layer 7B stack, the
# 80-layer 72B stack, and eight concurrent 7B streams.
WORKLOADS = {
    "toy": Shape(4, 1, 64, 16, 32, 8, kind="toy"),
    "qwen7b_layer": Shape(28, 4, 128, 196, 1568, 64),
    "qwen7b_stack": Shape(28, 4, 128, 196, 2048, 256, num_layers=28),
    "qwen72b_stack": Shape(64, 8, 128, 196, 4096, 512, num_layers=80),
    "qwen7b_8streams": Shape(28, 4, 128, 196, 2048, 1024, num_layers=28, num_streams=8),
}


def _seed(seed: int, stream: int, layer: int, frame: int, tag: str) -> int:
    h = hashlib.blake2b(f"{seed}/{stream}/{layer}/{frame}/{tag}".encode(), digest_size=8)
    return int.from_bytes(h.digest(), "little") & ((1 << 63) - 1)


def _gen(device, seed, stream, layer, frame, tag) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(_seed(seed, stream, layer, frame, tag))
    return g


def _rotary(x: torch.Tensor, positions: torch.Tensor, theta: float) -> torch.Tensor:
    """Rotate-half rotary embedding of x [T][H][d] (fp32) at the given positions."""
    d = x.shape[-1]
    half = d // 2
    i = torch.arange(half, device=x.device, dtype=torch.float64)
    inv_freq = theta ** (-2.0 * i / d)
    ang = positions.to(torch.float64)[:, None] * inv_freq[None, :]
    cos = torch.cos(ang).to(torch.float32)[:, None, :]
    sin = torch.sin(ang).to(torch.float32)[:, None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return torch.cat([x1 * cos - x2 * sin, x2 * cos + x1 * sin], dim=-1)


def frame_qkv(shape: Shape, frame: int, *, layer: int = 0, stream: int = 0, seed: int = 0,
              device="cpu", kind: str | None = None):
    """Q [T][Hq][d], K [T][Hkv][d], V [T][Hkv][d] (bf16) of frame ``frame`` (1-based)."""
    kind = kind or shape.kind
    T, Hq, Hkv, d = shape.tokens_per_frame, shape.num_q_heads, shape.num_kv_heads, shape.head_dim
    args = (device, seed, stream, layer, frame)
    q = torch.randn((T, Hq, d), generator=_gen(*args, "q"), device=device, dtype=torch.float32)
    k = torch.randn((T, Hkv, d), generator=_gen(*args, "k"), device=device, dtype=torch.float32)
    v = torch.randn((T, Hkv, d), generator=_gen(*args, "v"), device=device, dtype=torch.float32)
    if kind == "toy":
        salient = torch.tensor([0, T // 2], device=device)
        k[salient] *= 4.0
    elif kind in ("qwen", "peaked"):
        if kind == "qwen":
            sigma = d ** -0.5
            q, k, v = q * sigma, k * sigma, v * sigma
        nboost = int(round(0.05 * T))
        if nboost > 0:
            u = torch.rand((Hkv, T), generator=_gen(*args, "boost"), device=device)
            idx = torch.argsort(u, dim=1)[:, :nboost]  # nboost distinct tokens per KV head
            mult = torch.ones((Hkv, T), device=device)
            mult.scatter_(1, idx, 3.0)
            k = k * mult.t()[:, :, None]
        positions = (frame - 1) * T + torch.arange(T, device=device)
        q = _rotary(q, positions, ROPE_THETA)
        k = _rotary(k, positions, ROPE_THETA)
    else:
        raise ValueError(f"unknown input kind {kind!r}")
    return (q.to(torch.bfloat16).contiguous(), k.to(torch.bfloat16).contiguous(),
            v.to(torch.bfloat16).contiguous())


def batch_qkv(shape: Shape, frame: int, *, streams, layers, seed: int = 0, device="cpu",
              kind: str | None = None):
    """Inputs of one frame for several (stream, layer) units, in the call layout
    [streams][layers][T][H][d] that ``statekv_prefill_frame`` reads.

    ``frame`` may be an int (same frame index for every stream) or a sequence
    with one frame index per stream.
    """
    streams = list(streams)
    layers = list(layers)
    frames = frame if isinstance(frame, (list, tuple)) else [frame] * len(streams)
    qs, ks, vs = [], [], []
    for s, f in zip(streams, frames):
        for l in layers:
            q, k, v = frame_qkv(shape, f, layer=l, stream=s, seed=seed, device=device, kind=kind)
            qs.append(q)
            ks.append(k)
            vs.append(v)
    S, L = len(streams), len(layers)
    T, Hq, Hkv, d = shape.tokens_per_frame, shape.num_q_heads, shape.num_kv_heads, shape.head_dim
    return (torch.stack(qs).view(S, L, T, Hq, d), torch.stack(ks).view(S, L, T, Hkv, d),
            torch.stack(vs).view(S, L, T, Hkv, d))


# ------------------------------------------------------------ transformer block
@dataclass(frozen=True)
class BlockShape:
    """Widths of the decoder layer around the StateKV step (Qwen2 naming)."""

    hidden: int
    intermediate: int
    weight_std: float = 0.02
    rms_eps: float = 1e-6
    rope_theta: float = ROPE_THETA


BLOCKS = {
    "qwen7b": BlockShape(3584, 18944),
    "tiny": BlockShape(128, 256, weight_std=0.08),
}


def block_weights(shape: Shape, block: BlockShape, *, seed: int = 0, device="cpu",
                  bias: bool = True, layers=None):
    """Synthetic (random-init) bf16 weights of every layer, torch.nn.Linear
    layout [out][in]: dicts with norm_attn, w_qkv, b_qkv, w_o, norm_mlp,
    w_gate_up (gate rows, then up rows), w_down."""
    Hq, Hkv, d = shape.num_q_heads, shape.num_kv_heads, shape.head_dim
    H, I, sd = block.hidden, block.intermediate, block.weight_std
    out = []
    for l in (range(shape.num_layers) if layers is None else layers):
        g = _gen(device, seed, 0, l, 0, "block")
        r = lambda *s: (torch.randn(s, generator=g, device=device) * sd).to(torch.bfloat16)
        norm = lambda: (1.0 + 0.1 * torch.randn((H,), generator=g, device=device)).to(torch.bfloat16)
        out.append({
            "norm_attn": norm(),
            "w_qkv": r((Hq + 2 * Hkv) * d, H),
            "b_qkv": r((Hq + 2 * Hkv) * d) if bias else None,
            "w_o": r(H, Hq * d),
            "norm_mlp": norm(),
            "w_gate_up": r(2 * I, H),
            "w_down": r(H, I),
        })
    return out


def block_input(shape: Shape, block: BlockShape, frame: int, *, seed: int = 0, device="cpu"):
    """The frame's input hidden states (the vision tokens' embeddings), bf16
    [streams][T][hidden], N(0, 1)."""
    xs = []
    for s in range(shape.num_streams):
        g = _gen(device, seed, s, -1, frame, "x")
        xs.append(torch.randn((shape.tokens_per_frame, block.hidden), generator=g, device=device))
    return torch.stack(xs).to(torch.bfloat16).contiguous()
