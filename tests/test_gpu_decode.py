"""statekv_decode_step: decoding over the detailed cache (Sec. 3.2 / 3.3).

After a video has been prefilled frame by frame, text tokens (a prompt, then
one generated token per call) attend to every row of the decode cache and
causally to each other.  The output must equal the oracle's exact attention
over the video frames' K/V (taken from the input generator) followed by the
text tokens' K/V; the cache rows must be bit copies of every input; once a
(stream, layer) has decoded, prefill is refused and the cache capacity holds.
"""
import dataclasses

import numpy as np
import pytest
import torch

import oracle
from paper_2605_31598_gb300 import StateKV, make_config
from paper_2605_31598_gb300.inputs import WORKLOADS, batch_qkv

from .parity import OUT_ATOL


def _text_tokens(shape, n, seed, device):
    """Seeded synthetic text-token Q/K/V, [S][L][n][H][d] bf16, N(0,1)/sqrt(d)."""
    g = torch.Generator(device="cpu").manual_seed(seed)
    S, L, d = shape.num_streams, shape.num_layers, shape.head_dim
    mk = lambda h: (torch.randn((S, L, n, h, d), generator=g) * d ** -0.5).to(torch.bfloat16)
    return (mk(shape.num_q_heads).to(device), mk(shape.num_kv_heads).to(device),
            mk(shape.num_kv_heads).to(device))


@pytest.mark.gpu
@pytest.mark.parametrize("name,frames,steps,units", [
    ("toy", 4, (5, 1, 1, 1), [(0, 0)]),
    # end of a 12-frame video on the 28-layer stack: 2352 video rows, a 32-token
    # prompt, then two generated tokens
    ("qwen7b_stack", 12, (32, 1, 1), [(0, 0), (0, 27)]),
])
def test_decode_matches_exact_oracle(name, frames, steps, units):
    import __graft_entry__ as g

    g.build()
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    base = WORKLOADS[name]
    T = base.tokens_per_frame
    extra = -(-sum(steps) // T)  # frames of capacity the text rows need
    shape = dataclasses.replace(base, max_frames=frames + extra)
    S, L = shape.num_streams, shape.num_layers
    eng = StateKV(make_config(shape))
    hist = {u: ([], []) for u in units}
    for n in range(1, frames + 1):
        q, k, v = batch_qkv(shape, n, streams=range(S), layers=range(L), device="cuda")
        for u in units:
            hist[u][0].append(oracle.as_bf16_bits(k[u]))
            hist[u][1].append(oracle.as_bf16_bits(v[u]))
        assert eng.prefill_frame(q, k, v, torch.empty_like(q)) == 0
    done = frames * T
    for i, nt in enumerate(steps):
        q, k, v = _text_tokens(shape, nt, seed=100 + i, device="cuda")
        out = torch.full_like(q, float("nan"))
        assert eng.decode_step(q, k, v, out) == 0
        torch.cuda.synchronize()
        for u in units:
            ks = np.concatenate(hist[u][0] + [oracle.as_bf16_bits(k[u])])
            vs = np.concatenate(hist[u][1] + [oracle.as_bf16_bits(v[u])])
            ref = oracle.full_attention(oracle.as_bf16_bits(q[u]), ks, vs, done, causal=True)
            got = out[u].float().cpu().numpy()
            assert np.isfinite(got).all()
            err = float(np.abs(got - ref).max())
            assert err <= OUT_ATOL, f"step {i} ({nt} tokens) unit {u}: max |O - O_exact| = {err}"
            hist[u][0].append(oracle.as_bf16_bits(k[u]))
            hist[u][1].append(oracle.as_bf16_bits(v[u]))
        done += nt
    # the cache holds every row, bit for bit, and reports its length
    for u in units:
        ck, cv, info = eng.cache(*u)
        assert info.length == done
        assert np.array_equal(oracle.as_bf16_bits(ck[:, :done].transpose(0, 1)),
                              np.concatenate(hist[u][0]))
        assert np.array_equal(oracle.as_bf16_bits(cv[:, :done].transpose(0, 1)),
                              np.concatenate(hist[u][1]))
    # the video part is closed once a (stream, layer) has decoded
    q, k, v = batch_qkv(shape, frames + 1, streams=range(S), layers=range(L), device="cuda")
    assert eng.prefill_frame(q, k, v, torch.empty_like(q)) == 1  # INVALID_ARG
    assert eng.sync() == 0


@pytest.mark.gpu
def test_decode_refuses_rows_beyond_the_cache():
    import __graft_entry__ as g

    g.build()
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    shape = dataclasses.replace(WORKLOADS["toy"], max_frames=3)  # 48 rows
    S, L, T = shape.num_streams, shape.num_layers, shape.tokens_per_frame
    eng = StateKV(make_config(shape))
    for n in range(1, 3):
        q, k, v = batch_qkv(shape, n, streams=range(S), layers=range(L), device="cuda")
        assert eng.prefill_frame(q, k, v, torch.empty_like(q)) == 0
    q, k, v = _text_tokens(shape, T + 1, seed=7, device="cuda")  # 32 + 17 > 48
    assert eng.decode_step(q, k, v, torch.empty_like(q)) == 3  # CACHE_FULL
    q, k, v = _text_tokens(shape, T, seed=8, device="cuda")     # exactly fills it
    assert eng.decode_step(q, k, v, torch.empty_like(q)) == 0
    q, k, v = _text_tokens(shape, 1, seed=9, device="cuda")
    assert eng.decode_step(q, k, v, torch.empty_like(q)) == 3
    assert eng.sync() == 0
