"""Pins of the CPU oracle against what the paper and the mathematics fix.

None of these checks re-types the oracle's loops: they compare it with a
library routine used on the textbook definition (scaled_dot_product_attention
in fp64, with an identity value matrix to read the attention weights back),
closed forms, a hand-worked example, brute-force subset search and invariants.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle
from oracle import OracleLayer, bf16_bits_to_f64

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def bits(x):
    """float array -> bf16 bit patterns (values must be exact in bf16 or are rounded)."""
    t = torch.as_tensor(np.asarray(x, np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16).copy()


def rand_bits(rng, shape, sigma=1.0):
    return bits(rng.standard_normal(shape) * sigma)


def sdpa_weights_and_out(q, k, v, mask, scale):
    """Textbook attention through the library routine, fp64.

    q [nq][d], k [nk][d], v [nk][dv], mask [nq][nk] bool (True = visible).
    Returns (A [nq][nk], O [nq][dv]).  A is read back by attending over an
    identity value matrix.
    """
    F = torch.nn.functional
    qt = torch.as_tensor(q, dtype=torch.float64)[None, None]
    kt = torch.as_tensor(k, dtype=torch.float64)[None, None]
    vt = torch.as_tensor(v, dtype=torch.float64)[None, None]
    m = torch.as_tensor(mask)[None, None]
    eye = torch.eye(k.shape[0], dtype=torch.float64)[None, None]
    A = F.scaled_dot_product_attention(qt, kt, eye, attn_mask=m, scale=scale)[0, 0]
    O = F.scaled_dot_product_attention(qt, kt, vt, attn_mask=m, scale=scale)[0, 0]
    return A.numpy(), O.numpy()


def test_oracle_builds():
    path = oracle.build()
    assert os.path.exists(path)


def test_hand_worked_example_w1():
    """Hand-derived two-frame example (tests/golden/w1_hand_example.json)."""
    with open(os.path.join(GOLDEN, "w1_hand_example.json")) as f:
        g = json.load(f)
    s = g["shape"]
    lay = OracleLayer(s["n_q"], s["n_kv"], s["d"], s["T"], s["B"], max_frames=2,
                      causal=bool(s["causal"]), scale=math.log(3.0))
    for fr in g["frames"]:
        T = s["T"]
        q = bits(np.array(fr["q"]).reshape(T, 1, 1))
        k = bits(np.array(fr["k"]).reshape(T, 1, 1))
        v = bits(np.array(fr["v"]).reshape(T, 1, 1))
        b_before = int(lay.count[0])
        out, imp, kept = lay.prefill_frame(q, k, v)
        np.testing.assert_allclose(out.reshape(-1), fr["out"], rtol=0, atol=1e-12)
        np.testing.assert_allclose(imp[0, :b_before], fr["importance_state"], atol=1e-12)
        np.testing.assert_allclose(imp[0, s["B"]:], fr["importance_frame"], atol=1e-12)
        assert list(lay.state_positions(0)) == fr["state_positions_after"]
        c = int(lay.count[0])
        np.testing.assert_array_equal(bf16_bits_to_f64(lay.sk[0, :c, 0]), fr["state_k_after"])
        np.testing.assert_array_equal(bf16_bits_to_f64(lay.sv[0, :c, 0]), fr["state_v_after"])
    L = g["virtual_len_after"]
    assert lay.virtual_len == L
    np.testing.assert_array_equal(bf16_bits_to_f64(lay.dk[0, :L, 0]), g["cache_k_after"])
    np.testing.assert_array_equal(bf16_bits_to_f64(lay.dv[0, :L, 0]), g["cache_v_after"])


def _run_stream(n_q, n_kv, d, T, B, N, seed, sigma=1.0, causal=True):
    rng = np.random.default_rng(seed)
    lay = OracleLayer(n_q, n_kv, d, T, B, max_frames=N, causal=causal)
    frames = []
    for n in range(N):
        q = rand_bits(rng, (T, n_q, d), sigma)
        k = rand_bits(rng, (T, n_kv, d), sigma)
        v = rand_bits(rng, (T, n_kv, d))
        pre = (lay.count.copy(), lay.pos.copy(), lay.sk.copy(), lay.sv.copy(), lay.virtual_len)
        out, imp, kept = lay.prefill_frame(q, k, v)
        frames.append(dict(q=q, k=k, v=v, out=out, imp=imp, kept=kept, pre=pre))
    return lay, frames


@pytest.mark.parametrize("causal", [True, False])
def test_full_attention_when_capacity_covers_stream(causal):
    """B >= N*T: every token stays, so frame n's queries attend to the whole
    prefix (the full self-attention the paper calls exact, Sec. 4)."""
    n_q, n_kv, d, T, N = 6, 2, 16, 5, 4
    G = n_q // n_kv
    lay, frames = _run_stream(n_q, n_kv, d, T, B=N * T, N=N, seed=1, causal=causal)
    scale = 1.0 / math.sqrt(d)
    allk = np.concatenate([bf16_bits_to_f64(f["k"]) for f in frames])  # [N*T][n_kv][d]
    allv = np.concatenate([bf16_bits_to_f64(f["v"]) for f in frames])
    for n, f in enumerate(frames):
        nk = (n + 1) * T
        qpos = n * T + np.arange(T)
        kpos = np.arange(nk)
        if causal:
            mask = kpos[None, :] <= qpos[:, None]
        else:
            mask = (kpos[None, :] < n * T) | (kpos[None, :] >= n * T)
        q = bf16_bits_to_f64(f["q"])
        for h in range(n_kv):
            colsum = np.zeros(nk)
            for g in range(G):
                hq = h * G + g
                A, O = sdpa_weights_and_out(q[:, hq], allk[:nk, h], allv[:nk, h], mask, scale)
                np.testing.assert_allclose(f["out"][:, hq], O, rtol=1e-11, atol=1e-12)
                colsum += A.sum(axis=0)
            # state columns are in position order (= positions 0..nT-1 here)
            np.testing.assert_allclose(f["imp"][h, : n * T], colsum[: n * T], rtol=1e-11, atol=1e-13)
            np.testing.assert_allclose(f["imp"][h, N * T:], colsum[n * T:], rtol=1e-11, atol=1e-13)
    assert np.all(lay.count == N * T)
    for h in range(n_kv):
        assert list(lay.state_positions(h)) == list(range(N * T))


@pytest.mark.parametrize("causal", [True, False])
def test_full_attention_function_matches_uncompressed_stream(causal):
    """oracle.full_attention (numpy matrix form) against the C loops of the
    stream whose state never evicts: the same exact attention two ways."""
    import oracle

    n_q, n_kv, d, T, N = 6, 2, 16, 5, 4
    lay, frames = _run_stream(n_q, n_kv, d, T, B=N * T, N=N, seed=3, causal=causal)
    for n, f in enumerate(frames):
        ks = np.concatenate([fr["k"] for fr in frames[: n + 1]])
        vs = np.concatenate([fr["v"] for fr in frames[: n + 1]])
        o = oracle.full_attention(f["q"], ks, vs, n * T, causal=causal)
        np.testing.assert_allclose(o, f["out"], rtol=1e-11, atol=1e-12)


@pytest.mark.parametrize("B", [7, 10, 13])
def test_recency_window_keeps_the_latest_tokens(B):
    """policy 1 (the recency-window baseline): the state holds the B most
    recent tokens, so frame n attends exactly to the last min(B, (n-1)T)
    earlier tokens plus itself (B multiple of T and not)."""
    import oracle

    n_q, n_kv, d, T, N = 4, 2, 16, 5, 6
    rng = np.random.default_rng(11)
    lay = OracleLayer(n_q, n_kv, d, T, B, max_frames=N, policy=1)
    ks, vs = [], []
    for n in range(N):
        q = rand_bits(rng, (T, n_q, d))
        k = rand_bits(rng, (T, n_kv, d))
        v = rand_bits(rng, (T, n_kv, d))
        out, _, _ = lay.prefill_frame(q, k, v)
        prev_k = np.concatenate(ks) if ks else np.zeros((0, n_kv, d), np.uint16)
        prev_v = np.concatenate(vs) if vs else np.zeros((0, n_kv, d), np.uint16)
        w = min(B, n * T)
        ref = oracle.full_attention(q, np.concatenate([prev_k[len(prev_k) - w:], k]),
                                    np.concatenate([prev_v[len(prev_v) - w:], v]), w)
        np.testing.assert_allclose(out, ref, rtol=1e-11, atol=1e-12)
        ks.append(k)
        vs.append(v)
        total = (n + 1) * T
        for h in range(n_kv):
            assert list(lay.state_positions(h)) == list(range(max(0, total - B), total))


def test_attention_over_selected_state_matches_library():
    """B < N*T: each frame's output is attention over exactly the pre-frame
    state's keys (looked up by position in the full stream) followed by the
    frame's keys, and the importance is the column sums of those weights."""
    n_q, n_kv, d, T, B, N = 4, 2, 8, 6, 7, 6
    G = n_q // n_kv
    lay, frames = _run_stream(n_q, n_kv, d, T, B, N, seed=2, sigma=1.5)
    scale = 1.0 / math.sqrt(d)
    allk = np.concatenate([bf16_bits_to_f64(f["k"]) for f in frames])
    allv = np.concatenate([bf16_bits_to_f64(f["v"]) for f in frames])
    for n, f in enumerate(frames):
        count, pos, _, _, L = f["pre"]
        assert L == n * T
        q = bf16_bits_to_f64(f["q"])
        for h in range(n_kv):
            b = int(count[h])
            spos = pos[h, :b]
            keys = np.concatenate([spos, n * T + np.arange(T)])
            mask = np.ones((T, b + T), bool)
            mask[:, b:] = np.tril(np.ones((T, T), bool))
            colsum = np.zeros(b + T)
            for g in range(G):
                hq = h * G + g
                A, O = sdpa_weights_and_out(q[:, hq], allk[keys, h], allv[keys, h], mask, scale)
                np.testing.assert_allclose(f["out"][:, hq], O, rtol=1e-11, atol=1e-12)
                colsum += A.sum(axis=0)
            np.testing.assert_allclose(f["imp"][h, :b], colsum[:b], rtol=1e-11, atol=1e-13)
            np.testing.assert_allclose(f["imp"][h, B:], colsum[b:], rtol=1e-11, atol=1e-13)


def test_selection_is_the_best_subset_brute_force():
    """The kept set maximises the summed score over every B-subset of the pool
    (Eq. 6's TopK), checked by enumerating all subsets on tiny pools."""
    n_q, n_kv, d, T, B, N = 2, 1, 4, 3, 2, 5
    lay, frames = _run_stream(n_q, n_kv, d, T, B, N, seed=3, sigma=2.0)
    for n, f in enumerate(frames):
        count = int(f["pre"][0][0])
        scores = list(f["imp"][0, :count]) + list(f["imp"][0, B:])
        cols = list(range(count)) + [B + t for t in range(T)]
        kept = [c for c in cols if f["kept"][0, c]]
        if len(scores) <= B:
            assert len(kept) == len(scores)
            continue
        best = max(itertools.combinations(range(len(scores)), B),
                   key=lambda s: sum(scores[i] for i in s))
        assert sorted(kept) == sorted(cols[i] for i in best)


def test_uniform_attention_closed_form_and_tie_break():
    """Q = 0: every visible key scores 0, so attention is uniform.

    O[i] = mean of the visible V; a state key receives
    G * sum_{i<T} 1/(b+i+1) and frame token t receives G * sum_{i>=t} 1/(b+i+1).
    All state keys tie with frame token 0; the older-wins tie-break then keeps
    the current state once it is full."""
    n_q, n_kv, d, T, B, N = 3, 1, 4, 4, 6, 4
    G = n_q // n_kv
    rng = np.random.default_rng(4)
    lay = OracleLayer(n_q, n_kv, d, T, B, max_frames=N)
    allv = []
    for n in range(N):
        q = np.zeros((T, n_q, d), np.uint16)
        k = rand_bits(rng, (T, n_kv, d))
        v = rand_bits(rng, (T, n_kv, d))
        allv.append(bf16_bits_to_f64(v))
        b = int(lay.count[0])
        spos = lay.state_positions(0)
        svals = bf16_bits_to_f64(lay.sv[0, :b])
        out, imp, kept = lay.prefill_frame(q, k, v)
        inv = 1.0 / (b + np.arange(T) + 1)
        np.testing.assert_allclose(imp[0, :b], G * inv.sum(), rtol=1e-13)
        for t in range(T):
            np.testing.assert_allclose(imp[0, B + t], G * inv[t:].sum(), rtol=1e-13)
        fv = bf16_bits_to_f64(v)[:, 0]
        for i in range(T):
            vis = np.concatenate([svals, fv[: i + 1]])
            for hq in range(n_q):
                np.testing.assert_allclose(out[i, hq], vis.mean(axis=0), rtol=1e-12, atol=1e-15)
        # selection: fill, then keep all state + the oldest frame tokens; once full, unchanged
        new_pos = lay.state_positions(0)
        if b + T <= B:
            assert list(new_pos) == list(spos) + [n * T + t for t in range(T)]
        elif b < B:
            assert list(new_pos) == list(spos) + [n * T + t for t in range(B - b)]
        else:
            assert list(new_pos) == list(spos)
    assert list(lay.state_positions(0)) == [0, 1, 2, 3, 4, 5]


def test_zero_capacity_means_no_cross_frame_context():
    """B = 0: each frame attends to itself only (in-frame causal attention)."""
    n_q, n_kv, d, T, N = 4, 2, 8, 5, 3
    G = n_q // n_kv
    lay, frames = _run_stream(n_q, n_kv, d, T, B=0, N=N, seed=5)
    scale = 1.0 / math.sqrt(d)
    mask = np.tril(np.ones((T, T), bool))
    for f in frames:
        q, k, v = (bf16_bits_to_f64(f[x]) for x in ("q", "k", "v"))
        for h in range(n_kv):
            colsum = np.zeros(T)
            for g in range(G):
                A, O = sdpa_weights_and_out(q[:, h * G + g], k[:, h], v[:, h], mask, scale)
                np.testing.assert_allclose(f["out"][:, h * G + g], O, rtol=1e-11, atol=1e-12)
                colsum += A.sum(axis=0)
            np.testing.assert_allclose(f["imp"][h], colsum, rtol=1e-11)
        assert np.all(lay.count == 0)


@pytest.mark.parametrize("kind", ["toy", "qwen", "peaked"])
def test_invariants_on_generated_inputs(kind):
    """Capacity, mass conservation, unique positions, bit-copied rows and the
    append-only decode cache, over a run long enough to evict."""
    from paper_2605_31598_gb300.inputs import Shape, frame_qkv

    shape = Shape(4, 2, 32, 12, 20, 8, kind=kind)
    n_q, n_kv, d, T, B, N = 4, 2, 32, 12, 20, 8
    G = n_q // n_kv
    lay = OracleLayer(n_q, n_kv, d, T, B, max_frames=N)
    ks, vs = [], []
    for n in range(1, N + 1):
        q, k, v = (oracle.as_bf16_bits(x) for x in frame_qkv(shape, n, layer=1, stream=2))
        ks.append(k)
        vs.append(v)
        b = lay.count.copy()
        out, imp, kept = lay.prefill_frame(q, k, v)
        L = n * T
        for h in range(n_kv):
            assert lay.count[h] == min(B, b[h] + T)
            np.testing.assert_allclose(imp[h].sum(), G * T, rtol=1e-12)
            assert np.all(imp[h, b[h]:B] == 0)
            p = lay.state_positions(h)
            assert len(set(p.tolist())) == len(p)
            assert np.all(np.diff(p) > 0) and p.min() >= 0 and p.max() < L
            allk = np.concatenate(ks)[:, h]
            allv = np.concatenate(vs)[:, h]
            np.testing.assert_array_equal(lay.sk[h, : len(p)], allk[p])
            np.testing.assert_array_equal(lay.sv[h, : len(p)], allv[p])
            assert kept[h].sum() == lay.count[h]
        np.testing.assert_array_equal(lay.dk[:, :L], np.concatenate(ks).transpose(1, 0, 2))
        np.testing.assert_array_equal(lay.dv[:, :L], np.concatenate(vs).transpose(1, 0, 2))
    assert lay.virtual_len == N * T


def test_cache_overflow_is_refused():
    lay = OracleLayer(1, 1, 4, 2, 2, max_frames=1)
    z = np.zeros((2, 1, 4), np.uint16)
    lay.prefill_frame(z, z, z)
    with pytest.raises(RuntimeError):
        lay.prefill_frame(z, z, z)
