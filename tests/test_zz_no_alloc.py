"""The allocation-free attention entry point (statekv_frame_attention_noalloc).

Some callers cannot call cudaMalloc -- a plugin bound to its host
application's memory budget, or code that runs while another component is
capturing a stream.  For them the library offers one entry point whose scratch
lives in fixed device arrays inside the library; the caller passes only its
inputs and outputs.  These tests check that it refuses shapes beyond that
fixed scratch, and that on two calls in a row it returns the same attention
output and importance as the handle-based statekv_prefill_frame and as the
oracle, then on calls of other shapes that reuse the same scratch.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
from paper_2605_31598_gb300 import StateKV, make_config, statekv
from paper_2605_31598_gb300.inputs import WORKLOADS, Shape, batch_qkv

from .parity import IMP_ATOL, IMP_RTOL, OUT_ATOL


def _call(cfg, q, k, v, sk, sv, count, out, imp):
    stream = torch.cuda.current_stream().cuda_stream if torch.cuda.is_available() else 0
    ptr = lambda t: t.data_ptr() if t is not None else None
    return statekv.statekv_frame_attention_noalloc(
        cfg, q.data_ptr(), k.data_ptr(), v.data_ptr(), ptr(sk), ptr(sv), count,
        out.data_ptr(), imp.data_ptr(), stream)


def _check_against_oracle(shape, q, k, v, sk, sv, pos, count, vlen, out, imp):
    """The call's output and importance against the oracle started from the
    same state (slot order mapped through the positions)."""
    T, Hq, Hkv, d, B = (shape.tokens_per_frame, shape.num_q_heads, shape.num_kv_heads,
                        shape.head_dim, shape.state_capacity)
    lay = oracle.OracleLayer(Hq, Hkv, d, T, B, shape.max_frames)
    if B > 0:
        lay.set_state(np.full(Hkv, count, np.int32), pos, oracle.as_bf16_bits(sk),
                      oracle.as_bf16_bits(sv), vlen)
    o_ref, imp_ref, _ = lay.prefill_frame(*(oracle.as_bf16_bits(x) for x in (q, k, v)))
    err = float(np.abs(out.float().cpu().numpy() - o_ref).max())
    assert err <= OUT_ATOL, f"max |dO| = {err} against the oracle"
    g = imp.cpu().numpy().astype(np.float64)
    for h in range(Hkv):
        order = {int(p): i for i, p in enumerate(np.sort(pos[h, :count]))} if B > 0 else {}
        ref = np.array([imp_ref[h, order[int(pos[h, j])]] for j in range(count)] + list(imp_ref[h, B:]))
        got = np.concatenate([g[h, :count], g[h, B:]])
        assert np.all(np.abs(got - ref) <= IMP_RTOL * np.abs(ref) + IMP_ATOL), f"head {h}: importance"
        assert np.all(g[h, count:B] == 0), f"head {h}: empty state columns not 0"


def test_noalloc_refuses_shapes_beyond_its_fixed_scratch():
    """4 KV heads x 11 query tiles x (B + 196) partials must fit in 2^20 floats;
    B = 24000 does not.  The check happens before any device work."""
    from paper_2605_31598_gb300 import build_ext

    build_ext.build()
    shape = WORKLOADS["qwen7b_layer"]
    big = make_config(shape)
    big.state_capacity = 24000
    lib = statekv.lib()
    rc = lib.statekv_frame_attention_noalloc(ctypes.byref(big), 16, 16, 16, 16, 16, 0, 16, 16, None)
    assert rc == 2  # STATEKV_ERR_UNSUPPORTED
    rc = lib.statekv_frame_attention_noalloc(None, 16, 16, 16, 16, 16, 0, 16, 16, None)
    assert rc == 1  # STATEKV_ERR_INVALID_ARG


@pytest.mark.gpu
def test_noalloc_matches_prefill_frame_and_oracle():
    """Two 7B-layer calls in a row (a full state), each checked against the
    handle path's statekv_prefill_frame on the same pre-frame state and
    against the oracle; then, on the same shared scratch, a toy-shaped call
    (d 64, B 32, state half full) and a call with no state (B 0, null state
    pointers), both against the oracle."""
    import __graft_entry__ as g

    g.build()
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    shape = WORKLOADS["qwen7b_layer"]
    cfg = make_config(shape)
    T, Hq, Hkv, d, B = (shape.tokens_per_frame, shape.num_q_heads, shape.num_kv_heads,
                        shape.head_dim, shape.state_capacity)
    eng = StateKV(cfg)
    for n in range(1, 10):  # nine frames: the state holds 1568 of them
        q, k, v = batch_qkv(shape, n, streams=[0], layers=[0], device="cuda")
        assert eng.prefill_frame(q, k, v, torch.empty_like(q)) == 0
    for n in (10, 11):  # two calls in a row, each against the handle path
        q, k, v = batch_qkv(shape, n, streams=[0], layers=[0], device="cuda")
        torch.cuda.synchronize()
        kk, vv, pp, info = eng.state(0, 0)
        sk, sv, count = kk.clone(), vv.clone(), info.count  # pre-frame state
        pos, vlen = pp.cpu().numpy().astype(np.int64), info.virtual_len
        out_ref = torch.empty_like(q)
        imp_ref = torch.empty((1, 1, Hkv, B + T), device="cuda")
        assert eng.prefill_frame(q, k, v, out_ref, imp_ref) == 0
        out = torch.full_like(q[0, 0], float("nan"))
        imp = torch.full((Hkv, B + T), float("nan"), device="cuda")
        rc = _call(cfg, q[0, 0], k[0, 0], v[0, 0], sk, sv, count, out, imp)
        assert rc == 0, f"frame {n}: statekv_frame_attention_noalloc returned {rc}"
        torch.cuda.synchronize()
        assert (out.float() - out_ref[0, 0].float()).abs().max().item() <= OUT_ATOL
        ref = imp_ref[0, 0].double()
        assert ((imp.double() - ref).abs() <= IMP_RTOL * ref.abs() + IMP_ATOL).all()
        _check_against_oracle(shape, q[0, 0], k[0, 0], v[0, 0], sk, sv, pos, count, vlen, out, imp)
    assert eng.sync() == 0

    # toy shape, state half full (count 16 < B 32): d 64 and a smaller pool
    # than the previous call left in the scratch
    toy = WORKLOADS["toy"]
    tcfg = make_config(toy)
    teng = StateKV(tcfg)
    q, k, v = batch_qkv(toy, 1, streams=[0], layers=[0], device="cuda")
    assert teng.prefill_frame(q, k, v, torch.empty_like(q)) == 0
    q, k, v = batch_qkv(toy, 2, streams=[0], layers=[0], device="cuda")
    torch.cuda.synchronize()
    kk, vv, pp, info = teng.state(0, 0)
    assert info.count == 16
    out = torch.full_like(q[0, 0], float("nan"))
    imp = torch.full((toy.num_kv_heads, toy.state_capacity + toy.tokens_per_frame), float("nan"),
                     device="cuda")
    assert _call(tcfg, q[0, 0], k[0, 0], v[0, 0], kk, vv, info.count, out, imp) == 0
    torch.cuda.synchronize()
    _check_against_oracle(toy, q[0, 0], k[0, 0], v[0, 0], kk, vv,
                          pp.cpu().numpy().astype(np.int64), info.count, info.virtual_len, out, imp)
    assert teng.sync() == 0

    # no state at all: B = 0, null state pointers (in-frame causal attention)
    b0 = Shape(4, 2, 64, 40, 0, 2)
    bcfg = make_config(b0)
    q, k, v = batch_qkv(b0, 1, streams=[0], layers=[0], device="cuda", kind="peaked")
    out = torch.full_like(q[0, 0], float("nan"))
    imp = torch.full((2, 40), float("nan"), device="cuda")
    assert _call(bcfg, q[0, 0], k[0, 0], v[0, 0], None, None, 0, out, imp) == 0
    torch.cuda.synchronize()
    _check_against_oracle(b0, q[0, 0], k[0, 0], v[0, 0], None, None, None, 0, 0, out, imp)
