"""The allocation-free attention entry point (statekv_frame_attention_noalloc).

Some callers cannot call cudaMalloc -- a plugin bound to its host
application's memory budget, or code that runs while another component is
capturing a stream.  For them the library offers one entry point whose scratch
lives in fixed device arrays inside the library; the caller passes only its
inputs and outputs.  These tests check that it refuses shapes beyond that
fixed scratch, and that on two calls in a row it returns the same attention
output and importance as the handle-based statekv_prefill_frame.
"""
import ctypes

import pytest
import torch

from paper_2605_31598_gb300 import StateKV, make_config, statekv
from paper_2605_31598_gb300.inputs import WORKLOADS, batch_qkv

from .parity import IMP_ATOL, IMP_RTOL, OUT_ATOL


def _call(cfg, q, k, v, sk, sv, count, out, imp):
    stream = torch.cuda.current_stream().cuda_stream if torch.cuda.is_available() else 0
    return statekv.statekv_frame_attention_noalloc(
        cfg, q.data_ptr(), k.data_ptr(), v.data_ptr(), sk.data_ptr(), sv.data_ptr(), count,
        out.data_ptr(), imp.data_ptr(), stream)


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
def test_noalloc_matches_prefill_frame_on_two_calls():
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
        kk, vv, pp, info = eng.state(0, 0)
        sk, sv, count = kk.clone(), vv.clone(), info.count  # pre-frame state
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
    assert eng.sync() == 0
