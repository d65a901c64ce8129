"""Plain CPU oracle of the StateKV per-frame cache-builder step (fp64).

TEST INFRASTRUCTURE ONLY: only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package.  The product path
(``paper_2605_31598_gb300``) never imports it and shares no code with it.

The arithmetic lives in ``statekv_oracle.c`` (plain loops, fp64); this module
only compiles it with gcc and marshals numpy arrays.  What it follows:

* Sec. 3.3, Eq. 5 -- attention of the frame's queries over [state ; frame]
  with every state token visible and in-frame causal order;
* Sec. 3.1, Eq. 1 / Sec. 3.3 -- importance = attention received, summed over
  the frame's queries and the query heads of a KV head (App. A keeps sinks per
  layer and KV head), each weight taken as exp(score - LSE) (App. B.1);
* Sec. 3.3, Eq. 6 -- keep the top B of the pool (state + frame tokens);
* Sec. 3.2/3.3 -- append the frame's K, V to the decode cache; L_n += T.
* Sec. 2 / Sec. 4 -- the recency-window baseline the method is compared with
  (``policy=1``): the state keeps the B most recent tokens instead.
* Sec. 4.1 / App. B -- the full self-attention baseline: the frame's queries
  attend to every earlier token and to the frame (causal within it), which
  is Eq. 5 with nothing ever evicted (``full_attention``, numpy matrix form).

Readings of silent points: score ties keep the older token; a pool of at most
B tokens is kept whole; the state is stored in ascending position.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "statekv_oracle.c")
_OUT_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_OUT_DIR, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle into ``oracle/_build/liboracle.so`` (gcc, -O2)."""
    os.makedirs(_OUT_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + ".tmp.%d" % os.getpid()
    # -O2 without -ffast-math: the fp64 loops keep IEEE semantics.
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            u16p = ctypes.POINTER(ctypes.c_uint16)
            i32p = ctypes.POINTER(ctypes.c_int32)
            i64p = ctypes.POINTER(ctypes.c_int64)
            f64p = ctypes.POINTER(ctypes.c_double)
            lib.oracle_prefill_frame.restype = ctypes.c_int
            lib.oracle_prefill_frame.argtypes = [
                ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                ctypes.c_int, ctypes.c_double, ctypes.c_int64,
                u16p, u16p, u16p, i32p, i64p, u16p, u16p, f64p, f64p, i32p]
            lib.oracle_prefill_frame_policy.restype = ctypes.c_int
            lib.oracle_prefill_frame_policy.argtypes = [
                ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                ctypes.c_int, ctypes.c_double, ctypes.c_int64,
                u16p, u16p, u16p, i32p, i64p, u16p, u16p, f64p, f64p, i32p, ctypes.c_int]
            lib.oracle_append_cache.restype = ctypes.c_int
            lib.oracle_append_cache.argtypes = [
                ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int64, ctypes.c_int64,
                u16p, u16p, u16p, u16p]
            _lib = lib
    return _lib


def _ptr(a: np.ndarray, ctype):
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data_as(ctypes.POINTER(ctype))


def as_bf16_bits(x) -> np.ndarray:
    """bf16 torch tensor (any device) -> C-contiguous numpy uint16 bit patterns."""
    import torch  # local: the oracle itself needs only numpy

    t = x.detach().to("cpu").contiguous()
    assert t.dtype == torch.bfloat16
    return t.view(torch.int16).numpy().view(np.uint16).copy()


def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float64."""
    u = bits.astype(np.uint32) << np.uint32(16)
    return u.view(np.float32).astype(np.float64)


class OracleLayer:
    """State of one (stream, layer): compressed state C and decode cache D.

    ``count[h]``, ``pos[h, :count]`` (ascending), ``sk/sv[h, :count]`` (bf16
    bits) hold the compressed state per KV head; ``dk/dv[h, :length]`` the
    detailed (decode) cache; ``virtual_len`` is L_n.
    """

    def __init__(self, n_q, n_kv, d, T, B, max_frames, causal=True, scale=None, policy=0):
        """policy 0: the method's top-B importance selection (Eq. 6); policy 1:
        the recency window (keep the B most recent tokens), the baseline."""
        self.n_q, self.n_kv, self.d, self.T, self.B = n_q, n_kv, d, T, B
        self.policy = int(policy)
        self.causal = 1 if causal else 0
        self.scale = float(scale) if scale else 1.0 / np.sqrt(d)
        self.count = np.zeros(n_kv, np.int32)
        self.pos = np.full((n_kv, max(B, 1)), -1, np.int64)
        self.sk = np.zeros((n_kv, max(B, 1), d), np.uint16)
        self.sv = np.zeros((n_kv, max(B, 1), d), np.uint16)
        self.capacity = max_frames * T
        self.dk = np.zeros((n_kv, self.capacity, d), np.uint16)
        self.dv = np.zeros((n_kv, self.capacity, d), np.uint16)
        self.virtual_len = 0

    def set_state(self, count, pos, sk, sv, virtual_len):
        """Teacher forcing: start the next frame from an externally given state.

        Entries may come in any slot order; they are stored here by position.
        """
        B = self.B
        self.count[:] = count
        self.pos[:] = -1
        for h in range(self.n_kv):
            c = int(count[h])
            order = np.argsort(pos[h, :c], kind="stable")
            self.pos[h, :c] = pos[h, :c][order]
            if B > 0:
                self.sk[h, :c] = sk[h, :c][order]
                self.sv[h, :c] = sv[h, :c][order]
        self.virtual_len = int(virtual_len)

    def prefill_frame(self, q_bits, k_bits, v_bits):
        """Run one frame.  q: [T][n_q][d], k/v: [T][n_kv][d] bf16 bits.

        Returns (out [T][n_q][d] f64, imp [n_kv][B+T] f64, kept [n_kv][B+T] i32).
        """
        lib = _load()
        T, n_q, n_kv, d, B = self.T, self.n_q, self.n_kv, self.d, self.B
        q = np.ascontiguousarray(q_bits, np.uint16).reshape(T, n_q, d)
        k = np.ascontiguousarray(k_bits, np.uint16).reshape(T, n_kv, d)
        v = np.ascontiguousarray(v_bits, np.uint16).reshape(T, n_kv, d)
        out = np.zeros((T, n_q, d), np.float64)
        imp = np.zeros((n_kv, B + T), np.float64)
        kept = np.zeros((n_kv, B + T), np.int32)
        rc = lib.oracle_append_cache(n_kv, d, T, self.virtual_len, self.capacity,
                                     _ptr(k, ctypes.c_uint16), _ptr(v, ctypes.c_uint16),
                                     _ptr(self.dk, ctypes.c_uint16),
                                     _ptr(self.dv, ctypes.c_uint16))
        if rc != 0:
            raise RuntimeError("oracle: decode cache full")
        rc = lib.oracle_prefill_frame_policy(
            n_q, n_kv, d, T, B, self.causal, self.scale, self.virtual_len,
            _ptr(q, ctypes.c_uint16), _ptr(k, ctypes.c_uint16), _ptr(v, ctypes.c_uint16),
            _ptr(self.count, ctypes.c_int32), _ptr(self.pos, ctypes.c_int64),
            _ptr(self.sk, ctypes.c_uint16), _ptr(self.sv, ctypes.c_uint16),
            _ptr(out, ctypes.c_double), _ptr(imp, ctypes.c_double),
            _ptr(kept, ctypes.c_int32), self.policy)
        if rc != 0:
            raise RuntimeError("oracle: bad arguments")
        self.virtual_len += T
        return out, imp, kept

    def state_positions(self, h):
        return self.pos[h, : int(self.count[h])].copy()


def full_attention(q_bits: np.ndarray, k_bits: np.ndarray, v_bits: np.ndarray, n_prefix: int,
                   causal: bool = True, scale: float | None = None) -> np.ndarray:
    """Exact softmax attention of one frame (fp64), the full-SA baseline.

    q: [T][n_q][d]; k, v: [n_prefix + T][n_kv][d] bf16 bits, the earlier
    tokens in order followed by the frame's own.  Query i of the frame sees
    every earlier token and frame token j iff j <= i (all frame tokens when
    not causal); query head h reads KV head h // (n_q / n_kv).  Returns O
    [T][n_q][d] float64.
    """
    q = bf16_bits_to_f64(q_bits)
    k = bf16_bits_to_f64(k_bits)
    v = bf16_bits_to_f64(v_bits)
    T, n_q, d = q.shape
    n_kv = k.shape[1]
    G = n_q // n_kv
    sc = float(scale) if scale else 1.0 / np.sqrt(d)
    visible = np.ones((T, n_prefix + T), dtype=bool)
    if causal:
        visible[:, n_prefix:] = np.tril(np.ones((T, T), dtype=bool))
    out = np.empty((T, n_q, d))
    for h in range(n_q):
        s = (q[:, h, :] @ k[:, h // G, :].T) * sc
        s = np.where(visible, s, -np.inf)
        s -= s.max(axis=1, keepdims=True)
        w = np.exp(s)
        w /= w.sum(axis=1, keepdims=True)
        out[:, h, :] = w @ v[:, h // G, :]
    return out
