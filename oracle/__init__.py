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
* App. A -- layer-level selection (``policy=2``: one ranking per layer by the
  attention summed over all heads, applied to every KV head) and the
  assumption diagnostics computed from the full-attention baseline's
  layer-level scores: the concentration C_{n,B} of historical attention in
  its top-B tokens (App. A.1), and candidate-pool recall, weighted recall,
  retention and churn of consecutive top-B oracle states (App. A.2).

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
        the recency window (keep the B most recent tokens), the baseline;
        policy 2: layer-level selection (App. A), one top-B by the importance
        summed over every KV head, shared by all heads."""
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
                   causal: bool = True, scale: float | None = None,
                   return_scores: bool = False):
    """Exact softmax attention of one frame (fp64), the full-SA baseline.

    q: [T][n_q][d]; k, v: [n_prefix + T][n_kv][d] bf16 bits, the earlier
    tokens in order followed by the frame's own.  Query i of the frame sees
    every earlier token and frame token j iff j <= i (all frame tokens when
    not causal); query head h reads KV head h // (n_q / n_kv).  Returns O
    [T][n_q][d] float64; with ``return_scores``, also the layer-level score
    of every key (App. A's shared protocol: the attention weights summed over
    the frame's queries within each head, then over all heads), float64
    [n_prefix + T].
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
    scores = np.zeros(n_prefix + T)
    for h in range(n_q):
        s = (q[:, h, :] @ k[:, h // G, :].T) * sc
        s = np.where(visible, s, -np.inf)
        s -= s.max(axis=1, keepdims=True)
        w = np.exp(s)
        w /= w.sum(axis=1, keepdims=True)
        out[:, h, :] = w @ v[:, h // G, :]
        scores += w.sum(axis=0)
    return (out, scores) if return_scores else out


# ---------------------------------------------------------------------------
# App. A diagnostics, on layer-level scores (one float per key position).

def top_b(scores: np.ndarray, B: int) -> np.ndarray:
    """Positions of the B highest scores, ties to the lower position (the
    older token), ascending.  Every position is kept when there are <= B."""
    scores = np.asarray(scores, np.float64)
    n = scores.shape[0]
    order = np.lexsort((np.arange(n), -scores))  # last key is the primary one
    return np.sort(order[: min(B, n)])


def concentration(hist_scores: np.ndarray, budgets) -> np.ndarray:
    """App. A.1: C_{n,B} = (sum of the B largest historical scores) / (sum of
    all historical scores), for each B in ``budgets``.  ``hist_scores`` are
    the layer-level scores of the keys of frames before n."""
    hist_scores = np.asarray(hist_scores, np.float64)
    mass = hist_scores.sum()
    return np.array([hist_scores[top_b(hist_scores, B)].sum() / mass for B in budgets])


def state_metrics(scores_n: np.ndarray, scores_next: np.ndarray, B: int) -> dict:
    """App. A.2 on consecutive oracle states.

    ``scores_n``: layer-level scores of frame n over every token seen up to
    and including frame n (positions 0 .. len - 1); ``scores_next``: those of
    frame n + 1 over every token up to and including it, so the tokens of
    frame n + 1 are the positions len(scores_n) .. len(scores_next) - 1.
    S_n and S_{n+1} are the top-B sets of each; the candidate pool is
    P_{n+1} = S_n + frame n + 1.  Returns recall |S_{n+1} & P| / |S_{n+1}|,
    weighted recall (weights = scores_next), retention |S_n & S_{n+1}| / |S_n|
    and churn |S_{n+1} - S_n| / |S_{n+1}|.
    """
    scores_next = np.asarray(scores_next, np.float64)
    n_seen = len(scores_n)
    s_n = set(top_b(scores_n, B).tolist())
    s_next = set(top_b(scores_next, B).tolist())
    pool = s_n | set(range(n_seen, len(scores_next)))
    hit = s_next & pool
    w_all = sum(scores_next[j] for j in s_next)
    w_hit = sum(scores_next[j] for j in hit)
    return {
        "recall": len(hit) / len(s_next),
        "weighted_recall": w_hit / w_all,
        "retention": len(s_n & s_next) / len(s_n),
        "churn": len(s_next - s_n) / len(s_next),
    }
