"""ctypes binding of ``include/statekv.h`` (argument marshalling only).

Every function of the C ABI is exposed under its own name; ``StateKV`` is a
small convenience owner that allocates the device arena with torch (PyTorch
is used for device memory and streams only) and passes raw pointers through.
Every step of the path runs in the CUDA library; there is no fallback: if the
library is missing the first call raises.
"""
from __future__ import annotations

import ctypes
import os
import threading

PKG = os.path.dirname(os.path.abspath(__file__))
# STATEKV_DEBUG=1 in the environment (before the first call) loads the debug
# build (bounds checks and arena guard bands; build_ext.build(debug=True))
LIB_PATH = os.path.join(PKG, "libstatekv_debug.so" if os.environ.get("STATEKV_DEBUG") == "1"
                        else "libstatekv.so")

STATEKV_OK = 0
STATUS_NAMES = {
    0: "STATEKV_OK", 1: "STATEKV_ERR_INVALID_ARG", 2: "STATEKV_ERR_UNSUPPORTED",
    3: "STATEKV_ERR_CACHE_FULL", 4: "STATEKV_ERR_CUDA", 5: "STATEKV_ERR_DEVICE_TIMEOUT",
    6: "STATEKV_ERR_ARENA_TOO_SMALL", 7: "STATEKV_ERR_DEVICE_FAULT",
}
EXPORTED = ("statekv_arena_bytes", "statekv_init", "statekv_prefill_frame",
            "statekv_prefill_frame_host", "statekv_prefill_frames_host",
            "statekv_full_attention_frame", "statekv_decode_step",
            "statekv_state_view", "statekv_cache_view",
            "statekv_profile_enable", "statekv_profile_read", "statekv_sync",
            "statekv_device_error", "statekv_watchdog_selftest", "statekv_frame_attention_noalloc",
            "statekv_debug_check",
            "statekv_scores_workspace_bytes", "statekv_full_attention_scores",
            "statekv_topb_mask", "statekv_concentration_sums", "statekv_state_metrics",
            "statekv_block_workspace_bytes", "statekv_block_frame",
            "statekv_destroy", "statekv_status_string")


class statekv_config(ctypes.Structure):
    _fields_ = [("num_streams", ctypes.c_int32), ("num_layers", ctypes.c_int32),
                ("num_q_heads", ctypes.c_int32), ("num_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("tokens_per_frame", ctypes.c_int32),
                ("state_capacity", ctypes.c_int32), ("max_frames", ctypes.c_int32),
                ("causal_in_frame", ctypes.c_int32), ("host_staging", ctypes.c_int32),
                ("softmax_scale", ctypes.c_float), ("watchdog_ms", ctypes.c_uint32),
                ("selection", ctypes.c_int32)]


class statekv_decode_args(ctypes.Structure):
    _fields_ = [("stream_begin", ctypes.c_int32), ("stream_count", ctypes.c_int32),
                ("layer_begin", ctypes.c_int32), ("layer_count", ctypes.c_int32),
                ("num_tokens", ctypes.c_int32),
                ("q", ctypes.c_void_p), ("k", ctypes.c_void_p), ("v", ctypes.c_void_p),
                ("out", ctypes.c_void_p)]


class statekv_block_config(ctypes.Structure):
    _fields_ = [("hidden", ctypes.c_int32), ("intermediate", ctypes.c_int32),
                ("rms_eps", ctypes.c_float), ("rope_theta", ctypes.c_float),
                ("yarn_factor", ctypes.c_float), ("yarn_original_max", ctypes.c_int32)]


class statekv_block_weights(ctypes.Structure):
    _fields_ = [("norm_attn", ctypes.c_void_p), ("w_qkv", ctypes.c_void_p),
                ("b_qkv", ctypes.c_void_p), ("w_o", ctypes.c_void_p),
                ("norm_mlp", ctypes.c_void_p), ("w_gate_up", ctypes.c_void_p),
                ("w_down", ctypes.c_void_p)]


class statekv_frame_args(ctypes.Structure):
    _fields_ = [("stream_begin", ctypes.c_int32), ("stream_count", ctypes.c_int32),
                ("layer_begin", ctypes.c_int32), ("layer_count", ctypes.c_int32),
                ("q", ctypes.c_void_p), ("k", ctypes.c_void_p), ("v", ctypes.c_void_p),
                ("out", ctypes.c_void_p), ("importance", ctypes.c_void_p)]


class statekv_state_info(ctypes.Structure):
    _fields_ = [("k", ctypes.c_void_p), ("v", ctypes.c_void_p), ("positions", ctypes.c_void_p),
                ("count", ctypes.c_int32), ("frames", ctypes.c_int32),
                ("virtual_len", ctypes.c_int64)]


class statekv_cache_info(ctypes.Structure):
    _fields_ = [("k", ctypes.c_void_p), ("v", ctypes.c_void_p), ("length", ctypes.c_int64),
                ("capacity", ctypes.c_int64)]


class statekv_profile(ctypes.Structure):
    _fields_ = [("launches", ctypes.c_int64 * 5), ("milliseconds", ctypes.c_double * 5)]


_lock = threading.Lock()
_lib = None


def lib() -> ctypes.CDLL:
    """The loaded C library (raises if it has not been built)."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise RuntimeError(
                    f"{LIB_PATH} is missing: build the CUDA library first "
                    "(python -c 'import __graft_entry__ as g; g.build()')")
            L = ctypes.CDLL(LIB_PATH)
            P = ctypes.POINTER
            st = ctypes.c_int
            L.statekv_arena_bytes.argtypes = [P(statekv_config), P(ctypes.c_size_t)]
            L.statekv_arena_bytes.restype = st
            L.statekv_init.argtypes = [P(statekv_config), ctypes.c_void_p, ctypes.c_size_t,
                                       P(ctypes.c_void_p)]
            L.statekv_init.restype = st
            for name in ("statekv_prefill_frame", "statekv_prefill_frame_host",
                         "statekv_full_attention_frame"):
                fn = getattr(L, name)
                fn.argtypes = [ctypes.c_void_p, P(statekv_frame_args), ctypes.c_void_p]
                fn.restype = st
            L.statekv_prefill_frames_host.argtypes = [ctypes.c_void_p, P(statekv_frame_args),
                                                      ctypes.c_int32, ctypes.c_void_p]
            L.statekv_prefill_frames_host.restype = st
            L.statekv_debug_check.argtypes = [ctypes.c_void_p, ctypes.c_void_p]
            L.statekv_debug_check.restype = st
            L.statekv_watchdog_selftest.argtypes = [ctypes.c_void_p, ctypes.c_void_p]
            L.statekv_watchdog_selftest.restype = st
            L.statekv_decode_step.argtypes = [ctypes.c_void_p, P(statekv_decode_args),
                                              ctypes.c_void_p]
            L.statekv_decode_step.restype = st
            L.statekv_state_view.argtypes = [ctypes.c_void_p, ctypes.c_int32, ctypes.c_int32,
                                             P(statekv_state_info)]
            L.statekv_state_view.restype = st
            L.statekv_cache_view.argtypes = [ctypes.c_void_p, ctypes.c_int32, ctypes.c_int32,
                                             P(statekv_cache_info)]
            L.statekv_cache_view.restype = st
            L.statekv_profile_enable.argtypes = [ctypes.c_void_p, ctypes.c_int32]
            L.statekv_profile_enable.restype = st
            L.statekv_profile_read.argtypes = [ctypes.c_void_p, P(statekv_profile)]
            L.statekv_profile_read.restype = st
            L.statekv_sync.argtypes = [ctypes.c_void_p]
            L.statekv_sync.restype = st
            L.statekv_device_error.argtypes = [ctypes.c_void_p, P(ctypes.c_int32)]
            L.statekv_device_error.restype = st
            L.statekv_frame_attention_noalloc.argtypes = [
                P(statekv_config), ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int32, ctypes.c_void_p,
                ctypes.c_void_p, ctypes.c_void_p]
            L.statekv_frame_attention_noalloc.restype = st
            L.statekv_scores_workspace_bytes.argtypes = [ctypes.c_void_p, ctypes.c_int32,
                                                         ctypes.c_int32, P(ctypes.c_size_t)]
            L.statekv_scores_workspace_bytes.restype = st
            L.statekv_full_attention_scores.argtypes = [
                ctypes.c_void_p, P(statekv_frame_args), ctypes.c_void_p, ctypes.c_void_p,
                ctypes.c_size_t, ctypes.c_void_p]
            L.statekv_full_attention_scores.restype = st
            L.statekv_topb_mask.argtypes = [ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64,
                                            ctypes.c_int64, ctypes.c_int64, ctypes.c_void_p,
                                            ctypes.c_void_p]
            L.statekv_topb_mask.restype = st
            L.statekv_concentration_sums.argtypes = [ctypes.c_void_p, ctypes.c_void_p,
                                                     ctypes.c_int32, ctypes.c_int64,
                                                     ctypes.c_int64, ctypes.c_void_p,
                                                     ctypes.c_void_p]
            L.statekv_concentration_sums.restype = st
            L.statekv_state_metrics.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                                                ctypes.c_int32, ctypes.c_int64, ctypes.c_int32,
                                                ctypes.c_int64, ctypes.c_void_p, ctypes.c_void_p]
            L.statekv_state_metrics.restype = st
            L.statekv_block_workspace_bytes.argtypes = [ctypes.c_void_p, P(statekv_block_config),
                                                        ctypes.c_int32, P(ctypes.c_size_t)]
            L.statekv_block_workspace_bytes.restype = st
            L.statekv_block_frame.argtypes = [
                ctypes.c_void_p, P(statekv_block_config), P(statekv_block_weights),
                ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_void_p,
                ctypes.c_void_p, ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p]
            L.statekv_block_frame.restype = st
            L.statekv_destroy.argtypes = [ctypes.c_void_p]
            L.statekv_destroy.restype = None
            L.statekv_status_string.argtypes = [ctypes.c_int]
            L.statekv_status_string.restype = ctypes.c_char_p
            _lib = L
    return _lib


class StateKVError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        msg = lib().statekv_status_string(status).decode()
        super().__init__(f"{what}: {STATUS_NAMES.get(status, status)} ({msg})")


def check(status: int, what: str):
    if status != STATEKV_OK:
        raise StateKVError(status, what)


# ---------------------------------------------------------------- C ABI names
def statekv_arena_bytes(cfg: statekv_config) -> int:
    n = ctypes.c_size_t(0)
    check(lib().statekv_arena_bytes(ctypes.byref(cfg), ctypes.byref(n)), "statekv_arena_bytes")
    return n.value


def statekv_init(cfg: statekv_config, arena_ptr: int, arena_bytes: int) -> int:
    h = ctypes.c_void_p(0)
    check(lib().statekv_init(ctypes.byref(cfg), ctypes.c_void_p(arena_ptr), arena_bytes,
                             ctypes.byref(h)), "statekv_init")
    return h.value


def statekv_prefill_frame(handle: int, args: statekv_frame_args, stream: int) -> int:
    return lib().statekv_prefill_frame(handle, ctypes.byref(args), ctypes.c_void_p(stream))


def statekv_prefill_frame_host(handle: int, args: statekv_frame_args, stream: int) -> int:
    return lib().statekv_prefill_frame_host(handle, ctypes.byref(args), ctypes.c_void_p(stream))


def statekv_prefill_frames_host(handle: int, frames, n: int, stream: int) -> int:
    """``frames``: a ctypes array of ``n`` statekv_frame_args (host pointers)."""
    return lib().statekv_prefill_frames_host(handle, frames, n, ctypes.c_void_p(stream))


def statekv_full_attention_frame(handle: int, args: statekv_frame_args, stream: int) -> int:
    return lib().statekv_full_attention_frame(handle, ctypes.byref(args), ctypes.c_void_p(stream))


def statekv_decode_step(handle: int, args: statekv_decode_args, stream: int) -> int:
    return lib().statekv_decode_step(handle, ctypes.byref(args), ctypes.c_void_p(stream))


def statekv_state_view(handle: int, stream: int, layer: int) -> statekv_state_info:
    info = statekv_state_info()
    check(lib().statekv_state_view(handle, stream, layer, ctypes.byref(info)),
          "statekv_state_view")
    return info


def statekv_cache_view(handle: int, stream: int, layer: int) -> statekv_cache_info:
    info = statekv_cache_info()
    check(lib().statekv_cache_view(handle, stream, layer, ctypes.byref(info)),
          "statekv_cache_view")
    return info


def statekv_profile_enable(handle: int, enable: bool):
    check(lib().statekv_profile_enable(handle, 1 if enable else 0), "statekv_profile_enable")


def statekv_profile_read(handle: int) -> statekv_profile:
    prof = statekv_profile()
    check(lib().statekv_profile_read(handle, ctypes.byref(prof)), "statekv_profile_read")
    return prof


def statekv_sync(handle: int) -> int:
    return lib().statekv_sync(handle)


def statekv_device_error(handle: int) -> int:
    code = ctypes.c_int32(0)
    check(lib().statekv_device_error(handle, ctypes.byref(code)), "statekv_device_error")
    return code.value


def statekv_frame_attention_noalloc(cfg: statekv_config, q: int, k: int, v: int, state_k: int,
                                    state_v: int, state_count: int, out: int, importance: int,
                                    stream: int) -> int:
    """Attention + importance for one (stream, layer) without device allocation
    (scratch lives in fixed device arrays of the library); returns the status."""
    return lib().statekv_frame_attention_noalloc(
        ctypes.byref(cfg), ctypes.c_void_p(q), ctypes.c_void_p(k), ctypes.c_void_p(v),
        ctypes.c_void_p(state_k), ctypes.c_void_p(state_v), state_count, ctypes.c_void_p(out),
        ctypes.c_void_p(importance), ctypes.c_void_p(stream))


def statekv_scores_workspace_bytes(handle: int, stream_count: int, layer_count: int) -> int:
    n = ctypes.c_size_t(0)
    check(lib().statekv_scores_workspace_bytes(handle, stream_count, layer_count, ctypes.byref(n)),
          "statekv_scores_workspace_bytes")
    return n.value


def statekv_full_attention_scores(handle: int, args: statekv_frame_args, scores: int,
                                  workspace: int, workspace_bytes: int, stream: int) -> int:
    return lib().statekv_full_attention_scores(handle, ctypes.byref(args), ctypes.c_void_p(scores),
                                               ctypes.c_void_p(workspace), workspace_bytes,
                                               ctypes.c_void_p(stream))


def statekv_topb_mask(scores: int, rows: int, n: int, row_stride: int, B: int, mask: int,
                      stream: int) -> int:
    return lib().statekv_topb_mask(ctypes.c_void_p(scores), rows, n, row_stride, B,
                                   ctypes.c_void_p(mask), ctypes.c_void_p(stream))


def statekv_concentration_sums(scores: int, mask: int, rows: int, n: int, row_stride: int,
                               out: int, stream: int) -> int:
    return lib().statekv_concentration_sums(ctypes.c_void_p(scores), ctypes.c_void_p(mask), rows,
                                            n, row_stride, ctypes.c_void_p(out),
                                            ctypes.c_void_p(stream))


def statekv_state_metrics(mask_n: int, mask_n1: int, scores_n1: int, rows: int, n_seen: int,
                          T: int, row_stride: int, out: int, stream: int) -> int:
    return lib().statekv_state_metrics(ctypes.c_void_p(mask_n), ctypes.c_void_p(mask_n1),
                                       ctypes.c_void_p(scores_n1), rows, n_seen, T, row_stride,
                                       ctypes.c_void_p(out), ctypes.c_void_p(stream))


def statekv_block_workspace_bytes(handle: int, bc: statekv_block_config, stream_count: int) -> int:
    n = ctypes.c_size_t(0)
    check(lib().statekv_block_workspace_bytes(handle, ctypes.byref(bc), stream_count,
                                              ctypes.byref(n)), "statekv_block_workspace_bytes")
    return n.value


def statekv_block_frame(handle: int, bc: statekv_block_config, weights, stream_begin: int,
                        stream_count: int, layer_begin: int, layer_count: int, x_in: int,
                        x_out: int, workspace: int, workspace_bytes: int, stream: int) -> int:
    """``weights``: a ctypes array of statekv_block_weights, one per layer."""
    return lib().statekv_block_frame(handle, ctypes.byref(bc), weights, stream_begin, stream_count,
                                     layer_begin, layer_count, ctypes.c_void_p(x_in),
                                     ctypes.c_void_p(x_out), ctypes.c_void_p(workspace),
                                     workspace_bytes, ctypes.c_void_p(stream))


def block_weights_array(layers) -> ctypes.Array:
    """ctypes array of statekv_block_weights from per-layer dicts of device
    tensors (keys norm_attn, w_qkv, b_qkv (or None), w_o, norm_mlp, w_gate_up,
    w_down)."""
    arr = (statekv_block_weights * len(layers))()
    for i, w in enumerate(layers):
        arr[i] = statekv_block_weights(
            w["norm_attn"].data_ptr(), w["w_qkv"].data_ptr(),
            w["b_qkv"].data_ptr() if w.get("b_qkv") is not None else None, w["w_o"].data_ptr(),
            w["norm_mlp"].data_ptr(), w["w_gate_up"].data_ptr(), w["w_down"].data_ptr())
    return arr


def statekv_destroy(handle: int):
    lib().statekv_destroy(handle)


def statekv_status_string(status: int) -> str:
    return lib().statekv_status_string(status).decode()


# ---------------------------------------------------------------- owner object
SELECTION_IMPORTANCE = 0  # the method: top-B by importance (Eq. 6)
SELECTION_RECENCY = 1     # the baseline: the B most recent tokens
SELECTION_LAYER = 2       # App. A: one top-B per layer by the importance summed over heads


def make_config(shape, *, causal=True, host_staging=False, softmax_scale=0.0,
                watchdog_ms=0, selection=SELECTION_IMPORTANCE) -> statekv_config:
    """statekv_config from an ``inputs.Shape``-like object."""
    return statekv_config(shape.num_streams, shape.num_layers, shape.num_q_heads,
                          shape.num_kv_heads, shape.head_dim, shape.tokens_per_frame,
                          shape.state_capacity, shape.max_frames, 1 if causal else 0,
                          1 if host_staging else 0, softmax_scale, watchdog_ms, selection)


class StateKV:
    """Owns a handle and its torch-allocated device arena."""

    def __init__(self, cfg: statekv_config, device="cuda", arena=None):
        """``arena``: optional caller-owned uint8 device tensor of at least
        ``statekv_arena_bytes(cfg)`` bytes (its prior contents do not matter)."""
        import torch

        self.cfg = cfg
        self.nbytes = statekv_arena_bytes(cfg)
        if arena is None:
            arena = torch.empty(max(self.nbytes, 256), dtype=torch.uint8, device=device)
        assert arena.dtype == torch.uint8 and arena.numel() >= self.nbytes
        self.arena = arena
        self.handle = statekv_init(cfg, self.arena.data_ptr(), self.nbytes)

    def close(self):
        if getattr(self, "handle", None):
            statekv_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _args(self, q, k, v, out, importance, stream_begin, stream_count, layer_begin,
              layer_count):
        return statekv_frame_args(stream_begin, stream_count, layer_begin, layer_count,
                                  q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(),
                                  importance.data_ptr() if importance is not None else None)

    def prefill_frame(self, q, k, v, out, importance=None, *, stream_begin=0, stream_count=None,
                      layer_begin=0, layer_count=None, stream=None) -> int:
        """Enqueue one frame step on ``stream`` (torch current stream by default).

        Returns the C status code (0 = OK); the caller decides how to react."""
        import torch

        sc = self.cfg.num_streams - stream_begin if stream_count is None else stream_count
        lc = self.cfg.num_layers - layer_begin if layer_count is None else layer_count
        st = (stream or torch.cuda.current_stream()).cuda_stream
        args = self._args(q, k, v, out, importance, stream_begin, sc, layer_begin, lc)
        return statekv_prefill_frame(self.handle, args, st)

    def full_attention_frame(self, q, k, v, out, *, stream_begin=0, stream_count=None,
                             layer_begin=0, layer_count=None, stream=None) -> int:
        """Exact full self-attention of the next frame over the whole decode
        cache (the comparison baseline); changes no state.  Returns the C status."""
        import torch

        sc = self.cfg.num_streams - stream_begin if stream_count is None else stream_count
        lc = self.cfg.num_layers - layer_begin if layer_count is None else layer_count
        st = (stream or torch.cuda.current_stream()).cuda_stream
        args = self._args(q, k, v, out, None, stream_begin, sc, layer_begin, lc)
        return statekv_full_attention_frame(self.handle, args, st)

    def full_attention_scores(self, q, k, v, out, scores, workspace, *, stream_begin=0,
                              stream_count=None, layer_begin=0, layer_count=None,
                              stream=None) -> int:
        """Full self-attention of the next frame plus App. A's layer-level score
        of every key into ``scores`` (fp32 [S][L][max_frames * T]);
        ``workspace``: a uint8 device tensor of ``scores_workspace_bytes``.
        Changes no state.  Returns the C status."""
        import torch

        sc = self.cfg.num_streams - stream_begin if stream_count is None else stream_count
        lc = self.cfg.num_layers - layer_begin if layer_count is None else layer_count
        st = (stream or torch.cuda.current_stream()).cuda_stream
        args = self._args(q, k, v, out, None, stream_begin, sc, layer_begin, lc)
        return statekv_full_attention_scores(self.handle, args, scores.data_ptr(),
                                             workspace.data_ptr(), workspace.numel(), st)

    def scores_workspace_bytes(self, stream_count=None, layer_count=None) -> int:
        sc = self.cfg.num_streams if stream_count is None else stream_count
        lc = self.cfg.num_layers if layer_count is None else layer_count
        return statekv_scores_workspace_bytes(self.handle, sc, lc)

    def block_frame(self, bc, weights, x_in, x_out, workspace, *, stream_begin=0,
                    stream_count=None, layer_begin=0, layer_count=None, stream=None) -> int:
        """The next frame of the streams through layers [layer_begin, +count) of
        the transformer block (x: bf16 [S][T][hidden]); ``weights``: from
        ``block_weights_array``; ``workspace``: uint8 device tensor of
        ``block_workspace_bytes`` bytes.  Returns the C status."""
        import torch

        sc = self.cfg.num_streams - stream_begin if stream_count is None else stream_count
        lc = self.cfg.num_layers - layer_begin if layer_count is None else layer_count
        st = (stream or torch.cuda.current_stream()).cuda_stream
        return statekv_block_frame(self.handle, bc, weights, stream_begin, sc, layer_begin, lc,
                                   x_in.data_ptr(), x_out.data_ptr(), workspace.data_ptr(),
                                   workspace.numel(), st)

    def block_workspace_bytes(self, bc, stream_count=None) -> int:
        sc = self.cfg.num_streams if stream_count is None else stream_count
        return statekv_block_workspace_bytes(self.handle, bc, sc)

    def decode_step(self, q, k, v, out, *, stream_begin=0, stream_count=None, layer_begin=0,
                    layer_count=None, stream=None) -> int:
        """Enqueue ``q.shape[2]`` new tokens per (stream, layer) over the decode
        cache (q: [S][L][n][Hq][d] bf16, k/v: [S][L][n][Hkv][d]); their K/V are
        appended afterwards.  Returns the C status."""
        import torch

        sc = self.cfg.num_streams - stream_begin if stream_count is None else stream_count
        lc = self.cfg.num_layers - layer_begin if layer_count is None else layer_count
        st = (stream or torch.cuda.current_stream()).cuda_stream
        args = statekv_decode_args(stream_begin, sc, layer_begin, lc, int(q.shape[2]),
                                   q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr())
        return statekv_decode_step(self.handle, args, st)

    def prefill_frame_host(self, q, k, v, out, importance=None, *, stream_begin=0,
                           stream_count=None, layer_begin=0, layer_count=None,
                           stream=None) -> int:
        import torch

        sc = self.cfg.num_streams - stream_begin if stream_count is None else stream_count
        lc = self.cfg.num_layers - layer_begin if layer_count is None else layer_count
        st = (stream or torch.cuda.current_stream()).cuda_stream
        args = self._args(q, k, v, out, importance, stream_begin, sc, layer_begin, lc)
        return statekv_prefill_frame_host(self.handle, args, st)

    def prefill_frames_host(self, frames, *, stream_begin=0, stream_count=None, layer_begin=0,
                            layer_count=None, stream=None) -> int:
        """Consecutive frames from pinned host buffers, copies pipelined with the
        steps: ``frames`` is a sequence of (q, k, v, out, importance-or-None)
        CPU tensors laid out as for ``prefill_frame_host``.  Returns the C status."""
        import torch

        sc = self.cfg.num_streams - stream_begin if stream_count is None else stream_count
        lc = self.cfg.num_layers - layer_begin if layer_count is None else layer_count
        st = (stream or torch.cuda.current_stream()).cuda_stream
        arr = (statekv_frame_args * len(frames))()
        for i, (q, k, v, out, imp) in enumerate(frames):
            arr[i] = self._args(q, k, v, out, imp, stream_begin, sc, layer_begin, lc)
        return statekv_prefill_frames_host(self.handle, arr, len(frames), st)

    def _arena_view(self, ptr, nbytes, dtype, shape):
        import torch

        off = ptr - self.arena.data_ptr()
        assert 0 <= off and off + nbytes <= self.arena.numel()
        return self.arena[off: off + nbytes].view(dtype).view(shape)

    def state(self, stream: int, layer: int):
        """(k [Hkv][B][d] bf16, v, positions [Hkv][B] int32, info) views into the arena."""
        import torch

        c = self.cfg
        info = statekv_state_view(self.handle, stream, layer)
        H, B, d = c.num_kv_heads, c.state_capacity, c.head_dim
        if B == 0:
            e = torch.empty((H, 0, d), dtype=torch.bfloat16, device=self.arena.device)
            return e, e, torch.empty((H, 0), dtype=torch.int32, device=self.arena.device), info
        kk = self._arena_view(info.k, H * B * d * 2, torch.bfloat16, (H, B, d))
        vv = self._arena_view(info.v, H * B * d * 2, torch.bfloat16, (H, B, d))
        pp = self._arena_view(info.positions, H * B * 4, torch.int32, (H, B))
        return kk, vv, pp, info

    def cache(self, stream: int, layer: int):
        """(k [Hkv][capacity][d] bf16, v, info) views into the arena."""
        import torch

        c = self.cfg
        info = statekv_cache_view(self.handle, stream, layer)
        H, cap, d = c.num_kv_heads, info.capacity, c.head_dim
        kk = self._arena_view(info.k, H * cap * d * 2, torch.bfloat16, (H, cap, d))
        vv = self._arena_view(info.v, H * cap * d * 2, torch.bfloat16, (H, cap, d))
        return kk, vv, info

    def profile(self, enable: bool):
        statekv_profile_enable(self.handle, enable)

    def profile_read(self):
        p = statekv_profile_read(self.handle)
        return [(int(p.launches[i]), float(p.milliseconds[i])) for i in range(5)]

    def sync(self) -> int:
        return statekv_sync(self.handle)

    def device_error(self) -> int:
        """Raw device status word (0 = none); see statekv_device_error."""
        return statekv_device_error(self.handle)

    def debug_check(self, stream=None) -> int:
        """Enqueue the guard-band comparison of a debug build
        (statekv_debug_check); STATEKV_ERR_UNSUPPORTED from a release build."""
        import torch

        st = (stream or torch.cuda.current_stream()).cuda_stream
        return lib().statekv_debug_check(self.handle, ctypes.c_void_p(st))

    def watchdog_selftest(self, stream=None) -> int:
        """Enqueue the failure-detection self-test (statekv_watchdog_selftest):
        the attention kernel's bounded wait on a barrier nothing completes
        expires, and the handle reports DEVICE_TIMEOUT from then on."""
        import torch

        st = (stream or torch.cuda.current_stream()).cuda_stream
        return lib().statekv_watchdog_selftest(self.handle, ctypes.c_void_p(st))
