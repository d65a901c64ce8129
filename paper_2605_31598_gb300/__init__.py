"""GB300 (sm_103a) StateKV per-frame video-prefill step.

The compute path lives in the C-ABI library ``libstatekv.so`` (see
``include/statekv.h``); ``statekv`` is its ctypes binding and ``inputs`` the
seeded synthetic-input generator.
"""
from .statekv import StateKV, StateKVError, lib, make_config  # noqa: F401
