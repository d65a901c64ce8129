"""Layer-level selection (selection = 2, App. A): one top-B per (stream,
layer) by the importance summed over every KV head, applied to all heads.

Teacher-forced parity against the oracle's policy 2: outputs, per-head
importance, the kept set outside the 1e-3 band of the layer-level score,
identical positions in every head, and bit-exact state rows and cache.
"""
import dataclasses

import pytest

from paper_2605_31598_gb300.inputs import WORKLOADS

from .parity import run_parity


@pytest.mark.gpu
def test_layer_selection_toy_all_frames():
    stats = {}
    run_parity(WORKLOADS["toy"], 8, selection=2, stats=stats)
    assert stats["decisions"] > 0


@pytest.mark.gpu
def test_layer_selection_peaked_7b_layer():
    """Peaked inputs (C2 shapes without the 1/sqrt(d) factor) admit tens of
    frame tokens per frame, so most decisions fall outside the band."""
    shape = dataclasses.replace(WORKLOADS["qwen7b_layer"], max_frames=14)
    stats = {}
    run_parity(shape, 14, kind="peaked", check_frames=[9, 10, 11, 14], selection=2, stats=stats)
    print("layer-level peaked", stats)
    assert stats["band_candidates"] < stats["decisions"]


@pytest.mark.gpu
def test_layer_selection_multi_layer_split_calls():
    shape = dataclasses.replace(WORKLOADS["toy"], num_streams=2, num_layers=3)
    run_parity(shape, 5, call_layers=[(0, 2), (2, 1)], selection=2, kind="peaked")
