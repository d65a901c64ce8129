"""App. A assumption diagnostics over device tensors (argument marshalling).

The paper checks its two assumptions on the full-attention baseline: layer-level
scores (attention summed over the frame's queries within each head, then over
the heads), the concentration C_{n,B} of historical attention in the top-B
historical tokens (App. A.1), and the candidate-pool recall, weighted recall,
retention and churn of consecutive top-B oracle states (App. A.2).  The sums
and the top-B sets are computed by the library's kernels
(``statekv_topb_mask``, ``statekv_concentration_sums``,
``statekv_state_metrics``); this module passes device pointers and divides the
returned sums.
"""
from __future__ import annotations

from .statekv import (check, statekv_concentration_sums, statekv_state_metrics,
                      statekv_topb_mask)


def _stream(stream):
    import torch

    return (stream or torch.cuda.current_stream()).cuda_stream


def topb_mask(scores, n: int, B: int, *, stream=None):
    """uint8 mask [rows][stride] of the top-B of ``scores[:, :n]`` (fp32
    [rows][stride], device), ties to the lower position."""
    import torch

    rows, stride = scores.shape
    mask = torch.empty((rows, stride), dtype=torch.uint8, device=scores.device)
    check(statekv_topb_mask(scores.data_ptr(), rows, n, stride, B, mask.data_ptr(),
                            _stream(stream)), "statekv_topb_mask")
    return mask


def concentration(scores, n_hist: int, budgets, *, stream=None):
    """C_{n,B} per row for each budget: fp64 numpy [rows][len(budgets)].
    ``scores``: layer-level scores of frame n (fp32 [rows][stride], device),
    whose first ``n_hist`` columns are the keys of earlier frames."""
    import numpy as np
    import torch

    rows, stride = scores.shape
    out = torch.empty((len(budgets), rows, 2), dtype=torch.float64, device=scores.device)
    for i, B in enumerate(budgets):
        mask = topb_mask(scores, n_hist, B, stream=stream)
        check(statekv_concentration_sums(scores.data_ptr(), mask.data_ptr(), rows, n_hist, stride,
                                         out[i].data_ptr(), _stream(stream)),
              "statekv_concentration_sums")
    o = out.cpu().numpy()
    return (o[:, :, 0] / o[:, :, 1]).T.copy()


def state_metrics(scores_n, scores_next, n_seen: int, T: int, B: int, *, stream=None) -> dict:
    """App. A.2 per row.  ``scores_n``: frame n's layer-level scores over the
    ``n_seen`` tokens seen up to and including frame n; ``scores_next``: frame
    n + 1's over ``n_seen + T`` tokens (both fp32 [rows][stride], device).
    Returns numpy arrays: recall, weighted_recall, retention, churn."""
    import torch

    rows, stride = scores_next.shape
    s_n = topb_mask(scores_n, n_seen, B, stream=stream)
    s_next = topb_mask(scores_next, n_seen + T, B, stream=stream)
    out = torch.empty((rows, 6), dtype=torch.float64, device=scores_next.device)
    check(statekv_state_metrics(s_n.data_ptr(), s_next.data_ptr(), scores_next.data_ptr(), rows,
                                n_seen, T, stride, out.data_ptr(), _stream(stream)),
          "statekv_state_metrics")
    o = out.cpu().numpy()
    return {
        "recall": o[:, 0] / o[:, 1],
        "weighted_recall": o[:, 2] / o[:, 3],
        "retention": o[:, 4] / o[:, 5],
        "churn": (o[:, 1] - o[:, 4]) / o[:, 1],
    }
