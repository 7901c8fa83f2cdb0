"""Comparison of CUDA-path outputs with oracle outputs (test helper).

Reading of "codes identical except at rounding ties" used throughout: a code
that differs from the oracle's is accepted when it is
  (a) a tie: the oracle's w/scale lies within tau (in grid steps) of a
      rounding boundary, or its group's zero point was a tie;
  (b) downstream of an accepted tie: later in the same row (the OBS feedback
      carries the other rounding decision forward along the row), or, when
      Block-GD is on, in a later column block than the tie (the gradient
      couples all rows after every block).
Everything else is an unexplained mismatch and fails the test.
"""
from __future__ import annotations

import numpy as np


def unpack(codes: np.ndarray, n: int) -> np.ndarray:
    lo = (codes & 15).astype(np.int64)
    hi = (codes >> 4).astype(np.int64)
    return np.stack([lo, hi], axis=2).reshape(codes.shape[0], -1)[:, :n]


def compare_codes(gpu_codes: np.ndarray, orc: dict, block_size: int, group_size: int, bgd: bool, tau: float = 1e-3):
    ref = orc["codes"]
    m, n = ref.shape
    g = group_size if group_size > 0 else n
    mism = gpu_codes != ref
    tie = orc["margin"] < tau
    ztie = np.repeat(orc["zero_margin"] < tau, g, axis=1)[:, :n]
    tie = tie | ztie
    explained = np.zeros_like(mism)
    first_block = None
    unexplained_first = []
    for i in np.nonzero(mism.any(axis=1))[0]:
        j0 = int(np.nonzero(mism[i])[0][0])
        if tie[i, j0]:
            explained[i, j0:] = True
            b = j0 // block_size
            first_block = b if first_block is None else min(first_block, b)
        else:
            unexplained_first.append((int(i), j0, float(orc["margin"][i, j0])))
    if bgd and first_block is not None:
        explained[:, (first_block + 1) * block_size:] = True
    unexpl = mism & ~explained
    compare_codes.last_explained = explained
    return {
        "frac_equal": 1.0 - float(mism.mean()),
        "n_mismatch": int(mism.sum()),
        "n_unexplained": int(unexpl.sum()),
        "unexplained_first": unexplained_first[:10],
        "n_ties_total": int(tie.sum()),
    }


def scale_agreement(gpu_scale: np.ndarray, orc_scale: np.ndarray, group_size: int, rtol: float = 1e-5,
                    explained: np.ndarray = None, adam_bound: np.ndarray = None):
    """(fraction of groups within rtol, median relative error, groups off by more
    than rtol that are neither downstream of an accepted tie nor within
    adam_bound).

    adam_bound (per group, absolute): a scale is (xmax - xmin) / (2^b - 1); an
    optimizer step whose gradient entry is within rounding of zero may take the
    other sign, moving that weight by 2 lr, so a group whose extreme weight had
    such an entry before its parameters were computed can differ by up to
    2 * 2 lr * steps / (2^b - 1).  The test passes that bound in."""
    diff = np.abs(gpu_scale.astype(np.float64) - orc_scale.astype(np.float64))
    rel = diff / np.abs(orc_scale.astype(np.float64))
    bad = rel > rtol
    if adam_bound is not None:
        bad = bad & (diff > adam_bound)
    n_unexpl = int(bad.sum())
    if explained is not None:
        m, n = explained.shape
        g = group_size if group_size > 0 else n
        first_cols = np.arange(gpu_scale.shape[1]) * g
        n_unexpl = int((bad & ~explained[:, first_cols]).sum())
    return float((~bad).mean()), float(np.median(rel)), n_unexpl
