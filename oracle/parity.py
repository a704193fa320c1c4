"""Parity criteria between the CUDA path and the oracle -- TEST
INFRASTRUCTURE, imported only by tests/, __graft_entry__.smoke() and the
oracle leg of bench.py.  It holds comparison rules, none of the archive's
arithmetic.

* RVQ indices (Sec. 3 "Setup"): equal wherever the oracle's top-2 distance
  gap exceeds 1e-4 of the stage residual's squared norm; stage s is compared
  only where stages < s agreed (a different earlier choice changes the
  residual); closer ties that differ are counted as near-tie mismatches.
* Reconstructed K/V: a fp16/bf16 output rounded on the GPU from a float32
  stage sum must equal the oracle's float64 sum rounded to nearest-even,
  except where the float32 summation error bound straddles a rounding
  boundary (those are counted as borderline cases).
"""
from __future__ import annotations

import numpy as np

GAP = 1e-4


def compare_rvq(gpu, ora, gap, band: float = GAP):
    """gpu, ora: [n, S] indices; gap: the oracle's [n, S] gaps.
    Returns (hard mismatches, near-tie mismatches, compared entries)."""
    gpu = np.asarray(gpu)
    ora = np.asarray(ora)
    n, S = ora.shape
    prefix = np.ones(n, bool)
    hard = near = seen = 0
    for s in range(S):
        diff = (gpu[:, s] != ora[:, s]) & prefix
        h = diff & (gap[:, s] > band)
        hard += int(h.sum())
        near += int((diff & ~h).sum())
        seen += int(prefix.sum())
        prefix &= ~diff
    return hard, near, seen


def rounded_mismatches(got, ref64, dtype, absum):
    """got: the GPU's fp16/bf16 outputs as float64; ref64: the oracle's
    float64 sums; absum: the float64 sums of |c_s| (the float32 summation
    error bound is 4 * 2^-24 * absum, plus 1e-6 relative).  Returns
    (hard differences, borderline differences, compared values)."""
    from . import round_to
    got = np.asarray(got, np.float64)
    want = round_to(ref64, dtype)
    ok = got == want
    if ok.all():
        return 0, 0, got.size
    eps = 4 * 2.0 ** -24 * absum + 1e-6 * np.abs(ref64)
    borderline = round_to(ref64 - eps, dtype) != round_to(ref64 + eps, dtype)
    bad = ~(ok | borderline)
    return int(bad.sum()), int((~ok & borderline).sum()), got.size
