"""The span decoder's arctangent polynomial (decode_core.cuh kAtan, from
paper_2607_07144_gb300/csrc/fit_atan.py) against numpy's float64 arctan: its
float32 evaluation stays inside the 1.2e-5 rad the sector test's threshold
assumes, and the octant reflections rebuild atan2 over the whole circle."""
import os
import re
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2607_07144_gb300", "csrc")
sys.path.insert(0, CSRC)
import fit_atan  # noqa: E402

BOUND = 1.2e-5     # the arctangent term of the error bound in fkv_create and classify


def kernel_coefficients():
    src = open(os.path.join(CSRC, "decode_core.cuh")).read()
    body = re.search(r"kAtan\[5\]\s*=\s*\{([^}]*)\}", src).group(1)
    return np.array([float(x.strip().rstrip("f")) for x in body.split(",")], dtype=np.float32)


def test_coefficients_match_the_fit():
    assert np.array_equal(kernel_coefficients(), fit_atan.fit())


def test_float32_error_within_bound():
    err = fit_atan.max_error(kernel_coefficients())
    assert err < BOUND
    # endpoints and the octant edge
    c = kernel_coefficients()
    assert fit_atan.horner32(c, np.array([0.0]))[0] == 0.0
    assert abs(float(fit_atan.horner32(c, np.array([1.0]))[0]) - np.pi / 4) < BOUND


def test_reflections_rebuild_the_angle():
    """Octant reduction and reflections as the kernel does them (float32),
    over directions all around the circle, against arctan2."""
    c = kernel_coefficients()
    rng = np.random.default_rng(5)
    th = rng.uniform(-np.pi, np.pi, 200000)
    th = np.concatenate([th, np.arange(-8, 9) * np.pi / 4])      # axes and diagonals
    x = np.cos(th).astype(np.float32)
    y = np.sin(th).astype(np.float32)
    ax, ay = np.abs(x), np.abs(y)
    mx, mn = np.maximum(ax, ay), np.minimum(ax, ay)
    u = np.where(mx > 0, mn / np.where(mx > 0, mx, 1), 0).astype(np.float32)
    ph = fit_atan.horner32(c, u)
    ph = np.where(ay > ax, np.float32(1.57079637) - ph, ph).astype(np.float32)
    ph = np.where(x < 0, np.float32(3.14159274) - ph, ph).astype(np.float32)
    ph = np.where(y < 0, -ph, ph).astype(np.float32)
    ref = np.arctan2(y.astype(np.float64), x.astype(np.float64))
    d = np.abs(ph.astype(np.float64) - ref)
    d = np.minimum(d, 2 * np.pi - d)                              # -pi and pi are one direction
    assert d.max() < BOUND + 1.5e-6
