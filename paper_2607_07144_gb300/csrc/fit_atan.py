"""Coefficients of the span decoder's arctangent (decode_core.cuh, kAtan).

The decoder's sector test needs the angle of a direction to about 1e-5 rad.
After an octant reduction the argument u = min(|x|, |y|) / max(|x|, |y|) lies
in [0, 1], and atan u is approximated by the odd polynomial
    u (a1 + a3 u^2 + a5 u^4 + a7 u^6 + a9 u^8).
The coefficients come from least squares at Chebyshev nodes of [0, 1],
reweighted toward the points of largest error until the error is close to
equal-ripple (a cheap stand-in for a minimax fit), then rounded to float32.
The script prints them and the largest error of the float32 Horner evaluation
the kernel performs, against numpy's float64 arctan, on 2^22 + 1 points of
[0, 1].

Run: python fit_atan.py
"""
import numpy as np

TERMS = 5          # a1, a3, a5, a7, a9
NODES = 4000
ROUNDS = 30


def fit():
    k = np.arange(NODES)
    u = 0.5 - 0.5 * np.cos(np.pi * (k + 0.5) / NODES)
    A = np.stack([u ** (2 * i + 1) for i in range(TERMS)], axis=1)
    y = np.arctan(u)
    w = np.ones(NODES)
    for _ in range(ROUNDS):
        c, *_ = np.linalg.lstsq(A * w[:, None], y * w, rcond=None)
        e = np.abs(A @ c - y)
        w = w * (1.0 + 50.0 * e / e.max())
        w /= w.max()
    return c.astype(np.float32)


def horner32(c32: np.ndarray, u: np.ndarray) -> np.ndarray:
    """u (a1 + u^2 (a3 + ...)) in float32, one rounding per operation, as the
    kernel evaluates it (its fused multiply-adds round once, so they are no
    less accurate than this)."""
    u = u.astype(np.float32)
    u2 = (u * u).astype(np.float32)
    p = np.float32(c32[-1])
    for a in c32[-2::-1]:
        p = (p * u2 + a).astype(np.float32)
    return (p * u).astype(np.float32)


def max_error(c32: np.ndarray, points: int = (1 << 22) + 1) -> float:
    u = np.linspace(0.0, 1.0, points)
    return float(np.max(np.abs(horner32(c32, u).astype(np.float64) - np.arctan(u.astype(np.float32)))))


if __name__ == "__main__":
    c = fit()
    for i, a in enumerate(c):
        print("a%d = %.9e" % (2 * i + 1, a))
    print("max |error| = %.3e rad" % max_error(c))
