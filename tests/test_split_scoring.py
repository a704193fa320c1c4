"""A CPU model of the tensor-core scoring in the RVQ kernels (Sec. 3 "Setup":
the nearest codeword of every stage), against exact float64 scores.

The kernels score s_j = ||c_j||^2 - 2 r.c_j as fp16 x fp16 products
accumulated in float32: the row operand t = r 2^-(e+er) and the codeword
operand -2 c 2^-e each split into hi = fp16(v) and lo = fp16(v - hi), the
products hi*hi + lo*hi + hi*lo taken (lo*lo dropped), plus ||c_j||^2 2^-2e
in three fp16 parts against the row's 2^(10-er).  This model makes the same
splits and one float32 rounding per 16-wide K step, in the kernels' order
(norm term; per 64-wide K block hi*hi and lo*hi, then hi*lo), and checks that
its score error stays an order of magnitude inside the half tie band (5e-5 of
the stage residual's squared norm) that the parity rule excuses: the GPU can
then differ from the oracle only on near ties.  Test infrastructure: it
shares nothing with the kernels or with the oracle."""
import numpy as np
import pytest

import synth

HALF_BAND = 5e-5


def _split(v32):
    hi = v32.astype(np.float16)
    lo = (v32 - hi.astype(np.float32)).astype(np.float16)
    return hi.astype(np.float64), lo.astype(np.float64)


def _stage_scale(cb):
    """e with max |c| 2^-e in [2^8, 2^9)."""
    return int(np.frexp(float(np.abs(cb).max()))[1]) - 9


def model_scores(r, cb):
    """||c_j||^2 - 2 r.c_j as the tensor cores accumulate it, rescaled to r's units."""
    e = _stage_scale(cb)
    t = (r * 2.0 ** -e).astype(np.float32)
    m = np.abs(t).max(axis=1)
    er = np.where(m >= 4096.0, np.frexp(m)[1] - 12, 0)             # keeps |t| below 2^12
    t = (t * (2.0 ** -er)[:, None]).astype(np.float32)
    th, tl = _split(t)
    bh, bl = _split((np.float32(-2.0) * (cb.astype(np.float32) * np.float32(2.0 ** -e))).astype(np.float32))
    rest = ((cb.astype(np.float64) * 2.0 ** -e) ** 2).sum(axis=1) * 2.0 ** -10
    parts = []
    for _ in range(3):
        p = rest.astype(np.float16).astype(np.float64)
        parts.append(p)
        rest = rest - p
    aug = (2.0 ** (10 - er)).astype(np.float16).astype(np.float64)
    acc = (aug[:, None] * (parts[0] + parts[1] + parts[2])[None, :]).astype(np.float32)
    for kb in range(r.shape[1] // 64):
        steps = [slice(kb * 64 + 16 * k, kb * 64 + 16 * k + 16) for k in range(4)]
        for sl in steps:                                             # the hi piece: hi*hi, lo*hi
            acc = (acc + (th[:, sl] @ bh[:, sl].T).astype(np.float32)).astype(np.float32)
            acc = (acc + (tl[:, sl] @ bh[:, sl].T).astype(np.float32)).astype(np.float32)
        for sl in steps:                                             # the lo piece: hi*lo
            acc = (acc + (th[:, sl] @ bl[:, sl].T).astype(np.float32)).astype(np.float32)
    return acc.astype(np.float64) * (2.0 ** (2 * e + er))[:, None]


def exact_scores(r, cb):
    return (cb.astype(np.float64) ** 2).sum(axis=1)[None, :] - 2.0 * r @ cb.astype(np.float64).T


def _rows(cfg, n):
    """n head vectors of (layer 0, head 0), storage values as float64."""
    pos = np.arange(n)
    x = synth.kv_elements(cfg, 0, 0, pos // cfg.seq % cfg.batch, 0, pos % cfg.seq)
    return synth.storage_to_f64(x, cfg.dtype)


@pytest.mark.parametrize("base", [synth.CFG3, synth.CFG1], ids=["d128-bf16", "d64-fp16"])
def test_split_scores_inside_the_tie_band(base):
    cfg = synth.small_config(base, 900 + base.cfg_id, n_layers=1, batch=2, seq=300)
    cbs = np.asarray(synth.codebooks(cfg, 0))[0, 0]                  # [S, 256, D]
    r = _rows(cfg, 512)
    r[:8] *= 1e4                                                     # rows that take a shift er > 0
    worst = 0.0
    for s in range(cbs.shape[0]):
        cb = cbs[s]
        ex = exact_scores(r, cb)
        mo = model_scores(r, cb)
        rn = (r ** 2).sum(axis=1)
        rel = np.abs(mo - ex).max(axis=1) / rn
        worst = max(worst, float(rel.max()))
        assert rel.max() < HALF_BAND / 10, (s, rel.max())
        # a different argmin only where the exact top-2 gap is inside the band
        im, ie = mo.argmin(axis=1), ex.argmin(axis=1)
        diff = np.flatnonzero(im != ie)
        gap = ex[diff, im[diff]] - ex[diff, ie[diff]]
        assert np.all(gap <= 2 * HALF_BAND * rn[diff]), (s, gap / rn[diff])
        r = r - cb[ie]                                               # the next stage's residual
    assert worst > 0.0                                               # the model does round


def test_model_matches_exact_on_representable_operands():
    """Operands exact in fp16 with a codebook whose norms split exactly: the
    model has no rounding left and equals the exact scores."""
    rng = np.random.default_rng(3)
    cb = rng.integers(-64, 64, size=(256, 64)).astype(np.float64) * 2.0   # max |c| 2^-e in [2^8, 2^9) for e = -2
    cb[0, 0] = 256.0 * 2 ** -2 * 1.5
    r = rng.integers(-32, 32, size=(64, 64)).astype(np.float64)
    mo, ex = model_scores(r, cb), exact_scores(r, cb)
    assert np.array_equal(mo.argmin(axis=1), ex.argmin(axis=1))
    assert np.abs(mo - ex).max() <= 1e-9 * np.abs(ex).max()
