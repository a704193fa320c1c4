"""The bounded device waits' failure path: a wait on an mbarrier that nothing
completes gives up, raises the kernel's abort flag, lets the other waiter
leave, releases TMEM and reports FKV_ETIMEOUT through the status word; the
context then keeps working (a span encode after it is bit-exact)."""
import numpy as np
import pytest
import torch

from paper_2607_07144_gb300._binding import ETIMEOUT, OK

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def fkv():
    import paper_2607_07144_gb300 as m
    m.lib()
    return m


@pytest.mark.parametrize("limit_ns", [200_000, 20_000_000])
def test_wait_gives_up_and_reports_timeout(fkv, oracle_mod, limit_ns):
    ctx = fkv.Context(256)
    assert ctx.sync_status() == OK
    res = ctx.check_bounded_wait(limit_ns)
    # [first waiter, second waiter, second left on the flag, completed phase,
    #  open phase, teardown ran]
    assert res == [0, 0, 1, 1, 0, 1]
    assert ctx.sync_status() == ETIMEOUT
    assert ctx.sync_status() == OK            # the status word was cleared
    # the context and the device stay usable
    rng = np.random.default_rng(3)
    sym = rng.integers(0, 256, size=(2, 1000)).astype(np.uint8)
    pts = ctx.span_encode(torch.from_numpy(sym).cuda()).cpu().numpy()
    assert ctx.sync_status() == OK
    want = np.stack([oracle_mod.span_encode(s, 256, ctx.r, ctx.L) for s in sym])
    assert np.array_equal(pts.view(np.uint64), want.view(np.uint64))


def test_wait_limit_is_checked(fkv):
    ctx = fkv.Context(256)
    for bad in (0, 99_999, 1_000_000_001):
        with pytest.raises(fkv.FkvError):
            ctx.check_bounded_wait(bad)
