"""The C-ABI library builds, loads and exports every symbol include/fkv.h
declares; its host-only geometry helpers agree with the oracle.  No kernel
launches (no GPU needed)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "fkv.h")


def _declared():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(fkv_[a-z_0-9]+)\s*\(", src)))


@pytest.fixture(scope="module")
def libfkv():
    from paper_2607_07144_gb300 import build
    build.build()
    return ctypes.CDLL(build.LIB)


def test_every_declared_symbol_is_exported(libfkv):
    names = _declared()
    assert len(names) >= 20
    for n in names:
        assert hasattr(libfkv, n), n


def test_binding_covers_the_header():
    from paper_2607_07144_gb300 import _binding
    assert set(_declared()) == set(_binding.SIGNATURES)


def test_host_geometry_matches_oracle(libfkv, oracle_mod):
    from paper_2607_07144_gb300 import _binding
    L = _binding.lib()
    for N in [3, 4, 5, 6, 8, 16, 64, 100, 256, 257, 512, 1000, 1024]:
        assert L.fkv_packing_ratio(N) == oracle_mod.packing_ratio(N)
        r = oracle_mod.packing_ratio(N)
        assert L.fkv_max_span_len(r) == oracle_mod.max_span_len(r)
    assert L.fkv_packing_ratio(2) == 0.0 and L.fkv_packing_ratio(1025) == 0.0
    assert L.fkv_max_span_len(0.0) == 0 and L.fkv_max_span_len(0.6) == 0


def test_create_rejects_bad_parameters_without_touching_the_gpu(libfkv):
    from paper_2607_07144_gb300 import _binding
    L = _binding.lib()
    h = ctypes.c_void_p()
    r4 = L.fkv_packing_ratio(4)
    assert L.fkv_create(2, 0.5, 4, None, ctypes.byref(h)) == _binding.EINVAL
    assert L.fkv_create(4, r4 * 1.001, 4, None, ctypes.byref(h)) == _binding.EINVAL   # r > r_N
    assert L.fkv_create(4, r4, 45, None, ctypes.byref(h)) == _binding.EINVAL          # span too long
    assert L.fkv_create(4, r4, 0, None, ctypes.byref(h)) == _binding.EINVAL
    assert L.fkv_create(1025, 0.003, 4, None, ctypes.byref(h)) == _binding.EINVAL     # N above 1024
    assert L.fkv_symbol_bytes(None) == 0
    assert not h.value
