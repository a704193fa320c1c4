"""GB300-native fractal KV-cache archive (arXiv 2607.07144).

The library is libfkv.so (C ABI in include/fkv.h, CUDA kernels for sm_103a);
this package is its thin Python binding.  Build with
``paper_2607_07144_gb300.build.build()`` or ``__graft_entry__.build()``.
"""
from ._binding import (BF16, F16, F32, Context, FkvError, Streams, cache_view, lib,  # noqa: F401
                       max_span_len, measure_fp64_rate, packing_ratio)

__all__ = ["Context", "Streams", "FkvError", "lib", "packing_ratio", "max_span_len", "cache_view", "measure_fp64_rate",
           "F32", "F16", "BF16"]
