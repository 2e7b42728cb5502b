"""CPU oracle for the Spectral-LSH compression pass (arXiv 2607.19368).

TEST INFRASTRUCTURE ONLY.  This package is the plain, slow, obviously correct
statement of what the compression pass computes.  Only the tests, the package
smoke check and the benchmark's CPU-baseline leg may import it; the product
path (the CUDA library and its Python binding) never does, and shares no code
with it.

Everything is numpy, float64 unless the method fixes a precision (SimHash's
float32 chain).  Each function cites the part of the paper it follows.  Where
the paper is silent or ambiguous the reading taken is stated in the docstring.

Parity pins: every function here is pinned by tests under ``tests/`` against
something other than itself (closed forms, dense eigendecompositions, the
RFF expectation, collision statistics, invariants, brute force on tiny inputs,
and values printed in the paper).  The paper's end metrics (perplexity, KL)
need models and datasets that are not available: parity unpinned, not built.
"""
from .spectral_lsh import *  # noqa: F401,F403
from .spectral_lsh import __all__  # noqa: F401
