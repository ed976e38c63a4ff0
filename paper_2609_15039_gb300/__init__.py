"""SpliTEE masked-linear hot path on GB300 (sm_103a).

The compute lives in ``libspl.so``: hand-written CUDA kernels behind a C ABI
(declared in ``include/spl.h``).  ``paper_2609_15039_gb300.spl`` is the thin
ctypes binding with the same function names; it loads the library on first
use and raises if it is missing.  ``workloads`` draws the seeded synthetic
inputs.  Importing this package loads nothing compiled.
"""
