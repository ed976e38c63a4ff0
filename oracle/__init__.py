"""fp64 CPU oracle for the SpliTEE masked-linear path (TEST INFRASTRUCTURE).

This package is a plain, slow, obviously-correct restatement of what the
GPU path computes, written from the paper (arxiv 2609.15039):

* ``philox``      -- the counter-based generator and the noise transforms
                     (Gaussian mechanism, Prop. "eps-GDP mechanism", Sec. 4.4;
                     Laplace at the same scale as a configured alternative).
* ``linear``      -- masking x + eta, the masked product W(x + eta), the
                     correction W eta and the unmask r - W eta (Sec. 3.3.1,
                     Eq. add-and-then-subtract).
* ``bounds``      -- the floating-point cancellation bounds (Thm. 4 and
                     Eq. fp-log-bound, Sec. 4.5) and fp32 emulations of the
                     three dot products the theorem compares.
* ``sensitivity`` -- global l2 sensitivities (Thms. 1-3, Sec. 4.3).
* ``stats``       -- Kolmogorov-Smirnov statistic against closed-form CDFs.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py`` (its
``cpu_baseline`` leg and ``--impl reference`` arm) may import this package.
The CUDA product path never imports, links or runs anything from here, and
nothing here imports the CUDA path: the two share no code.
"""

from . import bounds, linear, philox, sensitivity, stats  # noqa: F401
