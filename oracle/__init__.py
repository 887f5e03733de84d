"""CPU oracle for QSVD's latent-attention path (arxiv 2510.16292).

TEST INFRASTRUCTURE ONLY.  This package is the plain, slow, obviously correct
definition of what the GPU path computes, written from the paper in numpy
(fp64 for real arithmetic, int64 for integer arithmetic; fp32 steps the
quantizer fixes are emulated by rounding each fp64 result to fp32).  Only the
tests, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` / reference leg of
``bench.py`` may import it.  It shares no code with the CUDA library and
imports nothing from it; the only module both sides use is ``synthetic``
(seeded random inputs, none of the method's arithmetic).

Modules and the passages they follow:

* ``svd``       -- rank-r truncated SVD (Eq. 1), joint QKV SVD and the beta
                   split (Eq. 2-4), with a one-sided Jacobi SVD of our own.
* ``quant``     -- per-token / per-channel symmetric round-to-nearest
                   quantizers (Sec. 4 experimental setup; Eq. 11-12), the int4
                   group variant and nibble packing of the latent cache.
* ``latent``    -- the quantized down-projection C = Q(X) Q(W_d) (Eq. 12),
                   its dequantization and per-token requantization into the
                   latent cache (Eq. 11, Q(C_qkv)); cache append.
* ``attention`` -- decode attention over the latent cache with K = C W_k^u,
                   V = C W_v^u materialised explicitly (Eq. 5), plus the
                   absorbed form used only as a cross-check.
* ``cost``      -- weight / cache / FLOP counts and the R1, R2 ratios
                   (Sec. 3.1, Eq. 15).
* ``pipeline``  -- a workload driver: prefill, then decode steps.

Parity status: every function here is pinned by ``tests/test_oracle_*.py``
against closed forms, brute force, library routines used as independent
checks, or values the paper prints (``tests/golden``).
"""
from . import svd, quant, latent, attention, cost, pipeline  # noqa: F401
