"""fp64 CPU oracle for the SubZero+ subspace zeroth-order weight path.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path may import, call or
execute this package: only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline / ``--impl reference`` legs of ``bench.py`` use it.  It shares no
code with the CUDA library (``paper_2608_15665_gb300/csrc``): the two sides
implement the same published definitions independently.

What it computes, in plain fp64 numpy, one matrix at a time, in the paper's
order (SubZero+, arXiv 2608.15665):

* ``rng``      -- the counter-based Gaussian contract: Philox4x32-10 (Salmon et
                  al., SC'11) and Box-Muller; the seeds of Alg. 2 / Alg. 3.
* ``rounding`` -- rounding of an exact fp64 value to the weight storage dtype
                  (bf16 / fp32, round-to-nearest-even, one rounding per pass).
* ``haar``     -- Alg. 1 (Haar-distributed bases): thin Householder QR of a Gaussian
                  matrix followed by the sign correction of Eq. (11).
* ``subzero``  -- Alg. 2 (the in-place perturbation) as a fused pass W <- rnd(W + U C V^T),
                  the multi-query estimator of Eq. (6), the subspace Adam of
                  Eqs. (7)-(10), and the Alg. 3 schedule driver.
* ``mezo``     -- the full-space SPSA perturbation of Eq. (1) (MeZO's baseline):
                  W <- rnd(W + coef Z) with Z i.i.d. N(0,1) per element.

Pins (tests/test_oracle_*.py) tie each function to something other than
itself: published known-answer vectors, closed forms, uniqueness of the
positive-diagonal QR, brute-force Haar moments, a hand-computed 2x2 Adam step.
"""

from . import rng, rounding, haar, subzero, mezo  # noqa: F401
