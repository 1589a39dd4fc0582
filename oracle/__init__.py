"""CPU oracle for speculative-diffusion verification (test infrastructure only).

This package is a plain, slow, fp64 restatement of what the paper computes:

* ``philox``  - Philox4x32-10 counter-based generator (Salmon et al., SC'11) and
  the uniform / Box-Muller transforms that turn its words into the random
  numbers the method draws (coins, the residual uniform, Gaussian noise).
* ``verify``  - per-step Gaussian log density ratios (Appendix A.2 log form),
  sample verification (Algorithm "token-verification"), block verification
  (Algorithm "block-verification"), the Psi_alpha CDF (Eq. u-cdf), the
  bisection U-sampler (Algorithm "u-sample"), the decomposition residual
  (Algorithm "decomposition-res") and the reflection residual (Algorithm
  "reflect-res").
* ``sampler`` - the end-to-end speculative sampler of Algorithm
  "full-block-verification" on an analytic Gaussian-mixture target with the
  Free / Frozen drafters (Section 3.3, Eq. frozen-draft-drift).

It shares no code with the CUDA path and imports nothing from it.  Only the
tests, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` / reference legs of
``bench.py`` may import it; the product path never calls it.

Parity status: every function here is pinned by a ``-m "not gpu"`` test against
closed forms, published test vectors, brute-force enumeration or statistical
identities the paper proves (see tests/test_oracle_*.py).
"""
