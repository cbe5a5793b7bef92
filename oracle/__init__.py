"""CPU oracle for the WorldDynCache cached denoising rollout.

TEST INFRASTRUCTURE ONLY.  This package is a plain, slow, fp64 restatement of
the method, written from the paper, that the CUDA path is checked against.  Only
``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` / reference
legs of ``bench.py`` may import it.  The product path (the C-ABI library and its
Python binding) never imports, links or calls anything here, and this package
imports nothing from the product path; the two share no arithmetic.  Random
inputs are generated elsewhere and passed in.

Modules (each function cites the passage it follows):

* ``schedule``  -- flow-matching Euler schedule and the scheduler transition
                   Psi_t of Eq. 1.
* ``summary``   -- the lift Phi (Eq. 2), RMS normalisation, the fixed
                   256-dimensional summary s(.) and cosine similarity.
* ``surrogate`` -- transition retrieval (Eq. 3), scheduler scaling and lifted
                   evolution (Eq. 4), kernelised observation (Eq. 5).
* ``controller``-- defect proxy (Eq. 6), counterfactual defect (Eq. 7),
                   online calibration (Eq. 8), risk accumulation (Eq. 9),
                   reliability decision (Eq. 10).
* ``rollout``   -- the exact-transition bank and the cached / native rollouts
                   (section "Inference and Complexity").
* ``dit``       -- the adaLN DiT denoiser F_theta used as the exact branch.
* ``ablation``  -- the ablation variants of Tables 3 and 4 (section
                   "Ablation Study"), as switches of the steps above.
* ``diagnostics`` -- the synthetic transition diagnostics of Fig. 2 and
                   Fig. 3a.
* ``batch``     -- batched and guided rollouts (serving extensions: a batch of
                   independent trajectories; classifier-free guidance).

Parity status: the controller constants and the lift's normalisation details
are not printed in the paper (it defers them to supplementary material that is
not available).  Each such reading is stated in the docstring of the function
that makes it.  Absolute values fixed only by those readings (d_hat, R, eta_d,
the realised anchor pattern) are "parity unpinned"; the structure around them
is pinned by the tests in ``tests/test_oracle_*.py``.
"""

from . import schedule, summary, surrogate, controller, rollout, dit  # noqa: F401
from .params import CacheParams, DiTConfig  # noqa: F401
