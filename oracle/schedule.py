"""Flow-matching Euler schedule and the scheduler transition Psi_t (Eq. 1).

Test infrastructure only (see the package docstring).

The paper writes the exact transition as z_{t-1} = Psi_t(z_t, F_theta(z_t,t,c))
(Eq. 1, section "Overview"; also the Introduction) and leaves Psi_t to the
backbone.  The workloads here use a flow-matching Euler scheduler.  Index
convention: step k = 0..T-1 maps z_k to z_{k+1}; the paper's t counts down, so
its z_t is z_k with k = T - t.
"""
import numpy as np


def sigmas(T, shift=1.0):
    """Noise levels sigma_k = 1 - k/T for k = 0..T (fp64).

    With shift s != 1 the usual flow-matching time shift
    sigma' = s*sigma / (1 + (s-1)*sigma) is applied.  Reading: the paper does
    not name its schedule; these are the textbook flow-matching Euler values.
    """
    if T <= 0:
        raise ValueError("T must be positive")
    s = 1.0 - np.arange(T + 1, dtype=np.float64) / float(T)
    if shift != 1.0:
        s = shift * s / (1.0 + (shift - 1.0) * s)
    return s


def model_timestep(sigma):
    """Timestep fed to the denoiser: t = 1000 * sigma."""
    return 1000.0 * np.asarray(sigma, dtype=np.float64)


def phase(sigma):
    """Normalised scheduler phase q.

    Section "Condition-Aware Lifted State": when no scheduler phase is
    available the normalised timestep replaces it; here q_k = sigma_k in [0,1].
    """
    return np.asarray(sigma, dtype=np.float64)


def psi(z, v, sigma_k, sigma_k1):
    """Scheduler transition Psi (Eq. 1): Euler step z + (sigma_{k+1}-sigma_k) v."""
    return np.asarray(z, dtype=np.float64) + (float(sigma_k1) - float(sigma_k)) * np.asarray(v, dtype=np.float64)
