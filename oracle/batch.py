"""Batched and guided cached rollouts: serving extensions around the method.

Test infrastructure only (see the package docstring).

The paper rolls out one trajectory at a time (section "Inference and
Complexity") and never mentions classifier-free guidance.  The readings the
CUDA path is checked against:

* A batch is a set of independent trajectories.  Sample b keeps its own
  exact-transition bank, risk state and controller constants, and its rollout
  is the single-trajectory cached rollout of Eq. 1-10 on its own latent and
  condition; running several samples' exact steps in one denoiser call changes
  how the work is scheduled, not what any sample computes.
* Classifier-free guidance: the velocity of a guided sample is
      v = F(z, t, null) + g (F(z, t, c) - F(z, t, null)),
  with ``null`` the all-zero condition-token set.  That v is the F_theta of
  Eq. 1 for the sample: it drives the exact transition Psi and the
  counterfactual defect of Eq. 7.

Parity status: pinned by the closed forms of the guidance formula (g = 1 gives
the conditional velocity, g = 0 the unconditional one, the result is affine in
g, a zero condition makes it independent of g) and by batch equivariance
(permuting the samples permutes the results; a batch of one is the single
rollout), ``tests/test_oracle_batch.py``.
"""
import numpy as np

from . import dit
from .rollout import cached_rollout


def null_tokens(cfg):
    """The null condition of guidance: all-zero condition tokens."""
    return np.zeros((cfg.cond_tokens, cfg.cond_dim), dtype=np.float64)


def guided_velocity(v_cond, v_null, g):
    """v = v_null + g (v_cond - v_null), in fp64."""
    v_cond = np.asarray(v_cond, dtype=np.float64)
    v_null = np.asarray(v_null, dtype=np.float64)
    return v_null + g * (v_cond - v_null)


def denoiser(Wt, cfg, tokens, guidance=None):
    """F_theta(z, t, c) of the DiT with fixed condition tokens, as the
    ``denoiser(z, t, cond, k)`` the rollouts take; with ``guidance`` g the
    guided velocity of the same tokens against the null condition."""
    shape = (cfg.in_ch, cfg.frames, cfg.height, cfg.width)

    def F(z, t, c, k):
        zz = np.asarray(z).reshape(shape)
        vc = dit.forward(Wt, cfg, zz, t, tokens)
        if guidance is None:
            return vc
        return guided_velocity(vc, dit.forward(Wt, cfg, zz, t, null_tokens(cfg)), guidance)

    return F


def rollout_batch(z_Ts, denoisers, conds, sigmas, params):
    """Cached rollouts of B independent samples: sample b starts from
    z_Ts[b], runs its exact steps through denoisers[b] with conds[b] and
    controller constants params[b].  Returns (finals, decisions, traces),
    one entry per sample."""
    finals, decisions, traces = [], [], []
    for z, F, c, p in zip(z_Ts, denoisers, conds, params):
        zf, dec, tr = cached_rollout(z, F, c, sigmas, p)
        finals.append(zf)
        decisions.append(dec)
        traces.append(tr)
    return finals, decisions, traces
