"""Synthetic latent-transition diagnostics (section "Motivation and
Observations", Fig. 2; section "Transition Risk Controller", Fig. 3),
computed with the oracle's own rollout pieces.

Test infrastructure only (see the package docstring).

The paper defers the experimental details to supplementary material; these
are the readings used (the CUDA-side counterpart in the package follows the
same text):

* Single-injection downstream impact (Observation 1, Fig. 2a-b).  Run the
  all-exact trajectory z_0..z_T with the cache's bookkeeping active (tau_risk
  < 0, so every step is exact but a counterfactual candidate z_hat_t is built
  whenever the bank is non-empty).  For an injection step t, commit z_hat_t
  instead of the exact z_{t+1} and resume exact inference to the end:
      d_t      = mean|z_{t+1} - z_hat_t| / (mean|z_{t+1}| + eps)   (Eq. 7 form)
      D_down_t = ||z_T^inj - z_T|| / ||z_T||                         (relative L2)
  together with the controller's d_hat_t, w_t and Delta_t = w_t d_hat_t at
  that step.  With thresholds tau_d, tau_D an injection is a false-safe case
  of the instantaneous criterion when d_t <= tau_d but D_down_t > tau_D, and
  of the future-weighted criterion when w_t d_t <= tau_d but D_down_t > tau_D
  (rates over all injections).
* Direction error over a cache streak (Observation 2, Fig. 2c).  Roll out
  with periodic placement (exact every P steps); at every step with a
  candidate, from the same current state z_t, the angle between the
  approximate increment z_hat_t - z_t and the exact increment
  Psi(z_t, F(z_t)) - z_t, binned by the streak position (the pre-decision age).
* Predicted versus counterfactual defect at exact anchors (Fig. 3a): the
  pairs (d_hat_t, d_cf_t) of a cached rollout's exact steps that had a
  supported, finite candidate, with their Pearson and Spearman correlations.
"""
import numpy as np

from . import rollout as ro
from . import schedule as sch


def _rel_l2(a, b):
    a = np.asarray(a, dtype=np.float64).reshape(-1)
    b = np.asarray(b, dtype=np.float64).reshape(-1)
    return float(np.linalg.norm(a - b) / np.linalg.norm(b))


def _angle(u, v):
    """Angle between two increments; a zero increment carries no direction
    and counts as orthogonal (pi/2)."""
    u = np.asarray(u, dtype=np.float64).reshape(-1)
    v = np.asarray(v, dtype=np.float64).reshape(-1)
    nu, nv = np.linalg.norm(u), np.linalg.norm(v)
    if nu == 0.0 or nv == 0.0:
        return float(np.pi / 2)
    c = float(np.dot(u, v) / (nu * nv))
    return float(np.arccos(min(1.0, max(-1.0, c))))


def _ranks(x):
    x = np.asarray(x, dtype=np.float64)
    order = np.argsort(x, kind="stable")
    r = np.empty(len(x))
    r[order] = np.arange(len(x), dtype=np.float64)
    return r


def correlations(a, b):
    """(Pearson, Spearman) of two equal-length samples (no ties expected)."""
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    pear = float(np.corrcoef(a, b)[0, 1])
    spear = float(np.corrcoef(_ranks(a), _ranks(b))[0, 1])
    return pear, spear


def all_exact_with_candidates(z_T, denoiser, conds, sigmas, p):
    """The all-exact run with the cache's bookkeeping (tau_risk < 0).  Returns
    (latents z_0..z_T as float32, per-step infos, per-step candidates or None)."""
    T = len(sigmas) - 1
    z = ro._f32(z_T).reshape(-1)
    state = ro.CacheState.initial(z, sigmas, p)
    zs, infos, cands = [z], [], []
    for k in range(T):
        c = conds[k] if isinstance(conds, (list, tuple)) else conds
        z_hat, info = ro.surrogate_step(state, z, k, c, sigmas, p)
        assert info["decision"] == 0
        v = denoiser(z, float(sch.model_timestep(sigmas[k])), c, k)
        z = ro.exact_step(state, z, v, z_hat, k, c, sigmas, p, info)
        zs.append(z)
        infos.append(info)
        cands.append(z_hat if (z_hat is not None and info["supported"] and info["finite"]) else None)
    return zs, infos, cands


def native_from(z, k0, denoiser, conds, sigmas):
    """Exact inference from latent z at step k0 to the end."""
    T = len(sigmas) - 1
    z = ro._f32(z).reshape(-1)
    for k in range(k0, T):
        c = conds[k] if isinstance(conds, (list, tuple)) else conds
        v = denoiser(z, float(sch.model_timestep(sigmas[k])), c, k)
        z = ro._f32(sch.psi(z, np.asarray(v).reshape(-1), sigmas[k], sigmas[k + 1]))
    return z


def downstream_impact(z_T, denoiser, conds, sigmas, p, steps=None, tau_d=0.025, tau_D=0.06):
    """Single-injection diagnostics (module docstring).  ``p.tau_risk`` must be
    negative.  Returns a dict with per-injection rows and the false-safe rates."""
    assert p.tau_risk < 0
    zs, infos, cands = all_exact_with_candidates(z_T, denoiser, conds, sigmas, p)
    rows = []
    for t, zh in enumerate(cands):
        if zh is None or (steps is not None and t not in steps):
            continue
        z_inj = native_from(zh, t + 1, denoiser, conds, sigmas)
        info = infos[t]
        rows.append({"t": t, "d": float(info["d_cf"]), "D_down": _rel_l2(z_inj, zs[-1]),
                     "d_hat": float(info["d_hat"]), "w": float(info["w"]), "delta": float(info["delta"])})
    n = max(1, len(rows))
    inst = sum(1 for r in rows if r["d"] <= tau_d and r["D_down"] > tau_D) / n
    fut = sum(1 for r in rows if r["w"] * r["d"] <= tau_d and r["D_down"] > tau_D) / n
    return {"rows": rows, "false_safe_instantaneous": inst, "false_safe_future_weighted": fut}


def proxy_vs_counterfactual(z_T, denoiser, conds, sigmas, p):
    """(d_hat_t, d_cf_t) at the exact anchors of a cached rollout (Fig. 3a)."""
    _, _, trace = ro.cached_rollout(z_T, denoiser, conds, sigmas, p)
    return [(float(i["d_hat"]), float(i["d_cf"])) for i in trace if i["decision"] == 0 and np.isfinite(i["d_cf"])]


def direction_errors(z_T, denoiser, conds, sigmas, p):
    """Direction error over cache streaks (module docstring); ``p`` should use
    periodic placement.  Returns per-step rows (k, streak position, angle,
    decision) and the mean angle per streak position."""
    T = len(sigmas) - 1
    z = ro._f32(z_T).reshape(-1)
    state = ro.CacheState.initial(z, sigmas, p)
    rows = []
    for k in range(T):
        c = conds[k] if isinstance(conds, (list, tuple)) else conds
        age = state.age
        z_hat, info = ro.surrogate_step(state, z, k, c, sigmas, p)
        v = denoiser(z, float(sch.model_timestep(sigmas[k])), c, k)
        z_ex = ro._f32(sch.psi(z, np.asarray(v).reshape(-1), sigmas[k], sigmas[k + 1]))
        if z_hat is not None and info["supported"] and info["finite"]:
            rows.append({"k": k, "streak": age, "angle": _angle(z_hat.astype(np.float64) - z, z_ex.astype(np.float64) - z),
                         "decision": info["decision"]})
        if info["decision"] == 1:
            z = z_hat
        else:
            z = ro.exact_step(state, z, v, z_hat, k, c, sigmas, p, info)
    by = {}
    for r in rows:
        by.setdefault(r["streak"], []).append(r["angle"])
    return {"rows": rows, "mean_by_streak": {s: float(np.mean(a)) for s, a in sorted(by.items())}}
