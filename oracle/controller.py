"""Transition risk controller (Eq. 6-10).

Test infrastructure only (see the package docstring).

Section "Transition Risk Controller":
* Eq. 6  predicted defect d_hat = eta_d * p_t with the proxy
         p_t = w_z d_z + w_age d_age + w_phase d_phase + w_cam d_cam + w_depth d_depth;
* Eq. 7  counterfactual defect d_cf = mean|z_exact - z_cf| / (mean|z_exact| + eps);
* Eq. 8  eta_d <- clamp(beta_d eta_d + (1-beta_d) d_cf/(p_t+eps), eta_min, eta_max);
* Eq. 9  w_t = min{2, 1 + a_cam u_cam + a_depth u_depth + a_phase u_phase},
         Delta_t = w_t d_hat, R_cand = lambda R + Delta_t;
* Eq. 10 Surrogate iff Available_t and R_cand <= tau_risk, else Exact.

Readings of the signals the paper defers to its supplementary material
(parity unpinned for their absolute values):
* d_z     = rms(z_t - z_a) / (rms(z_a) + eps)
* d_age   = number of consecutive surrogate steps since the latest exact step
* d_phase = |q_{t-1} - q_a|  (phase distance from the anchor to the target)
* d_cam   = ||cam_t - cam_a||_2,  d_depth = ||depth_t - depth_a||_2
* u_cam   = ||cam_t||_2, u_depth = ||depth_t||_2, u_phase = q_t (remaining
            noise fraction: earlier errors have more transitions to propagate
            through, Observation 1)
"""
import numpy as np


def proxy_signals(rms_z_minus_za, rms_za, age, q_next, q_a, cam, cam_a, depth, depth_a, p):
    """The five pre-decision signals of Eq. 6 (readings in the module docstring)."""
    cam = np.asarray(cam, dtype=np.float64)
    depth = np.asarray(depth, dtype=np.float64)
    return {
        "d_z": float(rms_z_minus_za / (rms_za + p.eps)),
        "d_age": float(age),
        "d_phase": float(abs(q_next - q_a)),
        "d_cam": float(np.linalg.norm(cam - np.asarray(cam_a, dtype=np.float64))),
        "d_depth": float(np.linalg.norm(depth - np.asarray(depth_a, dtype=np.float64))),
    }


def defect_proxy(sig, p):
    """p_t of Eq. 6 (a fixed non-negative combination of the signals)."""
    return (p.w_z * sig["d_z"] + p.w_age * sig["d_age"] + p.w_phase * sig["d_phase"]
            + p.w_cam * sig["d_cam"] + p.w_depth * sig["d_depth"])


def impact_weight(cam, depth, q_t, p):
    """w_t = min{2, 1 + a_cam u_cam + a_depth u_depth + a_phase u_phase} (Eq. 9)."""
    u_cam = float(np.linalg.norm(np.asarray(cam, dtype=np.float64)))
    u_depth = float(np.linalg.norm(np.asarray(depth, dtype=np.float64)))
    u_phase = float(q_t)
    return min(2.0, 1.0 + p.a_cam * u_cam + p.a_depth * u_depth + p.a_phase * u_phase)


def candidate_risk(R, w, d_hat, p):
    """Delta_t = w_t d_hat and R_cand = lambda R + Delta_t (Eq. 9)."""
    delta = w * d_hat
    return delta, p.lam * R + delta


def counterfactual_defect(z_exact, z_cf, p, chunk=1 << 24):
    """d_cf = mean|z_exact - z_cf| / (mean|z_exact| + eps) (Eq. 7), fp64."""
    ze = np.asarray(z_exact).reshape(-1)
    zc = np.asarray(z_cf).reshape(-1)
    n = ze.size
    num = 0.0
    den = 0.0
    for s0 in range(0, n, chunk):
        a = ze[s0:s0 + chunk].astype(np.float64)
        b = zc[s0:s0 + chunk].astype(np.float64)
        num += float(np.sum(np.abs(a - b)))
        den += float(np.sum(np.abs(a)))
    return (num / n) / (den / n + p.eps)


def calibrate(eta, d_cf, p_t, p):
    """eta_d <- clamp(beta_d eta_d + (1 - beta_d) d_cf / (p_t + eps), eta_min, eta_max) (Eq. 8)."""
    v = p.beta_d * eta + (1.0 - p.beta_d) * d_cf / (p_t + p.eps)
    return float(min(max(v, p.eta_min), p.eta_max))


def available(k, T, n_bank, age, q_t, q_a, finite, supported, p):
    """Available_t of Eq. 10 (section "Reliability Decision").

    The conjunction of: a non-empty bank; an anchor of pre-decision age at most
    max_age; a compatible scheduler phase |q_t - q_a| <= q_gap_max; a finite
    candidate; adequate retrieval support; and k outside the mandatory-exact
    initialisation (k < n_init_exact) and refinement (k >= T - n_final_exact)
    phases.  Returns (flag, dict of the individual terms).
    """
    terms = {
        "bank": n_bank > 0,
        "age": age <= p.max_age,
        "phase": abs(q_t - q_a) <= p.q_gap_max,
        "finite": bool(finite),
        "support": bool(supported),
        "window": (k >= p.n_init_exact) and (k < T - p.n_final_exact),
    }
    return all(terms.values()), terms


def decide(avail, R_cand, p):
    """a_t of Eq. 10: True (Surrogate) iff Available_t and R_cand <= tau_risk."""
    return bool(avail) and (R_cand <= p.tau_risk)
