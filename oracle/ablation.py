"""Ablation variants of the method (section "Ablation Study", Tables 3 and 4).

Test infrastructure only (see the package docstring).

The paper names the variants and defers their definitions to supplementary
material; the readings below are the ones this implementation adopts
(parity unpinned for the paper's quality numbers, which need its weights).

Controller variants (Table 3, "Risk controller"; Tables 3-4 "Periodic"):
* periodic placement (ABL_PERIODIC): the risk test of Eq. 10 is replaced by a
  fixed period P -- after an exact step, at most P - 1 surrogate steps
  follow: Surrogate iff Available_t and age_t + 1 < P.  Available_t is kept
  (a candidate must exist and be finite).  P is chosen by the caller to
  match the risk controller's exact-call budget ("matched budget");
* instantaneous risk (ABL_INSTANT_RISK): R_cand = Delta_t, i.e. Eq. 9 with
  lambda = 0 (and R <- 0 at exact steps);
* w/o impact weighting (ABL_NO_IMPACT): w_t = 1 in Eq. 9;
* w/o CF calibration (ABL_NO_CALIB): eta_d stays eta_init (Eq. 8 is not
  applied; d_cf of Eq. 7 is still measured and reported);
* w/o support constraint (ABL_NO_SUPPORT): the compatibility filter of the
  retrieval is dropped -- N_t is the whole bank (Eq. 3's softmax runs over
  every record) and the support term of Available_t always holds.

Surrogate variants (Table 3, "Surrogate design"; Tables 3-4 "native latent
secant"):
* native latent secant (ABL_SECANT): the candidate extrapolates the latest
  exact latent displacement in the original latent space,
      z_hat = z_t + alpha_t (z_a - z_a,in),
  with z_a the latest exact output, z_a,in its input and alpha_t the
  scheduler scaling of Eq. 4; it uses no retrieval, so its support term is
  satisfied whenever the bank is non-empty;
* linear observation (ABL_LINEAR_OBS): Eq. 5's query-dependent softmax
  weights are replaced by a linear readout of the evolved summary: the
  coefficients beta that best reproduce s(phi_hat) from the bank's output
  summaries in the least-squares sense (ridge-regularised),
      (G + rho I) beta = S_out s(phi_hat),  G_ij = s_out_i . s_out_j,
      rho = ridge * trace(G) / |M_t|,
  and z_hat = sum_i beta_i z_out_i;
* no condition (ABL_NO_COND): the camera and depth descriptors are left out
  of the lifted state (their four entries each of s(phi) are zero for the
  query and for the records); the controller still sees them (Eq. 6, 9).
"""
import numpy as np

from .params import (ABL_INSTANT_RISK, ABL_LINEAR_OBS, ABL_NO_CALIB, ABL_NO_COND, ABL_NO_IMPACT,
                     ABL_NO_SUPPORT, ABL_PERIODIC, ABL_SECANT)


def lift_descriptors(cam, depth, p):
    """The condition descriptors as they enter the lifted state (Eq. 2)."""
    if p.has(ABL_NO_COND):
        return np.zeros(4), np.zeros(4)
    return cam, depth


def risk_decay(p):
    """lambda of Eq. 9 (0 for instantaneous risk)."""
    return 0.0 if p.has(ABL_INSTANT_RISK) else p.lam


def impact_weight(w_full, p):
    """w_t of Eq. 9, or 1 without impact weighting."""
    return 1.0 if p.has(ABL_NO_IMPACT) else w_full


def calibrates(p):
    """Whether Eq. 8 updates eta_d."""
    return not p.has(ABL_NO_CALIB)


def compat_filter(p):
    """Whether the retrieval restricts Eq. 3 to the compatible subset N_t."""
    return not p.has(ABL_NO_SUPPORT)


def periodic_decision(avail, age, p):
    """Surrogate iff Available_t and age_t + 1 < period (periodic placement)."""
    return bool(avail) and (age + 1 < p.period)


def secant_candidate(z_t, z_a, z_a_in, alpha):
    """z_hat = z_t + alpha (z_a - z_a,in), fp64 from the stored float32 latents."""
    z_t = np.asarray(z_t, dtype=np.float64).reshape(-1)
    z_a = np.asarray(z_a, dtype=np.float64).reshape(-1)
    z_a_in = np.asarray(z_a_in, dtype=np.float64).reshape(-1)
    return z_t + alpha * (z_a - z_a_in)


def linear_readout(s_hat, bank, p):
    """beta of the ridge least-squares readout of s(phi_hat) from the records'
    output summaries (linear observation); zeros when every s_out is 0."""
    S = np.array([rec.s_out for rec in bank], dtype=np.float64)      # [K, 256]
    G = S @ S.T
    K = len(bank)
    tr = float(np.trace(G))
    if tr == 0.0:
        return np.zeros(K)
    rho = p.ridge * tr / K
    return np.linalg.solve(G + rho * np.eye(K), S @ np.asarray(s_hat, dtype=np.float64))


__all__ = ["ABL_PERIODIC", "ABL_SECANT", "ABL_INSTANT_RISK", "ABL_NO_IMPACT", "ABL_NO_CALIB",
           "ABL_NO_SUPPORT", "ABL_LINEAR_OBS", "ABL_NO_COND", "lift_descriptors", "risk_decay",
           "impact_weight", "calibrates", "compat_filter", "periodic_decision", "secant_candidate",
           "linear_readout"]
