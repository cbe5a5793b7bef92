"""Cached denoising rollout (section "Inference and Complexity") and its
per-step pieces, plus the native rollout it replaces.

Test infrastructure only (see the package docstring).

One step k (z_k -> z_{k+1}, phase q_k = sigma_k, target q_{k+1}):

1. Lift the current state: s(phi_k) with the current anchor z_a and history
   h(H) (Eq. 2).
2. If the bank is non-empty, run the surrogate head (Eq. 3-5); if N_t gives
   adequate support, build the candidate z_hat = sum kappa_i z_out_i (Eq. 5).
   The candidate is built at every step with a non-empty bank, mandatory-exact
   steps included, so exact steps always have their pre-insertion
   counterfactual (section "Transition Risk Controller", Eq. 7).
3. Proxy p_k, prediction d_hat = eta p_k (Eq. 6), weight w, increment Delta,
   candidate risk R_cand (Eq. 9), Available (Eq. 10), decision.
4. Surrogate: R <- R_cand, age += 1, commit z_hat.
   Exact: z_ex = Psi(z_k, F(z_k, t_k, c)), R <- lambda R; with a supported
   finite counterfactual, d_cf (Eq. 7) and the calibration of Eq. 8; insert
   the record (lifted with the pre-insertion anchor and history, so there is
   no self-retrieval) into the FIFO bank; the anchor becomes z_ex, age = 0.

Latents are stored as float32 between steps (the storage type of the CUDA
path); all arithmetic is fp64.
"""
from dataclasses import dataclass, field

import numpy as np

from . import ablation as ab
from . import controller as ctl
from . import schedule as sch
from .params import OBS_RESIDUAL
from . import summary as sm
from . import surrogate as sg


def _f32(x):
    return np.asarray(x, dtype=np.float64).astype(np.float32)


@dataclass
class CacheState:
    """Controller and memory state carried across steps (D1/D2 of the method)."""
    bank: list = field(default_factory=list)   # oldest first, newest last
    z_a: np.ndarray = None                     # latest exact anchor (float32)
    q_a_in: float = 1.0                        # latest exact interval q_{a} -> q_{a-1}
    q_a_out: float = 1.0
    z_a_in: np.ndarray = None                  # input latent of the latest exact step (secant ablation)
    cam_a: np.ndarray = field(default_factory=lambda: np.zeros(4))
    depth_a: np.ndarray = field(default_factory=lambda: np.zeros(4))
    R: float = 0.0
    eta: float = 1.0
    age: int = 0

    @classmethod
    def initial(cls, z0, sigmas, p):
        """State before the first step: empty bank, anchor z_a := z_T (the
        initial latent), interval collapsed to the initial phase."""
        q0 = float(sch.phase(sigmas[0]))
        return cls(bank=[], z_a=_f32(z0).reshape(-1), q_a_in=q0, q_a_out=q0,
                   R=0.0, eta=float(p.eta_init), age=0)

    def history(self, T, p):
        return sm.history_summary(list(reversed(self.bank)), T, p.bank_capacity)


def _cond_desc(cond):
    cam = np.zeros(4) if cond is None or cond.get("cam") is None else np.asarray(cond["cam"], dtype=np.float64)
    depth = np.zeros(4) if cond is None or cond.get("depth") is None else np.asarray(cond["depth"], dtype=np.float64)
    return cam, depth


def surrogate_step(state, z_k, k, cond, sigmas, p):
    """Steps 1-4 up to the decision.  Returns (z_hat or None, info).

    On a Surrogate decision the state is advanced (R <- R_cand, age += 1);
    on Exact the caller completes the step with ``exact_step``.
    """
    T = len(sigmas) - 1
    q_k = float(sch.phase(sigmas[k]))
    q_next = float(sch.phase(sigmas[k + 1]))
    cam, depth = _cond_desc(cond)
    lcam, ldepth = ab.lift_descriptors(cam, depth, p)
    z_k = np.asarray(z_k).reshape(-1)
    h = state.history(T, p)
    s_phi = sm.summary_of_state(z_k, state.z_a, lcam, ldepth, q_k, h, p.eps_nu, p.sketch_seed)

    info = {"k": k, "q": q_k, "s_phi": s_phi, "h": h, "n_bank": len(state.bank),
            "supported": False, "finite": False, "alpha": 0.0, "n_compat": 0,
            "kappa": np.zeros(0), "pi": np.zeros(0), "margins": []}
    z_hat = None
    if state.bank and p.has(ab.ABL_SECANT):
        # native latent secant (ablation): no retrieval, extrapolate z_a - z_a,in
        alpha = sg.scheduler_scaling(q_k, q_next, state.q_a_in, state.q_a_out, p)
        z_hat = _f32(ab.secant_candidate(z_k, state.z_a, state.z_a_in, alpha))
        info.update({"alpha": alpha, "supported": True, "n_compat": len(state.bank),
                     "finite": bool(np.all(np.isfinite(z_hat)))})
        info["margins"].append(abs(p.q_gap_max - abs(q_k - state.q_a_out)))
    elif state.bank:
        head = sg.surrogate_head(s_phi, q_k, q_next, state.bank, state.q_a_in, state.q_a_out, p)
        info.update({"alpha": head["alpha"], "kappa": head["kappa"], "pi": head["pi"],
                     "sim_in": head["sim"], "sim_out": head["sim_out"], "s_hat": head["s_hat"],
                     "n_compat": head["n_compat"], "supported": head["supported"]})
        for i in range(len(state.bank)):
            info["margins"].append(abs(head["sim"][i] - p.sim_min))
            info["margins"].append(abs(p.q_gap_max - abs(head["dq"][i])))
        info["margins"].append(abs(p.q_gap_max - abs(q_k - state.q_a_out)))
        if head["supported"]:
            if p.has(OBS_RESIDUAL):
                z_hat = _f32(sg.observe_residual(head["kappa"], state.bank, z_k))
            else:
                z_hat = _f32(sg.observe(head["kappa"], state.bank))
            info["finite"] = bool(np.all(np.isfinite(z_hat)))

    rms_dz = sm.rms(z_k.astype(np.float64) - state.z_a.astype(np.float64))
    rms_za = sm.rms(state.z_a)
    sig = ctl.proxy_signals(rms_dz, rms_za, state.age, q_next, state.q_a_out,
                            cam, state.cam_a, depth, state.depth_a, p)
    p_t = ctl.defect_proxy(sig, p)
    d_hat = state.eta * p_t
    w = ab.impact_weight(ctl.impact_weight(cam, depth, q_k, p), p)
    delta = w * d_hat
    R_cand = ab.risk_decay(p) * state.R + delta                      # Eq. 9
    avail, terms = ctl.available(k, T, len(state.bank), state.age, q_k, state.q_a_out,
                                 info["finite"], info["supported"], p)
    if p.has(ab.ABL_PERIODIC):
        surrogate = ab.periodic_decision(avail, state.age, p)
    else:
        surrogate = ctl.decide(avail, R_cand, p)
        if all(v for key, v in terms.items()):
            info["margins"].append(abs(R_cand - p.tau_risk))
    info.update({"p": p_t, "d_hat": d_hat, "w": w, "delta": delta, "R_cand": R_cand,
                 "available": avail, "terms": terms, "decision": 1 if surrogate else 0,
                 "d_cf": float("nan"), "age": state.age, **sig})
    if surrogate:
        state.R = R_cand
        state.age += 1
    info["R"] = state.R
    info["eta"] = state.eta
    return z_hat, info


def exact_step(state, z_k, v, z_hat, k, cond, sigmas, p, info):
    """Complete an Exact step: Psi, counterfactual calibration, bank insertion.

    Returns z_{k+1} = z_ex (float32).  ``info`` from ``surrogate_step`` is
    updated in place with d_cf, R and eta.
    """
    T = len(sigmas) - 1
    q_k = float(sch.phase(sigmas[k]))
    q_next = float(sch.phase(sigmas[k + 1]))
    cam, depth = _cond_desc(cond)
    z_k = np.asarray(z_k).reshape(-1)
    z_ex = _f32(sch.psi(z_k, np.asarray(v).reshape(-1), sigmas[k], sigmas[k + 1]))

    state.R = ab.risk_decay(p) * state.R
    if z_hat is not None and info["supported"] and info["finite"]:
        d_cf = ctl.counterfactual_defect(z_ex, z_hat, p)
        if ab.calibrates(p):
            state.eta = ctl.calibrate(state.eta, d_cf, info["p"], p)
        info["d_cf"] = d_cf

    h = state.history(T, p)            # pre-insertion history
    s_in = info["s_phi"]
    lcam, ldepth = ab.lift_descriptors(cam, depth, p)
    s_out = sm.summary_of_state(z_ex, state.z_a, lcam, ldepth, q_next, h, p.eps_nu, p.sketch_seed)
    r = sm.rms(z_ex.astype(np.float64) - z_k.astype(np.float64)) / (sm.rms(z_k) + p.eps)
    rec = sg.Record(s_in=np.array(s_in), s_out=s_out, s_dphi=s_out - s_in, z_out=z_ex, z_in=_f32(z_k),
                    q_in=q_k, q_out=q_next, r=r, cam=cam.copy(), depth=depth.copy())
    state.bank.append(rec)
    if len(state.bank) > p.bank_capacity:
        state.bank.pop(0)
    state.z_a = z_ex
    state.z_a_in = _f32(z_k)
    state.q_a_in, state.q_a_out = q_k, q_next
    state.cam_a, state.depth_a = cam.copy(), depth.copy()
    state.age = 0
    info["R"] = state.R
    info["eta"] = state.eta
    info["r"] = r
    return z_ex


def cached_rollout(z_T, denoiser, conds, sigmas, p, trace=None):
    """WorldDynCache rollout.  ``denoiser(z, t, cond, k)`` returns v; ``conds``
    is a list with one dict per step (or a single dict used for every step),
    each with optional "cam"/"depth" descriptors and whatever the denoiser
    needs.  Returns (z_final float32, decisions list, trace list)."""
    T = len(sigmas) - 1
    z = _f32(z_T).reshape(-1)
    state = CacheState.initial(z, sigmas, p)
    decisions, infos = [], []
    for k in range(T):
        c = conds[k] if isinstance(conds, (list, tuple)) else conds
        z_hat, info = surrogate_step(state, z, k, c, sigmas, p)
        if info["decision"] == 1:
            z = z_hat
        else:
            v = denoiser(z, float(sch.model_timestep(sigmas[k])), c, k)
            z = exact_step(state, z, v, z_hat, k, c, sigmas, p, info)
        decisions.append(info["decision"])
        infos.append(info)
    if trace is not None:
        trace.extend(infos)
    return z, decisions, infos


def native_rollout(z_T, denoiser, conds, sigmas):
    """The uncached rollout: an exact transition at every step (Eq. 1)."""
    T = len(sigmas) - 1
    z = _f32(z_T).reshape(-1)
    for k in range(T):
        c = conds[k] if isinstance(conds, (list, tuple)) else conds
        v = denoiser(z, float(sch.model_timestep(sigmas[k])), c, k)
        z = _f32(sch.psi(z, np.asarray(v).reshape(-1), sigmas[k], sigmas[k + 1]))
    return z
