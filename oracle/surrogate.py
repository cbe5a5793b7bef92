"""Latent dynamics surrogate G_t (Eq. 3-5): retrieval, lifted evolution and
kernelised observation over the exact-transition bank.

Test infrastructure only (see the package docstring).

Section "Local Lifted Evolution": a FIFO bank B_t of exact transitions, each
record holding the lifted input and output, their increment, the exact output
latent and the scheduler phases; the retrieval view (phi_in, dphi) is filtered
to the locally compatible subset N_t and weighted by Eq. 3; Eq. 4 rescales by
the scheduler interval and evolves the lifted state.  Section "Kernelized
Nonlinear Observation": Eq. 5 maps the evolved state back to a latent with a
softmax over the exact-output view M_t of the same bank (all records).

Records keep the summaries s(phi_in), s(phi_out), s(dphi) (s is linear, so
s(dphi) = s(phi_out) - s(phi_in) and s(phi_hat) = s(phi_t) + alpha *
sum pi_i s(dphi_i) -- the lifted state is never materialised in full).

Readings (the paper defers thresholds and temperatures): compatibility is
sim >= sim_min and |q_t - q_in| <= q_gap_max; support means |N_t| >=
min_support; with no compatible record the evolution is skipped.
"""
from dataclasses import dataclass, field

import numpy as np

from . import ablation as ab
from .summary import cosine


@dataclass
class Record:
    """One exact transition z_in -> z_out in the bank (section "Local Lifted Evolution")."""
    s_in: np.ndarray            # s(phi_in), 256
    s_out: np.ndarray           # s(phi_out), 256
    s_dphi: np.ndarray          # s(phi_out) - s(phi_in), 256
    z_out: np.ndarray           # exact output latent (stored as float32)
    q_in: float
    q_out: float
    r: float = 0.0              # rms(z_out - z_in) / rms(z_in), feeds h(H)
    cam: np.ndarray = field(default_factory=lambda: np.zeros(4))
    depth: np.ndarray = field(default_factory=lambda: np.zeros(4))
    z_in: np.ndarray = None     # exact input latent (float32; read only by the residual reading)


def _softmax(x):
    x = np.asarray(x, dtype=np.float64)
    if x.size == 0:
        return x
    e = np.exp(x - np.max(x))
    return e / np.sum(e)


def retrieve(s_phi, q_t, bank, p):
    """Transition retrieval (Eq. 3).

    Returns a dict with per-record ``sim`` = sim(s(phi_t), s(phi_in_i)),
    ``compat`` (membership in N_t), ``ell`` (retrieval score
    sim - gamma_q (q_t - q_in)^2), ``pi`` (softmax of ell/tau_in over N_t, 0
    outside it) and ``supported`` (|N_t| >= min_support).
    """
    K = len(bank)
    sims = np.array([cosine(s_phi, rec.s_in) for rec in bank], dtype=np.float64)
    dq = np.array([q_t - rec.q_in for rec in bank], dtype=np.float64)
    if ab.compat_filter(p):
        compat = np.array([(sims[i] >= p.sim_min) and (abs(dq[i]) <= p.q_gap_max) for i in range(K)], dtype=bool)
    else:
        compat = np.ones(K, dtype=bool)          # w/o support constraint: N_t = the whole bank
    ell = sims - p.gamma_q * dq * dq
    pi = np.zeros(K, dtype=np.float64)
    if compat.any():
        pi[compat] = _softmax(ell[compat] / p.tau_in)
    return {"sim": sims, "dq": dq, "compat": compat, "ell": ell, "pi": pi,
            "n_compat": int(compat.sum()), "supported": int(compat.sum()) >= p.min_support}


def scheduler_scaling(q_t, q_next, q_a_in, q_a_out, p):
    """alpha_t = clip(|q_{t-1} - q_t| / (|q_{a-1} - q_a| + eps), alpha_min, alpha_max) (Eq. 4).

    (q_a_in -> q_a_out) is the latest exact transition interval a -> a-1.
    """
    raw = abs(q_next - q_t) / (abs(q_a_out - q_a_in) + p.eps)
    return float(min(max(raw, p.alpha_min), p.alpha_max))


def evolve_summary(s_phi, alpha, pi, bank):
    """s(phi_hat_{t-1}) = s(phi_t) + alpha * sum_{i in N_t} pi_i s(dphi_i) (Eq. 4, via linearity of s)."""
    out = np.array(s_phi, dtype=np.float64, copy=True)
    for i, rec in enumerate(bank):
        if pi[i] != 0.0:
            out += alpha * pi[i] * rec.s_dphi
    return out


def observation_weights(s_hat, bank, p):
    """kappa_i = softmax_i(sim(s(phi_hat), s(phi_out_i)) / tau) over all records (Eq. 5)."""
    sims = np.array([cosine(s_hat, rec.s_out) for rec in bank], dtype=np.float64)
    return _softmax(sims / p.tau_obs), sims


def observe(kappa, bank, chunk=1 << 24):
    """z_hat = sum_i kappa_i z_out_i (Eq. 5), accumulated in fp64."""
    n = bank[0].z_out.size
    out = np.zeros(n, dtype=np.float64)
    for s0 in range(0, n, chunk):
        acc = np.zeros(min(chunk, n - s0), dtype=np.float64)
        for i, rec in enumerate(bank):
            acc += kappa[i] * rec.z_out.reshape(-1)[s0:s0 + chunk].astype(np.float64)
        out[s0:s0 + chunk] = acc
    return out


def observe_residual(kappa, bank, z_t, chunk=1 << 24):
    """Residual reading of Eq. 5: z_hat = z_t + sum_i kappa_i (z_out_i - z_in_i),
    accumulated in fp64.  Eq. 5 as printed blends the stored outputs
    themselves (``observe``), a convex combination that cannot move past the
    bank; this reading blends the records' exact displacements and applies
    them to the current latent."""
    z_t = np.asarray(z_t).reshape(-1)
    n = z_t.size
    out = np.zeros(n, dtype=np.float64)
    for s0 in range(0, n, chunk):
        acc = z_t[s0:s0 + chunk].astype(np.float64)
        for i, rec in enumerate(bank):
            zo = rec.z_out.reshape(-1)[s0:s0 + chunk].astype(np.float64)
            zi = rec.z_in.reshape(-1)[s0:s0 + chunk].astype(np.float64)
            acc = acc + kappa[i] * (zo - zi)
        out[s0:s0 + chunk] = acc
    return out


def surrogate_head(s_phi, q_t, q_next, bank, q_a_in, q_a_out, p):
    """The scalar part of G_t: Eq. 3, Eq. 4 and the weights of Eq. 5.

    Returns a dict with the retrieval results, alpha, s_hat and kappa.  With no
    compatible record the evolution term is empty (s_hat = s(phi_t)).
    """
    ret = retrieve(s_phi, q_t, bank, p)
    alpha = scheduler_scaling(q_t, q_next, q_a_in, q_a_out, p)
    s_hat = evolve_summary(s_phi, alpha, ret["pi"], bank)
    kappa, sims_out = observation_weights(s_hat, bank, p)
    if p.has(ab.ABL_LINEAR_OBS):
        kappa = ab.linear_readout(s_hat, bank, p)   # linear observation (ablation)
    ret.update({"alpha": alpha, "s_hat": s_hat, "kappa": kappa, "sim_out": sims_out})
    return ret
