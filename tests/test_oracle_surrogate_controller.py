"""Pins of the oracle's surrogate (Eq. 3-5) and controller (Eq. 6-10) against
closed forms, the model-class exactness properties and library routines."""
import json
import os

import numpy as np
import pytest
from scipy.special import softmax

from oracle import controller as ctl
from oracle import summary as sm
from oracle import surrogate as sg
from oracle.params import CacheParams

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rec(s_in, s_out, z_out, q_in, q_out, r=0.0):
    s_in = np.asarray(s_in, dtype=np.float64)
    s_out = np.asarray(s_out, dtype=np.float64)
    return sg.Record(s_in=s_in, s_out=s_out, s_dphi=s_out - s_in, z_out=np.asarray(z_out, dtype=np.float32),
                     q_in=q_in, q_out=q_out, r=r)


# ------------------------------------------------------------------ Eq. 3
def test_retrieval_softmax_matches_scipy_on_compatible_subset():
    p = CacheParams(sim_min=0.0, q_gap_max=0.25, gamma_q=10.0, tau_in=0.1)
    g = np.random.default_rng(0)
    s_phi = g.standard_normal(256)
    bank = []
    for i, q_in in enumerate([0.80, 0.70, 0.30, 0.75]):
        s_in = s_phi + 0.8 * g.standard_normal(256)
        if i == 1:
            s_in = -s_phi                         # sim = -1: incompatible by similarity
        bank.append(_rec(s_in, s_in, np.zeros(8), q_in, q_in - 0.1))
    ret = sg.retrieve(s_phi, 0.8, bank, p)
    assert ret["compat"].tolist() == [True, False, False, True]   # q gap 0.5 > 0.25 for record 2
    ell = np.array([sm.cosine(s_phi, r.s_in) - 10.0 * (0.8 - r.q_in) ** 2 for r in bank])
    want = np.zeros(4)
    want[[0, 3]] = softmax(ell[[0, 3]] / 0.1)
    assert np.allclose(ret["pi"], want, atol=1e-14)
    assert ret["supported"] and ret["n_compat"] == 2


def test_retrieval_phase_penalty_is_monotone():
    p = CacheParams(q_gap_max=1.0)
    s = np.ones(256)
    bank = [_rec(s, s, np.zeros(4), 0.5, 0.4), _rec(s, s, np.zeros(4), 0.6, 0.5)]
    pi = sg.retrieve(s, 0.5, bank, p)["pi"]
    assert pi[0] > pi[1]                           # equal similarity, larger phase gap -> smaller weight


def test_unsupported_when_nothing_compatible():
    p = CacheParams(min_support=1)
    s = np.ones(256)
    bank = [_rec(-s, s, np.zeros(4), 0.5, 0.4)]
    ret = sg.retrieve(s, 0.5, bank, p)
    assert not ret["supported"] and np.all(ret["pi"] == 0.0)


# ------------------------------------------------------------------ Eq. 4
def test_scheduler_scaling_ratio_and_clip():
    p = CacheParams(alpha_min=0.5, alpha_max=2.0, eps=1e-8)
    assert abs(sg.scheduler_scaling(0.6, 0.57, 0.7, 0.66, p) - 0.03 / (0.04 + 1e-8)) < 1e-12
    assert sg.scheduler_scaling(0.6, 0.59, 0.7, 0.6, p) == 0.5       # 0.1 -> clipped up
    assert sg.scheduler_scaling(0.6, 0.2, 0.7, 0.66, p) == 2.0       # 10  -> clipped down


def test_lemma_summary_space_evolution_equals_full_lift():
    # s is linear, so evolving the full lifted state and summarising it equals
    # evolving the summaries (the shortcut every kernel uses).
    g = np.random.default_rng(1)
    n, seed, eps_nu = 128 * 40 + 13, 77, 1e-12
    lifts = []
    for _ in range(4):
        z, za = g.standard_normal(n), g.standard_normal(n)
        lifts.append(sm.lift_full(z, za, g.standard_normal(4), g.standard_normal(4), g.uniform(), g.standard_normal(7), eps_nu))
    phi_t, ins, outs = lifts[0], lifts[1:3], [lifts[3], lifts[1]]
    pi, alpha = np.array([0.3, 0.7]), 1.37
    full = phi_t + alpha * sum(pi[i] * (outs[i] - ins[i]) for i in range(2))
    bank = [_rec(sm.summarize_full(ins[i], n, seed), sm.summarize_full(outs[i], n, seed), np.zeros(4), 0.5, 0.4) for i in range(2)]
    got = sg.evolve_summary(sm.summarize_full(phi_t, n, seed), alpha, pi, bank)
    assert np.allclose(got, sm.summarize_full(full, n, seed), atol=1e-11)


def test_P3_lifted_evolution_exact_in_model_class():
    # Trajectory whose lifted increments are proportional to the phase step:
    # phi_{k+1} - phi_k = c (q_{k+1} - q_k) u.  Then phi_hat equals the true
    # next lifted state for any retrieval weights when alpha is unclipped.
    g = np.random.default_rng(2)
    u = g.standard_normal(256)
    phi0, c = g.standard_normal(256), 3.0
    q = np.array([1.0, 0.9, 0.8, 0.7, 0.6])
    phi = [phi0 + c * (q[k] - q[0]) * u for k in range(5)]
    bank = [_rec(phi[k], phi[k + 1], np.zeros(4), q[k], q[k + 1]) for k in range(3)]
    p = CacheParams(alpha_min=0.0, alpha_max=10.0, eps=0.0)
    alpha = sg.scheduler_scaling(q[3], q[4], q[2], q[3], p)
    for pi in [np.array([1.0, 0.0, 0.0]), np.array([0.2, 0.5, 0.3])]:
        got = sg.evolve_summary(phi[3], alpha, pi, bank)
        assert np.allclose(got, phi[4], atol=1e-12)


# ------------------------------------------------------------------ Eq. 5
def test_P1_identical_outputs_give_that_output():
    g = np.random.default_rng(3)
    Z = g.standard_normal(1000).astype(np.float32)
    bank = [_rec(g.standard_normal(256), g.standard_normal(256), Z, 0.5, 0.4) for _ in range(3)]
    kappa, _ = sg.observation_weights(g.standard_normal(256), bank, CacheParams())
    assert abs(kappa.sum() - 1.0) < 1e-14
    assert np.allclose(sg.observe(kappa, bank), Z.astype(np.float64), atol=1e-12)


def test_P2_small_temperature_is_one_hot():
    g = np.random.default_rng(4)
    bank = [_rec(g.standard_normal(256), g.standard_normal(256), g.standard_normal(100), 0.5, 0.4) for _ in range(4)]
    p = CacheParams(tau_obs=1e-4)
    kappa, _ = sg.observation_weights(bank[2].s_out, bank, p)
    assert np.allclose(kappa, [0, 0, 1, 0], atol=1e-12)
    assert np.allclose(sg.observe(kappa, bank), bank[2].z_out.astype(np.float64), atol=1e-12)


def test_P4_single_record():
    g = np.random.default_rng(5)
    rec = _rec(g.standard_normal(256), g.standard_normal(256), g.standard_normal(64), 0.8, 0.7)
    p = CacheParams(sim_min=-1.0)
    head = sg.surrogate_head(g.standard_normal(256), 0.7, 0.6, [rec], 0.8, 0.7, p)
    assert np.allclose(head["pi"], [1.0]) and np.allclose(head["kappa"], [1.0])
    assert np.array_equal(sg.observe(head["kappa"], [rec]), rec.z_out.astype(np.float64))


def test_observation_weights_match_scipy_softmax():
    g = np.random.default_rng(6)
    bank = [_rec(g.standard_normal(256), g.standard_normal(256), np.zeros(4), 0.5, 0.4) for _ in range(4)]
    s_hat = g.standard_normal(256)
    kappa, sims = sg.observation_weights(s_hat, bank, CacheParams(tau_obs=0.05))
    assert np.allclose(kappa, softmax(np.array([sm.cosine(s_hat, r.s_out) for r in bank]) / 0.05), atol=1e-14)


# ------------------------------------------------------------------ Eq. 6-10
def test_impact_weight_cap():
    consts = json.load(open(os.path.join(GOLDEN, "structural_constants.json")))
    p = CacheParams()
    assert ctl.impact_weight(np.zeros(4), np.zeros(4), 0.0, p) == 1.0
    assert ctl.impact_weight(np.full(4, 10.0), np.zeros(4), 1.0, p) == consts["impact_weight_cap"]["value"]
    w = ctl.impact_weight(np.array([0.3, 0, 0, 0.4]), np.zeros(4), 0.2, p)
    assert abs(w - (1 + 0.5 * 0.5 + 1.0 * 0.2)) < 1e-15


def test_risk_equals_defining_geometric_sum():
    p = CacheParams(lam=0.83)
    R0 = 0.4
    deltas = [0.01, 0.2, 0.05, 0.13, 0.0, 0.07]
    R = R0
    for d in deltas:
        _, R = ctl.candidate_risk(R, 1.0, d, p)
    n = len(deltas)
    closed = p.lam ** n * R0 + sum(p.lam ** (n - 1 - j) * deltas[j] for j in range(n))
    assert abs(R - closed) < 1e-15


def test_calibration_fixed_point_and_rate():
    p = CacheParams(beta_d=0.8, eta_min=0.1, eta_max=10.0, eps=0.0)
    r, eta0 = 2.5, 1.0
    eta = eta0
    for n in range(1, 30):
        eta = ctl.calibrate(eta, r * 0.3, 0.3, p)
        assert abs(abs(eta - r) - p.beta_d ** n * abs(eta0 - r)) < 1e-12
    assert ctl.calibrate(1.0, 1e6, 1.0, p) == p.eta_max             # clamp high
    eta = 1.0
    for _ in range(200):
        eta = ctl.calibrate(eta, 0.0, 1.0, p)
    assert eta == p.eta_min                                         # clamp low


def test_counterfactual_defect():
    p = CacheParams(eps=1e-8)
    g = np.random.default_rng(7)
    z = g.standard_normal(1000).astype(np.float32)
    assert ctl.counterfactual_defect(z, z, p) == 0.0
    m = np.mean(np.abs(z.astype(np.float64)))
    assert abs(ctl.counterfactual_defect(z, np.zeros_like(z), p) - m / (m + 1e-8)) < 1e-15
    assert abs(ctl.counterfactual_defect(2 * z, z, p) - 0.5 * (2 * m) / (2 * m + 1e-8)) < 1e-12


def test_proxy_and_decision_tie():
    consts = json.load(open(os.path.join(GOLDEN, "structural_constants.json")))
    p = CacheParams(w_z=1.0, w_age=0.05, w_phase=1.0, w_cam=0.5, w_depth=0.5)
    sig = ctl.proxy_signals(0.2, 1.0, 3, 0.5, 0.56, np.ones(4), np.zeros(4), np.zeros(4), np.zeros(4), p)
    assert abs(sig["d_cam"] - 2.0) < 1e-15 and abs(sig["d_phase"] - 0.06) < 1e-15
    assert abs(ctl.defect_proxy(sig, p) - (0.2 / (1 + 1e-8) + 0.15 + 0.06 + 1.0)) < 1e-12
    assert consts["decision_tie"]["value"] == "surrogate"
    assert ctl.decide(True, 0.5, CacheParams(tau_risk=0.5)) is True
    assert ctl.decide(True, 0.5000001, CacheParams(tau_risk=0.5)) is False
    assert ctl.decide(False, 0.0, CacheParams(tau_risk=0.5)) is False


def test_available_terms():
    p = CacheParams(max_age=6, q_gap_max=0.25, n_init_exact=1, n_final_exact=2)
    ok, _ = ctl.available(3, 10, 2, 6, 0.5, 0.6, True, True, p)
    assert ok
    assert not ctl.available(3, 10, 2, 7, 0.5, 0.6, True, True, p)[0]     # age 7 > 6
    assert not ctl.available(0, 10, 2, 0, 0.5, 0.6, True, True, p)[0]     # initial phase
    assert not ctl.available(8, 10, 2, 0, 0.5, 0.6, True, True, p)[0]     # final refinement phase
    assert not ctl.available(3, 10, 2, 0, 0.5, 0.8, True, True, p)[0]     # phase gap 0.3
    assert not ctl.available(3, 10, 0, 0, 0.5, 0.6, True, True, p)[0]     # empty bank
    assert not ctl.available(3, 10, 2, 0, 0.5, 0.6, False, True, p)[0]    # non-finite
    assert not ctl.available(3, 10, 2, 0, 0.5, 0.6, True, False, p)[0]    # unsupported
