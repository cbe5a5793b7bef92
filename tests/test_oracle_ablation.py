"""Pins of the oracle's ablation variants (section "Ablation Study", Tables 3
and 4) against closed forms, library routines and the invariants each
variant's definition fixes."""
import math

import numpy as np
from scipy.special import softmax

from oracle import ablation as ab
from oracle import rollout as ro
from oracle import schedule as sch
from oracle import summary as sm
from oracle import surrogate as sg
from oracle.params import CacheParams
from paper_2608_01845_gb300 import synth


def _lin_denoiser(z, t, c, k):
    z = np.asarray(z, dtype=np.float64)
    return -0.8 * z + 0.05 * np.sin(np.arange(z.size) * 0.01 + 0.001 * t)


def _rollout(p, T=20, n=2048, seed=5, denoiser=_lin_denoiser, conds=None, shift=1.0):
    s = sch.sigmas(T, shift)
    z0 = synth.latent(seed, (n,))
    return ro.cached_rollout(z0, denoiser, conds if conds is not None else {}, s, p)


def _rec(s_out, z_out, q_in=0.9, q_out=0.8):
    s_out = np.asarray(s_out, dtype=np.float64)
    return sg.Record(s_in=np.zeros(256), s_out=s_out, s_dphi=s_out.copy(),
                     z_out=np.asarray(z_out, dtype=np.float32), q_in=q_in, q_out=q_out)


# ------------------------------------------------------------------ periodic placement
def test_periodic_places_exact_steps_every_period():
    # the risk test would never accept (tau < 0); the period alone decides
    for P in (2, 3, 4, 8):
        p = CacheParams(tau_risk=-1.0, sim_min=-1.0, q_gap_max=1.0, flags=ab.ABL_PERIODIC, period=P)
        _, dec, _ = _rollout(p, T=24)
        assert [k for k, d in enumerate(dec) if d == 0] == list(range(0, 24, P))


def test_periodic_period_one_is_bitwise_native():
    p = CacheParams(tau_risk=1e9, sim_min=-1.0, flags=ab.ABL_PERIODIC, period=1)
    s = sch.sigmas(12)
    z0 = synth.latent(9, (1024,))
    zc, dec, _ = ro.cached_rollout(z0, _lin_denoiser, {}, s, p)
    assert dec == [0] * 12
    assert np.array_equal(zc, ro.native_rollout(z0, _lin_denoiser, {}, s))


def test_periodic_keeps_availability():
    # nothing compatible -> no candidate -> exact, whatever the period says
    p = CacheParams(tau_risk=1e9, sim_min=2.0, flags=ab.ABL_PERIODIC, period=4)
    _, dec, _ = _rollout(p, T=10)
    assert dec == [0] * 10


# ------------------------------------------------------------------ native latent secant
def test_secant_is_exact_for_a_constant_velocity_field():
    # v(z) = c: the exact step is z + dsigma_k c and the latest exact
    # displacement is dsigma_e c, so z_t + alpha (z_a - z_a,in) with
    # alpha = |dsigma_k| / |dsigma_e| is the exact step.  A shifted schedule
    # makes the steps unequal (alpha != 1, inside the clip), so an inverted
    # alpha, a sign error or the wrong latent pair all break the equality.
    g = np.random.default_rng(3)
    c = g.standard_normal(1536)
    F = lambda z, t, cond, k: c
    T, shift = 16, 1.7
    s = sch.sigmas(T, shift)
    p = CacheParams(tau_risk=-1.0, sim_min=-1.0, q_gap_max=1.0, flags=ab.ABL_PERIODIC | ab.ABL_SECANT, period=4)
    z0 = synth.latent(8, (1536,))
    zc, dec, tr = ro.cached_rollout(z0, F, {}, s, p)
    assert sum(dec) == 12
    zn = ro.native_rollout(z0, F, {}, s)
    assert np.max(np.abs(zc - zn)) < 1e-5 * (1 + np.max(np.abs(zn)))
    alphas = [t["alpha"] for t in tr if t["decision"] == 1]
    assert 0.5 < min(alphas) and max(alphas) < 2.0          # unclipped
    assert min(alphas) < 0.95 or max(alphas) > 1.05         # and not all 1


def test_secant_candidate_formula_and_counterfactual():
    T = 10
    s = sch.sigmas(T)
    p = CacheParams(tau_risk=-1.0, sim_min=-1.0, flags=ab.ABL_SECANT)
    z0 = synth.latent(11, (1024,))
    st = ro.CacheState.initial(z0, s, p)
    z = z0.reshape(-1)
    for k in range(4):
        zh, info = ro.surrogate_step(st, z, k, {}, s, p)
        if k == 0:
            assert zh is None
        else:
            alpha = sg.scheduler_scaling(float(s[k]), float(s[k + 1]), st.q_a_in, st.q_a_out, p)
            want = z.astype(np.float64) + alpha * (st.z_a.astype(np.float64) - st.z_a_in.astype(np.float64))
            assert np.allclose(zh, want, rtol=0, atol=1e-6)
            assert info["supported"] and info["finite"]
        z = ro.exact_step(st, z, _lin_denoiser(z, 0, None, k), zh, k, {}, s, p, info)
        assert (k == 0) == math.isnan(info["d_cf"])


# ------------------------------------------------------------------ controller variants
def test_instantaneous_risk_has_no_memory():
    p = CacheParams(tau_risk=0.3, sim_min=-1.0, flags=ab.ABL_INSTANT_RISK)
    _, dec, tr = _rollout(p, T=30)
    assert 0 < sum(dec) < 30
    for t in tr:
        assert t["R_cand"] == t["delta"]
        assert t["R"] == (t["delta"] if t["decision"] == 1 else 0.0)


def test_no_impact_weighting_sets_w_to_one():
    conds = [{"cam": np.full(4, 0.3), "depth": np.full(4, 0.2)}] * 20
    p_full = CacheParams(tau_risk=0.5, sim_min=-1.0)
    _, _, tr_full = _rollout(p_full, conds=conds)
    assert all(t["w"] > 1.0 for t in tr_full)
    p = CacheParams(tau_risk=0.5, sim_min=-1.0, flags=ab.ABL_NO_IMPACT)
    _, _, tr = _rollout(p, conds=conds)
    assert all(t["w"] == 1.0 for t in tr)
    assert all(t["delta"] == t["d_hat"] for t in tr)


def test_no_calibration_keeps_eta_fixed_but_measures_d_cf():
    p = CacheParams(tau_risk=0.3, sim_min=-1.0, eta_init=1.7, flags=ab.ABL_NO_CALIB)
    _, _, tr = _rollout(p, T=30)
    assert all(t["eta"] == 1.7 for t in tr)
    assert sum(1 for t in tr if np.isfinite(t["d_cf"])) >= 3
    p_full = CacheParams(tau_risk=0.3, sim_min=-1.0, eta_init=1.7)
    _, _, tr_full = _rollout(p_full, T=30)
    assert any(t["eta"] != 1.7 for t in tr_full)


def test_no_support_constraint_retrieves_from_the_whole_bank():
    g = np.random.default_rng(4)
    s_phi = g.standard_normal(256)
    bank = [_rec(g.standard_normal(256), g.standard_normal(64), q_in=q) for q in (0.9, 0.5, 0.1)]
    for r in bank:
        r.s_in = g.standard_normal(256)
    p = CacheParams(sim_min=2.0, q_gap_max=0.25, gamma_q=10.0, tau_in=0.1)
    assert not sg.retrieve(s_phi, 0.8, bank, p)["supported"]
    p_ns = CacheParams(sim_min=2.0, q_gap_max=0.25, gamma_q=10.0, tau_in=0.1, flags=ab.ABL_NO_SUPPORT)
    ret = sg.retrieve(s_phi, 0.8, bank, p_ns)
    assert ret["supported"] and ret["n_compat"] == 3
    sims = np.array([sm.cosine(s_phi, r.s_in) for r in bank])
    ell = sims - 10.0 * (0.8 - np.array([0.9, 0.5, 0.1])) ** 2
    assert np.allclose(ret["pi"], softmax(ell / 0.1), rtol=1e-13, atol=0)
    # in a rollout where nothing is ever compatible, the variant still skips
    _, dec_full, _ = _rollout(CacheParams(tau_risk=1e9, sim_min=2.0), T=12)
    _, dec_ns, _ = _rollout(CacheParams(tau_risk=1e9, sim_min=2.0, flags=ab.ABL_NO_SUPPORT), T=12)
    assert dec_full == [0] * 12 and sum(dec_ns) > 0


# ------------------------------------------------------------------ linear observation
def test_linear_readout_orthogonal_closed_form():
    # orthogonal output summaries: G is diagonal, beta_i = s_hat.s_i / (|s_i|^2 + rho)
    g = np.random.default_rng(5)
    Q, _ = np.linalg.qr(g.standard_normal((256, 3)))
    scales = np.array([1.0, 2.5, 0.4])
    S = (Q * scales).T
    bank = [_rec(S[i], np.zeros(8)) for i in range(3)]
    s_hat = g.standard_normal(256)
    p = CacheParams(ridge=1e-3)
    rho = 1e-3 * np.sum(scales ** 2) / 3
    want = (S @ s_hat) / (scales ** 2 + rho)
    assert np.allclose(ab.linear_readout(s_hat, bank, p), want, rtol=1e-12, atol=0)


def test_linear_readout_is_least_squares_and_reproduces_a_record():
    g = np.random.default_rng(6)
    S = g.standard_normal((4, 256))
    bank = [_rec(S[i], np.zeros(8)) for i in range(4)]
    s_hat = g.standard_normal(256)
    p0 = CacheParams(ridge=0.0)
    beta_ls = np.linalg.lstsq(S.T, s_hat, rcond=None)[0]
    assert np.allclose(ab.linear_readout(s_hat, bank, p0), beta_ls, rtol=1e-10, atol=1e-12)
    assert np.allclose(ab.linear_readout(S[2], bank, p0), [0, 0, 1, 0], atol=1e-12)
    # the default ridge perturbs that by ~1e-6 only
    assert np.allclose(ab.linear_readout(S[2], bank, CacheParams()), [0, 0, 1, 0], atol=1e-5)


def test_linear_observation_in_the_surrogate_head():
    g = np.random.default_rng(7)
    bank = [_rec(g.standard_normal(256), g.standard_normal(32), q_in=0.9, q_out=0.8) for _ in range(3)]
    for r in bank:
        r.s_in = g.standard_normal(256)
        r.s_dphi = r.s_out - r.s_in
    s_phi = g.standard_normal(256)
    p = CacheParams(sim_min=-1.0, flags=ab.ABL_LINEAR_OBS)
    head = sg.surrogate_head(s_phi, 0.8, 0.7, bank, 0.9, 0.8, p)
    assert np.allclose(head["kappa"], ab.linear_readout(head["s_hat"], bank, p), rtol=1e-14, atol=0)
    full = sg.surrogate_head(s_phi, 0.8, 0.7, bank, 0.9, 0.8, CacheParams(sim_min=-1.0))
    assert np.allclose(full["s_hat"], head["s_hat"], rtol=0, atol=0)     # evolution unchanged
    assert abs(np.sum(full["kappa"]) - 1.0) < 1e-14


# ------------------------------------------------------------------ no condition
def test_no_condition_drops_descriptors_from_the_lift_only():
    g = np.random.default_rng(8)
    conds_a = [{"cam": g.standard_normal(4) * 0.1, "depth": g.standard_normal(4) * 0.1} for _ in range(16)]
    conds_b = [{"cam": c["cam"] * 3.0, "depth": -c["depth"]} for c in conds_a]
    p = CacheParams(tau_risk=-1.0, sim_min=-1.0, flags=ab.ABL_NO_COND)
    z0 = synth.latent(12, (1024,))
    s = sch.sigmas(16)
    _, _, tr_a = ro.cached_rollout(z0, _lin_denoiser, conds_a, s, p)
    _, _, tr_b = ro.cached_rollout(z0, _lin_denoiser, conds_b, s, p)
    for ta, tb in zip(tr_a, tr_b):
        assert np.all(ta["s_phi"][sm.OFF_CAM:sm.OFF_Q] == 0.0)
        assert np.array_equal(ta["s_phi"], tb["s_phi"])       # the lift ignores the descriptors
        assert np.array_equal(ta["kappa"], tb["kappa"])
        if ta["k"] > 1:
            assert ta["p"] != tb["p"]                          # the controller still sees them


# ------------------------------------------------------------------ residual reading of Eq. 5
def test_residual_observation_closed_forms():
    g = np.random.default_rng(9)
    z_t = g.standard_normal(512).astype(np.float32)
    D = g.standard_normal(512).astype(np.float32)
    # every record carries the same displacement: z_t + D for any weights summing to 1
    bank = []
    for i in range(3):
        zi = g.standard_normal(512).astype(np.float32)
        r = _rec(np.zeros(256), (zi.astype(np.float64) + D).astype(np.float32))
        r.z_in = zi
        bank.append(r)
    kap = np.array([0.2, 0.5, 0.3])
    want = z_t.astype(np.float64) + sum(kap[i] * (bank[i].z_out.astype(np.float64) - bank[i].z_in) for i in range(3))
    got = sg.observe_residual(kap, bank, z_t)
    assert np.allclose(got, want, rtol=0, atol=1e-12)
    assert np.allclose(got, z_t.astype(np.float64) + D, rtol=0, atol=1e-5)
    # a single record: z_t + (z_out - z_in)
    one = sg.observe_residual(np.array([1.0]), bank[:1], z_t)
    assert np.allclose(one, z_t.astype(np.float64) + bank[0].z_out.astype(np.float64) - bank[0].z_in, atol=1e-12)


def test_residual_reading_is_exact_for_a_constant_velocity_field():
    # uniform schedule, v(z) = c: every exact displacement is dsigma c, so
    # z_t + sum kappa_i (z_out_i - z_in_i) is the exact Euler step whatever
    # the weights; Eq. 5 as printed instead returns a blend of past latents
    from oracle.params import OBS_RESIDUAL
    g = np.random.default_rng(10)
    c = g.standard_normal(1024)
    F = lambda z, t, cond, k: c
    s = sch.sigmas(16)
    z0 = synth.latent(13, (1024,))
    p = CacheParams(tau_risk=1e9, sim_min=-1.0, q_gap_max=1.0, flags=OBS_RESIDUAL)
    zc, dec, _ = ro.cached_rollout(z0, F, {}, s, p)
    assert sum(dec) >= 10
    zn = ro.native_rollout(z0, F, {}, s)
    assert np.max(np.abs(zc - zn)) < 1e-5 * (1 + np.max(np.abs(zn)))
    zp, dec_p, _ = ro.cached_rollout(z0, F, {}, s, CacheParams(tau_risk=1e9, sim_min=-1.0, q_gap_max=1.0))
    assert dec_p == dec and np.max(np.abs(zp - zn)) > 0.1        # the printed reading does not advance
