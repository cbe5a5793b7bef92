"""Pins of the oracle's synthetic diagnostics (Fig. 2, Fig. 3a readings):
library correlations, and closed-form cases where the injected or
approximate transition is exact."""
import numpy as np
from scipy.stats import pearsonr, spearmanr

from oracle import diagnostics as dg
from oracle import rollout as ro
from oracle import schedule as sch
from oracle.params import ABL_PERIODIC, ABL_SECANT, OBS_RESIDUAL, CacheParams
from paper_2608_01845_gb300 import synth


def test_correlations_match_scipy():
    g = np.random.default_rng(0)
    a = g.standard_normal(40)
    b = 0.7 * a + 0.3 * g.standard_normal(40)
    pe, sp = dg.correlations(a, b)
    assert abs(pe - pearsonr(a, b)[0]) < 1e-12
    assert abs(sp - spearmanr(a, b)[0]) < 1e-12


def _const_field(n, seed=3):
    c = np.random.default_rng(seed).standard_normal(n)
    return lambda z, t, cond, k: c


def test_exact_injection_has_no_downstream_impact():
    # v(z) = c, uniform schedule, residual reading: every candidate is the
    # exact next latent, so d_t = 0 and D_down = 0 up to float32 storage; an
    # off-by-one in the resume step would give D_down ~ ||c|| dsigma / ||z_T||.
    F = _const_field(1024)
    s = sch.sigmas(12)
    z0 = synth.latent(4, (1024,))
    p = CacheParams(tau_risk=-1.0, sim_min=-1.0, q_gap_max=1.0, flags=OBS_RESIDUAL)
    r = dg.downstream_impact(z0, F, {}, s, p)
    assert len(r["rows"]) == 11
    for row in r["rows"]:
        assert row["d"] < 1e-6 and row["D_down"] < 1e-6
    assert r["false_safe_instantaneous"] == 0.0


def test_printed_reading_injection_is_measured_against_the_exact_end():
    # the printed Eq. 5 returns a past latent: injecting at the last step
    # leaves the final latent at the candidate, so D_down = ||z_hat - z_T|| / ||z_T||
    F = _const_field(1024)
    s = sch.sigmas(8)
    z0 = synth.latent(5, (1024,))
    p = CacheParams(tau_risk=-1.0, sim_min=-1.0, q_gap_max=1.0)
    zs, infos, cands = dg.all_exact_with_candidates(z0, F, {}, s, p)
    r = dg.downstream_impact(z0, F, {}, s, p, steps={7})
    (row,) = r["rows"]
    want = np.linalg.norm(cands[7].astype(np.float64) - zs[-1]) / np.linalg.norm(zs[-1].astype(np.float64))
    assert abs(row["D_down"] - want) < 1e-12
    d_want = np.mean(np.abs(zs[8].astype(np.float64) - cands[7])) / (np.mean(np.abs(zs[8].astype(np.float64))) + p.eps)
    assert abs(row["d"] - d_want) < 1e-12


def test_direction_error_zero_for_exact_increments_and_large_for_past_latents():
    F = _const_field(2048)
    s = sch.sigmas(12)
    z0 = synth.latent(6, (2048,))
    for flags in (ABL_SECANT, OBS_RESIDUAL):
        p = CacheParams(tau_risk=1e9, sim_min=-1.0, q_gap_max=1.0, flags=ABL_PERIODIC | flags, period=4)
        r = dg.direction_errors(z0, F, {}, s, p)
        assert len(r["rows"]) >= 10 and sorted(r["mean_by_streak"]) == [0, 1, 2, 3]
        assert max(x["angle"] for x in r["rows"]) < 1e-3
    p = CacheParams(tau_risk=1e9, sim_min=-1.0, q_gap_max=1.0, flags=ABL_PERIODIC, period=4)
    r = dg.direction_errors(z0, F, {}, s, p)
    assert min(r["mean_by_streak"].values()) > 0.5          # blends of past latents point elsewhere
