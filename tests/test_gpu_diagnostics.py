"""Synthetic diagnostics (Fig. 2, Fig. 3a readings) on the GPU against the
CPU oracle's, on the 2-layer parity model (D=256, latent 16x4x16x16, fp32
parity mode): single-injection local and downstream defects, the
predicted / counterfactual defect pairs, and the direction error per streak
position."""
import numpy as np
import pytest
import torch

from helpers import params_for_both
from oracle import diagnostics as odg
from oracle import dit
from oracle import schedule as sch
from oracle.params import DiTConfig
from paper_2608_01845_gb300 import diagnostics as gdg
from paper_2608_01845_gb300 import synth, wdc

pytestmark = pytest.mark.gpu
PARITY_MODEL = dict(layers=2, hidden=256, heads=4, head_dim=64, mlp=1024, temb_dim=256, freq_dim=256, in_ch=16, frames=4,
            height=16, width=16, patch=2, cond_tokens=16, cond_dim=256, dual_stream=0)
T = 10


@pytest.fixture(scope="module")
def model():
    W = synth.dit_weights(PARITY_MODEL, 0, std=0.02)
    z0 = synth.latent(1, (16, 4, 16, 16)).reshape(-1)
    ct = synth.cond_tokens(2, 16, 256)
    desc = synth.cond_descriptors(3)
    cfg = DiTConfig(**PARITY_MODEL)
    F = lambda z, t, c, k: dit.forward(W, cfg, np.asarray(z).reshape(16, 4, 16, 16), t, ct)
    return W, z0, ct, desc, F


def _ctx(W, cp):
    ctx = wdc.Context(wdc.make_config(dtype=wdc.F32, **PARITY_MODEL), T, params=cp)
    ctx.set_weights(W)
    return ctx


def test_downstream_impact_matches_oracle(model):
    W, z0, ct, desc, F = model
    op, cp = params_for_both(tau_risk=-1.0, sim_min=-1.0)
    ref = odg.downstream_impact(z0, F, desc, sch.sigmas(T), op)
    ctx = _ctx(W, cp)
    ct_d = torch.from_numpy(ct).cuda()
    got = gdg.downstream_impact(ctx, torch.from_numpy(z0.copy()).cuda(), [wdc.make_cond(ct_d, desc["cam"], desc["depth"])],
                                ct_d)
    assert [r["t"] for r in got["rows"]] == [r["t"] for r in ref["rows"]] and len(ref["rows"]) >= 8
    for a, b in zip(got["rows"], ref["rows"]):
        for key in ["d", "D_down", "d_hat", "w", "delta"]:
            assert abs(a[key] - b[key]) <= 1e-4 * max(1e-3, abs(b[key])), (a["t"], key, a[key], b[key])
    assert got["false_safe_instantaneous"] == ref["false_safe_instantaneous"]
    assert ctx.device_errors() == 0


def test_proxy_vs_counterfactual_matches_oracle(model):
    W, z0, ct, desc, F = model
    op, cp = params_for_both(tau_risk=0.5)          # both decisions, margins checked by the rollout tests
    ref = odg.proxy_vs_counterfactual(z0, F, desc, sch.sigmas(T), op)
    ctx = _ctx(W, cp)
    ct_d = torch.from_numpy(ct).cuda()
    got = gdg.proxy_vs_counterfactual(ctx, torch.from_numpy(z0.copy()).cuda(),
                                      wdc.make_cond(ct_d, desc["cam"], desc["depth"]))
    assert len(got) == len(ref) >= 3
    assert np.allclose(np.array(got), np.array(ref), rtol=1e-4, atol=1e-7)


@pytest.mark.parametrize("flags", [wdc.ABL_SECANT, wdc.OBS_RESIDUAL, wdc.OBS_RESIDUAL | wdc.ABL_NO_COND])
def test_direction_errors_match_oracle(model, flags):
    W, z0, ct, desc, F = model
    op, cp = params_for_both(tau_risk=1e9, sim_min=-1.0, q_gap_max=1.0, flags=wdc.ABL_PERIODIC | flags, period=4)
    ref = odg.direction_errors(z0, F, desc, sch.sigmas(T), op)
    ctx = _ctx(W, cp)
    ct_d = torch.from_numpy(ct).cuda()
    got = gdg.direction_errors(ctx, torch.from_numpy(z0.copy()).cuda(),
                               [wdc.make_cond(ct_d, desc["cam"], desc["depth"])], ct_d)
    assert [(r["k"], r["streak"], r["decision"]) for r in got["rows"]] == \
        [(r["k"], r["streak"], r["decision"]) for r in ref["rows"]]
    assert sorted(got["mean_by_streak"]) == [0, 1, 2, 3]
    for a, b in zip(got["rows"], ref["rows"]):
        assert abs(a["angle"] - b["angle"]) <= 1e-4, (a["k"], a["angle"], b["angle"])


@pytest.mark.parametrize("n,with_c", [(16 * 4 * 16 * 16, True), (16 * 4 * 16 * 16, False)])
def test_latent_pair_stats_match_fp64_sums(n, with_c):
    """The device reductions behind the diagnostics (wdc_latent_pair_stats)
    against fp64 sums of the same fp32 latents, 1e-6 relative."""
    W = synth.dit_weights(PARITY_MODEL, 0, std=0.02)
    op, cp = params_for_both()
    ctx = _ctx(W, cp)
    g = np.random.default_rng(5)
    a, b, c = (g.standard_normal(n).astype(np.float32) for _ in range(3))
    dev = [torch.from_numpy(x.copy()).cuda() for x in (a, b, c)]
    got = ctx.latent_pair_stats(dev[0], dev[1], dev[2] if with_c else None)
    a64, b64 = a.astype(np.float64), b.astype(np.float64)
    c64 = c.astype(np.float64) if with_c else np.zeros(n)
    want = [np.sum((a64 - c64) ** 2), np.sum((b64 - c64) ** 2), np.sum((a64 - c64) * (b64 - c64)),
            np.sum((a64 - b64) ** 2), np.sum(b64 ** 2)]
    for k in range(5):
        assert abs(got[k] - want[k]) <= 1e-6 * max(abs(want[k]), 1e-3 * want[0]), (k, got[k], want[k])
