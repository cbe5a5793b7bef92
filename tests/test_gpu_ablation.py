"""Ablation variants (section "Ablation Study", Tables 3 and 4) and the
residual reading of Eq. 5 on the GPU against the CPU oracle: the 2-layer parity model (D=256, latent
16x4x16x16, fp32 parity mode) rolled out under each variant, one flag at a
time plus the core factorization (periodic / risk x secant / lifted).  The
decision sequence must be identical and the final latent within 1e-5
relative L2; the per-step controller scalars within 1e-4."""
import numpy as np
import pytest
import torch

from helpers import params_for_both, rel_l2
from oracle import dit
from oracle import rollout as ro
from oracle import schedule as sch
from oracle.params import DiTConfig
from paper_2608_01845_gb300 import synth, wdc

pytestmark = pytest.mark.gpu
PARITY_MODEL = dict(layers=2, hidden=256, heads=4, head_dim=64, mlp=1024, temb_dim=256, freq_dim=256, in_ch=16, frames=4,
            height=16, width=16, patch=2, cond_tokens=16, cond_dim=256, dual_stream=0)
T = 10

VARIANTS = {
    "periodic+secant": dict(flags=wdc.ABL_PERIODIC | wdc.ABL_SECANT, period=3),
    "risk+secant": dict(flags=wdc.ABL_SECANT),
    "periodic+lifted": dict(flags=wdc.ABL_PERIODIC, period=3),
    "instantaneous": dict(flags=wdc.ABL_INSTANT_RISK),
    "no_impact": dict(flags=wdc.ABL_NO_IMPACT),
    "no_calibration": dict(flags=wdc.ABL_NO_CALIB),
    "no_support": dict(flags=wdc.ABL_NO_SUPPORT, sim_min=0.3),
    "linear_obs": dict(flags=wdc.ABL_LINEAR_OBS),
    "no_condition": dict(flags=wdc.ABL_NO_COND),
    "residual": dict(flags=wdc.OBS_RESIDUAL),
    "residual+linear_obs": dict(flags=wdc.OBS_RESIDUAL | wdc.ABL_LINEAR_OBS),
}


@pytest.fixture(scope="module")
def model():
    W = synth.dit_weights(PARITY_MODEL, 0, std=0.02)
    z0 = synth.latent(1, (16, 4, 16, 16))
    ct = synth.cond_tokens(2, 16, 256)
    desc = synth.cond_descriptors(3)
    cfg = DiTConfig(**PARITY_MODEL)
    cache = {}

    def F(z, t, c, k):
        key = (np.asarray(z, dtype=np.float32).tobytes(), t)
        if key not in cache:
            cache[key] = dit.forward(W, cfg, np.asarray(z).reshape(16, 4, 16, 16), t, ct)
        return cache[key]

    return W, z0, ct, desc, F


def _oracle_with_margin(kw, z0, desc, F):
    """The first threshold for which the oracle's rollout takes both
    decisions with every tie margin above 1e-4 (chosen from the oracle only)."""
    for tau in (0.5, 0.3, 0.8, 1.2, 0.2):
        op, cp = params_for_both(tau_risk=tau, **kw)
        zf, dec, tr = ro.cached_rollout(z0, F, desc, sch.sigmas(T), op)
        if not 0 < sum(dec) < T:
            continue
        if all(min(t["margins"]) > 1e-4 for t in tr if t["margins"]):
            return op, cp, zf, dec, tr
    pytest.fail(f"no threshold separates the decisions for {kw}")


@pytest.mark.parametrize("name", sorted(VARIANTS))
def test_ablation_rollout_matches_oracle(model, name):
    W, z0, ct, desc, F = model
    op, cp, zf_o, dec_o, tr_o = _oracle_with_margin(VARIANTS[name], z0, desc, F)
    ctx = wdc.Context(wdc.make_config(dtype=wdc.F32, **PARITY_MODEL), T, params=cp)
    ctx.set_weights(W)
    c = wdc.make_cond(torch.from_numpy(ct).cuda(), desc["cam"], desc["depth"])
    out = torch.empty(z0.size, dtype=torch.float32, device="cuda")
    dec, tr = ctx.rollout(torch.from_numpy(z0.ravel().copy()).cuda(), c, out)
    assert dec == dec_o
    assert rel_l2(out.cpu().numpy(), zf_o) <= 1e-5
    for a, b in zip(tr, tr_o):
        for key in ["p", "d_hat", "w", "R_cand", "R", "eta", "alpha"]:
            assert abs(a[key] - b[key]) <= 1e-4 * max(1.0, abs(b[key])), (name, a["k"], key)
        if not np.isnan(b["d_cf"]):
            assert abs(a["d_cf"] - b["d_cf"]) <= 1e-4 * max(1.0, b["d_cf"]), (name, a["k"])
        assert bool(a["supported"]) == bool(b["supported"]), (name, a["k"])
    assert ctx.device_errors() == 0


def test_periodic_placement_pattern_on_gpu(model):
    # tau_risk < 0: only the period places surrogate steps
    W, z0, ct, desc, F = model
    _, cp = params_for_both(tau_risk=-1.0, q_gap_max=1.0, sim_min=-1.0, flags=wdc.ABL_PERIODIC, period=4)
    ctx = wdc.Context(wdc.make_config(dtype=wdc.F32, **PARITY_MODEL), T, params=cp)
    ctx.set_weights(W)
    c = wdc.make_cond(torch.from_numpy(ct).cuda(), desc["cam"], desc["depth"])
    out = torch.empty(z0.size, dtype=torch.float32, device="cuda")
    dec, _ = ctx.rollout(torch.from_numpy(z0.ravel().copy()).cuda(), c, out)
    assert [k for k, d in enumerate(dec) if d == 0] == list(range(0, T, 4))


def test_linear_readout_weights_match_oracle_at_larger_bank():
    # the surrogate step alone, bank of 6 records, linear observation: the
    # readout coefficients (reported as kappa) against the oracle's solve
    from helpers import make_state, state_to_host
    from oracle import surrogate as sg
    n, K, k = 1 << 16, 6, 20
    op, cp = params_for_both(tau_risk=10.0, bank_capacity=8, sim_min=-1.0, flags=wdc.ABL_LINEAR_OBS)
    s = sch.sigmas(50)
    z = synth.latent(21, (n,)).reshape(-1)
    st = make_state(22, z, K, n, float(s[k]), 50, p=op)
    ctx = wdc.Context(wdc.make_config(in_ch=1, frames=1, height=1, width=n), 50, params=cp)
    zb = [torch.from_numpy(r.z_out.copy()).cuda() for r in st.bank]
    zc = torch.from_numpy(z.copy()).cuda()
    ctx.state_set(state_to_host(st), zb, zc)
    zh_o, info_o = ro.surrogate_step(st, z, k, {}, s, op)
    zh = torch.empty(n, dtype=torch.float32, device="cuda")
    info = ctx.surrogate_step(k, wdc.make_cond(), zh)
    beta = np.array(list(info.kappa)[:K])
    assert np.allclose(beta, info_o["kappa"], rtol=1e-5, atol=1e-9)     # s_hat carries the fp32 sketch sums
    assert rel_l2(zh.cpu().numpy(), zh_o) <= 1e-5
    assert abs(np.sum(beta) - 1.0) > 1e-6            # not a convex combination: a genuine linear readout
