"""Teacher-forced replay of the full-size cached rollouts against the CPU
oracle: the Aether-5B-like workload (42 layers, 48 x 64 heads, latent
16x13x60x90, 23 exact steps of 50) and the HunyuanVoyager-13B-like one (60
dual-stream layers, 24 x 128 heads, latent 16x13x64x64, 10 exact steps),
exactly as the benchmark runs them (same weights seed, inputs and frozen
tau_risk).

A CPU forward of these models costs about 3e14 flop, so the oracle cannot run
the denoiser.  Instead the GPU rollout is driven through the C ABI's step
calls (wdc_surrogate_step, wdc_dit_forward, wdc_risk_update), which must give
the same decisions and the bitwise-same final latent as wdc_rollout, and the
velocity v_k of every exact step is recorded.  The oracle then replays the
method itself -- lift, retrieval, evolution, observation (Eq. 2-5), proxy,
calibration, risk and decision (Eq. 6-10) and Psi (Eq. 1) -- in fp64 with those
v_k in place of its own denoiser.  Bar: the identical decision sequence (every
oracle decision clear of its threshold by a guard band), the controller's
scalars of every step within 1e-5 relative, and the final latent within 2e-2
relative L2 (fp32 storage on both sides: ~1e-6 expected)."""
import numpy as np
import pytest
import torch

from helpers import device_view, params_for_both, rel_l2
from oracle import rollout as ro
from oracle import schedule as sch
from paper_2608_01845_gb300 import wdc

pytestmark = pytest.mark.gpu
TOL = 1e-5
LATENT_TOL = 2e-2
GUARD = 1e-5          # a decision margin below this could flip on fp32 reductions


def _stepped_rollout(ctx, zT_d, cond, tokens):
    """The cached rollout driven step by step through the C ABI, as
    wdc_rollout runs it; returns (decisions, per-step infos, final latent,
    {k: v_k on the host} for the exact steps)."""
    T = ctx.sched.T
    sig = ctx.sigmas()
    n = ctx.numel
    cand = [torch.empty(n, dtype=torch.float32, device="cuda") for _ in range(2)]
    v = torch.empty(n, dtype=torch.float32, device="cuda")
    cur = zT_d.clone()
    ctx.state_reset(cur)
    ci = 1
    dec, infos, vs = [], [], {}
    for k in range(T):
        zh = cand[ci]
        info = ctx.surrogate_step(k, cond, zh)
        d = info.as_dict()
        if info.decision == 1:
            cur = zh
            ci ^= 1
        else:
            ctx.dit_forward(cur, float(1000.0 * sig[k]), tokens, v)
            vs[k] = v.cpu().numpy().copy()
            full = wdc.StepInfo()
            ok = bool(info.supported and info.finite)
            nxt = ctx.risk_update(k, cond, cur, v, zh if ok else None, full)
            d.update(d_cf=full.d_cf, R=full.R, eta=full.eta, r=full.r)
            cur = device_view(nxt, n)         # the bank slot holding z_exact
            ci = 0
        dec.append(info.decision)
        infos.append(d)
    return dec, infos, cur.cpu().numpy().copy(), vs


@pytest.mark.parametrize("name", ["5b", "13b"])
def test_full_size_rollout_teacher_forced_replay(name):
    import bench
    w = bench.WORKLOADS[name]
    T = w["T"]
    op, cp = params_for_both(tau_risk=w["tau_risk"])
    ctx = wdc.Context(bench.dit_config(w), T, params=cp)
    try:
        ctx.init_weights(w["weight_seed"], 0.02)
        zT, ct, desc = bench.inputs(w, 0)
        zT_d = torch.from_numpy(zT).cuda()
        ct_d = torch.from_numpy(ct).cuda()
        cond = wdc.make_cond(ct_d, desc["cam"], desc["depth"])

        # the benchmark's own call
        out = torch.empty_like(zT_d)
        dec_r, tr_r = ctx.rollout(zT_d, cond, out)
        assert T - sum(dec_r) == w["target_exact"]
        # the same rollout through the step calls, recording v_k
        dec_s, tr_s, z_s, vs = _stepped_rollout(ctx, zT_d, cond, ct_d)
        assert dec_s == dec_r
        assert np.array_equal(z_s, out.cpu().numpy())
        assert ctx.device_errors() == 0
        sig = ctx.sigmas()
    finally:
        ctx.close()
        torch.cuda.empty_cache()

    def recorded(z, t, c, k):
        assert k in vs, f"the oracle takes an exact step at k={k} where the GPU did not"
        return vs[k]

    sig_o = sch.sigmas(T)
    assert np.allclose(sig, sig_o, rtol=0, atol=1e-15)
    zf_o, dec_o, tr_o = ro.cached_rollout(zT, recorded, desc, sig_o, op)
    margins = [min(i["margins"]) for i in tr_o if i["margins"]]
    assert min(margins) > GUARD, min(margins)
    assert dec_o == dec_r
    for a, b in zip(tr_r, tr_o):
        assert a["supported"] == int(b["supported"]) and a["n_compat"] == b["n_compat"], a["k"]
        for key in ["p", "d_hat", "w", "R_cand", "R", "eta", "alpha"]:
            assert abs(a[key] - b[key]) <= TOL * max(1.0, abs(b[key])), (a["k"], key)
        if not np.isnan(b["d_cf"]):
            assert abs(a["d_cf"] - b["d_cf"]) <= TOL * max(1.0, abs(b["d_cf"])), a["k"]
    err = rel_l2(z_s, zf_o)
    assert err <= LATENT_TOL
    print(f"{name}: {T - sum(dec_o)} exact steps, final latent rel L2 {err:.2e}, "
          f"smallest decision margin {min(margins):.2e}")
