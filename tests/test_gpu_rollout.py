"""Cached rollout on the GPU against the CPU oracle (2-layer D=256 model,
latent 16x4x16x16, fp32 parity mode): the anchor/skip decision sequence must
be identical and the final latent within 1e-5 relative L2 (fp32 kernels vs
fp64), for the host-driven rollout and for the device-side control flow.
Plus the invariants: all-exact == native bitwise, host-pointer API ==
device-pointer API, and the printed 7-of-50 exact-call budget."""
import json
import os

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
GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
PARITY_MODEL = dict(layers=2, hidden=256, heads=4, head_dim=64, mlp=1024, temb_dim=256, freq_dim=256, in_ch=16, frames=4,
            height=16, width=16, patch=2, cond_tokens=16, cond_dim=256, dual_stream=0)


def _setup(T, **pkw):
    op, cp = params_for_both(**pkw)
    W = synth.dit_weights(PARITY_MODEL, 0, std=0.02)
    ctx = wdc.Context(wdc.make_config(dtype=wdc.F32, **PARITY_MODEL), T, params=cp)
    ctx.set_weights(W)
    z0 = synth.latent(1, (16, 4, 16, 16))
    ct = synth.cond_tokens(2, 16, 256)
    desc = synth.cond_descriptors(3)
    return op, cp, W, ctx, z0, ct, desc


def _oracle(op, W, z0, ct, desc, T):
    cfg = DiTConfig(**PARITY_MODEL)
    F = lambda z, t, c, k: dit.forward(W, cfg, np.asarray(z).reshape(16, 4, 16, 16), t, ct)
    return ro.cached_rollout(z0, F, desc, sch.sigmas(T), op)


def test_cfg0_decisions_and_latent_match_oracle():
    T = 10
    op, cp, W, ctx, z0, ct, desc = _setup(T, tau_risk=0.5)
    zf_o, dec_o, tr_o = _oracle(op, W, z0, ct, desc, T)
    assert 0 < sum(dec_o) < T                       # both decisions occur
    for info in tr_o:
        if info["margins"]:
            assert min(info["margins"]) > 1e-4
    c = wdc.make_cond(torch.from_numpy(ct).cuda(), desc["cam"], desc["depth"])
    out = torch.empty(z0.size, dtype=torch.float32, device="cuda")
    dec, tr = ctx.rollout(torch.from_numpy(z0.ravel().copy()).cuda(), c, out)
    assert dec == dec_o
    assert rel_l2(out.cpu().numpy(), zf_o) <= TOL
    _check_trace(tr, tr_o)


TOL = 1e-5


def _check_trace(tr, tr_o, d_cf=True):
    for a, b in zip(tr, tr_o):
        assert a["decision"] == b["decision"]
        for key in ["p", "d_hat", "w", "R_cand", "R", "eta"]:
            assert abs(a[key] - b[key]) <= TOL * max(1.0, abs(b[key])), (a["k"], key)
        if d_cf and not np.isnan(b["d_cf"]):
            assert abs(a["d_cf"] - b["d_cf"]) <= TOL * max(1.0, b["d_cf"])


@pytest.mark.parametrize("flags", [0, wdc.ABL_SECANT])
def test_graph_rollout_matches_oracle(flags):
    """wdc_rollout_graph (device-side control flow) against the CPU oracle's
    cached rollout directly: the same decision sequence, the final latent
    within 1e-5 relative L2 and the controller scalars of every step within
    1e-5 relative."""
    T = 10
    op, cp, W, ctx, z0, ct, desc = _setup(T, tau_risk=0.5, flags=flags)
    zf_o, dec_o, tr_o = _oracle(op, W, z0, ct, desc, T)
    assert 0 < sum(dec_o) < T
    for info in tr_o:
        if info["margins"]:
            assert min(info["margins"]) > 1e-4
    c = wdc.make_cond(torch.from_numpy(ct).cuda(), desc["cam"], desc["depth"])
    out = torch.empty(z0.size, dtype=torch.float32, device="cuda")
    dec, tr = ctx.rollout_graph(torch.from_numpy(z0.ravel().copy()).cuda(), c, out)
    assert dec == dec_o
    assert rel_l2(out.cpu().numpy(), zf_o) <= TOL
    _check_trace(tr, tr_o)
    assert ctx.device_errors() == 0


def test_all_exact_equals_native_bitwise():
    T = 6
    op, cp, W, ctx, z0, ct, desc = _setup(T, tau_risk=-1.0)
    c = wdc.make_cond(torch.from_numpy(ct).cuda(), desc["cam"], desc["depth"])
    zT = torch.from_numpy(z0.ravel().copy()).cuda()
    a = torch.empty_like(zT)
    b = torch.empty_like(zT)
    dec, _ = ctx.rollout(zT, c, a)
    ctx.native_rollout(zT, c, b)
    torch.cuda.synchronize()
    assert dec == [0] * T
    assert torch.equal(a, b)


def test_host_pointer_rollout_equals_device_rollout():
    T = 10
    op, cp, W, ctx, z0, ct, desc = _setup(T, tau_risk=0.5)
    zT = torch.from_numpy(z0.ravel().copy())
    dev_out = torch.empty(zT.numel(), dtype=torch.float32, device="cuda")
    c_dev = wdc.make_cond(torch.from_numpy(ct).cuda(), desc["cam"], desc["depth"])
    d1, _ = ctx.rollout(zT.cuda(), c_dev, dev_out)
    host_in = zT.pin_memory()
    host_out = torch.empty(zT.numel(), dtype=torch.float32).pin_memory()
    ct_host = torch.from_numpy(ct.copy()).pin_memory()
    c_host = wdc.make_cond(ct_host, desc["cam"], desc["depth"])
    d2, _ = ctx.rollout(host_in, c_host, host_out)
    assert d1 == d2
    assert torch.equal(host_out, dev_out.cpu())


def test_host_condition_staging_grows_and_is_reused():
    """Host condition tokens go through the context's staging buffer: one
    condition, then one per step (the buffer grows), then one again; each
    rollout equals the same rollout from device tokens bitwise."""
    T = 10
    op, cp, W, ctx, z0, ct, desc = _setup(T, tau_risk=0.5)
    zT = torch.from_numpy(z0.ravel().copy()).cuda()
    cts = [synth.cond_tokens(10 + k, 16, 256) for k in range(T)]
    for tokens in ([ct], cts, [ct]):
        dev = [wdc.make_cond(torch.from_numpy(x).cuda(), desc["cam"], desc["depth"]) for x in tokens]
        host = [wdc.make_cond(torch.from_numpy(x.copy()).pin_memory(), desc["cam"], desc["depth"]) for x in tokens]
        a = torch.empty_like(zT)
        b = torch.empty_like(zT)
        d1, _ = ctx.rollout(zT, dev, a)
        d2, _ = ctx.rollout(zT, host, b)
        assert d1 == d2
        assert torch.equal(a, b)


def test_age_convention_budget_on_gpu():
    gold = json.load(open(os.path.join(GOLDEN, "age_convention.json")))
    T = gold["T"]
    op, cp, W, ctx, z0, ct, desc = _setup(T, tau_risk=1e9, sim_min=-2.0, q_gap_max=1.0, max_age=gold["max_age"])
    c = wdc.make_cond(torch.from_numpy(ct).cuda(), desc["cam"], desc["depth"])
    out = torch.empty(z0.size, dtype=torch.float32, device="cuda")
    dec, _ = ctx.rollout(torch.from_numpy(z0.ravel().copy()).cuda(), c, out)
    assert [k for k, d in enumerate(dec) if d == 0] == gold["exact_steps"]
    assert torch.isfinite(out).all()


@pytest.mark.parametrize("flags", [0, wdc.ABL_SECANT, wdc.OBS_RESIDUAL])
def test_graph_rollout_equals_host_rollout(flags):
    """wdc_rollout_graph (device-side control flow: WHILE / SWITCH / IF graph
    nodes, decisions set on the device) against the host-driven rollout of
    the same context: identical decisions and trace, bitwise-identical latent;
    a second call reuses the graph."""
    T = 10
    op, cp, W, ctx, z0, ct, desc = _setup(T, tau_risk=0.5, flags=flags)
    c = wdc.make_cond(torch.from_numpy(ct).cuda(), desc["cam"], desc["depth"])
    zT = torch.from_numpy(z0.ravel().copy()).cuda()
    out_h = torch.empty(z0.size, dtype=torch.float32, device="cuda")
    dec_h, tr_h = ctx.rollout(zT, c, out_h)
    assert 0 < sum(dec_h) < T
    for rep in range(2):
        out_g = torch.empty_like(out_h)
        dec_g, tr_g = ctx.rollout_graph(zT, c, out_g)
        assert dec_g == dec_h
        assert torch.equal(out_g, out_h)
        for a, b in zip(tr_g, tr_h):
            for key in ["decision", "n_bank", "age", "p", "d_hat", "w", "R_cand", "R", "eta", "alpha"]:
                assert a[key] == b[key], (rep, a["k"], key)
    assert ctx.device_errors() == 0


def test_graph_rollout_all_exact_is_native_and_host_buffers():
    T = 6
    op, cp, W, ctx, z0, ct, desc = _setup(T, tau_risk=-1.0)
    c = wdc.make_cond(torch.from_numpy(ct).cuda(), desc["cam"], desc["depth"])
    zT = torch.from_numpy(z0.ravel().copy()).cuda()
    nat = torch.empty_like(zT)
    ctx.native_rollout(zT, c, nat)
    zh = torch.from_numpy(z0.ravel().copy()).pin_memory()
    outh = torch.empty_like(zh).pin_memory()
    ch = wdc.make_cond(torch.from_numpy(ct).pin_memory(), desc["cam"], desc["depth"])
    dec, _ = ctx.rollout_graph(zh, ch, outh)
    assert dec == [0] * T
    assert torch.equal(outh, nat.cpu())


def test_graph_rollout_dual_stream_bf16_equals_host():
    """bf16 dual-stream model: the captured forward forks the condition rows
    onto a second stream; graph and host rollouts agree bitwise."""
    T = 8
    cfg = dict(PARITY_MODEL, dual_stream=1)
    W = synth.dit_weights(cfg, 0, std=0.02)
    _, cp = params_for_both(tau_risk=0.5)
    ctx = wdc.Context(wdc.make_config(dtype=wdc.BF16, **cfg), T, params=cp)
    ctx.set_weights(W)
    z0 = synth.latent(1, (16, 4, 16, 16))
    ct = synth.cond_tokens(2, 16, 256)
    desc = synth.cond_descriptors(3)
    c = wdc.make_cond(torch.from_numpy(ct).cuda(), desc["cam"], desc["depth"])
    zT = torch.from_numpy(z0.ravel().copy()).cuda()
    out_h = torch.empty_like(zT)
    dec_h, _ = ctx.rollout(zT, c, out_h)
    out_g = torch.empty_like(zT)
    dec_g, _ = ctx.rollout_graph(zT, c, out_g)
    assert dec_g == dec_h and torch.equal(out_g, out_h)
