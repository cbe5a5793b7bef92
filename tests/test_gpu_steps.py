"""Parity of the fused step kernels (skip pass: Eq. 2-6, 9, 10; anchor pass:
Eq. 1, 7, 8 and the bank insertion) with the CPU oracle, element by element,
on seeded synthetic banks with smooth drift.  Tolerance: 1e-5 relative for the
fp32 latents and the reduced statistics; decisions and integer fields exact."""
import copy
import math

import numpy as np
import pytest
import torch

from helpers import device_view, make_state, params_for_both, rel_l2, state_to_host
from oracle import rollout as ro
from oracle import schedule as sch
from paper_2608_01845_gb300 import synth, wdc

pytestmark = pytest.mark.gpu
TOL = 1e-5


def _ctx(n, cp, T):
    cfg = wdc.make_config(layers=0, in_ch=1, frames=1, height=1, width=n)
    return wdc.Context(cfg, T, params=cp)


def _setup(n, K, seed, T=50, k=20, **pkw):
    op, cp = params_for_both(bank_capacity=max(K, 1), **pkw)
    sig = sch.sigmas(T)
    q_k = float(sig[k])
    z_k = synth.latent(seed, (n,))
    st = make_state(seed + 7, z_k, K, n, q_k, T, p=op)
    cond = synth.cond_descriptors(seed + 3)
    return op, cp, sig, z_k, st, cond


def _run_skip(n, K, seed, tau_shift=None, T=50, k=20, **pkw):
    op, cp, sig, z_k, st, cond = _setup(n, K, seed, T, k, **pkw)
    # decide tau_risk from the oracle's own R_cand so both decisions are exercised
    probe = copy.deepcopy(st)
    _, info0 = ro.surrogate_step(probe, z_k, k, cond, sig, op)
    if tau_shift is not None:
        op.tau_risk = info0["R_cand"] + tau_shift
        cp.tau_risk = op.tau_risk
    st_o = copy.deepcopy(st)
    zh_o, info_o = ro.surrogate_step(st_o, z_k, k, cond, sig, op)
    assert min(info_o["margins"]) > 1e-4          # guard band for an exact decision match

    ctx = _ctx(n, cp, T)
    dev = torch.device("cuda")
    bank = [torch.from_numpy(r.z_out.copy()).to(dev) for r in st.bank]
    zc = torch.from_numpy(z_k.copy()).to(dev)
    ctx.state_set(state_to_host(st), bank, zc)
    zh = torch.empty(n, dtype=torch.float32, device=dev)
    c = wdc.make_cond(cam=cond["cam"], depth=cond["depth"])
    info = ctx.surrogate_step(k, c, zh)
    return ctx, op, cp, sig, z_k, st, st_o, cond, zh, zh_o, info, info_o, c, bank, zc


def _check_skip(info, info_o, zh, zh_o, K):
    assert info.decision == info_o["decision"]
    assert info.supported == int(info_o["supported"]) and info.n_compat == info_o["n_compat"]
    assert info.finite == int(info_o["finite"])
    for key in ["alpha", "p", "d_hat", "w", "delta", "R_cand", "R", "eta", "d_z"]:
        assert abs(getattr(info, key) - info_o[key]) <= TOL * max(1.0, abs(info_o[key])), key
    if info_o["supported"]:
        assert np.allclose(list(info.kappa)[:K], info_o["kappa"], atol=TOL)
        assert np.allclose(list(info.pi)[:K], info_o["pi"], atol=TOL)
        assert rel_l2(zh.cpu().numpy(), zh_o) <= TOL


@pytest.mark.parametrize("n,K", [(128 * 1000 + 37, 1), (128 * 1000 + 36, 2), (1 << 20, 3), (1 << 20, 4),
                                 (4096 * 3 + 128 * 5 + 64, 8), (1 << 24, 4)])
@pytest.mark.parametrize("tau_shift", [-0.05, 0.05])
def test_skip_pass_parity(n, K, tau_shift):
    (ctx, op, cp, sig, z_k, st, st_o, cond, zh, zh_o, info, info_o, *_rest) = _run_skip(n, K, 11 + K, tau_shift)
    _check_skip(info, info_o, zh, zh_o, K)
    assert info.decision == (1 if tau_shift > 0 else 0)
    # state after the decision, and the candidate statistics the next lift uses
    s = ctx.state_get()
    assert abs(s.R - st_o.R) <= TOL * max(1.0, abs(st_o.R))
    from oracle import summary as sm
    assert np.allclose(np.array(s.s_phi), sm.summary_of_state(z_k, st.z_a, cond["cam"], cond["depth"], float(sig[20]),
                                                             st.history(50, op), op.eps_nu, op.sketch_seed), atol=TOL)
    if info.decision == 1:
        zf = zh_o.astype(np.float64)
        want = sm.sketch(zh_o, op.sketch_seed) / math.sqrt(120.0 / n)
        assert rel_l2(np.array(s.cur_sketch), want) <= TOL
        assert abs(s.cur_sumsq - float(np.sum(zf * zf))) <= TOL * float(np.sum(zf * zf))
        d = zf - st.z_a.astype(np.float64)
        assert abs(s.cur_sumsq_anchor - float(np.sum(d * d))) <= TOL * float(np.sum(d * d))


def test_skip_pass_full_size_64M():
    (ctx, op, cp, sig, z_k, st, st_o, cond, zh, zh_o, info, info_o, *_rest) = _run_skip(1 << 26, 4, 5, 0.05)
    _check_skip(info, info_o, zh, zh_o, 4)


@pytest.mark.parametrize("K", [2, 4])
def test_skip_pass_2e28_sampled_and_reductions(K):
    """The sweep's largest launch (2^28 elements, the bench's bank recipe and
    launch): every output checked by what holds at any size.  The observation
    (Eq. 5) on 2^20 sampled elements plus both ends equals sum_i kappa_i z_i
    with the kernel's own kappa (fp64, 1e-6 of the terms' magnitude); kappa is
    a softmax (non-negative, sums to 1); the statistics the next lift reads --
    the sum of squares of z_hat and of z_hat - z_a, and the signed sketch of
    z_hat -- equal fp64 sums of the kernel's z_hat (the sketch through the
    oracle's sketch) within 1e-5."""
    from oracle import summary as sm
    n, T, k = 1 << 28, 50, 20
    # every record compatible, as in the bench's sweep; a risk threshold no
    # candidate reaches, so the pass commits the candidate's statistics
    op, cp = params_for_both(bank_capacity=K, sim_min=-1.0, q_gap_max=1.0, tau_risk=1e9)
    ctx = _ctx(n, cp, T)
    bank = synth.drift_bank_device(n % 1000003 + K, n, K)
    st = wdc.StateHost()
    st.n_bank, st.R, st.eta = K, 0.1, 1.0
    g = np.random.default_rng(0)
    for i in range(K):
        a = g.standard_normal(256)
        for j in range(256):
            st.rec[i].s_in[j] = a[j]
            st.rec[i].s_out[j] = a[j] + 0.1
            st.rec[i].s_dphi[j] = 0.1
        st.rec[i].q_in = 0.6 + 0.02 * (K - i)
        st.rec[i].q_out = st.rec[i].q_in - 0.02
    st.q_a_in, st.q_a_out = st.rec[K - 1].q_in, st.rec[K - 1].q_out
    zc = bank[-1] + 0.01
    ctx.state_set(st, bank, zc)
    zh = torch.empty(n, device="cuda")
    info = ctx.surrogate_step(k, wdc.make_cond(), zh)
    assert info.supported == 1 and info.finite == 1 and info.decision == 1
    kap = np.array(list(info.kappa)[:K], dtype=np.float64)
    assert np.all(kap >= 0.0) and abs(kap.sum() - 1.0) <= 1e-6
    gen = torch.Generator(device="cuda").manual_seed(3)
    idx = torch.cat([torch.arange(4096, device="cuda"), torch.arange(n - 4096, n, device="cuda"),
                     torch.randint(0, n, (1 << 20,), device="cuda", generator=gen)])
    terms = torch.stack([float(kap[i]) * bank[i][idx].double() for i in range(K)])
    want = terms.sum(0)
    scale = terms.abs().sum(0) + 1e-30
    assert float(((zh[idx].double() - want).abs() / scale).max()) <= 1e-6
    s = ctx.state_get()
    zd = zh.double()
    ss = float((zd * zd).sum())
    assert abs(s.cur_sumsq - ss) <= 1e-5 * ss
    d = zd - bank[-1].double()
    sa = float((d * d).sum())
    assert abs(s.cur_sumsq_anchor - sa) <= 1e-5 * sa
    del zd, d
    want_sk = sm.sketch(zh.cpu().numpy(), op.sketch_seed) / math.sqrt(120.0 / n)
    assert rel_l2(np.array(s.cur_sketch), want_sk) <= 1e-5


@pytest.mark.parametrize("n,K", [(128 * 1000 + 37, 1), (1 << 20, 4), (4096 * 3 + 128 * 5 + 64, 8)])
def test_anchor_pass_parity(n, K):
    (ctx, op, cp, sig, z_k, st, st_o, cond, zh, zh_o, info, info_o, c, bank, zc) = _run_skip(n, K, 23 + K, -0.05)
    assert info.decision == 0
    v = synth.normal(99, (n,), 1.0)
    k = 20
    z_ex_o = ro.exact_step(st_o, z_k, v, zh_o, k, cond, sig, op, info_o)
    vt = torch.from_numpy(v).cuda()
    out_info = wdc.StepInfo()
    addr = ctx.risk_update(k, c, zc, vt, zh if info.supported and info.finite else None, out_info)
    # read z_exact through its device address
    s = ctx.state_get()
    got = device_view(addr, n).clone()
    assert rel_l2(got.cpu().numpy(), z_ex_o) <= 1e-6
    if info_o["supported"] and info_o["finite"]:
        assert abs(out_info.d_cf - info_o["d_cf"]) <= TOL * max(1.0, abs(info_o["d_cf"]))
    assert abs(out_info.eta - st_o.eta) <= TOL * st_o.eta
    assert abs(out_info.R - st_o.R) <= TOL * max(1.0, st_o.R)
    assert abs(out_info.r - info_o["r"]) <= TOL * max(1.0, info_o["r"])
    # the inserted record (newest) and the FIFO order
    assert s.n_bank == len(st_o.bank)
    for i, rec in enumerate(st_o.bank):
        h = s.rec[i]
        # phases are held in fp32 on the device (2^-24 relative)
        assert h.q_in == pytest.approx(rec.q_in, abs=1e-7) and h.q_out == pytest.approx(rec.q_out, abs=1e-7)
    new = s.rec[s.n_bank - 1]
    ref = st_o.bank[-1]
    assert rel_l2(np.array(new.s_in), ref.s_in) <= TOL
    assert rel_l2(np.array(new.s_out), ref.s_out) <= TOL
    assert rel_l2(np.array(new.s_dphi), ref.s_dphi) <= 10 * TOL
    assert s.age == 0 and s.cur_sumsq_anchor == 0.0


def test_nonfinite_bank_forces_exact():
    n, K = 128 * 64, 2
    op, cp, sig, z_k, st, cond = _setup(n, K, 41, tau_risk=1e9)
    st.bank[0].z_out = st.bank[0].z_out.copy()
    st.bank[0].z_out[77] = np.inf                           # host-injected fault
    st_o = copy.deepcopy(st)
    zh_o, info_o = ro.surrogate_step(st_o, z_k, 20, cond, sig, op)
    ctx = _ctx(n, cp, 50)
    bank = [torch.from_numpy(r.z_out.copy()).cuda() for r in st.bank]
    ctx.state_set(state_to_host(st), bank, torch.from_numpy(z_k.copy()).cuda())
    zh = torch.empty(n, dtype=torch.float32, device="cuda")
    info = ctx.surrogate_step(20, wdc.make_cond(cam=cond["cam"], depth=cond["depth"]), zh)
    assert info_o["decision"] == 0 and info.decision == 0
    assert info.supported == 1 and info.finite == 0


def test_empty_bank_and_order_errors():
    n = 4096
    _, cp = params_for_both()
    ctx = _ctx(n, cp, 10)
    z = torch.randn(n, device="cuda")
    ctx.state_reset(z)
    zh = torch.empty_like(z)
    info = ctx.surrogate_step(0, wdc.make_cond(), zh)
    assert info.decision == 0 and info.supported == 0 and info.n_bank == 0
    with pytest.raises(wdc.WdcError) as e:
        ctx.risk_update(3, wdc.make_cond(), z, z, None)     # not preceded by surrogate_step(3)
    assert e.value.status == 6
    with pytest.raises(wdc.WdcError) as e:
        ctx.surrogate_step(10, wdc.make_cond(), zh)         # k out of range
    assert e.value.status == 1
    with pytest.raises(wdc.WdcError) as e:
        ctx.surrogate_step(1, wdc.make_cond(), zh[1:])      # misaligned
    assert e.value.status == 1


def test_scheduler_step_is_one_fma():
    n = 100003
    _, cp = params_for_both()
    ctx = _ctx(n, cp, 7)
    z = torch.randn(n, device="cuda")
    v = torch.randn(n, device="cuda")
    out = torch.empty_like(z)
    ctx.scheduler_step(3, z, v, out)
    sig = sch.sigmas(7)
    dsig = np.float32(sig[4] - sig[3])
    zn, vn = z.cpu().numpy().astype(np.float64), v.cpu().numpy().astype(np.float64)
    want = (zn + float(dsig) * vn)                          # fma: one rounding of the exact value
    assert np.array_equal(out.cpu().numpy(), want.astype(np.float32))


def test_bounded_wait_times_out_and_context_stays_usable():
    """A device wait on an mbarrier that nothing completes gives up after its
    limit, reports the timeout bit, and the context keeps working (the wait
    machinery every tensor-core kernel uses; no GPU fault involved)."""
    import time
    ctx = _ctx(1 << 16, wdc.make_params(), 50)
    assert ctx.device_errors() == 0
    t0 = time.perf_counter()
    ctx.selftest_wait_timeout(2_000_000)            # 2 ms
    bits = ctx.device_errors()                     # synchronises
    assert bits == 1
    assert time.perf_counter() - t0 < 5.0
    assert ctx.device_errors() == 0                # cleared by the read
    with pytest.raises(wdc.WdcError):
        ctx.selftest_wait_timeout(10)              # limit out of range: rejected before launch
    # the context still runs a full step afterwards
    z = torch.randn(1 << 16, device="cuda")
    ctx.state_reset(z)
    zh = torch.empty_like(z)
    info = ctx.surrogate_step(0, wdc.make_cond(), zh)
    assert info.decision == 0 and ctx.device_errors() == 0
