"""Synthetic latent-transition diagnostics on the GPU (section "Motivation
and Observations", Fig. 2; section "Transition Risk Controller", Fig. 3).

Every transition runs through the C ABI (the fused step passes and the
denoiser), and so does every reduction: the latent sums behind the downstream
impact and the direction error come from wdc_latent_pair_stats, the local
defect d_t from the anchor pass (Eq. 7), the schedule from
wdc_schedule_sigmas and the correlations from wdc_correlations.  This module
only sequences the calls and combines a few reduced scalars.  Readings (the
paper defers the details to supplementary material):

* Single-injection downstream impact (Observation 1).  The all-exact
  trajectory is rolled out with the cache's bookkeeping active (tau_risk < 0:
  every step exact, a counterfactual candidate z_hat_t built whenever the
  bank is non-empty).  For an injection step t, z_hat_t replaces the exact
  z_{t+1} and exact inference resumes to the end:
      d_t      = mean|z_{t+1} - z_hat_t| / (mean|z_{t+1}| + eps)   (Eq. 7 form)
      D_down_t = ||z_T^inj - z_T|| / ||z_T||
  with the controller's d_hat_t, w_t, Delta_t at that step.  A false-safe
  case of the instantaneous criterion has d_t <= tau_d but D_down_t > tau_D;
  of the future-weighted criterion, w_t d_t <= tau_d but D_down_t > tau_D.
* Direction error over a cache streak (Observation 2): with periodic
  placement, at every step with a candidate, the angle between z_hat_t - z_t
  and the exact increment Psi(z_t, F(z_t)) - z_t from the same state, binned
  by the streak position (pre-decision age).
* Predicted versus counterfactual defect at exact anchors (Fig. 3a): the
  (d_hat_t, d_cf_t) pairs of a cached rollout's exact steps that had a
  supported, finite candidate, with Pearson and Spearman correlations.
"""
import argparse
import json
import time

import numpy as np

from . import wdc


def downstream_rel(ctx, z_inj, z_ref):
    """||z_inj - z_ref|| / ||z_ref|| from the device sums of wdc_latent_pair_stats."""
    s = ctx.latent_pair_stats(z_inj, z_ref)
    return float(np.sqrt(s[3] / s[4]))


def increment_angle(ctx, z_hat, z_ex, z):
    """Angle between the increments z_hat - z and z_ex - z from the device
    sums of wdc_latent_pair_stats; an increment of zero length has no
    direction and is reported as pi/2."""
    s = ctx.latent_pair_stats(z_hat, z_ex, z)
    if s[0] == 0.0 or s[1] == 0.0:
        return float(np.pi / 2)
    return float(np.arccos(np.clip(s[2] / np.sqrt(s[0] * s[1]), -1.0, 1.0)))


class _Stepper:
    """Step-level driving of one context: current latent, candidate and
    velocity buffers on the device."""

    def __init__(self, ctx, cond_list, cond_tokens):
        import torch
        self.torch = torch
        self.ctx = ctx
        self.conds = cond_list
        self.tokens = cond_tokens
        n = ctx.numel
        dev = torch.device("cuda")
        self.zbuf = [torch.empty(n, device=dev) for _ in range(2)]
        self.zh = torch.empty(n, device=dev)
        self.v = torch.empty(n, device=dev)
        self.zex = torch.empty(n, device=dev)
        self.sigmas = None

    def cond(self, k):
        return self.conds[k] if len(self.conds) > 1 else self.conds[0]

    def tok(self, k):
        return self.tokens[k] if isinstance(self.tokens, (list, tuple)) else self.tokens

    def velocity(self, k, z):
        self.ctx.dit_forward(z, 1000.0 * self.sigmas[k], self.tok(k), self.v)

    def native_from(self, z0, k0):
        """Exact inference from z0 (device) at step k0 to the end; returns the
        device buffer holding the final latent."""
        T = len(self.sigmas) - 1
        cur = self.zbuf[0]
        cur.copy_(z0)
        for k in range(k0, T):
            self.velocity(k, cur)
            self.ctx.scheduler_step(k, cur, self.v, cur)
        return cur


def _view(ptr, n):
    import torch

    class _A:
        def __init__(self):
            self.__cuda_array_interface__ = {"shape": (n,), "typestr": "<f4", "data": (int(ptr), False), "version": 2}

    return torch.as_tensor(_A(), device="cuda")


def downstream_impact(ctx, z_T, conds, cond_tokens, steps=None, tau_d=0.025, tau_D=0.06):
    """Single-injection diagnostics on the GPU (module docstring).  The
    context's tau_risk must be negative.  Returns the same dict layout as the
    CPU oracle's ``downstream_impact``."""
    assert ctx.params.tau_risk < 0
    torch = __import__("torch")
    T = ctx.sched.T
    st = _Stepper(ctx, conds, cond_tokens)
    st.sigmas = ctx.sigmas()
    n = ctx.numel
    ctx.state_reset(z_T)
    cur = z_T
    infos, cands = [], []
    for k in range(T):
        info = ctx.surrogate_step(k, st.cond(k), st.zh)
        assert info.decision == 0
        ok = bool(info.supported and info.finite)
        cands.append(st.zh.clone() if ok else None)
        st.velocity(k, cur)
        full = wdc.StepInfo()
        nxt = ctx.risk_update(k, st.cond(k), cur, st.v, st.zh if ok else None, full)
        d = info.as_dict()
        d["d_cf"] = full.d_cf
        infos.append(d)
        cur = _view(nxt, n).clone()
    z_final = cur.clone()
    rows = []
    for t, zh in enumerate(cands):
        if zh is None or (steps is not None and t not in steps):
            continue
        z_inj = st.native_from(zh, t + 1)
        i = infos[t]
        rows.append({"t": t, "d": float(i["d_cf"]), "D_down": downstream_rel(ctx, z_inj, z_final),
                     "d_hat": float(i["d_hat"]), "w": float(i["w"]), "delta": float(i["delta"])})
        torch.cuda.synchronize()
    m = max(1, len(rows))
    inst = sum(1 for r in rows if r["d"] <= tau_d and r["D_down"] > tau_D) / m
    fut = sum(1 for r in rows if r["w"] * r["d"] <= tau_d and r["D_down"] > tau_D) / m
    return {"rows": rows, "false_safe_instantaneous": inst, "false_safe_future_weighted": fut}


def proxy_vs_counterfactual(ctx, z_T, conds):
    """(d_hat_t, d_cf_t) at the exact anchors of one cached rollout (Fig. 3a)."""
    torch = __import__("torch")
    out = torch.empty_like(z_T)
    _, trace = ctx.rollout(z_T, conds, out)
    return [(float(i["d_hat"]), float(i["d_cf"])) for i in trace if i["decision"] == 0 and np.isfinite(i["d_cf"])]


def direction_errors(ctx, z_T, conds, cond_tokens):
    """Direction error over cache streaks on the GPU (module docstring); the
    context's parameters should select periodic placement."""
    T = ctx.sched.T
    st = _Stepper(ctx, conds, cond_tokens)
    st.sigmas = ctx.sigmas()
    n = ctx.numel
    ctx.state_reset(z_T)
    cur = z_T.clone()
    rows = []
    cand = [st.zh, st.zbuf[1]]
    ci = 0
    for k in range(T):
        zh = cand[ci]
        age = ctx.state_get().age
        info = ctx.surrogate_step(k, st.cond(k), zh)
        st.velocity(k, cur)
        ctx.scheduler_step(k, cur, st.v, st.zex)
        if info.supported and info.finite:
            rows.append({"k": k, "streak": age, "decision": info.decision,
                         "angle": increment_angle(ctx, zh, st.zex, cur)})
        if info.decision == 1:
            cur = zh.clone()
            ci ^= 1
        else:
            nxt = ctx.risk_update(k, st.cond(k), cur, st.v, zh if (info.supported and info.finite) else None)
            cur = _view(nxt, n).clone()
    by = {}
    for r in rows:
        by.setdefault(r["streak"], []).append(r["angle"])
    return {"rows": rows, "mean_by_streak": {s: float(np.mean(a)) for s, a in sorted(by.items())}}


def main():
    """Diagnostics at the 5B-scale shape (random-init weights): a few
    single injections and the direction error per strategy."""
    import torch
    ap = argparse.ArgumentParser()
    ap.add_argument("--inject", type=int, nargs="*", default=[5, 15, 25, 35, 45])
    ap.add_argument("--period", type=int, default=5)
    ap.add_argument("--tau-d", type=float, default=0.025)
    ap.add_argument("--tau-D", type=float, default=0.06)
    args = ap.parse_args()
    from . import synth
    cfg = wdc.make_config(layers=42, hidden=3072, heads=48, head_dim=64, mlp=12288, temb_dim=512, freq_dim=256,
                          in_ch=16, frames=13, height=60, width=90, patch=2, cond_tokens=226, cond_dim=3072,
                          dual_stream=0, dtype=wdc.BF16)
    T = 50
    z0 = synth.latent(0, (16, 13, 60, 90)).reshape(-1)
    ct = torch.from_numpy(synth.cond_tokens(1, 226, 3072)).cuda()
    desc = synth.cond_descriptors(2)
    cond = [wdc.make_cond(ct, desc["cam"], desc["depth"])]
    zT = torch.from_numpy(z0.copy()).cuda()
    out = {}
    t0 = time.perf_counter()
    ctx = wdc.Context(cfg, T, params=wdc.make_params(tau_risk=-1.0))
    ctx.init_weights(0, 0.02)
    r = downstream_impact(ctx, zT, cond, ct, steps=set(args.inject), tau_d=args.tau_d, tau_D=args.tau_D)
    out["downstream"] = {"rows": r["rows"], "false_safe_instantaneous": r["false_safe_instantaneous"],
                         "false_safe_future_weighted": r["false_safe_future_weighted"],
                         "seconds": time.perf_counter() - t0}
    t1 = time.perf_counter()
    ctx.set_cache_params(wdc.make_params(tau_risk=0.1))
    pairs = proxy_vs_counterfactual(ctx, zT, cond)
    pe, sp = wdc.correlations(*zip(*pairs)) if len(pairs) > 2 else (None, None)
    out["proxy_vs_cf"] = {"pairs": len(pairs), "pearson": pe, "spearman": sp, "seconds": time.perf_counter() - t1}
    strategies = {"native secant": wdc.ABL_SECANT, "lifted, no condition": wdc.ABL_NO_COND,
                  "lifted (Eq. 5 as printed)": 0, "lifted, residual reading": wdc.OBS_RESIDUAL}
    out["direction"] = {}
    for name, fl in strategies.items():
        t1 = time.perf_counter()
        ctx.set_cache_params(wdc.make_params(tau_risk=1e9, flags=wdc.ABL_PERIODIC | fl, period=args.period))
        d = direction_errors(ctx, zT, cond, ct)
        out["direction"][name] = {"mean_angle_by_streak": d["mean_by_streak"], "seconds": time.perf_counter() - t1}
    print(json.dumps(out))


if __name__ == "__main__":
    main()
