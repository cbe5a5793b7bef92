"""Batched and guided forwards and rollouts on the GPU (serving extensions:
the paper rolls out one trajectory at a time and is silent on classifier-free
guidance).

* A batched forward gives each sample bitwise the velocity of a forward on it
  alone (fp32 SIMT and bf16 tcgen05 paths; single and dual stream; a case
  whose condition-token GEMM moves from the single-CTA to the CTA-pair kernel
  when batched).
* The guided forward against the oracle's guided velocity (fp32 parity
  model, rel L2 <= 1e-5 against fp64).
* wdc_rollout_batch against the oracle's per-sample cached rollouts: three
  samples with their own latents, conditions and thresholds (so that their
  exact steps differ), with and without guidance; decisions identical, final
  latents within 1e-5 relative L2, controller scalars within 1e-4.
* wdc_rollout_batch on the bf16 model equals each sample's wdc_rollout alone,
  bitwise.
* Argument errors: batch above max_batch, a context shared by two samples,
  contexts of different latent size.
* The largest batch (16 forwards, and 8 guided pairs) on the bf16 model.
* Per-step conditions (n_cond = T) and pinned host latents in a batched
  rollout, against each sample's single rollout."""
import numpy as np
import pytest
import torch

from helpers import params_for_both, rel_l2
from oracle import batch as ob
from oracle import dit
from oracle import schedule as sch
from oracle.params import DiTConfig
from paper_2608_01845_gb300 import synth, wdc

pytestmark = pytest.mark.gpu
PARITY_MODEL = dict(layers=2, hidden=256, heads=4, head_dim=64, mlp=1024, temb_dim=256, freq_dim=256, in_ch=16,
                    frames=4, height=16, width=16, patch=2, cond_tokens=16, cond_dim=256, dual_stream=0)
DUAL_128 = dict(PARITY_MODEL, layers=1, heads=2, head_dim=128, dual_stream=1)
WIDE_COND = dict(PARITY_MODEL, layers=1, cond_tokens=96)          # 96 rows alone, 288 in a batch of 3
SHAPE = (16, 4, 16, 16)
N = 16 * 4 * 16 * 16
T = 10


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).cuda()


def _ctx(cfgd, dtype, max_batch, W, params=None):
    ctx = wdc.Context(wdc.make_config(dtype=dtype, max_batch=max_batch, **cfgd), T, params=params)
    ctx.set_weights(W)
    return ctx


@pytest.mark.parametrize("dtype", [wdc.F32, wdc.BF16])
@pytest.mark.parametrize("model", ["single", "dual128", "wide_cond"])
def test_batched_forward_equals_single_forwards(dtype, model):
    cfgd = {"single": PARITY_MODEL, "dual128": DUAL_128, "wide_cond": WIDE_COND}[model]
    W = synth.dit_weights(cfgd, 7, std=0.02, bias_std=0.02)
    ctx = _ctx(cfgd, dtype, 4, W)
    B = 3
    zs = [_dev(synth.latent(30 + b, SHAPE)) for b in range(B)]
    cts = [_dev(synth.cond_tokens(40 + b, cfgd["cond_tokens"], 256)) for b in range(B)]
    vs = [torch.empty(N, device="cuda") for _ in range(B)]
    ctx.dit_forward_batch(zs, 731.0, cts, vs)
    for b in range(B):
        ref = torch.empty(N, device="cuda")
        ctx.dit_forward(zs[b], 731.0, cts[b], ref)
        torch.cuda.synchronize()
        assert torch.equal(vs[b], ref), (model, b)
    assert ctx.device_errors() == 0


def test_guided_forward_matches_oracle():
    W = synth.dit_weights(PARITY_MODEL, 8, std=0.02, bias_std=0.02)
    ctx = _ctx(PARITY_MODEL, wdc.F32, 4, W)
    cfg = DiTConfig(**PARITY_MODEL)
    g = 2.5
    zs = [synth.latent(50 + b, SHAPE) for b in range(2)]
    cts = [synth.cond_tokens(60 + b, 16, 256) for b in range(2)]
    vs = [torch.empty(N, device="cuda") for _ in range(2)]
    ctx.dit_forward_batch([_dev(z) for z in zs], 640.0, [_dev(c) for c in cts], vs, cfg=True, guidance=g)
    torch.cuda.synchronize()
    for b in range(2):
        want = ob.guided_velocity(dit.forward(W, cfg, zs[b], 640.0, cts[b]),
                                  dit.forward(W, cfg, zs[b], 640.0, ob.null_tokens(cfg)), g)
        assert rel_l2(vs[b].cpu().numpy(), want) <= 1e-5


@pytest.fixture(scope="module")
def parity():
    W = synth.dit_weights(PARITY_MODEL, 0, std=0.02)
    cfg = DiTConfig(**PARITY_MODEL)
    zs = [synth.latent(1 + b, SHAPE) for b in range(3)]
    cts = [synth.cond_tokens(2 + 7 * b, 16, 256) for b in range(3)]
    descs = [synth.cond_descriptors(3 + b) for b in range(3)]
    return W, cfg, zs, cts, descs


def _memo(F):
    cache = {}

    def G(z, t, c, k):
        key = (np.asarray(z, dtype=np.float32).tobytes(), t)
        if key not in cache:
            cache[key] = F(z, t, c, k)
        return cache[key]

    return G


def _oracle_sample(z, F, desc, taus):
    """The first threshold for which the oracle's rollout of this sample takes
    both decisions with every tie margin above 1e-4 (chosen from the oracle)."""
    from oracle import rollout as ro
    for tau in taus:
        op, cp = params_for_both(tau_risk=tau)
        zf, dec, tr = ro.cached_rollout(z, F, desc, sch.sigmas(T), op)
        if 0 < sum(dec) < T and all(min(t["margins"]) > 1e-4 for t in tr if t["margins"]):
            return cp, zf, dec, tr
    pytest.fail("no threshold separates the decisions")


@pytest.mark.parametrize("guided", [False, True])
def test_rollout_batch_matches_oracle(parity, guided):
    W, cfg, zs, cts, descs = parity
    g = 1.8 if guided else None
    taus = [(0.3, 0.5, 0.8), (0.8, 1.2, 0.5), (0.2, 0.3, 0.5)]
    want, cps = [], []
    for b in range(3):
        F = _memo(ob.denoiser(W, cfg, cts[b], guidance=g))
        cp, zf, dec, tr = _oracle_sample(zs[b], F, descs[b], taus[b])
        want.append((zf, dec, tr))
        cps.append(cp)
    ctxs = [_ctx(PARITY_MODEL, wdc.F32, 6, W, params=cps[0])]
    ctxs += [wdc.Context(wdc.make_config(in_ch=16, frames=4, height=16, width=16), T, params=cps[b])
             for b in (1, 2)]
    ct_d = [_dev(c) for c in cts]
    conds = [wdc.make_cond(ct_d[b], descs[b]["cam"], descs[b]["depth"]) for b in range(3)]
    outs = [torch.empty(N, device="cuda") for _ in range(3)]
    decs, traces = wdc.rollout_batch(ctxs, [_dev(z) for z in zs], conds, outs, cfg=guided, guidance=g or 1.0)
    for b in range(3):
        zf, dec, tr = want[b]
        assert decs[b] == dec, b
        assert rel_l2(outs[b].cpu().numpy(), zf) <= 1e-5, b
        for a, o in zip(traces[b], tr):
            for key in ["p", "d_hat", "w", "R_cand", "R", "eta", "alpha"]:
                assert abs(a[key] - o[key]) <= 1e-4 * max(1.0, abs(o[key])), (b, a["k"], key)
            if not np.isnan(o["d_cf"]):
                assert abs(a["d_cf"] - o["d_cf"]) <= 1e-4 * max(1.0, o["d_cf"]), (b, a["k"])
    # the samples' exact steps differ, so the exact batch size varies
    assert any(len({decs[b][k] for b in range(3)}) > 1 for k in range(T))
    for c in ctxs:
        assert c.device_errors() == 0


def test_rollout_batch_equals_single_rollouts_bf16():
    cfgd = dict(PARITY_MODEL, layers=1)
    W = synth.dit_weights(cfgd, 11, std=0.02, bf16=True)
    B = 3
    zs = [_dev(synth.latent(70 + b, SHAPE)) for b in range(B)]
    cts = [_dev(synth.cond_tokens(80 + b, 16, 256, bf16=True)) for b in range(B)]
    descs = [synth.cond_descriptors(90 + b) for b in range(B)]
    taus = [0.3, 0.6, 1.0]
    conds = [wdc.make_cond(cts[b], descs[b]["cam"], descs[b]["depth"]) for b in range(B)]
    ctxs = [_ctx(cfgd, wdc.BF16, B, W, params=wdc.make_params(tau_risk=taus[0]))]
    ctxs += [wdc.Context(wdc.make_config(in_ch=16, frames=4, height=16, width=16), T,
                         params=wdc.make_params(tau_risk=taus[b])) for b in range(1, B)]
    outs = [torch.empty(N, device="cuda") for _ in range(B)]
    decs, traces = wdc.rollout_batch(ctxs, zs, conds, outs)
    single = _ctx(cfgd, wdc.BF16, 1, W)
    for b in range(B):
        single.set_cache_params(wdc.make_params(tau_risk=taus[b]))
        out = torch.empty(N, device="cuda")
        dec, tr = single.rollout(zs[b], conds[b], out)
        assert dec == decs[b], b
        assert torch.equal(out, outs[b]), b
        assert [t["R"] for t in tr] == [t["R"] for t in traces[b]]


def test_batch_argument_errors(parity):
    W, cfg, zs, cts, descs = parity
    ctx = _ctx(PARITY_MODEL, wdc.F32, 2, W)
    z = [_dev(zs[0]) for _ in range(3)]
    c = [_dev(cts[0]) for _ in range(3)]
    v = [torch.empty(N, device="cuda") for _ in range(3)]
    with pytest.raises(wdc.WdcError) as e:
        ctx.dit_forward_batch(z, 500.0, c, v)                     # 3 > max_batch
    assert e.value.status == 1
    with pytest.raises(wdc.WdcError) as e:
        ctx.dit_forward_batch(z[:2], 500.0, c[:2], v[:2], cfg=True)   # 2 guided = 4 > max_batch
    assert e.value.status == 1
    cond = wdc.make_cond(c[0])
    with pytest.raises(wdc.WdcError) as e:
        wdc.rollout_batch([ctx, ctx], z[:2], [cond, cond], v[:2])     # one context for two samples
    assert e.value.status == 1
    other = wdc.Context(wdc.make_config(in_ch=16, frames=4, height=16, width=8), T)
    with pytest.raises(wdc.WdcError) as e:
        wdc.rollout_batch([ctx, other], z[:2], [cond, cond], v[:2])   # latent sizes differ
    assert e.value.status == 1
    # the context stays usable
    ctx.dit_forward_batch(z[:2], 500.0, c[:2], v[:2])
    torch.cuda.synchronize()
    assert torch.equal(v[0], v[1])


def test_batched_forward_at_max_batch_bf16():
    W = synth.dit_weights(PARITY_MODEL, 9, std=0.02, bias_std=0.02, bf16=True)
    ctx = _ctx(PARITY_MODEL, wdc.BF16, wdc.MAX_BATCH, W)
    B = wdc.MAX_BATCH
    zs = [_dev(synth.latent(100 + b, SHAPE)) for b in range(B)]
    cts = [_dev(synth.cond_tokens(200 + b, 16, 256, bf16=True)) for b in range(B)]
    vs = [torch.empty(N, device="cuda") for _ in range(B)]
    ctx.dit_forward_batch(zs, 420.0, cts, vs)
    for b in (0, 7, B - 1):
        ref = torch.empty(N, device="cuda")
        ctx.dit_forward(zs[b], 420.0, cts[b], ref)
        torch.cuda.synchronize()
        assert torch.equal(vs[b], ref), b
    # a guided batch of 8 pairs fills the same 16 slots
    gv = [torch.empty(N, device="cuda") for _ in range(B // 2)]
    ctx.dit_forward_batch(zs[:B // 2], 420.0, cts[:B // 2], gv, cfg=True, guidance=3.0)
    torch.cuda.synchronize()
    zero = torch.zeros(16, 256, device="cuda")
    for b in (0, B // 2 - 1):
        vc, vu = torch.empty(N, device="cuda"), torch.empty(N, device="cuda")
        ctx.dit_forward(zs[b], 420.0, cts[b], vc)
        ctx.dit_forward(zs[b], 420.0, zero, vu)
        torch.cuda.synchronize()
        assert torch.allclose(gv[b], vu + 3.0 * (vc - vu), rtol=1e-6, atol=1e-6), b
    assert ctx.device_errors() == 0


def test_rollout_batch_per_step_conditions_and_host_latents(parity):
    W, cfg, zs, cts, _ = parity
    B = 2
    descs = [synth.cond_descriptors(300 + b, T, static=False) for b in range(B)]
    ct_d = [_dev(c) for c in cts[:B]]
    conds = [[wdc.make_cond(ct_d[b], d["cam"], d["depth"]) for d in descs[b]] for b in range(B)]
    taus = [0.5, 0.3]
    ctxs = [_ctx(PARITY_MODEL, wdc.F32, B, W, params=wdc.make_params(tau_risk=taus[0]))]
    ctxs.append(wdc.Context(wdc.make_config(in_ch=16, frames=4, height=16, width=16), T,
                            params=wdc.make_params(tau_risk=taus[1])))
    outs = [torch.empty(N, device="cuda") for _ in range(B)]
    decs, tr = wdc.rollout_batch(ctxs, [_dev(z) for z in zs[:B]], conds, outs)
    # host (pinned) latents in and out give the same result
    zh = [torch.from_numpy(np.ascontiguousarray(z, dtype=np.float32).ravel()).pin_memory() for z in zs[:B]]
    oh = [torch.empty(N).pin_memory() for _ in range(B)]
    decs_h, _ = wdc.rollout_batch(ctxs, zh, conds, oh)
    assert decs_h == decs
    for b in range(B):
        assert torch.equal(oh[b], outs[b].cpu())
    # each sample alone, with its per-step conditions
    single = _ctx(PARITY_MODEL, wdc.F32, 1, W)
    for b in range(B):
        single.set_cache_params(wdc.make_params(tau_risk=taus[b]))
        out = torch.empty(N, device="cuda")
        dec, trs = single.rollout(_dev(zs[b]), conds[b], out)
        assert dec == decs[b]
        assert torch.equal(out, outs[b])
        assert [t["d_hat"] for t in trs] == [t["d_hat"] for t in tr[b]]
