"""Pins of the oracle's batched and guided rollouts (serving extensions; the
paper rolls out one trajectory at a time and is silent on guidance): the
closed forms of the guidance formula on a real DiT forward, and the batch's
independence of its samples."""
import numpy as np

from oracle import batch as ob
from oracle import dit
from oracle import rollout as ro
from oracle import schedule as sch
from oracle.params import CacheParams, DiTConfig
from paper_2608_01845_gb300 import synth

TINY = dict(layers=1, hidden=64, heads=2, head_dim=32, mlp=128, temb_dim=64, freq_dim=32, in_ch=4, frames=2,
            height=4, width=4, patch=2, cond_tokens=4, cond_dim=32, dual_stream=0)


def _model(seed=1):
    cfg = DiTConfig(**TINY)
    W = synth.dit_weights(TINY, seed, std=0.2, bias_std=0.05)
    z = synth.latent(seed + 1, (4, 2, 4, 4))
    ct = synth.cond_tokens(seed + 2, 4, 32)
    return cfg, W, z, ct


def test_guidance_closed_forms_on_the_dit():
    cfg, W, z, ct = _model()
    vc = dit.forward(W, cfg, z, 600.0, ct)
    vu = dit.forward(W, cfg, z, 600.0, ob.null_tokens(cfg))
    assert np.linalg.norm(vc - vu) > 1e-3 * np.linalg.norm(vc)          # the condition matters
    F = lambda g: ob.denoiser(W, cfg, ct, guidance=g)(z, 600.0, {}, 0)
    # g = 1: the conditional velocity; g = 0: the unconditional one
    assert np.allclose(F(1.0), vc, rtol=0, atol=1e-12 * np.abs(vc).max())
    assert np.array_equal(F(0.0), vu)
    # affine in g: v(g) = v(0) + g (v(1) - v(0))
    for g in (2.5, -0.5, 7.0):
        assert np.allclose(F(g), vu + g * (vc - vu), rtol=1e-12, atol=1e-12)
    # no guidance: the plain forward
    assert np.array_equal(ob.denoiser(W, cfg, ct)(z, 600.0, {}, 0), vc)


def test_null_condition_makes_guidance_inert():
    cfg, W, z, _ = _model(3)
    zero = ob.null_tokens(cfg)
    v1 = ob.denoiser(W, cfg, zero, guidance=1.0)(z, 300.0, {}, 0)
    v5 = ob.denoiser(W, cfg, zero, guidance=5.0)(z, 300.0, {}, 0)
    assert np.array_equal(v1, v5)


def test_null_tokens_shape_and_value():
    cfg = DiTConfig(**TINY)
    n = ob.null_tokens(cfg)
    assert n.shape == (4, 32) and not n.any()


def _lin(scale):
    def F(z, t, c, k):
        z = np.asarray(z, dtype=np.float64)
        return -scale * z + 0.05 * np.sin(np.arange(z.size) * 0.01 + 0.001 * t)
    return F


def test_batch_is_independent_samples():
    T, n = 16, 2048
    s = sch.sigmas(T)
    zs = [synth.latent(10 + b, (n,)) for b in range(3)]
    Fs = [_lin(0.8), _lin(0.6), _lin(1.1)]
    conds = [{}, {"cam": np.full(4, 0.1), "depth": np.zeros(4)}, {}]
    ps = [CacheParams(tau_risk=t, sim_min=-1.0) for t in (0.3, 0.8, 1e9)]
    finals, decs, _ = ob.rollout_batch(zs, Fs, conds, s, ps)
    for b in range(3):
        zf, dec, _ = ro.cached_rollout(zs[b], Fs[b], conds[b], s, ps[b])
        assert dec == decs[b] and np.array_equal(zf, finals[b])
    # permuting the samples permutes the results
    perm = [2, 0, 1]
    f2, d2, _ = ob.rollout_batch([zs[i] for i in perm], [Fs[i] for i in perm], [conds[i] for i in perm], s,
                                 [ps[i] for i in perm])
    for j, i in enumerate(perm):
        assert d2[j] == decs[i] and np.array_equal(f2[j], finals[i])
    # the samples' own constants give them different anchor patterns
    assert len({tuple(d) for d in decs}) > 1
