"""Pins of the oracle's DiT denoiser and of the cached / native rollouts
(Eq. 1, Eq. 10, section "Inference and Complexity") against brute force,
closed forms, invariants and the paper's printed budget arithmetic."""
import json
import math
import os

import numpy as np
import pytest
from scipy.special import erf

from oracle import dit
from oracle import rollout as ro
from oracle import schedule as sch
from oracle.params import CacheParams, DiTConfig
from paper_2608_01845_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ------------------------------------------------------------------ DiT pieces
def test_layer_norm_definition():
    x = np.random.default_rng(0).standard_normal((5, 64)) * 3 + 2
    y = dit.layer_norm(x)
    assert np.allclose(y.mean(axis=1), 0, atol=1e-12)
    assert np.allclose((y ** 2).mean(axis=1), 1.0 / (1.0 + 1e-6 / x.var(axis=1)), atol=1e-12)
    assert np.all(dit.layer_norm(np.full((2, 8), 3.0)) == 0.0)


def test_gelu_tanh_against_erf_gelu():
    x = np.linspace(-6, 6, 2001)
    exact = 0.5 * x * (1 + erf(x / math.sqrt(2)))
    assert dit.gelu_tanh(np.array([0.0]))[0] == 0.0
    assert np.max(np.abs(dit.gelu_tanh(x) - exact)) < 1e-3    # tanh form's known accuracy
    assert abs(dit.gelu_tanh(np.array([20.0]))[0] - 20.0) < 1e-12


def _attention_brute(q, k, v, heads):
    Lq, Dm = q.shape
    d = Dm // heads
    out = np.zeros((Lq, Dm))
    for h in range(heads):
        for i in range(Lq):
            scores = [sum(q[i, h * d + e] * k[j, h * d + e] for e in range(d)) / math.sqrt(d) for j in range(k.shape[0])]
            m = max(scores)
            ws = [math.exp(s - m) for s in scores]
            tot = sum(ws)
            for e in range(d):
                out[i, h * d + e] = sum(ws[j] * v[j, h * d + e] for j in range(k.shape[0])) / tot
    return out


def test_attention_brute_force():
    g = np.random.default_rng(1)
    q, k, v = g.standard_normal((5, 8)), g.standard_normal((7, 8)), g.standard_normal((7, 8))
    assert np.allclose(dit.attention(q, k, v, 2), _attention_brute(q, k, v, 2), atol=1e-12)


def test_attention_special_cases():
    g = np.random.default_rng(2)
    k, v = g.standard_normal((9, 4)), g.standard_normal((9, 4))
    # zero query: uniform weights -> mean of V
    assert np.allclose(dit.attention(np.zeros((3, 4)), k, v, 1), v.mean(axis=0)[None, :].repeat(3, 0), atol=1e-14)
    # one dominant key -> that value row
    k2 = k.copy()
    k2[4] = 1000.0 * np.ones(4)
    assert np.allclose(dit.attention(np.ones((1, 4)), k2, v, 1)[0], v[4], atol=1e-12)
    # key permutation invariance
    perm = g.permutation(9)
    q = g.standard_normal((2, 4))
    assert np.allclose(dit.attention(q, k[perm], v[perm], 1), dit.attention(q, k, v, 1), atol=1e-13)


def test_patchify_index_and_roundtrip():
    C, F, H, W, p = 3, 2, 4, 6, 2
    z = np.arange(C * F * H * W, dtype=np.float64).reshape(C, F, H, W)
    tok = dit.patchify(z, p)
    assert tok.shape == (F * (H // p) * (W // p), C * p * p)
    c, f, h, w = 2, 1, 3, 4
    assert tok[f * (H // p) * (W // p) + (h // p) * (W // p) + w // p, c * p * p + (h % p) * p + w % p] == z[c, f, h, w]
    assert np.array_equal(dit.unpatchify(tok, C, F, H, W, p), z)


def test_sinusoids():
    f = dit.timestep_features(0.0, 256)
    assert np.array_equal(f, np.concatenate([np.ones(128), np.zeros(128)]))
    pe = dit.position_embedding(3, 8)
    assert np.allclose(pe[0], [0, 1, 0, 1, 0, 1, 0, 1])
    assert abs(pe[2, 2] - math.sin(2 * 10000 ** (-2 / 8))) < 1e-15


def _tiny_cfg(**kw):
    base = dict(layers=2, hidden=32, heads=2, head_dim=16, mlp=64, temb_dim=32, in_ch=4, frames=2,
                height=4, width=4, patch=2, cond_tokens=3, cond_dim=32, dual_stream=0)
    base.update(kw)
    return DiTConfig(**base)


def test_zero_gates_make_block_identity():
    cfg = _tiny_cfg()
    W = synth.dit_weights(cfg.as_dict(), 3, std=0.2, bias_std=0.1)
    x = np.random.default_rng(3).standard_normal((cfg.tokens, cfg.hidden))
    mod = np.random.default_rng(4).standard_normal((6, cfg.hidden))
    mod[2] = 0.0
    mod[5] = 0.0
    assert np.array_equal(dit.block(x, W, cfg, 0, [mod]), x)


def test_linear_and_block_rows_consistency():
    cfg = _tiny_cfg()
    W = synth.dit_weights(cfg.as_dict(), 5, std=0.2, bias_std=0.1)
    x = np.random.default_rng(5).standard_normal((cfg.tokens, cfg.hidden))
    mod = np.random.default_rng(6).standard_normal((6, cfg.hidden)) * 0.3
    full = dit.block(x, W, cfg, 1, [mod])
    rows = np.array([0, 4, 7, cfg.tokens - 1])
    assert np.allclose(dit.block_rows(x, W, cfg, 1, [mod], rows), full[rows], atol=1e-12)
    # Linear against explicit loops
    Wl, b = W["L0.s0.o.w"], W["L0.s0.o.b"]
    y = dit.linear(x[:2], Wl, b)
    for i in range(2):
        for o in range(3):
            assert abs(y[i, o] - (sum(x[i, j] * float(Wl[o, j]) for j in range(cfg.hidden)) + float(b[o]))) < 1e-12


def test_dual_stream_block_rows_consistency():
    # condition rows (stream 1) and video rows (stream 0) against the full block
    cfg = _tiny_cfg(dual_stream=1)
    W = synth.dit_weights(cfg.as_dict(), 15, std=0.2, bias_std=0.1)
    x = np.random.default_rng(15).standard_normal((cfg.tokens, cfg.hidden))
    mods = [np.random.default_rng(16 + s).standard_normal((6, cfg.hidden)) * 0.3 for s in range(2)]
    full = dit.block(x, W, cfg, 1, mods)
    rows = np.array([0, cfg.cond_tokens - 1, cfg.cond_tokens, cfg.tokens - 1])
    assert np.allclose(dit.block_rows(x, W, cfg, 1, mods, rows), full[rows], atol=1e-12)


def test_zero_final_weights_give_bias_field():
    cfg = _tiny_cfg()
    W = synth.dit_weights(cfg.as_dict(), 7, std=0.2, bias_std=0.5)
    W["final.w"] = np.zeros_like(W["final.w"])
    z = np.random.default_rng(7).standard_normal((cfg.in_ch, cfg.frames, cfg.height, cfg.width))
    c = np.random.default_rng(8).standard_normal((cfg.cond_tokens, cfg.cond_dim))
    v = dit.forward(W, cfg, z, 500.0, c)
    tok = np.tile(W["final.b"].astype(np.float64), (cfg.video_tokens, 1))
    assert np.allclose(v, dit.unpatchify(tok, cfg.in_ch, cfg.frames, cfg.height, cfg.width, cfg.patch), atol=1e-12)


def test_dual_stream_with_equal_weights_equals_single_stream():
    cfg_single = _tiny_cfg(layers=1)
    cfg_dual = _tiny_cfg(layers=1, dual_stream=1)
    W2 = synth.dit_weights(cfg_dual.as_dict(), 9, std=0.2, bias_std=0.1)
    for key in list(W2):
        if key.startswith("L0.s1."):
            W2[key] = W2["L0.s0." + key[len("L0.s1."):]]
    W1 = {k: v for k, v in W2.items() if not k.startswith("L0.s1.")}
    z = np.random.default_rng(9).standard_normal((4, 2, 4, 4))
    c = np.random.default_rng(10).standard_normal((3, 32))
    assert np.allclose(dit.forward(W1, cfg_single, z, 300.0, c), dit.forward(W2, cfg_dual, z, 300.0, c), atol=1e-13)


# ------------------------------------------------------------------ rollouts
def _lin_denoiser(z, t, c, k):
    z = np.asarray(z, dtype=np.float64)
    return -0.8 * z + 0.05 * np.sin(np.arange(z.size) * 0.01 + 0.001 * t)


def test_all_exact_invariant_is_bitwise_native():
    cfg = _tiny_cfg()
    W = synth.dit_weights(cfg.as_dict(), 11, std=0.05, bias_std=0.01)
    z0 = synth.latent(1, (cfg.in_ch, cfg.frames, cfg.height, cfg.width))
    ct = synth.cond_tokens(2, cfg.cond_tokens, cfg.cond_dim)
    F = lambda z, t, c, k: dit.forward(W, cfg, np.asarray(z).reshape(cfg.in_ch, cfg.frames, cfg.height, cfg.width), t, ct)
    s = sch.sigmas(6)
    p = CacheParams(tau_risk=-1.0)
    zc, dec, _ = ro.cached_rollout(z0, F, synth.cond_descriptors(3), s, p)
    zn = ro.native_rollout(z0, F, synth.cond_descriptors(3), s)
    assert dec == [0] * 6
    assert np.array_equal(zc, zn)


def test_age_convention_reproduces_printed_budget():
    gold = json.load(open(os.path.join(GOLDEN, "age_convention.json")))
    T = gold["T"]
    s = sch.sigmas(T)
    p = CacheParams(tau_risk=1e9, max_age=gold["max_age"], n_init_exact=1, n_final_exact=0, sim_min=-1.0)
    z0 = synth.latent(4, (4096,))
    _, dec, _ = ro.cached_rollout(z0, _lin_denoiser, {}, s, p)
    exact = [k for k, d in enumerate(dec) if d == 0]
    assert exact == gold["exact_steps"]
    assert len(exact) == gold["exact_calls"]


def test_streaks_final_window_and_fifo():
    T = 30
    s = sch.sigmas(T)
    p = CacheParams(tau_risk=0.3, n_final_exact=3, bank_capacity=3, sim_min=-1.0)
    z0 = synth.latent(5, (2048,))
    z, dec, tr = ro.cached_rollout(z0, _lin_denoiser, {}, s, p)
    run = 0
    for d in dec:
        run = run + 1 if d == 1 else 0
        assert run <= p.max_age + 1
    assert dec[-3:] == [0, 0, 0] and dec[0] == 0
    assert 0 < sum(dec) < T                               # both decisions occur
    # replay the exact steps: the bank keeps the last 3 records, oldest first
    st = ro.CacheState.initial(z0, s, p)
    z = synth.latent(5, (2048,)).reshape(-1)
    for k in range(T):
        zh, info = ro.surrogate_step(st, z, k, {}, s, p)
        if info["decision"] == 1:
            z = zh
        else:
            z = ro.exact_step(st, z, _lin_denoiser(z, 0, None, k), zh, k, {}, s, p, info)
    exact_k = [k for k, d in enumerate(dec) if d == 0]
    assert [r.q_in for r in st.bank] == [float(s[k]) for k in exact_k[-3:]]


def test_no_self_retrieval_and_counterfactual_on_supported_steps():
    T = 12
    s = sch.sigmas(T)
    p = CacheParams(tau_risk=-1.0, sim_min=-1.0)
    z0 = synth.latent(6, (1024,))
    st = ro.CacheState.initial(z0, s, p)
    z = z0.reshape(-1)
    for k in range(T):
        zh, info = ro.surrogate_step(st, z, k, {}, s, p)
        n_before = len(st.bank)
        z = ro.exact_step(st, z, _lin_denoiser(z, 0, None, k), zh, k, {}, s, p, info)
        assert np.array_equal(st.bank[-1].s_in, info["s_phi"])      # record lifted pre-insertion
        if n_before == 0:
            assert math.isnan(info["d_cf"])                           # no counterfactual without memory
        else:
            assert np.isfinite(info["d_cf"])


def test_nonfinite_candidate_falls_back_to_exact():
    T = 10
    s = sch.sigmas(T)
    p = CacheParams(tau_risk=1e9, sim_min=-1.0)
    z0 = synth.latent(7, (1024,))
    st = ro.CacheState.initial(z0, s, p)
    z = z0.reshape(-1)
    zh, info = ro.surrogate_step(st, z, 0, {}, s, p)
    z = ro.exact_step(st, z, _lin_denoiser(z, 0, None, 0), zh, 0, {}, s, p, info)
    st.bank[-1].z_out = st.bank[-1].z_out.copy()
    st.bank[-1].z_out[17] = np.nan                       # host-injected fault
    zh, info = ro.surrogate_step(st, z, 1, {}, s, p)
    assert info["supported"] and not info["finite"] and info["decision"] == 0
    z = ro.exact_step(st, z, _lin_denoiser(z, 0, None, 1), zh, 1, {}, s, p, info)
    assert np.all(np.isfinite(z)) and math.isnan(info["d_cf"])
