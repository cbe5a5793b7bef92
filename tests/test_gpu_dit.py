"""Parity of the denoiser F_theta's CUDA kernels with the CPU oracle.

fp32 mode: full forward of the 2-layer D=256 model (and a dual-stream
variant), rel L2 <= 1e-5 against fp64.  bf16 mode: the GEMM and attention
operators on shapes spanning several tiles with ragged tails, and one block of
the 5B-scale model (L = 17776, D = 3072, 48 x 64 heads) on 256 sampled query
rows; rel L2 <= 2e-2 (bf16 operands, fp32 accumulation) against fp64."""
import numpy as np
import pytest
import torch

from helpers import rel_l2
from oracle import dit
from oracle.params import DiTConfig
from paper_2608_01845_gb300 import synth, wdc

pytestmark = pytest.mark.gpu
BF16_TOL = 2e-2

PARITY_MODEL = dict(layers=2, hidden=256, heads=4, head_dim=64, mlp=1024, temb_dim=256, freq_dim=256, in_ch=16, frames=4,
            height=16, width=16, patch=2, cond_tokens=16, cond_dim=256, dual_stream=0)


def _ctx(cfgd, dtype, T=10):
    cfg = wdc.make_config(dtype=dtype, **cfgd)
    return wdc.Context(cfg, T)


def _to_dev(a, dtype=torch.float32):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).cuda().to(dtype)


@pytest.mark.parametrize("dual", [0, 1])
def test_fp32_forward_matches_oracle(dual):
    cfgd = dict(PARITY_MODEL, dual_stream=dual, layers=2 if not dual else 1)
    W = synth.dit_weights(cfgd, 7, std=0.02, bias_std=0.02)
    ctx = _ctx(cfgd, wdc.F32)
    ctx.set_weights(W)
    z = synth.latent(3, (16, 4, 16, 16))
    ct = synth.cond_tokens(4, 16, 256)
    v = torch.empty(z.size, dtype=torch.float32, device="cuda")
    ctx.dit_forward(_to_dev(z), 731.0, _to_dev(ct), v)
    torch.cuda.synchronize()
    want = dit.forward(W, DiTConfig(**cfgd), z, 731.0, ct)
    assert rel_l2(v.cpu().numpy(), want) <= 1e-5


def test_fp32_modulation_matches_oracle():
    W = synth.dit_weights(PARITY_MODEL, 8, std=0.05, bias_std=0.02)
    ctx = _ctx(PARITY_MODEL, wdc.F32)
    ctx.set_weights(W)
    D = 256
    out = torch.empty(2 * 6 * D + 2 * D, dtype=torch.float32, device="cuda")
    ctx.dit_modulation(250.0, out)
    torch.cuda.synchronize()
    _, mods, fm = dit.conditioning(W, DiTConfig(**PARITY_MODEL), 250.0)
    want = np.concatenate([mods[(0, 0)].ravel(), mods[(1, 0)].ravel(), fm.ravel()])
    assert rel_l2(out.cpu().numpy(), want) <= 1e-5


def _bf(a):
    return synth.bf16_round(np.asarray(a, dtype=np.float32))


def _h(a):
    """fp16-rounded values (V^T of the bf16 model is stored in fp16)."""
    return np.asarray(a, dtype=np.float32).astype(np.float16).astype(np.float32)


@pytest.mark.parametrize("M,N,K", [(300, 384, 320), (128, 256, 64), (1000, 768, 1024), (17, 64, 128), (1, 32, 8),
                                   (257, 32, 8)])
@pytest.mark.parametrize("mode", ["store", "gelu", "resid"])
def test_bf16_gemm_matches_oracle(M, N, K, mode):
    """The tcgen05 GEMMs (one CTA per tile below 256 rows, CTA pairs from
    256) with each fused epilogue, down to the smallest shapes they take: one
    row, one 32-column chunk, one 8-element K step (one 64-wide K block,
    zero-filled past K), and a pair grid whose second 256-row tile holds a
    single row."""
    ctx = _ctx(dict(PARITY_MODEL, layers=1), wdc.BF16)
    A = _bf(synth.normal(1, (M, K)))
    W = _bf(synth.normal(2, (N, K), 0.05))
    b = synth.normal(3, (N,), 0.1)
    acc = A.astype(np.float64) @ W.astype(np.float64).T + b
    C = torch.empty(M, N, dtype=torch.bfloat16, device="cuda")
    kw = {}
    if mode == "gelu":
        kw["gelu"] = True
        want = dit.gelu_tanh(acc)
    elif mode == "resid":
        R = _bf(synth.normal(4, (M, N)))
        g = synth.normal(5, (N,), 1.0)
        Rt = _to_dev(R, torch.bfloat16)
        C = Rt                                      # in place, as in the block
        kw.update(res=Rt, gate=_to_dev(g))
        want = R.astype(np.float64) + g * acc
    else:
        want = acc
    ctx.op_gemm(_to_dev(A, torch.bfloat16), _to_dev(W, torch.bfloat16), C, bias=_to_dev(b), **kw)
    torch.cuda.synchronize()
    assert rel_l2(C.float().cpu().numpy(), want) <= 1e-2


@pytest.mark.parametrize("H,L,d", [(2, 1000, 64), (1, 1000, 128), (3, 264, 64), (1, 64, 128), (2, 4104, 64),
                                   (1, 2056, 128), (2, 300, 64), (1, 129, 128), (1, 40, 64), (2, 400, 64),
                                   (1, 1, 64), (2, 7, 128), (2, 100, 64)])
def test_bf16_attention_matches_oracle(H, L, d):
    """Every L runs the tcgen05 kernel, ragged against its 128-key steps and
    256-query CTAs (L = 40 and 400 leave the last CTA one partial query
    tile; L = 1 and 7 are a single ragged step, and at L = 1 the output is
    the one value row); V^T rows are padded to a multiple of 8 tokens, and the padding
    holds NaN to show it is never read."""
    ctx = _ctx(dict(PARITY_MODEL, layers=1), wdc.BF16)
    q = _bf(synth.normal(11, (H, L, d)))
    k = _bf(synth.normal(12, (H, L, d)))
    v = _h(synth.normal(13, (H, L, d)))
    o = torch.empty(L, H * d, dtype=torch.bfloat16, device="cuda")
    ldv = (L + 7) // 8 * 8
    vt = np.full((H, d, ldv), np.nan, dtype=np.float32)
    vt[:, :, :L] = v.transpose(0, 2, 1)
    ctx.op_attention(_to_dev(q, torch.bfloat16), _to_dev(k, torch.bfloat16), _to_dev(vt, torch.float16), o)
    torch.cuda.synchronize()
    qf = q.transpose(1, 0, 2).reshape(L, H * d).astype(np.float64)
    kf = k.transpose(1, 0, 2).reshape(L, H * d).astype(np.float64)
    vf = v.transpose(1, 0, 2).reshape(L, H * d).astype(np.float64)
    want = dit.attention(qf, kf, vf, H)
    assert rel_l2(o.float().cpu().numpy(), want) <= 1e-2


def test_bf16_shapes_outside_the_tensor_core_limits_are_errors():
    """A bf16 model runs on the tcgen05 kernels only: a GEMM shape they do not
    take is reported (WDC_ERR_UNSUPPORTED), never run on a slower path."""
    ctx = _ctx(dict(PARITY_MODEL, layers=1), wdc.BF16)
    launches = ctx.launches
    for M, N, K in [(64, 48, 64), (64, 64, 12)]:
        A = torch.zeros(M, K, dtype=torch.bfloat16, device="cuda")
        W = torch.zeros(N, K, dtype=torch.bfloat16, device="cuda")
        C = torch.empty(M, N, dtype=torch.bfloat16, device="cuda")
        with pytest.raises(wdc.WdcError) as e:
            ctx.op_gemm(A, W, C)
        assert e.value.status == 3 and "tcgen05" in str(e.value)
    assert ctx.launches == launches


@pytest.mark.parametrize("H,L,d", [(2, 300, 64), (2, 257, 128)])
def test_fp32_attention_matches_oracle(H, L, d):
    ctx = _ctx(dict(PARITY_MODEL, layers=1), wdc.F32)
    q, k, v = (synth.normal(s, (H, L, d)) for s in (21, 22, 23))
    o = torch.empty(L, H * d, dtype=torch.float32, device="cuda")
    ctx.op_attention(_to_dev(q), _to_dev(k), _to_dev(np.ascontiguousarray(v.transpose(0, 2, 1))), o)
    torch.cuda.synchronize()
    f = lambda a: a.transpose(1, 0, 2).reshape(L, H * d).astype(np.float64)
    assert rel_l2(o.cpu().numpy(), dit.attention(f(q), f(k), f(v), H)) <= 1e-5


BLOCK5B = dict(layers=1, hidden=3072, heads=48, head_dim=64, mlp=12288, temb_dim=512, freq_dim=256, in_ch=16,
               frames=13, height=60, width=90, patch=2, cond_tokens=226, cond_dim=3072, dual_stream=0)


def test_bf16_block_5b_scale_sampled_rows():
    """One block at the Aether-5B-like shape (L = 226 + 17550 = 17776 tokens),
    compared on 256 seeded rows (keys/values for all rows on the CPU)."""
    cfgd = BLOCK5B
    ctx = _ctx(cfgd, wdc.BF16)
    names = [f"L0.s0.{n}" for n in ["qkv.w", "qkv.b", "o.w", "o.b", "fc1.w", "fc1.b", "fc2.w", "fc2.b"]]
    W = synth.dit_weights(cfgd, 5, std=0.02, bias_std=0.02, bf16=True, names=names)
    ctx.set_weights(W)
    L, D = 17776, 3072
    x = _bf(synth.normal(31, (L, D)))
    mod = synth.normal(32, (6, D), 0.3)
    mod[2] = 1.0 + mod[2]                         # gates of order one: the block's delta dominates
    mod[5] = 1.0 + mod[5]
    xt = _to_dev(x, torch.bfloat16)
    ctx.dit_block_forward(0, xt, _to_dev(mod))
    torch.cuda.synchronize()
    rows = np.sort(np.random.default_rng(33).choice(L, 256, replace=False))
    got = xt.float().cpu().numpy()[rows]
    want = dit.block_rows(x.astype(np.float64), W, DiTConfig(**cfgd), 0, [mod.astype(np.float64)], rows)
    delta_got = got - x[rows]
    delta_want = want - x[rows]
    assert rel_l2(delta_got, delta_want) <= BF16_TOL
    assert rel_l2(got, want) <= BF16_TOL


def test_bench_model_forward_5b_sampled_tokens():
    """The bench's 5B-shape model as the device builds it -- wdc_init_weights
    with the bench's seed (the global tensors and layer 0 draw the same
    Philox streams in a 1-layer context as in the 42-layer one) -- run through
    one full forward (modulation, embeddings, one block in the bench's launch
    configuration, final layer, unpatchify) on the bench's synthetic inputs at
    the first step's timestep, and checked on 64 sampled video tokens (64
    latent entries each) against the oracle evaluated on the weights read back
    from the device."""
    import bench
    w = dict(bench.WORKLOADS["5b"], layers=1)
    keys = ["layers", "hidden", "heads", "head_dim", "mlp", "temb_dim", "freq_dim", "in_ch", "frames", "height",
            "width", "patch", "cond_tokens", "cond_dim", "dual_stream"]
    cfgd = {k: w[k] for k in keys}
    cfg = DiTConfig(**cfgd)
    ctx = _ctx(cfgd, wdc.BF16, T=w["T"])
    ctx.init_weights(w["weight_seed"], 0.02)
    W = ctx.get_weights(dit.param_shapes(cfg))
    for name in ["L0.s0.qkv.w", "L0.s0.fc2.w", "patch.w"]:          # N(0, 0.02^2), biases 0
        a = W[name]
        assert abs(a.std() - 0.02) < 5e-4 and abs(a.mean()) < 5e-4, name
    assert not W["L0.s0.qkv.b"].any()
    zT, ct, _ = bench.inputs(w, 0)
    C, F, H, Wd, p = cfg.in_ch, cfg.frames, cfg.height, cfg.width, cfg.patch
    t = 1000.0                                                       # sigma_0 = 1
    v = torch.empty(zT.size, dtype=torch.float32, device="cuda")
    ctx.dit_forward(_to_dev(zT), t, _to_dev(ct), v)
    torch.cuda.synchronize()
    assert ctx.device_errors() == 0
    Lc = cfg.cond_tokens
    toks = np.sort(np.random.default_rng(35).choice(cfg.video_tokens, 64, replace=False))
    _, mods, fmod = dit.conditioning(W, cfg, t)
    x0 = dit.embed(W, cfg, zT, ct)
    xr = dit.block_rows(x0, W, cfg, 0, [mods[(0, 0)]], Lc + toks)
    hr = dit.modulate(dit.layer_norm(xr), fmod[0], fmod[1])
    want = dit.linear(hr, W["final.w"], W["final.b"])               # [64 tokens, C*p*p]
    got = dit.patchify(v.cpu().numpy().reshape(C, F, H, Wd), p)[toks]
    assert rel_l2(got, want) <= BF16_TOL


BLOCK13B = dict(layers=1, hidden=3072, heads=24, head_dim=128, mlp=12288, temb_dim=512, freq_dim=256, in_ch=16,
                frames=13, height=64, width=64, patch=2, cond_tokens=256, cond_dim=3072, dual_stream=1)


def test_bf16_dual_stream_block_13b_scale_sampled_rows():
    """One dual-stream block at the HunyuanVoyager-13B-like shape (L = 256 +
    13312 = 13568 tokens, 24 x 128 heads): separate weights and modulation for
    the condition and video rows, joint attention; 256 seeded rows (both
    streams) compared with fp64."""
    cfgd = BLOCK13B
    ctx = _ctx(cfgd, wdc.BF16)
    names = [f"L0.s{s}.{n}" for s in range(2) for n in ["qkv.w", "qkv.b", "o.w", "o.b", "fc1.w", "fc1.b", "fc2.w", "fc2.b"]]
    W = synth.dit_weights(cfgd, 6, std=0.02, bias_std=0.02, bf16=True, names=names)
    ctx.set_weights(W)
    L, D = 13568, 3072
    x = _bf(synth.normal(41, (L, D)))
    mod = synth.normal(42, (12, D), 0.3)
    for g in (2, 5, 8, 11):                       # gates of order one in both streams
        mod[g] = 1.0 + mod[g]
    xt = _to_dev(x, torch.bfloat16)
    ctx.dit_block_forward(0, xt, _to_dev(mod))
    torch.cuda.synchronize()
    g = np.random.default_rng(43)
    rows = np.sort(np.concatenate([g.choice(256, 32, replace=False), 256 + g.choice(L - 256, 224, replace=False)]))
    got = xt.float().cpu().numpy()[rows]
    mods = [mod[:6].astype(np.float64), mod[6:].astype(np.float64)]
    want = dit.block_rows(x.astype(np.float64), W, DiTConfig(**cfgd), 0, mods, rows)
    assert rel_l2(got - x[rows], want - x[rows]) <= BF16_TOL
    assert rel_l2(got, want) <= BF16_TOL
    cond = rows < 256
    assert rel_l2(got[cond] - x[rows][cond], want[cond] - x[rows][cond]) <= BF16_TOL


@pytest.mark.parametrize("H,L,d", [(48, 17776, 64), (24, 13568, 128)])
def test_bf16_attention_full_size_sampled_rows(H, L, d):
    """The attention shapes of the 5B-scale (48 x 64 heads, L = 17776) and
    13B-scale (24 x 128 heads, L = 13568) models; 96 sampled query rows per
    head compared with fp64."""
    ctx = _ctx(dict(PARITY_MODEL, layers=1), wdc.BF16)
    g = np.random.default_rng(44)
    q = _bf(g.standard_normal((H, L, d), dtype=np.float32))
    k = _bf(g.standard_normal((H, L, d), dtype=np.float32))
    v = _h(g.standard_normal((H, L, d), dtype=np.float32))
    o = torch.empty(L, H * d, dtype=torch.bfloat16, device="cuda")
    ctx.op_attention(_to_dev(q, torch.bfloat16), _to_dev(k, torch.bfloat16),
                     _to_dev(np.ascontiguousarray(v.transpose(0, 2, 1)), torch.float16), o)
    torch.cuda.synchronize()
    got = o.float().cpu().numpy()
    rows = np.sort(g.choice(L, 96, replace=False))
    rows[-1] = L - 1
    for h in range(0, H, 7):
        want = dit.attention(q[h, rows].astype(np.float64), k[h].astype(np.float64), v[h].astype(np.float64), 1)
        assert rel_l2(got[rows, h * d:(h + 1) * d], want) <= 1e-2, h


@pytest.mark.parametrize("M,N,K", [(17776, 9216, 3072), (1000, 768, 1024)])
def test_bf16_gemm_sampled_full_size_and_no_device_errors(M, N, K):
    """Full 5B-scale QKV shape (the CTA-pair kernel) checked on 64 sampled rows;
    no kernel reported a timeout or a tensor-memory pair mismatch."""
    ctx = _ctx(dict(PARITY_MODEL, layers=1), wdc.BF16)
    g = np.random.default_rng(55)
    A = _bf(g.standard_normal((M, K), dtype=np.float32))
    W = _bf(0.05 * g.standard_normal((N, K), dtype=np.float32))
    C = torch.empty(M, N, dtype=torch.bfloat16, device="cuda")
    ctx.op_gemm(_to_dev(A, torch.bfloat16), _to_dev(W, torch.bfloat16), C)
    torch.cuda.synchronize()
    rows = np.sort(g.choice(M, 64, replace=False))
    rows[-1] = M - 1
    want = A[rows].astype(np.float64) @ W.astype(np.float64).T
    assert rel_l2(C.float().cpu().numpy()[rows], want) <= 1e-2
    assert ctx.device_errors() == 0


def test_profiler_times_every_launch_and_dual_stream_gemms_are_grouped():
    """The event profiler times every launch (all on the caller's stream); a
    dual-stream block issues each of its four GEMMs as one grouped launch over
    the video and the condition rows, and one LayerNorm launch per row range."""
    cfgd = dict(PARITY_MODEL, layers=1, dual_stream=1)
    ctx = _ctx(cfgd, wdc.BF16)
    ctx.init_weights(3, 0.02)
    z = _to_dev(synth.latent(3, (16, 4, 16, 16)))
    ct = _to_dev(synth.cond_tokens(4, 16, 256))
    v = torch.empty(z.numel(), dtype=torch.float32, device="cuda")
    ctx.dit_forward(z, 500.0, ct, v)
    torch.cuda.synchronize()
    n0 = ctx.launches
    ctx.profile_enable(True)
    ctx.dit_forward(z, 500.0, ct, v)
    prof = ctx.profile_read()
    ctx.profile_enable(False)
    # condition and patch embeddings, the block's 4 grouped GEMMs, the final GEMM
    assert prof["gemm"][1] == 7
    assert prof["attention"][1] == 1
    assert prof["norm"][1] == 5                    # 2 row ranges x 2 LayerNorms + the final one
    assert ctx.launches - n0 == sum(n for _, n in prof.values())
    assert all(ms > 0 for ms, n in prof.values() if n)


@pytest.mark.parametrize("dual", [0, 1])
def test_bf16_block_hidden_3072_few_ragged_rows(dual):
    """The D = 3072 kernels on a short ragged sequence: 5 condition + 272
    video tokens (277 rows: not a multiple of the LayerNorm's 8 rows per
    block nor of the attention's 128-row tiles; 272 video rows leave a
    16-row tail in the second 256-row GEMM tile pair; with dual-stream
    weights each GEMM is one grouped launch whose second problem has 5
    rows), the whole block against the fp64 oracle on every row."""
    cfgd = dict(layers=1, hidden=3072, heads=48, head_dim=64, mlp=12288, temb_dim=512, freq_dim=256, in_ch=16,
                frames=1, height=32, width=34, patch=2, cond_tokens=5, cond_dim=3072, dual_stream=dual)
    cfg = DiTConfig(**cfgd)
    ctx = _ctx(cfgd, wdc.BF16)
    S = 2 if dual else 1
    names = [f"L0.s{s}.{n}" for s in range(S) for n in ["qkv.w", "qkv.b", "o.w", "o.b", "fc1.w", "fc1.b", "fc2.w",
                                                         "fc2.b"]]
    W = synth.dit_weights(cfgd, 9, std=0.02, bias_std=0.02, bf16=True, names=names)
    ctx.set_weights(W)
    L, D = 277, 3072
    x = _bf(synth.normal(41, (L, D)))
    mods = [synth.normal(42 + s, (6, D), 0.3) for s in range(S)]
    for m in mods:
        m[2] += 1.0
        m[5] += 1.0
    xt = _to_dev(x, torch.bfloat16)
    ctx.dit_block_forward(0, xt, _to_dev(np.concatenate(mods, axis=0)))
    torch.cuda.synchronize()
    want = dit.block(x.astype(np.float64), W, cfg, 0, [m.astype(np.float64) for m in mods])
    got = xt.float().cpu().numpy()
    assert rel_l2(got - x, want - x) <= BF16_TOL
    assert ctx.device_errors() == 0


def test_bf16_v_beyond_fp16_range_is_saturated_and_reported():
    """V^T of a bf16 model is stored in fp16: a V value beyond +-65504 is
    saturated and reported through bit 8 of the device error word; the same
    block with ordinary weights reports nothing, and NaN input propagates
    (it is not turned into a finite value)."""
    cfgd = dict(PARITY_MODEL, layers=1)
    names = [f"L0.s0.{n}" for n in ["qkv.w", "qkv.b", "o.w", "o.b", "fc1.w", "fc1.b", "fc2.w", "fc2.b"]]
    W = synth.dit_weights(cfgd, 13, std=0.02, bf16=True, names=names)
    L, D = 16 + 4 * 8 * 8, 256
    x = _bf(synth.normal(51, (L, D)))
    mod = _to_dev(synth.normal(52, (6, D), 0.3))
    ctx = _ctx(cfgd, wdc.BF16)
    ctx.set_weights(W)
    ctx.dit_block_forward(0, _to_dev(x, torch.bfloat16), mod)
    assert ctx.device_errors() == 0
    big = dict(W)
    big["L0.s0.qkv.w"] = W["L0.s0.qkv.w"].copy()
    big["L0.s0.qkv.w"][2 * D:] *= 2.0 ** 24       # |V| ~ 1e6 > 65504
    ctx.set_weights(big)
    xt = _to_dev(x, torch.bfloat16)
    ctx.dit_block_forward(0, xt, mod)
    assert ctx.device_errors() == 8
    assert torch.isfinite(xt.float()).all()
    ctx.set_weights(W)
    xn = x.copy()
    xn[3, 5] = np.nan
    xt = _to_dev(xn, torch.bfloat16)
    ctx.dit_block_forward(0, xt, mod)
    assert ctx.device_errors() == 0
    assert torch.isnan(xt.float()).any()
