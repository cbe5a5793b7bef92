"""The exact denoiser F_theta: an adaLN-modulated DiT over video-latent tokens.

Test infrastructure only (see the package docstring).

The paper takes F_theta from the backbone ("a large transformer", Introduction
and Eq. 1; the DiT it cites) and does not print the architecture.  Reading
used by both this oracle and the CUDA path (all fp64 here):

* patchify: z [C,F,H,W] -> video tokens ordered (f, h', w'), patch features
  ordered (c, ph, pw); Linear C*p*p -> D (+bias); plus a 1-D sinusoidal
  position embedding over the video-token index, pe[n,2j] = sin(n w_j),
  pe[n,2j+1] = cos(n w_j), w_j = 10000^(-2j/D);
* condition tokens: Linear D_c -> D (+bias); the sequence is [cond; video];
* timestep: temb = W_t2 SiLU(W_t1 f(t) + b_t1) + b_t2 with f(t) the
  256-wide sinusoid [cos(t w_j), sin(t w_j)], w_j = exp(-ln(1e4) j/128);
* per block, [shift1, scale1, gate1, shift2, scale2, gate2] = W_mod SiLU(temb) + b_mod;
  x += gate1 * (W_o Attn(LN(x)(1+scale1) + shift1) + b_o)
  x += gate2 * (W_2 GELU_tanh(W_1 (LN(x)(1+scale2) + shift2) + b_1) + b_2)
  LN without affine, eps 1e-6; attention joint over all tokens, non-causal,
  scale 1/sqrt(d_head), no rotary embedding, no QK-norm;
* final: [shift_f, scale_f] = W_modf SiLU(temb) + b_modf;
  v = unpatchify(W_f (LN(x_video)(1+scale_f) + shift_f) + b_f);
* dual_stream: condition-token rows use a second set of block weights (QKV,
  out, MLP, modulation); attention stays joint.

Weights are a dict of fp64/fp32 arrays keyed as in ``param_shapes``; a Linear
weight has shape [out, in] and computes x @ W.T.
"""
import math

import numpy as np

LN_EPS = 1e-6


def param_shapes(cfg):
    """Name -> shape of every parameter of the model."""
    D, E, M, P = cfg.hidden, cfg.temb_dim, cfg.mlp, cfg.patch_dim
    shapes = {
        "patch.w": (D, P), "patch.b": (D,),
        "cond.w": (D, cfg.cond_dim), "cond.b": (D,),
        "t1.w": (E, cfg.freq_dim), "t1.b": (E,),
        "t2.w": (E, E), "t2.b": (E,),
        "final.mod.w": (2 * D, E), "final.mod.b": (2 * D,),
        "final.w": (P, D), "final.b": (P,),
    }
    for l in range(cfg.layers):
        for s in range(2 if cfg.dual_stream else 1):
            pre = f"L{l}.s{s}."
            shapes.update({
                pre + "mod.w": (6 * D, E), pre + "mod.b": (6 * D,),
                pre + "qkv.w": (3 * D, D), pre + "qkv.b": (3 * D,),
                pre + "o.w": (D, D), pre + "o.b": (D,),
                pre + "fc1.w": (M, D), pre + "fc1.b": (M,),
                pre + "fc2.w": (D, M), pre + "fc2.b": (D,),
            })
    return shapes


def silu(x):
    return x / (1.0 + np.exp(-x))


def gelu_tanh(x):
    """GELU, tanh form: 0.5 x (1 + tanh(sqrt(2/pi) (x + 0.044715 x^3)))."""
    return 0.5 * x * (1.0 + np.tanh(math.sqrt(2.0 / math.pi) * (x + 0.044715 * x ** 3)))


def layer_norm(x, eps=LN_EPS):
    """Row layer norm without affine parameters (biased variance)."""
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps)


def modulate(x, shift, scale):
    return x * (1.0 + scale) + shift


def timestep_features(t, dim=256):
    """f(t) = [cos(t w_j), sin(t w_j)], w_j = exp(-ln(10000) j / (dim/2))."""
    half = dim // 2
    w = np.exp(-math.log(10000.0) * np.arange(half, dtype=np.float64) / half)
    a = float(t) * w
    return np.concatenate([np.cos(a), np.sin(a)])


def position_embedding(n, D):
    """pe[i, 2j] = sin(i w_j), pe[i, 2j+1] = cos(i w_j), w_j = 10000^(-2j/D)."""
    j = np.arange(D // 2, dtype=np.float64)
    w = np.power(10000.0, -2.0 * j / D)
    a = np.arange(n, dtype=np.float64)[:, None] * w[None, :]
    pe = np.zeros((n, D), dtype=np.float64)
    pe[:, 0::2] = np.sin(a)
    pe[:, 1::2] = np.cos(a)
    return pe


def patchify(z, p):
    """[C,F,H,W] -> [F*(H/p)*(W/p), C*p*p] with tokens (f,h',w') and features (c,ph,pw)."""
    C, F, H, W = z.shape
    t = z.reshape(C, F, H // p, p, W // p, p)            # c f h' ph w' pw
    t = t.transpose(1, 2, 4, 0, 3, 5)                     # f h' w' c ph pw
    return t.reshape(F * (H // p) * (W // p), C * p * p)


def unpatchify(tok, C, F, H, W, p):
    """Inverse of ``patchify``."""
    t = tok.reshape(F, H // p, W // p, C, p, p)           # f h' w' c ph pw
    t = t.transpose(3, 0, 1, 4, 2, 5)                     # c f h' ph w' pw
    return t.reshape(C, F, H, W)


def linear(x, W, b):
    return x @ np.asarray(W, dtype=np.float64).T + np.asarray(b, dtype=np.float64)


def attention(q, k, v, heads):
    """Joint non-causal softmax attention: softmax(Q K^T / sqrt(d)) V per head.

    q: [Lq, heads*d]; k, v: [L, heads*d].  Returns [Lq, heads*d].
    """
    Lq, Dm = q.shape
    d = Dm // heads
    out = np.empty((Lq, Dm), dtype=np.float64)
    scale = 1.0 / math.sqrt(d)
    for h in range(heads):
        sl = slice(h * d, (h + 1) * d)
        s = (q[:, sl] @ k[:, sl].T) * scale
        s = s - s.max(axis=1, keepdims=True)
        e = np.exp(s)
        out[:, sl] = (e / e.sum(axis=1, keepdims=True)) @ v[:, sl]
    return out


def conditioning(Wt, cfg, t):
    """temb and the modulation vectors of every block (and the final layer)."""
    f = timestep_features(t, cfg.freq_dim)
    temb = linear(silu(linear(f, Wt["t1.w"], Wt["t1.b"])), Wt["t2.w"], Wt["t2.b"])
    st = silu(temb)
    mods = {}
    for l in range(cfg.layers):
        for s in range(2 if cfg.dual_stream else 1):
            pre = f"L{l}.s{s}."
            if pre + "mod.w" in Wt:
                mods[(l, s)] = linear(st, Wt[pre + "mod.w"], Wt[pre + "mod.b"]).reshape(6, cfg.hidden)
    final = linear(st, Wt["final.mod.w"], Wt["final.mod.b"]).reshape(2, cfg.hidden)
    return temb, mods, final


def _stream_rows(cfg, L):
    """Row ranges of the (video, condition) streams in the [cond; video] sequence."""
    return [(cfg.cond_tokens, L), (0, cfg.cond_tokens)] if cfg.dual_stream else [(0, L)]


def block(x, Wt, cfg, layer, mod):
    """One DiT block on the full sequence x [L, D] (fp64); ``mod[s]`` is [6, D] per stream."""
    L, D = x.shape
    rows = _stream_rows(cfg, L)
    h = np.empty_like(x)
    qkv = np.empty((L, 3 * D))
    for s, (r0, r1) in enumerate(rows):
        m = mod[s]
        h[r0:r1] = modulate(layer_norm(x[r0:r1]), m[0], m[1])
        pre = f"L{layer}.s{s}."
        qkv[r0:r1] = linear(h[r0:r1], Wt[pre + "qkv.w"], Wt[pre + "qkv.b"])
    o = attention(qkv[:, :D], qkv[:, D:2 * D], qkv[:, 2 * D:], cfg.heads)
    x = x.copy()
    for s, (r0, r1) in enumerate(rows):
        m = mod[s]
        pre = f"L{layer}.s{s}."
        x[r0:r1] += m[2] * linear(o[r0:r1], Wt[pre + "o.w"], Wt[pre + "o.b"])
        h2 = modulate(layer_norm(x[r0:r1]), m[3], m[4])
        x[r0:r1] += m[5] * linear(gelu_tanh(linear(h2, Wt[pre + "fc1.w"], Wt[pre + "fc1.b"])),
                                  Wt[pre + "fc2.w"], Wt[pre + "fc2.b"])
    return x


def block_rows(x, Wt, cfg, layer, mod, rows_idx):
    """The same block, evaluated only for the query rows ``rows_idx``.

    Keys and values are computed for every token (attention is joint), each
    token with its own stream's weights and modulation; queries, attention,
    out-projection and MLP only for the selected rows.  Returns
    [len(rows_idx), D].
    """
    L, D = x.shape
    rows = _stream_rows(cfg, L)
    rows_idx = np.asarray(rows_idx)
    stream_of = np.empty(L, dtype=np.int64)
    for s, (r0, r1) in enumerate(rows):
        stream_of[r0:r1] = s
    h = np.empty_like(x, dtype=np.float64)
    kv = np.empty((L, 2 * D))
    for s, (r0, r1) in enumerate(rows):
        m = mod[s]
        pre = f"L{layer}.s{s}."
        Wqkv = np.asarray(Wt[pre + "qkv.w"], dtype=np.float64)
        bqkv = np.asarray(Wt[pre + "qkv.b"], dtype=np.float64)
        h[r0:r1] = modulate(layer_norm(x[r0:r1]), m[0], m[1])
        kv[r0:r1] = h[r0:r1] @ Wqkv[D:].T + bqkv[D:]
    out = np.empty((len(rows_idx), D))
    for s, (r0, r1) in enumerate(rows):
        sel = np.nonzero(stream_of[rows_idx] == s)[0]
        if sel.size == 0:
            continue
        m = mod[s]
        pre = f"L{layer}.s{s}."
        Wqkv = np.asarray(Wt[pre + "qkv.w"], dtype=np.float64)
        bqkv = np.asarray(Wt[pre + "qkv.b"], dtype=np.float64)
        q = h[rows_idx[sel]] @ Wqkv[:D].T + bqkv[:D]
        o = attention(q, kv[:, :D], kv[:, D:], cfg.heads)
        xr = x[rows_idx[sel]].astype(np.float64)
        xr += m[2] * linear(o, Wt[pre + "o.w"], Wt[pre + "o.b"])
        h2 = modulate(layer_norm(xr), m[3], m[4])
        xr += m[5] * linear(gelu_tanh(linear(h2, Wt[pre + "fc1.w"], Wt[pre + "fc1.b"])), Wt[pre + "fc2.w"], Wt[pre + "fc2.b"])
        out[sel] = xr
    return out


def embed(Wt, cfg, z, cond_tokens):
    """Input sequence x0 = [Linear(cond); Linear(patchify(z)) + pe] (fp64)."""
    tok = patchify(np.asarray(z, dtype=np.float64).reshape(cfg.in_ch, cfg.frames, cfg.height, cfg.width), cfg.patch)
    xv = linear(tok, Wt["patch.w"], Wt["patch.b"]) + position_embedding(tok.shape[0], cfg.hidden)
    xc = linear(np.asarray(cond_tokens, dtype=np.float64).reshape(cfg.cond_tokens, cfg.cond_dim),
                Wt["cond.w"], Wt["cond.b"])
    return np.concatenate([xc, xv], axis=0)


def final_layer(Wt, cfg, x, final_mod):
    """v = unpatchify(W_f (LN(x_video)(1+scale_f) + shift_f) + b_f)."""
    xv = x[cfg.cond_tokens:]
    h = modulate(layer_norm(xv), final_mod[0], final_mod[1])
    out = linear(h, Wt["final.w"], Wt["final.b"])
    return unpatchify(out, cfg.in_ch, cfg.frames, cfg.height, cfg.width, cfg.patch)


def forward(Wt, cfg, z, t, cond_tokens):
    """F_theta(z, t, c) -> v with the latent's shape [C,F,H,W] (fp64)."""
    _, mods, fmod = conditioning(Wt, cfg, t)
    x = embed(Wt, cfg, z, cond_tokens)
    for l in range(cfg.layers):
        x = block(x, Wt, cfg, l, [mods[(l, s)] for s in range(2 if cfg.dual_stream else 1)])
    return final_layer(Wt, cfg, x, fmod)
