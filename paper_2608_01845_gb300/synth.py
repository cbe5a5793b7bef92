"""Seeded synthetic inputs for the cached rollout (latents, conditions, model
weights, bank contents).

This module holds no arithmetic of the method: it only draws numbers.  Tests
feed the same arrays to the CUDA path and to the CPU oracle, and ``bench.py``
uses it to build its workloads.  It imports neither of them.

Every generator is a pure function of its seed (numpy PCG64).
"""
import numpy as np

LATENT_STD = 1.0
WEIGHT_STD = 0.02


def rng(seed):
    return np.random.Generator(np.random.PCG64(int(seed) & 0xFFFFFFFFFFFFFFFF))


def normal(seed, shape, std=1.0):
    """N(0, std^2) float32 array."""
    return (rng(seed).standard_normal(size=shape, dtype=np.float32) * np.float32(std)).astype(np.float32)


def bf16_round(x):
    """Round float32 values to the nearest bfloat16 (ties to even); returns float32."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32).reshape(x.shape)


def dit_param_shapes(cfg):
    """Parameter names and shapes of the DiT denoiser ([out, in] for Linear weights).

    ``cfg`` is a mapping with hidden, temb_dim, mlp, in_ch, patch, cond_dim,
    layers, dual_stream and optionally freq_dim (default 256).
    """
    D, E, M = cfg["hidden"], cfg["temb_dim"], cfg["mlp"]
    P = cfg["in_ch"] * cfg["patch"] * cfg["patch"]
    Fd = cfg.get("freq_dim", 256)
    shapes = {
        "patch.w": (D, P), "patch.b": (D,),
        "cond.w": (D, cfg["cond_dim"]), "cond.b": (D,),
        "t1.w": (E, Fd), "t1.b": (E,),
        "t2.w": (E, E), "t2.b": (E,),
        "final.mod.w": (2 * D, E), "final.mod.b": (2 * D,),
        "final.w": (P, D), "final.b": (P,),
    }
    for l in range(cfg["layers"]):
        for s in range(2 if cfg.get("dual_stream", 0) else 1):
            pre = f"L{l}.s{s}."
            shapes.update({
                pre + "mod.w": (6 * D, E), pre + "mod.b": (6 * D,),
                pre + "qkv.w": (3 * D, D), pre + "qkv.b": (3 * D,),
                pre + "o.w": (D, D), pre + "o.b": (D,),
                pre + "fc1.w": (M, D), pre + "fc1.b": (M,),
                pre + "fc2.w": (D, M), pre + "fc2.b": (D,),
            })
    return shapes


def dit_weights(cfg, seed, std=WEIGHT_STD, bias_std=0.0, bf16=False, names=None):
    """All matrices N(0, std^2); biases N(0, bias_std^2) (0 by default).

    With ``bf16`` every value is rounded to a bfloat16-representable float32,
    so both sides of a comparison see the same bf16 model.  ``names`` restricts
    the output to a subset (each tensor has its own seed, derived from its
    name, so subsets are consistent with the full set).
    """
    out = {}
    for i, (name, shape) in enumerate(sorted(dit_param_shapes(cfg).items())):
        if names is not None and name not in names:
            continue
        sub = (int(seed) * 1000003 + i * 7919 + 17) & 0x7FFFFFFF
        if name.endswith(".b"):
            a = normal(sub, shape, bias_std) if bias_std > 0 else np.zeros(shape, dtype=np.float32)
        else:
            a = normal(sub, shape, std)
        out[name] = bf16_round(a) if bf16 else a
    return out


def latent(seed, shape):
    """z_T ~ N(0, 1), float32."""
    return normal(seed, shape, LATENT_STD)


def cond_tokens(seed, n_tokens, dim, bf16=False):
    a = normal(seed, (n_tokens, dim), 1.0)
    return bf16_round(a) if bf16 else a


def cond_descriptors(seed, T=None, std=0.1, static=True):
    """Camera / depth descriptors (4 + 4 values) per step; static by default."""
    if static or T is None:
        r = normal(seed, (8,), std)
        return {"cam": r[:4].astype(np.float64), "depth": r[4:].astype(np.float64)}
    r = normal(seed, (T, 8), std)
    return [{"cam": r[k, :4].astype(np.float64), "depth": r[k, 4:].astype(np.float64)} for k in range(T)]


def drift_bank(seed, n, K, delta=0.05):
    """Bank latents z_out_i = z0 + i * delta * sin(2 pi * 8 idx / n + phase_i),
    z0 ~ N(0,1) (smooth synthetic drift), float32 [K, n]."""
    g = rng(seed)
    z0 = g.standard_normal(size=n, dtype=np.float32)
    ph = g.uniform(0.0, 2.0 * np.pi, size=K)
    idx = np.arange(n, dtype=np.float64)
    out = np.empty((K, n), dtype=np.float32)
    for i in range(K):
        out[i] = z0 + np.float32(i * delta) * np.sin(2.0 * np.pi * 8.0 * idx / n + ph[i]).astype(np.float32)
    return out


def random_summaries(seed, K, dim=256):
    """Random record summaries s_in, s_out (float32 [K, dim])."""
    g = rng(seed)
    s_in = g.standard_normal(size=(K, dim), dtype=np.float32)
    s_out = s_in + np.float32(0.3) * g.standard_normal(size=(K, dim), dtype=np.float32)
    return s_in, s_out


def drift_bank_device(seed, n, K, delta=0.05):
    """drift_bank's recipe drawn on the current CUDA device with torch (for
    the bandwidth sweep's large latents): z0 ~ N(0,1) from a seeded torch
    generator, z_out_i = z0 + i * delta * sin(2 pi * 8 idx / n + phase_i);
    returns a list of K float32 tensors of n elements."""
    import torch
    g = torch.Generator(device="cuda").manual_seed(seed)
    z0 = torch.randn(n, device="cuda", generator=g)
    ph = torch.rand(K, device="cuda", generator=g, dtype=torch.float64) * (2.0 * np.pi)
    idx = torch.arange(n, device="cuda", dtype=torch.float64) * (2.0 * np.pi * 8.0 / n)
    out = []
    for i in range(K):
        out.append(z0 + (i * delta) * torch.sin(idx + ph[i]).float())
    del idx
    return out
