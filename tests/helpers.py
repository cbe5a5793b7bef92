"""Test helpers: move state between the CPU oracle's representation and the
C ABI's host structs; comparison utilities."""
import numpy as np

from oracle import surrogate as sg
from oracle.rollout import CacheState
from paper_2608_01845_gb300 import wdc


def rel_l2(a, b):
    a = np.asarray(a, dtype=np.float64).reshape(-1)
    b = np.asarray(b, dtype=np.float64).reshape(-1)
    den = np.linalg.norm(b)
    return float(np.linalg.norm(a - b) / (den if den > 0 else 1.0))


def params_for_both(**kw):
    """The same constants as an oracle CacheParams and a wdc_cache_params."""
    from oracle.params import CacheParams
    op = CacheParams(**kw)
    cp = wdc.make_params(**{k: v for k, v in op.as_dict().items()})
    return op, cp


def state_to_host(state):
    """oracle CacheState -> wdc.StateHost (records oldest first)."""
    s = wdc.StateHost()
    s.n_bank = len(state.bank)
    s.age = state.age
    s.R = state.R
    s.eta = state.eta
    s.q_a_in = state.q_a_in
    s.q_a_out = state.q_a_out
    for j in range(4):
        s.cam_a[j] = float(state.cam_a[j])
        s.depth_a[j] = float(state.depth_a[j])
    for i, r in enumerate(state.bank):
        h = s.rec[i]
        for j in range(256):
            h.s_in[j] = float(r.s_in[j])
            h.s_out[j] = float(r.s_out[j])
            h.s_dphi[j] = float(r.s_dphi[j])
        h.q_in, h.q_out, h.r = float(r.q_in), float(r.q_out), float(r.r)
        for j in range(4):
            h.cam[j] = float(r.cam[j])
            h.depth[j] = float(r.depth[j])
    return s


def make_state(seed, z_k, K, n, q_k, T, corr=(0.9, -0.9, 0.8, 0.85, 0.7, 0.9, 0.8, 0.75),
               q_offsets=(0.1, 0.2, 0.4, 0.15, 0.05, 0.3, 0.12, 0.22), R=0.2, eta=1.3, age=2, p=None,
               cam=None, depth=None, drift=0.05):
    """A synthetic but realistic bank of K records for the current latent z_k:
    bank latents with smooth drift around z_k, summaries correlated with the
    current lift by the given signs, phases offset from q_k."""
    from oracle import summary as sm
    from paper_2608_01845_gb300 import synth
    g = np.random.default_rng(seed)
    lat = synth.drift_bank(seed + 1, n, K, delta=drift)
    lat = lat + np.float32(0.02) * z_k.reshape(1, -1).astype(np.float32)
    za = lat[-1]
    st = CacheState(bank=[], z_a=za, q_a_in=q_k + q_offsets[0] + 0.02, q_a_out=q_k + q_offsets[0] - 0.02,
                    cam_a=np.zeros(4) if cam is None else g.standard_normal(4) * 0.1,
                    depth_a=np.zeros(4) if depth is None else g.standard_normal(4) * 0.1,
                    R=R, eta=eta, age=age)
    # provisional bank for the history term
    bank = []
    for i in range(K):
        # the newest record is the anchor of the current streak: close in phase
        qi = q_k + (0.06 if i == K - 1 else q_offsets[i % len(q_offsets)])
        bank.append(sg.Record(s_in=np.zeros(256), s_out=np.zeros(256), s_dphi=np.zeros(256), z_out=lat[i],
                              q_in=qi, q_out=qi - 0.04, r=0.05 + 0.01 * i,
                              cam=g.standard_normal(4) * 0.1, depth=g.standard_normal(4) * 0.1))
    st.bank = bank
    h = st.history(T, p)
    s_phi = sm.summary_of_state(z_k, za, np.zeros(4) if cam is None else cam, np.zeros(4) if depth is None else depth,
                                q_k, h, p.eps_nu, p.sketch_seed)
    for i, rec in enumerate(bank):
        c = corr[i % len(corr)]
        s_in = c * s_phi + 0.4 * np.linalg.norm(s_phi) / 16.0 * g.standard_normal(256)
        s_out = s_in + 0.3 * np.linalg.norm(s_phi) / 16.0 * g.standard_normal(256)
        rec.s_in = s_in.astype(np.float32).astype(np.float64)
        rec.s_out = s_out.astype(np.float32).astype(np.float64)
        rec.s_dphi = rec.s_out - rec.s_in
    st.q_a_in = bank[-1].q_in
    st.q_a_out = bank[-1].q_out
    return st


class _CudaArray:
    def __init__(self, ptr, n):
        self.__cuda_array_interface__ = {"shape": (n,), "typestr": "<f4", "data": (int(ptr), False), "version": 2}


def device_view(ptr, n):
    """A float32 torch view of n elements at a raw device address (no copy)."""
    import torch
    return torch.as_tensor(_CudaArray(ptr, n), device="cuda")
