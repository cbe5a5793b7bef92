"""The allocation-free entry point wdc_observe_noalloc against the regular
skip pass (wdc_surrogate_step), through the C ABI, on two calls in a row.

wdc_observe_noalloc serves callers that cannot call cudaMalloc (code running
under another framework's memory manager or inside a pre-sized arena): it keeps
its scratch in a file-scope device array instead of context memory.  Given the
weights kappa the skip pass chose, it must reproduce that pass's candidate and
the statistics the next lift uses, within the skip pass's 1e-5 tolerance.
This file is collected last so that a failure here cannot hide another test."""
import copy

import numpy as np
import pytest
import torch

from helpers import make_state, params_for_both, rel_l2, state_to_host
from oracle import schedule as sch
from paper_2608_01845_gb300 import synth, wdc

pytestmark = pytest.mark.gpu
TOL = 1e-5


@pytest.mark.parametrize("n,K", [(128 * 1000 + 36, 3), (1 << 20, 4)])
def test_observe_noalloc_matches_skip_pass(n, K):
    op, cp = params_for_both(bank_capacity=K, tau_risk=1e9)
    T, k = 50, 20
    sig = sch.sigmas(T)
    z_k = synth.latent(61, (n,))
    st = make_state(68, z_k, K, n, float(sig[k]), T, p=op)
    ctx = wdc.Context(wdc.make_config(layers=0, width=n), T, params=cp)
    bank = [torch.from_numpy(r.z_out.copy()).cuda() for r in st.bank]
    ctx.state_set(state_to_host(st), bank, torch.from_numpy(z_k.copy()).cuda())
    zh_ref = torch.empty(n, dtype=torch.float32, device="cuda")
    info = ctx.surrogate_step(k, wdc.make_cond(), zh_ref)
    assert info.supported == 1 and info.finite == 1 and info.decision == 1
    ref = ctx.state_get()                         # on Surrogate the candidate's statistics became current
    kappa = list(info.kappa)[:K]
    for call in range(2):                         # two calls in a row share the same scratch
        zh = torch.full((n,), float("nan"), dtype=torch.float32, device="cuda")
        stats = torch.full((123,), float("nan"), dtype=torch.float64, device="cuda")
        wdc.observe_noalloc(bank, kappa, bank[-1], zh, stats, sketch_seed=cp.sketch_seed)
        torch.cuda.synchronize()
        s = stats.cpu().numpy()
        assert rel_l2(zh.cpu().numpy(), zh_ref.cpu().numpy()) <= TOL, call
        assert rel_l2(s[:120], np.array(ref.cur_sketch)) <= TOL, call
        assert abs(s[120] - ref.cur_sumsq) <= TOL * ref.cur_sumsq, call
        assert abs(s[121] - ref.cur_sumsq_anchor) <= TOL * ref.cur_sumsq_anchor, call
        assert s[122] == 0.0, call


def _raw_call(z_out, kappa, z_a, z_hat, stats, n):
    """The C entry point itself, without the binding's argument checks."""
    import ctypes
    ptrs = (ctypes.c_void_p * len(z_out))(*[t.data_ptr() for t in z_out])
    kap = (ctypes.c_double * len(kappa))(*kappa)
    return wdc.LIB.wdc_observe_noalloc(ptrs, len(z_out), kap, ctypes.c_void_p(z_a.data_ptr()),
                                       ctypes.c_void_p(z_hat.data_ptr()), ctypes.c_void_p(stats.data_ptr()), n,
                                       0x2545F491, ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))


def test_observe_noalloc_rejects_sizes_beyond_its_limits():
    z = torch.zeros(1024, dtype=torch.float32, device="cuda")
    zh = torch.empty_like(z)
    st = torch.zeros(123, dtype=torch.float64, device="cuda")
    assert _raw_call([z] * 9, [0.1] * 9, z, zh, st, 1024) == 1              # K > 8
    assert _raw_call([z[1:]], [1.0], z, zh, st, 1023) == 1                  # misaligned latent
    assert _raw_call([z], [1.0], z, zh, st, 1 << 31) == 1                   # n beyond 32-bit indices
    assert _raw_call([z], [1.0], z, zh, st, 0) == 1                         # empty
    with pytest.raises(ValueError):
        wdc.observe_noalloc([z] * 9, [0.1] * 9, z, zh, st)
    with pytest.raises(ValueError):
        wdc.observe_noalloc([z], [1.0], z, zh, st[:120])                    # short statistics buffer


def test_observe_noalloc_allocates_no_device_memory():
    """The property the entry point exists for: after a first call (which
    looks up the scratch array's address), further calls leave the device's
    free memory unchanged."""
    n = 1 << 20
    g = torch.Generator(device="cuda").manual_seed(3)
    bank = [torch.randn(n, device="cuda", generator=g) for _ in range(4)]
    zh = torch.empty(n, dtype=torch.float32, device="cuda")
    stats = torch.empty(123, dtype=torch.float64, device="cuda")
    kappa = [0.1, 0.2, 0.3, 0.4]
    wdc.observe_noalloc(bank, kappa, bank[-1], zh, stats)
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    first = zh.clone()
    for _ in range(5):
        wdc.observe_noalloc(bank, kappa, bank[-1], zh, stats)
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0
    assert torch.equal(zh, first)
