"""Python binding of libwdc.so (the C ABI in include/wdc.h).

Argument marshalling only: every step of the cached rollout runs in the CUDA
kernels behind the C ABI.  PyTorch is used for device memory and streams.  If
the shared library is missing or cannot be loaded this module raises at
import time -- there is no fallback path.
"""
import ctypes
import os

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libwdc.so")

MAX_BANK = 8
MAX_BATCH = 16
SUMMARY_DIM = 256
SKETCH = 120
F32, BF16 = 0, 1

STATUS = {0: "ok", 1: "invalid argument", 2: "CUDA error", 3: "unsupported", 4: "device wait timed out",
          5: "non-finite value", 6: "call out of order", 7: "out of device memory"}

# tensor ids (enum wdc_tensor_id)
T_PATCH_W, T_PATCH_B, T_COND_W, T_COND_B, T_T1_W, T_T1_B, T_T2_W, T_T2_B = range(8)
T_FMOD_W, T_FMOD_B, T_FINAL_W, T_FINAL_B = 8, 9, 10, 11
T_MOD_W, T_MOD_B, T_QKV_W, T_QKV_B, T_O_W, T_O_B, T_FC1_W, T_FC1_B, T_FC2_W, T_FC2_B = range(12, 22)

# parameter names (as in the seeded generators) -> tensor ids
GLOBAL_TENSORS = {"patch.w": T_PATCH_W, "patch.b": T_PATCH_B, "cond.w": T_COND_W, "cond.b": T_COND_B,
                  "t1.w": T_T1_W, "t1.b": T_T1_B, "t2.w": T_T2_W, "t2.b": T_T2_B,
                  "final.mod.w": T_FMOD_W, "final.mod.b": T_FMOD_B, "final.w": T_FINAL_W, "final.b": T_FINAL_B}
LAYER_TENSORS = {"mod.w": T_MOD_W, "mod.b": T_MOD_B, "qkv.w": T_QKV_W, "qkv.b": T_QKV_B, "o.w": T_O_W,
                 "o.b": T_O_B, "fc1.w": T_FC1_W, "fc1.b": T_FC1_B, "fc2.w": T_FC2_W, "fc2.b": T_FC2_B}


class WdcError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__(f"{STATUS.get(status, status)}: {msg}")
        self.status = status


class DitConfig(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int) for n in
                ["layers", "hidden", "heads", "head_dim", "mlp", "temb_dim", "freq_dim", "in_ch", "frames",
                 "height", "width", "patch", "cond_tokens", "cond_dim", "dual_stream", "dtype", "max_batch"]]


class Schedule(ctypes.Structure):
    _fields_ = [("T", ctypes.c_int), ("shift", ctypes.c_double)]


class CacheParams(ctypes.Structure):
    _fields_ = ([("bank_capacity", ctypes.c_int), ("min_support", ctypes.c_int)]
                + [(n, ctypes.c_double) for n in ["sim_min", "q_gap_max", "gamma_q", "tau_in", "tau_obs",
                                                   "alpha_min", "alpha_max", "eps", "eps_nu"]]
                + [("sketch_seed", ctypes.c_uint32)]
                + [(n, ctypes.c_double) for n in ["w_z", "w_age", "w_phase", "w_cam", "w_depth", "eta_init",
                                                   "eta_min", "eta_max", "beta_d", "a_cam", "a_depth", "a_phase",
                                                   "lambda_", "tau_risk"]]
                + [(n, ctypes.c_int) for n in ["max_age", "n_init_exact", "n_final_exact", "flags", "period"]]
                + [("ridge", ctypes.c_double)])


# Ablation variants (wdc_cache_params.flags; definitions in include/wdc.h).
ABL_PERIODIC = 0x01
ABL_SECANT = 0x02
ABL_INSTANT_RISK = 0x04
ABL_NO_IMPACT = 0x08
ABL_NO_CALIB = 0x10
ABL_NO_SUPPORT = 0x20
ABL_LINEAR_OBS = 0x40
ABL_NO_COND = 0x80
OBS_RESIDUAL = 0x100      # residual reading of Eq. 5 (not an ablation)


class Cond(ctypes.Structure):
    _fields_ = [("tokens", ctypes.c_void_p), ("cam", ctypes.c_double * 4), ("depth", ctypes.c_double * 4)]


class StepInfo(ctypes.Structure):
    _fields_ = ([(n, ctypes.c_int) for n in ["k", "decision", "finite", "supported", "n_compat", "n_bank", "age"]]
                + [(n, ctypes.c_double) for n in ["q", "alpha", "p", "d_hat", "w", "delta", "R_cand", "R", "eta",
                                                   "d_cf", "d_z", "r"]]
                + [("kappa", ctypes.c_double * MAX_BANK), ("pi", ctypes.c_double * MAX_BANK)])

    def as_dict(self):
        d = {n: getattr(self, n) for n, _ in self._fields_ if n not in ("kappa", "pi")}
        d["kappa"] = list(self.kappa)
        d["pi"] = list(self.pi)
        return d


class RecordHost(ctypes.Structure):
    _fields_ = [("s_in", ctypes.c_double * SUMMARY_DIM), ("s_out", ctypes.c_double * SUMMARY_DIM),
                ("s_dphi", ctypes.c_double * SUMMARY_DIM), ("q_in", ctypes.c_double), ("q_out", ctypes.c_double),
                ("r", ctypes.c_double), ("cam", ctypes.c_double * 4), ("depth", ctypes.c_double * 4)]


class StateHost(ctypes.Structure):
    _fields_ = [("n_bank", ctypes.c_int), ("age", ctypes.c_int), ("R", ctypes.c_double), ("eta", ctypes.c_double),
                ("q_a_in", ctypes.c_double), ("q_a_out", ctypes.c_double), ("cam_a", ctypes.c_double * 4),
                ("depth_a", ctypes.c_double * 4), ("rec", RecordHost * MAX_BANK),
                ("cur_sketch", ctypes.c_double * SKETCH), ("cur_sumsq", ctypes.c_double),
                ("cur_sumsq_anchor", ctypes.c_double), ("anchor_sketch", ctypes.c_double * SKETCH),
                ("anchor_sumsq", ctypes.c_double), ("s_phi", ctypes.c_double * SUMMARY_DIM),
                ("cand_supported", ctypes.c_int), ("cand_finite", ctypes.c_int), ("cand_p", ctypes.c_double)]


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"libwdc.so not built at {LIB_PATH}; run `python -m paper_2608_01845_gb300.build`")
    lib = ctypes.CDLL(LIB_PATH)
    P, I, F, D, S = ctypes.c_void_p, ctypes.c_int, ctypes.c_float, ctypes.c_double, ctypes.c_size_t
    sig = {
        "wdc_status_string": (ctypes.c_char_p, [I]),
        "wdc_default_cache_params": (I, [ctypes.POINTER(CacheParams)]),
        "wdc_create": (I, [ctypes.POINTER(DitConfig), ctypes.POINTER(Schedule), ctypes.POINTER(CacheParams), I,
                           ctypes.POINTER(P)]),
        "wdc_destroy": (None, [P]),
        "wdc_set_cache_params": (I, [P, ctypes.POINTER(CacheParams)]),
        "wdc_profile_enable": (I, [P, I]),
        "wdc_device_errors": (I, [P, ctypes.POINTER(ctypes.c_uint)]),
        "wdc_selftest_wait_timeout": (I, [P, ctypes.c_ulonglong, P]),
        "wdc_profile_read": (I, [P, ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_ulonglong)]),
        "wdc_last_error": (ctypes.c_char_p, [P]),
        "wdc_latent_numel": (S, [P]),
        "wdc_launch_count": (ctypes.c_ulonglong, [P]),
        "wdc_set_tensor": (I, [P, I, I, I, P, S]),
        "wdc_get_tensor": (I, [P, I, I, I, P, S]),
        "wdc_init_weights": (I, [P, ctypes.c_ulonglong, F]),
        "wdc_dit_forward": (I, [P, P, F, P, P, P]),
        "wdc_dit_forward_batch": (I, [P, I, ctypes.POINTER(P), F, ctypes.POINTER(P), I, F, ctypes.POINTER(P), P]),
        "wdc_dit_block_forward": (I, [P, I, P, P, P]),
        "wdc_dit_modulation": (I, [P, F, P, P]),
        "wdc_scheduler_step": (I, [P, I, P, P, P, P]),
        "wdc_schedule_sigmas": (I, [P, ctypes.POINTER(D)]),
        "wdc_latent_pair_stats": (I, [P, P, P, P, ctypes.POINTER(D), P]),
        "wdc_correlations": (I, [ctypes.POINTER(D), ctypes.POINTER(D), I, ctypes.POINTER(D), ctypes.POINTER(D)]),
        "wdc_state_reset": (I, [P, P, P]),
        "wdc_state_get": (I, [P, ctypes.POINTER(StateHost), P]),
        "wdc_state_set": (I, [P, ctypes.POINTER(StateHost), P, P, P]),
        "wdc_surrogate_step": (I, [P, I, ctypes.POINTER(Cond), P, ctypes.POINTER(StepInfo), P]),
        "wdc_risk_update": (I, [P, I, ctypes.POINTER(Cond), P, P, P, ctypes.POINTER(P), ctypes.POINTER(StepInfo), P]),
        "wdc_rollout": (I, [P, P, ctypes.POINTER(Cond), I, P, ctypes.POINTER(I), ctypes.POINTER(StepInfo), P]),
        "wdc_rollout_graph": (I, [P, P, ctypes.POINTER(Cond), P, ctypes.POINTER(I), ctypes.POINTER(StepInfo), P]),
        "wdc_rollout_batch": (I, [ctypes.POINTER(P), I, ctypes.POINTER(P), ctypes.POINTER(Cond), I, I, F,
                                  ctypes.POINTER(P), ctypes.POINTER(I), ctypes.POINTER(StepInfo), P]),
        "wdc_native_rollout": (I, [P, P, ctypes.POINTER(Cond), I, P, P]),
        "wdc_op_gemm": (I, [P, P, P, P, P, I, I, I, I, P, P, P]),
        "wdc_op_attention": (I, [P, P, P, P, P, I, I, I, P]),
        "wdc_observe_noalloc": (I, [ctypes.POINTER(P), I, ctypes.POINTER(D), P, P, P, S, ctypes.c_uint32, P]),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    return lib


LIB = _load()


def default_params():
    p = CacheParams()
    LIB.wdc_default_cache_params(ctypes.byref(p))
    return p


def make_params(**overrides):
    """wdc_cache_params from the library defaults with overrides (``lam`` maps to lambda_)."""
    p = default_params()
    for k, v in overrides.items():
        k = "lambda_" if k == "lam" else k
        setattr(p, k, v)
    return p


def make_config(layers=0, hidden=0, heads=0, head_dim=0, mlp=0, temb_dim=0, freq_dim=256, in_ch=1, frames=1,
                height=1, width=1, patch=1, cond_tokens=0, cond_dim=0, dual_stream=0, dtype=F32, max_batch=1):
    return DitConfig(layers, hidden, heads, head_dim, mlp, temb_dim, freq_dim, in_ch, frames, height, width, patch,
                     cond_tokens, cond_dim, dual_stream, dtype, max_batch)


def _ptr(t):
    if t is None:
        return None
    return ctypes.c_void_p(t.data_ptr() if hasattr(t, "data_ptr") else int(t))


def _stream(s):
    if s is None:
        import torch
        return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    return ctypes.c_void_p(s.cuda_stream if hasattr(s, "cuda_stream") else int(s))


def make_cond(tokens=None, cam=None, depth=None):
    """wdc_cond for one step.  The returned object keeps ``tokens`` alive."""
    c = Cond()
    c.tokens = None if tokens is None else (tokens.data_ptr() if hasattr(tokens, "data_ptr") else
                                            tokens.ctypes.data)
    c._keep = tokens
    for j in range(4):
        c.cam[j] = 0.0 if cam is None else float(cam[j])
        c.depth[j] = 0.0 if depth is None else float(depth[j])
    return c


class Context:
    """Owns one wdc_ctx.  Method names follow the C entry points."""

    def __init__(self, cfg, T, params=None, shift=1.0, device=0):
        self._h = ctypes.c_void_p()
        self.cfg = cfg
        self.params = params if params is not None else default_params()
        self.sched = Schedule(T, shift)
        st = LIB.wdc_create(ctypes.byref(cfg), ctypes.byref(self.sched), ctypes.byref(self.params), device,
                            ctypes.byref(self._h))
        if st != 0:
            raise WdcError(st, "wdc_create failed")

    def close(self):
        if self._h:
            LIB.wdc_destroy(self._h)
            self._h = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _check(self, st, what):
        if st != 0:
            raise WdcError(st, f"{what}: {LIB.wdc_last_error(self._h).decode()}")

    @property
    def numel(self):
        return LIB.wdc_latent_numel(self._h)

    @property
    def launches(self):
        return LIB.wdc_launch_count(self._h)

    def set_cache_params(self, params):
        self._check(LIB.wdc_set_cache_params(self._h, ctypes.byref(params)), "set_cache_params")
        self.params = params

    def device_errors(self):
        """Error bits set by kernels since the last call (1 timeout, 4 TMEM pair
        mismatch, 8 a bf16 model's V saturated to fp16's range)."""
        b = ctypes.c_uint()
        self._check(LIB.wdc_device_errors(self._h, ctypes.byref(b)), "device_errors")
        return b.value

    def selftest_wait_timeout(self, limit_ns, stream=None):
        """wdc_selftest_wait_timeout: a bounded device wait that must time out."""
        self._check(LIB.wdc_selftest_wait_timeout(self._h, int(limit_ns), _stream(stream)), "selftest_wait_timeout")

    def profile_enable(self, on=True):
        self._check(LIB.wdc_profile_enable(self._h, int(on)), "profile_enable")

    def profile_read(self):
        """{class name: (ms, launches)} since the last enable/read."""
        ms = (ctypes.c_double * 6)()
        n = (ctypes.c_ulonglong * 6)()
        self._check(LIB.wdc_profile_read(self._h, ms, n), "profile_read")
        names = ["gemm", "attention", "norm", "skip", "anchor", "other"]
        return {names[i]: (ms[i], n[i]) for i in range(6)}

    def set_tensor(self, tensor_id, array, layer=0, stream=0):
        import numpy as np
        a = np.ascontiguousarray(array, dtype=np.float32)
        self._check(LIB.wdc_set_tensor(self._h, tensor_id, layer, stream, a.ctypes.data, a.size), "set_tensor")

    def get_tensor(self, tensor_id, shape, layer=0, stream=0):
        """wdc_get_tensor: one parameter tensor back as a float32 array."""
        import numpy as np
        a = np.empty(shape, dtype=np.float32)
        self._check(LIB.wdc_get_tensor(self._h, tensor_id, layer, stream, a.ctypes.data, a.size), "get_tensor")
        return a

    def get_weights(self, shapes):
        """{name: shape} (names as in set_weights) -> {name: float32 array} read from the device."""
        out = {}
        for name, shape in shapes.items():
            if name in GLOBAL_TENSORS:
                out[name] = self.get_tensor(GLOBAL_TENSORS[name], shape)
            else:
                lay, strm, rest = name.split(".", 2)
                out[name] = self.get_tensor(LAYER_TENSORS[rest], shape, layer=int(lay[1:]), stream=int(strm[1:]))
        return out

    def set_weights(self, weights):
        """Uploads a {name: array} dict (names as produced by the seeded generators)."""
        for name, arr in weights.items():
            if name in GLOBAL_TENSORS:
                self.set_tensor(GLOBAL_TENSORS[name], arr)
            else:
                lay, strm, rest = name.split(".", 2)
                self.set_tensor(LAYER_TENSORS[rest], arr, layer=int(lay[1:]), stream=int(strm[1:]))

    def init_weights(self, seed, std=0.02):
        self._check(LIB.wdc_init_weights(self._h, seed, std), "init_weights")

    def dit_forward(self, z_t, t, cond_tokens, v, stream=None):
        self._check(LIB.wdc_dit_forward(self._h, _ptr(z_t), float(t), _ptr(cond_tokens), _ptr(v), _stream(stream)),
                    "dit_forward")

    def dit_forward_batch(self, z_list, t, cond_list, v_list, cfg=False, guidance=1.0, stream=None):
        """wdc_dit_forward_batch: one batched (optionally guided) forward of
        len(z_list) latents at timestep t; cond_list may be None when the
        model has no condition tokens."""
        B = len(z_list)
        zs = (ctypes.c_void_p * B)(*[t_.data_ptr() for t_ in z_list])
        vs = (ctypes.c_void_p * B)(*[t_.data_ptr() for t_ in v_list])
        cs = None if cond_list is None else (ctypes.c_void_p * B)(*[t_.data_ptr() for t_ in cond_list])
        self._check(LIB.wdc_dit_forward_batch(self._h, B, zs, float(t), cs, int(bool(cfg)), float(guidance), vs,
                                              _stream(stream)), "dit_forward_batch")

    def dit_block_forward(self, layer, x, mod6, stream=None):
        self._check(LIB.wdc_dit_block_forward(self._h, layer, _ptr(x), _ptr(mod6), _stream(stream)),
                    "dit_block_forward")

    def dit_modulation(self, t, mod_out, stream=None):
        self._check(LIB.wdc_dit_modulation(self._h, float(t), _ptr(mod_out), _stream(stream)), "dit_modulation")

    def sigmas(self):
        """wdc_schedule_sigmas: the context's noise levels sigma_0..sigma_T."""
        T = self.sched.T
        out = (ctypes.c_double * (T + 1))()
        self._check(LIB.wdc_schedule_sigmas(self._h, out), "schedule_sigmas")
        return list(out)

    def latent_pair_stats(self, a, b, c=None, stream=None):
        """wdc_latent_pair_stats: [sum (a-c)^2, sum (b-c)^2, sum (a-c)(b-c),
        sum (a-b)^2, sum b^2] over three device latents (c may be None)."""
        out = (ctypes.c_double * 5)()
        self._check(LIB.wdc_latent_pair_stats(self._h, _ptr(a), _ptr(b), _ptr(c), out, _stream(stream)),
                    "latent_pair_stats")
        return list(out)

    def scheduler_step(self, k, z_t, v, z_next, stream=None):
        self._check(LIB.wdc_scheduler_step(self._h, k, _ptr(z_t), _ptr(v), _ptr(z_next), _stream(stream)),
                    "scheduler_step")

    def state_reset(self, z_T, stream=None):
        self._check(LIB.wdc_state_reset(self._h, _ptr(z_T), _stream(stream)), "state_reset")

    def state_get(self, stream=None):
        s = StateHost()
        self._check(LIB.wdc_state_get(self._h, ctypes.byref(s), _stream(stream)), "state_get")
        return s

    def state_set(self, state, z_out_list, z_cur, stream=None):
        arr = (ctypes.c_void_p * max(1, len(z_out_list)))(*[t.data_ptr() for t in z_out_list])
        self._check(LIB.wdc_state_set(self._h, ctypes.byref(state), arr, _ptr(z_cur), _stream(stream)), "state_set")

    def surrogate_step(self, k, cond, z_hat, stream=None):
        info = StepInfo()
        self._check(LIB.wdc_surrogate_step(self._h, k, ctypes.byref(cond), _ptr(z_hat), ctypes.byref(info),
                                           _stream(stream)), "surrogate_step")
        return info

    def risk_update(self, k, cond, z_t, v, z_cf, info=None, stream=None):
        """Returns the device address of z_exact (inside the context's bank)."""
        out = ctypes.c_void_p()
        self._check(LIB.wdc_risk_update(self._h, k, ctypes.byref(cond), _ptr(z_t), _ptr(v), _ptr(z_cf),
                                        ctypes.byref(out), ctypes.byref(info) if info is not None else None,
                                        _stream(stream)), "risk_update")
        return out.value

    def rollout(self, z_T, conds, z_out, trace=True, stream=None):
        """Cached rollout; z_T / z_out may be torch tensors on the device or pinned host tensors."""
        T = self.sched.T
        conds = conds if isinstance(conds, (list, tuple)) else [conds]
        carr = (Cond * len(conds))(*conds)
        dec = (ctypes.c_int * T)()
        tr = (StepInfo * T)() if trace else None
        self._check(LIB.wdc_rollout(self._h, _ptr(z_T), carr, len(conds), _ptr(z_out), dec, tr, _stream(stream)),
                    "rollout")
        return list(dec), ([tr[k].as_dict() for k in range(T)] if trace else None)

    def rollout_graph(self, z_T, cond, z_out, trace=True, stream=None):
        """wdc_rollout_graph: the cached rollout with device-side control flow (one condition)."""
        T = self.sched.T
        dec = (ctypes.c_int * T)()
        tr = (StepInfo * T)() if trace else None
        self._check(LIB.wdc_rollout_graph(self._h, _ptr(z_T), ctypes.byref(cond), _ptr(z_out), dec, tr,
                                          _stream(stream)), "rollout_graph")
        return list(dec), ([tr[k].as_dict() for k in range(T)] if trace else None)

    def native_rollout(self, z_T, conds, z_out, stream=None):
        conds = conds if isinstance(conds, (list, tuple)) else [conds]
        carr = (Cond * len(conds))(*conds)
        self._check(LIB.wdc_native_rollout(self._h, _ptr(z_T), carr, len(conds), _ptr(z_out), _stream(stream)),
                    "native_rollout")

    def op_gemm(self, A, W, C, bias=None, gelu=False, res=None, gate=None, stream=None):
        M, K = A.shape
        N = W.shape[0]
        self._check(LIB.wdc_op_gemm(self._h, _ptr(A), _ptr(W), _ptr(bias), _ptr(C), M, N, K, int(gelu), _ptr(res),
                                    _ptr(gate), _stream(stream)), "op_gemm")

    def op_attention(self, q, k, vt, o, stream=None):
        H, L, d = q.shape
        self._check(LIB.wdc_op_attention(self._h, _ptr(q), _ptr(k), _ptr(vt), _ptr(o), H, L, d, _stream(stream)),
                    "op_attention")


def correlations(x, y):
    """wdc_correlations: (Pearson, Spearman) of two equal-length samples."""
    n = len(x)
    if len(y) != n:
        raise ValueError("correlations: samples of different lengths")
    xs = (ctypes.c_double * n)(*[float(v) for v in x])
    ys = (ctypes.c_double * n)(*[float(v) for v in y])
    pe, sp = ctypes.c_double(), ctypes.c_double()
    st = LIB.wdc_correlations(xs, ys, n, ctypes.byref(pe), ctypes.byref(sp))
    if st != 0:
        raise WdcError(st, "wdc_correlations: needs n >= 2")
    return pe.value, sp.value


def rollout_batch(ctxs, z_T_list, conds, z_out_list, cfg=False, guidance=1.0, trace=True, stream=None):
    """wdc_rollout_batch: len(ctxs) cached rollouts in lockstep; ctxs[0] owns
    the denoiser, ctxs[b] holds sample b's cache state.  conds: one wdc_cond
    per sample (used for every step) or a list of T per sample.  Returns
    (decisions per sample, traces per sample or None)."""
    B = len(ctxs)
    T = ctxs[0].sched.T
    per = [c if isinstance(c, (list, tuple)) else [c] for c in conds]
    n_cond = len(per[0])
    flat = [c for p in per for c in p]
    carr = (Cond * len(flat))(*flat)
    hs = (ctypes.c_void_p * B)(*[c._h.value for c in ctxs])
    zs = (ctypes.c_void_p * B)(*[t.data_ptr() for t in z_T_list])
    outs = (ctypes.c_void_p * B)(*[t.data_ptr() for t in z_out_list])
    dec = (ctypes.c_int * (B * T))()
    tr = (StepInfo * (B * T))() if trace else None
    st = LIB.wdc_rollout_batch(hs, B, zs, carr, n_cond, int(bool(cfg)), float(guidance), outs, dec, tr,
                               _stream(stream))
    if st != 0:
        msgs = [LIB.wdc_last_error(c._h).decode() for c in ctxs]
        raise WdcError(st, "rollout_batch: " + " | ".join(f"sample {b}: {m}" for b, m in enumerate(msgs) if m))
    decs = [list(dec[b * T:(b + 1) * T]) for b in range(B)]
    traces = [[tr[b * T + k].as_dict() for k in range(T)] for b in range(B)] if trace else None
    return decs, traces


def observe_noalloc(z_out, kappa, z_a, z_hat, stats, sketch_seed=0x2545F491, stream=None):
    """wdc_observe_noalloc: z_hat = sum_i kappa_i z_out_i plus the next lift's
    statistics (stats: device float64 tensor of 123 values), with no device
    allocation inside the call (see include/wdc.h).

    The entry point has no context that knows the latent size, so the sizes of
    the tensors given here are its only guard: each is checked (dtype, element
    count, contiguity, device) before the call, and a mismatch raises
    ValueError."""
    import torch
    K = len(z_out)
    if len(kappa) != K:
        raise ValueError(f"observe_noalloc: {len(kappa)} weights for {K} latents")
    if not (1 <= K <= MAX_BANK):
        raise ValueError(f"observe_noalloc: K = {K} outside 1..{MAX_BANK}")
    if stats.dtype != torch.float64 or stats.numel() < SKETCH + 3 or not stats.is_contiguous():
        raise ValueError(f"observe_noalloc: stats must be a contiguous float64 tensor of >= {SKETCH + 3} values")
    n = z_hat.numel()
    lat = [("z_hat", z_hat), ("z_a", z_a)] + [(f"z_out[{i}]", t) for i, t in enumerate(z_out)]
    for name, t in lat:
        if t.dtype != torch.float32 or t.numel() != n or not t.is_contiguous():
            raise ValueError(f"observe_noalloc: {name} must be a contiguous float32 tensor of {n} elements")
    dev = torch.device("cuda", torch.cuda.current_device()) if torch.cuda.is_available() else None
    for name, t in lat + [("stats", stats)]:
        if dev is None or t.device != dev:
            raise ValueError(f"observe_noalloc: {name} must be on the current CUDA device")
    ptrs = (ctypes.c_void_p * K)(*[t.data_ptr() for t in z_out])
    kap = (ctypes.c_double * K)(*[float(x) for x in kappa])
    st = LIB.wdc_observe_noalloc(ptrs, K, kap, _ptr(z_a), _ptr(z_hat), _ptr(stats), z_hat.numel(), sketch_seed,
                                 _stream(stream))
    if st != 0:
        raise WdcError(st, "wdc_observe_noalloc failed")
