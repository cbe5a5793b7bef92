#!/usr/bin/env python
"""Benchmark of the WorldDynCache cached rollout on GB300.

Workload (one "step" of this benchmark = one full cached rollout): the
Aether-5B-like configuration -- a 42-layer random-init bf16 DiT (hidden 3072,
48 heads x 64, MLP 12288, ~5.15B parameters), latent 16x13x60x90 (2x2 patches
-> 17550 video tokens) plus 226 condition tokens, a 50-step flow-matching
Euler schedule, the surrogate + risk controller choosing anchors.  Inputs are
seeded synthetic tensors resident in HBM; the 10.3 GB of weights streamed per
forward are larger than L2, so no explicit flush is needed.

metric: denoising steps per second of the whole job (N replicas, one rollout
each per step: weak scaling).  Extra fields: the dominant kernel's roofline
(live CUDA-event durations inside the timed region), the DiT-block TFLOP/s,
the fused skip-pass GB/s at 2^28 fp32 elements (L2 flushed), the end-to-end
number through the C ABI with host buffers, the CPU oracle's baseline and the
clocks seen during the timed region.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]
"""
import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "cached-rollout steps/s; DiT-block bf16 TFLOP/s & skip-step GB/s vs peak"
UNIT = "steps/s"

# The Aether-5B-like cached rollout.  tau_risk was calibrated once on this
# seeded run to the paper's target exact-call ratio for Aether-5B (47%,
# section "Experimental Settings") and frozen.
WORKLOAD_5B = dict(
    name="cached rollout, 42-layer bf16 DiT 3072/48x64/12288 (~5.15B), latent 16x13x60x90 + 226 cond tokens, T=50",
    layers=42, hidden=3072, heads=48, head_dim=64, mlp=12288, temb_dim=512, freq_dim=256,
    in_ch=16, frames=13, height=60, width=90, patch=2, cond_tokens=226, cond_dim=3072, dual_stream=0,
    T=50, tau_risk=0.1, target_exact=23, weight_seed=1234, input_seed=77,
    paper_speedup=2.15,
)
# The HunyuanVoyager-13B-like cached rollout: 60 dual-stream layers (separate
# condition-token weights, joint attention), 24 heads x 128, latent 16x13x64x64
# (13312 video tokens) + 256 condition tokens.  Paper target exact-call ratio
# 20% (section "Experimental Settings").
WORKLOAD_13B = dict(
    name="cached rollout, 60-layer dual-stream bf16 DiT 3072/24x128/12288 (~14.7B), latent 16x13x64x64 + 256 cond tokens, T=50",
    layers=60, hidden=3072, heads=24, head_dim=128, mlp=12288, temb_dim=512, freq_dim=256,
    in_ch=16, frames=13, height=64, width=64, patch=2, cond_tokens=256, cond_dim=3072, dual_stream=1,
    T=50, tau_risk=0.8, target_exact=10, weight_seed=4321, input_seed=91,
    paper_speedup=4.92,
)
WORKLOADS = {"5b": WORKLOAD_5B, "13b": WORKLOAD_13B}
SKIP_SWEEP_N = 1 << 28          # fused skip pass measured at 2^28 fp32 elements, bank of 4

FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def dit_config(w):
    from paper_2608_01845_gb300 import wdc
    keys = ["layers", "hidden", "heads", "head_dim", "mlp", "temb_dim", "freq_dim", "in_ch", "frames", "height",
            "width", "patch", "cond_tokens", "cond_dim", "dual_stream"]
    return wdc.make_config(dtype=wdc.BF16, **{k: w[k] for k in keys})


def inputs(w, rank):
    from paper_2608_01845_gb300 import synth
    zT = synth.latent(w["input_seed"] + 1000 * rank, (w["in_ch"] * w["frames"] * w["height"] * w["width"],))
    ct = synth.cond_tokens(w["input_seed"] + 1, w["cond_tokens"], w["cond_dim"])
    desc = synth.cond_descriptors(w["input_seed"] + 2)
    return zT, ct, desc


def tokens(w):
    return w["cond_tokens"] + w["frames"] * (w["height"] // w["patch"]) * (w["width"] // w["patch"])


def block_flops(w):
    """Algorithmic flops of one DiT block: 4 GEMMs + joint attention."""
    L, D, M = tokens(w), w["hidden"], w["mlp"]
    gemm = 2 * L * D * 3 * D + 2 * L * D * D + 2 * 2 * L * D * M
    attn = 4 * w["heads"] * L * L * w["head_dim"]
    return gemm, attn


def weight_gb(w):
    """bf16 weight bytes read per forward (block matrices of every stream)."""
    D, M = w["hidden"], w["mlp"]
    per_stream = 3 * D * D + D * D + 2 * D * M
    return w["layers"] * (2 if w["dual_stream"] else 1) * per_stream * 2 / 1e9


def forward_flops(w):
    L, D = tokens(w), w["hidden"]
    Lv = L - w["cond_tokens"]
    P = w["in_ch"] * w["patch"] ** 2
    g, a = block_flops(w)
    extra = 2 * Lv * P * D * 2 + 2 * w["cond_tokens"] * w["cond_dim"] * D
    return w["layers"] * (g + a) + extra, w["layers"] * g + extra, w["layers"] * a


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return d, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


# ------------------------------------------------------------------ clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        try:
            self.p = subprocess.Popen(["nvidia-smi", "--query-gpu=" + self.FIELDS, "--format=csv,noheader,nounits",
                                       "-lms", "200", "-i", str(gpu_index)], stdout=self.f,
                                      stderr=subprocess.DEVNULL)
        except (OSError, ValueError):
            self.p = None

    def stop(self):
        if self.p is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.p.terminate()
        try:
            self.p.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.p.kill()
        self.f.flush()
        rows = []
        for line in open(self.f.name):
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append((float(parts[1]), float(parts[2]), parts[3], parts[5:9]))
            except ValueError:
                continue
        os.unlink(self.f.name)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i, v in enumerate(r[3]) if v.lower().startswith("active")})
        sm = [r[0] for r in rows]
        top = sorted(sm)[len(sm) // 4:] or sm          # drop idle samples at the edges
        return {"sm_mhz": statistics.median(top), "sm_max_mhz": max(r[1] for r in rows), "reasons": reasons,
                "samples": len(rows)}


# ------------------------------------------------------------------ CPU oracle timing
def cpu_sample(w, exact_steps, rows=16):
    """Times the CPU oracle on a bounded sample of the workload and scales it
    to steps/s: one DiT block evaluated for `rows` sampled query rows (keys and
    values for all 17776 tokens) gives the oracle's flop rate, which prices an
    exact forward; one surrogate step and one anchor step at the full latent
    size price the rest.  Returns (steps/s estimate, description, seconds)."""
    import numpy as np
    from oracle import dit
    from oracle import rollout as ro
    from oracle import schedule as sch
    from oracle.params import CacheParams, DiTConfig
    from paper_2608_01845_gb300 import synth
    cfgd = {k: w[k] for k in ["hidden", "heads", "head_dim", "mlp", "temb_dim", "freq_dim", "in_ch", "frames",
                              "height", "width", "patch", "cond_tokens", "cond_dim", "dual_stream"]}
    cfgd["layers"] = 1
    cfgd["dual_stream"] = 0      # the timing sample prices flops; a dual-stream block has the same count
    cfg = DiTConfig(**cfgd)
    names = [f"L0.s0.{n}" for n in ["qkv.w", "qkv.b", "o.w", "o.b", "fc1.w", "fc1.b", "fc2.w", "fc2.b"]]
    W = synth.dit_weights(cfgd, 5, bf16=True, names=names)
    L, D = tokens(w), w["hidden"]
    x = synth.normal(31, (L, D)).astype(np.float64)
    mod = synth.normal(32, (6, D), 0.3).astype(np.float64)
    idx = np.arange(rows) * (L // rows)
    t0 = time.perf_counter()
    dit.block_rows(x, W, cfg, 0, [mod], idx)
    t_blk = time.perf_counter() - t0
    g_full, a_full = block_flops(w)
    f = 2 * L * D * 2 * D + rows / L * (g_full - 2 * L * D * 2 * D) + rows / L * a_full
    rate = f / t_blk
    t_exact_fwd = forward_flops(w)[0] / rate
    # one surrogate step and one anchor step at the full latent size
    n = w["in_ch"] * w["frames"] * w["height"] * w["width"]
    T = w["T"]
    p = CacheParams(tau_risk=w["tau_risk"])
    sig = sch.sigmas(T)
    z = synth.latent(5, (n,))
    st = ro.CacheState.initial(z, sig, p)
    zh, info = ro.surrogate_step(st, z, 0, {}, sig, p)
    v = synth.normal(6, (n,))
    z1 = ro.exact_step(st, z, v, zh, 0, {}, sig, p, info)
    for k in range(1, 4):                    # fill the bank: 4 records
        zh, info = ro.surrogate_step(st, z1, k, {}, sig, p)
        z1 = ro.exact_step(st, z1, v, zh, k, {}, sig, p, info)
    t0 = time.perf_counter()
    zh, info = ro.surrogate_step(st, z1, 4, {}, sig, p)
    t_skip = time.perf_counter() - t0
    t0 = time.perf_counter()
    ro.exact_step(st, z1, v, zh, 4, {}, sig, p, info)
    t_anchor = time.perf_counter() - t0
    per_rollout = exact_steps * (t_exact_fwd + t_skip + t_anchor) + (T - exact_steps) * t_skip
    desc = (f"CPU oracle (fp64 numpy, {os.cpu_count()} BLAS threads): one DiT block for {rows} sampled query rows "
            f"({t_blk:.1f} s, {rate / 1e9:.1f} GFLOP/s) priced {exact_steps} exact forwards; one surrogate step "
            f"({t_skip:.2f} s) and one anchor step ({t_anchor:.2f} s) at {n} latent elements priced the rest; "
            f"scaled to a {T}-step rollout")
    return T / per_rollout, desc, t_blk + t_skip + t_anchor


def run_reference(args, rank, world):
    """The CPU oracle as the reference arm: each step is one bounded sample
    of the workload (one DiT block for 8 sampled query rows, one surrogate
    step and one anchor step at the full latent size), timed on the host
    cores; `value` is the full cached rollout's steps/s those samples price,
    `ms_per_step` the measured wall time of one sample."""
    if rank != 0:
        return
    w = WORKLOADS[args.workload]
    vals, walls = [], []
    desc = ""
    for i in range(args.warmup + args.steps):
        t0 = time.perf_counter()
        v, desc, _ = cpu_sample(w, w["target_exact"], rows=8)
        if i >= args.warmup:
            vals.append(v)
            walls.append(time.perf_counter() - t0)
    value = statistics.mean(vals)
    line = {"metric": METRIC, "value": value, "unit": UNIT, "impl": "reference", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000.0 * statistics.mean(walls),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": w["name"], "exact_steps_priced": w["target_exact"],
                       "step": "one bounded sample of the workload (ms_per_step is its measured wall time); "
                               "value = the full cached rollout's steps/s the samples price"},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
                             "sample": desc},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------ GPU arm
def kernel_hash(path):
    return hashlib.sha256(open(path, "rb").read()).hexdigest()[:16]


def traffic_for(kernel_file, workload):
    """DRAM bytes per launch from the committed ncu summary, if it was taken
    on this workload's launch and the kernel's source is unchanged since."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(p):
        return None
    d = json.load(open(p))
    e = d.get(os.path.basename(kernel_file))
    if not e or e.get("bench_workload") != workload:
        return None
    if e.get("source_sha256_16") != kernel_hash(kernel_file):
        return None
    return e.get("dram_bytes_per_launch")


def skip_pass_time(torch, wdc, n, K=4, secant=False, flush=True, reps=10, seed=0):
    """The fused skip pass alone at n fp32 elements with a bank of K records
    drawn by the sweep's recipe (z_out_i = z0 + 0.05 i sin(2 pi 8 idx/n +
    phase_i), z0 ~ N(0,1)), every record compatible so the pass streams;
    the average of `reps` launches timed with CUDA events on the launching
    stream, L2 flushed by a 512 MB write before each launch (or not, for the
    L2-resident figure).  With ``secant`` the native-latent-secant pass
    instead (reads z_t, the stored displacement and z_a, writes N).  Returns
    (ms per launch, algorithmic bytes, info of the last launch)."""
    import numpy as np
    from paper_2608_01845_gb300 import synth
    flags = wdc.ABL_SECANT if secant else 0
    ctx = wdc.Context(wdc.make_config(layers=0, width=n), 50,
                      params=wdc.make_params(bank_capacity=K, sim_min=-1.0, q_gap_max=1.0, flags=flags))
    bank = synth.drift_bank_device(seed + n % 1000003 + K, n, K)
    st = wdc.StateHost()
    st.n_bank, st.R, st.eta = K, 0.1, 1.0
    g = np.random.default_rng(seed)
    for i in range(K):
        a = g.standard_normal(256)
        for j in range(256):
            st.rec[i].s_in[j] = a[j]
            st.rec[i].s_out[j] = a[j] + 0.1
            st.rec[i].s_dphi[j] = 0.1
        st.rec[i].q_in = 0.6 + 0.02 * (K - i)
        st.rec[i].q_out = st.rec[i].q_in - 0.02
    st.q_a_in, st.q_a_out = st.rec[K - 1].q_in, st.rec[K - 1].q_out
    zc = bank[-1] + 0.01
    ctx.state_set(st, bank, zc)
    zh = torch.empty(n, device="cuda")
    buf = torch.empty(128 * 1024 * 1024, device="cuda") if flush else None
    cond = wdc.make_cond()
    for _ in range(3):
        if flush:
            buf.zero_()
        ctx.surrogate_step(20, cond, zh)
    ctx.profile_enable(True)
    for _ in range(reps):
        if flush:
            buf.zero_()
        info = ctx.surrogate_step(20, cond, zh)
    prof = ctx.profile_read()
    ctx.profile_enable(False)
    ms = prof["skip"][0] / prof["skip"][1]
    streams = 4 if secant else K + 1
    ctx.close()
    del bank, zc, zh, buf
    torch.cuda.empty_cache()
    return ms, streams * 4 * n, info


def skip_pass_gbps(torch, wdc, peaks, secant=False, n=SKIP_SWEEP_N, K=4, flush=True):
    ms, nbytes, info = skip_pass_time(torch, wdc, n, K, secant=secant, flush=flush)
    gbs = nbytes / (ms * 1e-3) / 1e9
    return {"gbps": gbs, "ms": ms, "n": n, "bank": K, "supported": bool(info.supported), "bytes": nbytes,
            "frac_of_measured_copy": gbs / peaks["hbm_gbs"], "l2": "flushed" if flush else "resident"}


def copy_ms(torch, nbytes, reps=10):
    """A plain device copy (torch's copy_) moving `nbytes` in all (half read,
    half written), L2 flushed before each, CUDA events, median of `reps`: the
    bandwidth a copy itself reaches at that size (the measured peak is a 2 GB
    copy; short copies pay their ramp and tail)."""
    n = max(1, nbytes // 8)
    a = torch.randn(n, device="cuda")
    b = torch.empty_like(a)
    buf = torch.empty(128 * 1024 * 1024, device="cuda")
    for _ in range(3):
        b.copy_(a)
    ts = []
    for _ in range(reps):
        buf.zero_()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        b.copy_(a)
        e1.record()
        torch.cuda.synchronize()
        ts.append(e0.elapsed_time(e1))
    del a, b, buf
    torch.cuda.empty_cache()
    return statistics.median(ts)


def oracle_step_gbps(n, K):
    """The CPU oracle's surrogate step and anchor step at n latent elements
    with a bank of K records (filled by K exact steps first), each timed once
    on the host cores, as GB/s of the same algorithmic bytes as the GPU
    passes: (K+1)*4n and 5*4n."""
    from oracle import rollout as ro
    from oracle import schedule as sch
    from oracle.params import CacheParams
    from paper_2608_01845_gb300 import synth
    p = CacheParams(tau_risk=0.5, bank_capacity=K)
    sig = sch.sigmas(50)
    z = synth.latent(5, (n,))
    v = synth.normal(6, (n,))
    st = ro.CacheState.initial(z, sig, p)
    for k in range(K):
        zh, info = ro.surrogate_step(st, z, k, {}, sig, p)
        z = ro.exact_step(st, z, v, zh, k, {}, sig, p, info)
    t0 = time.perf_counter()
    zh, info = ro.surrogate_step(st, z, K, {}, sig, p)
    t_skip = time.perf_counter() - t0
    t0 = time.perf_counter()
    ro.exact_step(st, z, v, zh, K, {}, sig, p, info)
    t_anchor = time.perf_counter() - t0
    return {"skip_gbps": (K + 1) * 4 * n / t_skip / 1e9, "anchor_gbps": 5 * 4 * n / t_anchor / 1e9,
            "cores": os.cpu_count(), "kind": "oracle"}


def skip_sweep(torch, wdc, peaks, workload_n, cpu=False):
    """The skipped-step kernel sweep: N in {2^20, 2^24, 2^26, 2^28} fp32
    elements x K in {2, 3, 4} bank records, L2 flushed before every launch;
    plus 2^20 L2-resident and the workload's own latent size.  Each row also
    gives a plain copy of the same byte count timed the same way, and the
    pass's time against it; with `cpu`, the 2^20 rows also give the CPU
    oracle's surrogate and anchor steps (larger sizes take the oracle minutes
    per bank fill)."""
    rows = []
    for e in (20, 24, 26, 28):
        for K in (2, 3, 4):
            r = skip_pass_gbps(torch, wdc, peaks, n=1 << e, K=K)
            cms = copy_ms(torch, r["bytes"])
            rows.append({"n": f"2^{e}", "K": K, "gbps": round(r["gbps"], 1), "ms": round(r["ms"], 5),
                         "frac_of_measured_copy": round(r["frac_of_measured_copy"], 4),
                         "same_bytes_copy_ms": round(cms, 5), "frac_of_same_bytes_copy": round(cms / r["ms"], 4)})
            if cpu and e == 20:
                rows[-1]["cpu_oracle"] = {k: (round(v, 4) if isinstance(v, float) else v)
                                          for k, v in oracle_step_gbps(1 << e, K).items()}
    r = skip_pass_gbps(torch, wdc, peaks, n=1 << 20, K=4, flush=False)
    rows.append({"n": "2^20", "K": 4, "l2": "resident", "gbps": round(r["gbps"], 1), "ms": round(r["ms"], 5),
                 "frac_of_measured_copy": round(r["frac_of_measured_copy"], 4)})
    r = skip_pass_gbps(torch, wdc, peaks, n=workload_n, K=4)
    rows.append({"n": workload_n, "K": 4, "note": "the rollout's own latent", "gbps": round(r["gbps"], 1),
                 "ms": round(r["ms"], 5), "frac_of_measured_copy": round(r["frac_of_measured_copy"], 4)})
    return {"bytes_per_launch": "(K+1)*4*N", "timing": "CUDA events on the launching stream, mean of 10",
            "same_bytes_copy": "torch copy_ of the same total bytes (half read, half written), median of 10",
            "rows": rows}


def block_tflops(torch, ctx, w, peaks):
    """One DiT block of the workload in place on [L, D]."""
    L, D = tokens(w), w["hidden"]
    x = torch.randn(L, D, device="cuda").bfloat16()
    mod = 0.1 * torch.randn((2 if w["dual_stream"] else 1) * 6, D, device="cuda")
    for _ in range(3):
        ctx.dit_block_forward(0, x, mod)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    reps = 10
    e0.record()
    for _ in range(reps):
        ctx.dit_block_forward(0, x, mod)
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / reps
    g, a = block_flops(w)
    tf = (g + a) / (ms * 1e-3) / 1e12
    return {"tflops": tf, "ms": ms, "frac_of_measured_burst": tf / peaks["bf16_tflops"]}


# The 2-layer parity model (the oracle-checked configuration): fp32, D = 256,
# 4 x 64 heads, MLP 1024, latent 16x4x16x16 + 16 condition tokens, T = 10.
WORKLOAD_CFG0 = dict(
    name="cached rollout, 2-layer fp32 DiT 256/4x64/1024, latent 16x4x16x16 + 16 cond tokens, T=10",
    layers=2, hidden=256, heads=4, head_dim=64, mlp=1024, temb_dim=256, freq_dim=256, in_ch=16, frames=4,
    height=16, width=16, patch=2, cond_tokens=16, cond_dim=256, dual_stream=0, T=10, tau_risk=0.5,
)


def surrogate_reading(flags):
    """Which reading of Eq. 5's observation the run used."""
    if flags & 0x02:
        return "native latent secant (ablation)"
    if flags & 0x100:
        return "residual reading of Eq. 5: z_t + sum_i kappa_i (z_out_i - z_in_i)"
    if flags & 0x40:
        return "linear observation (ablation): sum_i beta_i z_out_i, beta the ridge readout of the lifted summary"
    return "Eq. 5 as printed: sum_i kappa_i z_out_i"


def native_speedup(torch, ctx, w, zT_d, cond, cached_steps_per_s):
    """One uncached rollout (every step an exact forward, wdc_native_rollout)
    on the same context and inputs, CUDA events: its steps/s and the cached
    rollout's speedup over it, beside the paper's speedup for the model this
    workload is shaped like (8x A6000, context only)."""
    T = w["T"]
    nat = torch.empty_like(zT_d)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    ctx.native_rollout(zT_d, cond, nat)
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1)
    del nat
    native = T / (ms * 1e-3)
    return {"steps_per_s": native, "ms_per_rollout": ms, "speedup_cached_vs_native": cached_steps_per_s / native,
            "paper_speedup": w["paper_speedup"], "paper_hardware": "8x NVIDIA A6000 (context, not the target)"}


def rollout_component(torch, wdc, w, peaks, reps=2):
    """One workload's cached rollout on its own context: steps/s over `reps`
    timed rollouts after one warm-up, the exact-step count, and the dominant
    kernel class against the measured sustained bf16 peak (live CUDA-event
    durations)."""
    T = w["T"]
    ctx = wdc.Context(dit_config(w), T, params=wdc.make_params(tau_risk=w["tau_risk"]))
    ctx.init_weights(w["weight_seed"], 0.02)
    zT, ct, desc = inputs(w, 0)
    zT_d = torch.from_numpy(zT).cuda()
    ct_d = torch.from_numpy(ct).cuda()
    cond = wdc.make_cond(ct_d, desc["cam"], desc["depth"])
    out = torch.empty_like(zT_d)
    ctx.rollout(zT_d, cond, out, trace=False)
    torch.cuda.synchronize()
    ctx.profile_enable(True)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    exact = []
    for _ in range(reps):
        dec, _ = ctx.rollout(zT_d, cond, out, trace=False)
        exact.append(T - sum(dec))
    e1.record()
    torch.cuda.synchronize()
    prof = ctx.profile_read()
    ctx.profile_enable(False)
    ms = e0.elapsed_time(e1) / reps
    cls = {k: v[0] for k, v in prof.items()}
    dom = max(cls, key=cls.get)
    if dom == "attention":
        avg = prof["attention"][0] / prof["attention"][1]
        achieved = block_flops(w)[1] / (avg * 1e-3) / 1e12
    else:
        avg = None
        achieved = None
    native = native_speedup(torch, ctx, w, zT_d, cond, T / (ms * 1e-3))
    ctx.close()
    del zT_d, ct_d, out
    torch.cuda.empty_cache()
    res = {"workload": w["name"], "steps_per_s": T / (ms * 1e-3), "ms_per_rollout": ms, "exact_steps": exact,
           "tau_risk": w["tau_risk"], "dominant_kernel": dom,
           "time_share": {k: v / sum(cls.values()) for k, v in cls.items()}, "native_rollout": native}
    if achieved is not None:
        res.update({"attention_avg_launch_ms": avg, "attention_tflops": achieved,
                    "attention_frac_of_measured_sustained": achieved / peaks["bf16_tflops_sustained"]})
    return res


def cfg0_component(torch, wdc, cpu=True, reps=20):
    """The 2-layer fp32 parity model's cached rollout (T = 10): steps/s on the
    GPU (host-driven and graph rollout, median of `reps`), and the CPU oracle's
    own cached rollout of the same inputs timed on the host cores."""
    import numpy as np
    from paper_2608_01845_gb300 import synth
    w = WORKLOAD_CFG0
    keys = ["layers", "hidden", "heads", "head_dim", "mlp", "temb_dim", "freq_dim", "in_ch", "frames", "height",
            "width", "patch", "cond_tokens", "cond_dim", "dual_stream"]
    cfgd = {k: w[k] for k in keys}
    T = w["T"]
    W = synth.dit_weights(cfgd, 0, std=0.02)
    ctx = wdc.Context(wdc.make_config(dtype=wdc.F32, **cfgd), T, params=wdc.make_params(tau_risk=w["tau_risk"]))
    ctx.set_weights(W)
    z0 = synth.latent(1, (16, 4, 16, 16))
    ct = synth.cond_tokens(2, 16, 256)
    desc = synth.cond_descriptors(3)
    zT = torch.from_numpy(z0.ravel().copy()).cuda()
    cond = wdc.make_cond(torch.from_numpy(ct).cuda(), desc["cam"], desc["depth"])
    out = torch.empty_like(zT)
    res = {"workload": w["name"]}
    for mode, fn in [("host", lambda: ctx.rollout(zT, cond, out, trace=False)),
                     ("graph", lambda: ctx.rollout_graph(zT, cond, out, trace=False))]:
        for _ in range(3):
            dec, _ = fn()
        torch.cuda.synchronize()
        ts = []
        for _ in range(reps):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            fn()
            e1.record()
            torch.cuda.synchronize()
            ts.append(e0.elapsed_time(e1))
        ms = statistics.median(ts)
        res[mode] = {"steps_per_s": T / (ms * 1e-3), "ms_per_rollout": ms, "exact_steps": T - sum(dec)}
    res["decisions"] = dec
    ctx.close()
    if cpu:
        from oracle import dit
        from oracle import rollout as ro
        from oracle import schedule as sch
        from oracle.params import CacheParams, DiTConfig
        cfg = DiTConfig(**cfgd)
        F = lambda z, t, c, k: dit.forward(W, cfg, np.asarray(z).reshape(16, 4, 16, 16), t, ct)
        t0 = time.perf_counter()
        _, dec_o, _ = ro.cached_rollout(z0, F, desc, sch.sigmas(T), CacheParams(tau_risk=w["tau_risk"]))
        sec = time.perf_counter() - t0
        res["cpu_oracle"] = {"steps_per_s": T / sec, "s_per_rollout": sec, "cores": os.cpu_count(),
                             "kind": "oracle", "decisions_equal": dec_o == dec,
                             "sample": "the whole 10-step cached rollout (fp64 numpy)"}
    return res


# Ablation variants of Tables 3-4 (and the residual reading of Eq. 5) for
# `--ablation NAME` (the periodic
# controller at period 2 = 25 exact steps of 50, the closest period to the
# risk controller's 23 of 50: "matched budget").
ABLATIONS = {
    "full": dict(flags=0),
    "periodic+secant": dict(flags=0x01 | 0x02, period=2),
    "risk+secant": dict(flags=0x02),
    "periodic+lifted": dict(flags=0x01, period=2),
    "no_condition": dict(flags=0x80),
    "linear_obs": dict(flags=0x40),
    "instantaneous": dict(flags=0x04),
    "no_impact": dict(flags=0x08),
    "no_calibration": dict(flags=0x10),
    "no_support": dict(flags=0x20),
    "residual": dict(flags=0x100),                  # residual reading of Eq. 5 (not an ablation)
}


def max_over_ranks(x, world, device):
    """The slowest rank's figure: every rank contributes its own time, the
    job's time is the maximum (one all-reduce; nothing else crosses ranks)."""
    if world <= 1:
        return float(x)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_steps_per_s(world, T, rollouts, seconds):
    """Whole-job throughput of replicas: each of `world` ranks rolls out
    `rollouts` independent T-step rollouts in `seconds` (the max over ranks)."""
    return world * T * rollouts / seconds


def run_gpu(args, rank, world, local_rank):
    import torch
    import torch.distributed as dist
    from paper_2608_01845_gb300 import wdc
    torch.cuda.set_device(local_rank)
    w = WORKLOADS[args.workload]
    T = w["T"]
    peaks, peak_src = load_peaks()
    params = wdc.make_params(tau_risk=w["tau_risk"], **(ABLATIONS[args.ablation] if args.ablation else {}))
    ctx = wdc.Context(dit_config(w), T, params=params, device=local_rank)
    ctx.init_weights(w["weight_seed"], 0.02)
    zT, ct, desc = inputs(w, rank)
    zT_d = torch.from_numpy(zT).cuda()
    ct_d = torch.from_numpy(ct).cuda()
    cond = wdc.make_cond(ct_d, desc["cam"], desc["depth"])
    out = torch.empty_like(zT_d)

    def barrier():
        if world > 1:
            dist.barrier()

    for _ in range(args.warmup):
        decisions, _ = ctx.rollout(zT_d, cond, out, trace=False)
    torch.cuda.synchronize()

    # ---- timed region: K cached rollouts, inputs resident in HBM
    barrier()
    torch.cuda.synchronize()
    clocks = ClockSampler(local_rank)
    launches0 = ctx.launches
    ctx.profile_enable(True)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    all_dec = []
    for _ in range(args.steps):
        decisions, _ = ctx.rollout(zT_d, cond, out, trace=False)
        all_dec.append(decisions)
    e1.record()
    torch.cuda.synchronize()
    barrier()
    clk = clocks.stop()
    prof = ctx.profile_read()
    ctx.profile_enable(False)
    launches = ctx.launches - launches0
    ms = max_over_ranks(e0.elapsed_time(e1), world, "cuda")
    value = job_steps_per_s(world, T, args.steps, ms * 1e-3)
    exact = [T - sum(d) for d in all_dec]

    # ---- dominant kernel of the timed region and its roofline
    fwd_total, fwd_gemm, fwd_attn = forward_flops(w)
    n_fwd = sum(exact)
    cls_time = {k: v[0] for k, v in prof.items()}
    dom = max(cls_time, key=cls_time.get)
    if dom == "attention":
        avg_ms = prof["attention"][0] / prof["attention"][1]
        achieved = block_flops(w)[1] / (avg_ms * 1e-3) / 1e12
        kfile = os.path.join(ROOT, "paper_2608_01845_gb300", "csrc", "attn_tc.cu")
        kname = f"attn_tc_kernel<{w['head_dim']}, false> ({w['heads']} heads x {tokens(w)} tokens x {w['head_dim']})"
        traffic = traffic_for(kfile, args.workload)
    else:
        avg_ms = prof["gemm"][0] / prof["gemm"][1]
        if w["dual_stream"]:
            # the condition rows' block GEMMs run on the forked stream, untimed:
            # the timed GEMM work is the video rows' blocks plus the embeddings
            Lv = tokens(w) - w["cond_tokens"]
            g_all, _ = block_flops(w)
            fwd_gemm -= w["layers"] * g_all * (1.0 - Lv / tokens(w))
        achieved = n_fwd * fwd_gemm / (prof["gemm"][0] * 1e-3) / 1e12
        kfile = os.path.join(ROOT, "paper_2608_01845_gb300", "csrc", "gemm_tc.cu")
        kname = "gemm_tc2_kernel / gemm_tc_kernel (all denoiser GEMMs)"
        traffic = None          # an aggregate over several shapes has no per-launch capture
    peak = peaks["bf16_tflops_sustained"]
    roofline = {"bound": "tensor", "kernel": kname, "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                "frac": achieved / peak, "peak_source": f"{peak_src} sustained bf16 (kernel timed inside a long step)",
                "avg_launch_ms": avg_ms, "launches_timed": int(prof[dom][1]), "traffic": traffic,
                "time_share": {k: v / sum(cls_time.values()) for k, v in cls_time.items()}}

    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": w["name"] + (f", ablation {args.ablation}" if args.ablation else ""),
                       "T": T, "tau_risk": w["tau_risk"], "bank_capacity": 4,
                       "surrogate_reading": surrogate_reading(params.flags),
                       "l2": f"inputs larger than L2 ({weight_gb(w):.1f} GB of weights per forward)",
                       "parallelism": f"replicas x{world}"},
            "exact_steps_per_rollout": exact, "gpu_launches": launches, "clocks": clk, "roofline": roofline}

    # ---- end to end through the C ABI with host buffers
    zT_h = torch.from_numpy(zT).pin_memory()
    ct_h = torch.from_numpy(ct).pin_memory()
    out_h = torch.empty_like(zT_h).pin_memory()
    cond_h = wdc.make_cond(ct_h, desc["cam"], desc["depth"])
    barrier()
    torch.cuda.synchronize()
    # (at most 5 rollouts: each is seconds long, so the figure is settled by
    # then, and the bench's wall time stays within a few minutes)
    e2e_reps = min(args.steps, 5)
    t0 = time.perf_counter()
    for _ in range(e2e_reps):
        ctx.rollout(zT_h, cond_h, out_h, trace=False)
    torch.cuda.synchronize()
    et = max_over_ranks(time.perf_counter() - t0, world, "cuda")
    line["e2e"] = {"value": job_steps_per_s(world, T, e2e_reps, et), "unit": UNIT,
                   "h2d_bytes_per_step": zT.nbytes + ct.nbytes, "d2h_bytes_per_step": zT.nbytes,
                   "rollouts": e2e_reps,
                   "note": "without the per-launch event profiler the device-timed region runs for the roofline "
                           "(two events per launch, 0.2-0.4% of a rollout, measured), so it can read slightly above value"}

    # device-side control flow on the same workload (graph built by a first call)
    if rank == 0 and not args.ablation:
        ctx.rollout_graph(zT_d, cond, out, trace=False)
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        dec_g, _ = ctx.rollout_graph(zT_d, cond, out, trace=False)
        torch.cuda.synchronize()
        gt = time.perf_counter() - t0
        line["graph_rollout"] = {"steps_per_s": T / gt, "exact_steps": T - sum(dec_g),
                                 "note": "wdc_rollout_graph: no host synchronisation between steps"}
        line["native_rollout"] = native_speedup(torch, ctx, w, zT_d, cond, T * args.steps / (ms * 1e-3))

    if args.ablation and rank == 0:
        # mechanics of the variant on the random-init model: final latent
        # against the uncached rollout of the same inputs
        cached = out.cpu().numpy().astype("float64")
        nat = torch.empty_like(zT_d)
        ctx.native_rollout(zT_d, cond, nat)
        nat = nat.cpu().numpy().astype("float64")
        import numpy as np
        line["ablation"] = {"name": args.ablation, "flags": params.flags, "period": params.period,
                            "final_rel_l2_vs_native": float(np.linalg.norm(cached - nat) / np.linalg.norm(nat))}

    # ---- components named by the metric (rank 0 only)
    if rank == 0 and args.no_components:
        print(json.dumps(line), flush=True)
    elif rank == 0:
        line["components"] = {"dit_block": block_tflops(torch, ctx, w, peaks)}
        ctx.close()
        torch.cuda.empty_cache()
        if not args.ablation and not args.no_extra_rollouts:
            other = "13b" if args.workload == "5b" else "5b"
            line["components"][f"rollout_{other}"] = rollout_component(torch, wdc, WORKLOADS[other], peaks)
            line["components"]["rollout_cfg0"] = cfg0_component(torch, wdc,
                                                                cpu=world == 1 and not args.no_cpu_baseline)
        line["components"]["skip_pass"] = skip_pass_gbps(torch, wdc, peaks)
        line["components"]["secant_pass"] = skip_pass_gbps(torch, wdc, peaks, secant=True)
        line["components"]["skip_sweep"] = skip_sweep(torch, wdc, peaks,
                                                      w["in_ch"] * w["frames"] * w["height"] * w["width"],
                                                      cpu=world == 1 and not args.no_cpu_baseline)
        line["components"]["peaks"] = {"hbm_gbs": peaks["hbm_gbs"], "bf16_tflops": peaks["bf16_tflops"],
                                       "source": peak_src}
        if world == 1 and not args.no_cpu_baseline:
            v, d, secs = cpu_sample(w, int(round(statistics.mean(exact))))
            line["cpu_baseline"] = {"value": v, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
                                    "sample": d}
        print(json.dumps(line), flush=True)


def run_op(args):
    """One operator at its full 5B-scale shape, for profiler captures: a few
    launches, CUDA-event timing printed as JSON."""
    import torch
    from paper_2608_01845_gb300 import wdc
    w = WORKLOADS[args.workload]
    peaks, _ = load_peaks()
    L, D, H, d = tokens(w), w["hidden"], w["heads"], w["head_dim"]
    dev = torch.device("cuda")
    if args.op == "batch":
        return run_batch(args, w, peaks)
    one_layer = dict(w, layers=1)
    ctx = wdc.Context(dit_config(one_layer), w["T"])
    ev = lambda: torch.cuda.Event(enable_timing=True)
    if args.op == "attention":
        q = torch.randn(H, L, d, device=dev).bfloat16()
        k = torch.randn(H, L, d, device=dev).bfloat16()
        vt = torch.randn(H, d, L, device=dev).half()           # V^T is fp16 in the bf16 model
        o = torch.empty(L, H * d, device=dev, dtype=torch.bfloat16)
        fn, work, unit = (lambda: ctx.op_attention(q, k, vt, o)), 4 * H * L * L * d, "TFLOP/s"
    elif args.op == "gemm":
        A = torch.randn(L, D, device=dev).bfloat16()
        Wt = (0.02 * torch.randn(3 * D, D, device=dev)).bfloat16()
        C = torch.empty(L, 3 * D, device=dev, dtype=torch.bfloat16)
        fn, work, unit = (lambda: ctx.op_gemm(A, Wt, C)), 2 * L * 3 * D * D, "TFLOP/s"
    elif args.op == "block":
        ctx.init_weights(1, 0.02)
        x = torch.randn(L, D, device=dev).bfloat16()
        mod = 0.1 * torch.randn((2 if w["dual_stream"] else 1) * 6, D, device=dev)
        fn, work, unit = (lambda: ctx.dit_block_forward(0, x, mod)), sum(block_flops(w)), "TFLOP/s"
    elif args.op == "control":
        # host-driven vs device-side control flow (wdc_rollout vs
        # wdc_rollout_graph) on the 2-layer D=256 parity model, T = 50,
        # where the per-step host synchronisation is visible
        from paper_2608_01845_gb300 import synth
        small = dict(layers=2, hidden=256, heads=4, head_dim=64, mlp=1024, temb_dim=256, freq_dim=256, in_ch=16,
                     frames=4, height=16, width=16, patch=2, cond_tokens=16, cond_dim=256, dual_stream=0)
        T = 50
        res = {}
        for dt, name in [(wdc.F32, "fp32"), (wdc.BF16, "bf16")]:
            cx = wdc.Context(wdc.make_config(dtype=dt, **small), T, params=wdc.make_params(tau_risk=0.5))
            cx.init_weights(3, 0.02)
            zT = torch.from_numpy(synth.latent(1, (16 * 4 * 16 * 16,))).cuda()
            cd = wdc.make_cond(torch.from_numpy(synth.cond_tokens(2, 16, 256)).cuda(), [0.1] * 4, [0.05] * 4)
            out = torch.empty_like(zT)
            row = {}
            for mode, fn in [("host", lambda: cx.rollout(zT, cd, out, trace=False)),
                             ("graph", lambda: cx.rollout_graph(zT, cd, out, trace=False))]:
                for _ in range(3):
                    dec, _ = fn()
                torch.cuda.synchronize()
                ts = []
                for _ in range(max(args.reps, 5)):
                    t0 = time.perf_counter()
                    fn()
                    torch.cuda.synchronize()
                    ts.append(time.perf_counter() - t0)
                ms = 1e3 * statistics.median(ts)
                row[mode] = {"ms_per_rollout": ms, "steps_per_s": T / (ms * 1e-3), "exact_steps": T - sum(dec)}
            res[name] = row
            cx.close()
        print(json.dumps({"op": "control", "model": "2-layer D=256 (parity model shape), T=50", **res}))
        return
    elif args.op == "gemms":
        # the block's four GEMMs with their epilogues, one line per shape
        M = L
        out = {}
        for name, N, K, kw in [("qkv", 3 * D, D, {}), ("out", D, D, {"resid": True}),
                               ("mlp_up", w["mlp"], D, {"gelu": True}), ("mlp_down", D, w["mlp"], {"resid": True})]:
            A = torch.randn(M, K, device=dev).bfloat16()
            Wt = (0.02 * torch.randn(N, K, device=dev)).bfloat16()
            C = torch.randn(M, N, device=dev).bfloat16()
            b = torch.zeros(N, device=dev)
            gate = torch.ones(N, device=dev)
            extra = {"gelu": True} if kw.get("gelu") else ({"res": C, "gate": gate} if kw.get("resid") else {})
            f = lambda: ctx.op_gemm(A, Wt, C, bias=b, **extra)
            for _ in range(3):
                f()
            torch.cuda.synchronize()
            ts = []
            for _ in range(args.reps):
                a, e = ev(), ev()
                a.record()
                f()
                e.record()
                torch.cuda.synchronize()
                ts.append(a.elapsed_time(e))
            ms = statistics.median(ts)
            out[f"{name} {M}x{N}x{K}"] = {"ms": ms, "TFLOP/s": 2 * M * N * K / (ms * 1e-3) / 1e12}
            del A, Wt, C
        print(json.dumps({"op": "gemms", "workload": args.workload, **out}))
        return
    elif args.op == "skip_sweep":
        print(json.dumps({"op": "skip_sweep", **skip_sweep(torch, wdc, peaks, 16 * 13 * 60 * 90)}))
        return
    else:
        r = skip_pass_gbps(torch, wdc, peaks, secant=args.op == "secant", n=args.n, K=args.bank)
        print(json.dumps({"op": args.op, **r}))
        return
    for _ in range(2):
        fn()
    torch.cuda.synchronize()
    ts = []
    for _ in range(args.reps):
        a, b = ev(), ev()
        a.record()
        fn()
        b.record()
        torch.cuda.synchronize()
        ts.append(a.elapsed_time(b))
    ms = statistics.median(ts)
    print(json.dumps({"op": args.op, "workload": args.workload, "ms": ms, unit: work / (ms * 1e-3) / 1e12}))


def run_batch(args, w, peaks):
    """Batched cached rollout (wdc_rollout_batch) of --batch samples of the
    workload, each from its own latent, against the same samples rolled out
    one at a time (a batch of one each).  With --cfg every exact step runs the
    guided velocity (conditional + null-condition forward in one batch)."""
    import torch
    from paper_2608_01845_gb300 import wdc
    B = args.batch
    cfg = dit_config(w)
    cfg.max_batch = 2 * B if args.cfg else B
    T = w["T"]
    prm = lambda: wdc.make_params(tau_risk=w["tau_risk"])
    ctxs = [wdc.Context(cfg, T, params=prm())]
    ctxs[0].init_weights(w["weight_seed"], 0.02)
    lat = wdc.make_config(in_ch=w["in_ch"], frames=w["frames"], height=w["height"], width=w["width"])
    ctxs += [wdc.Context(lat, T, params=prm()) for _ in range(1, B)]
    _, ct, desc = inputs(w, 0)
    ct = torch.from_numpy(ct).cuda()
    zs = [torch.from_numpy(inputs(w, b)[0]).cuda() for b in range(B)]
    conds = [wdc.make_cond(ct, desc["cam"], desc["depth"]) for _ in range(B)]
    outs = [torch.empty_like(z) for z in zs]
    kw = dict(cfg=args.cfg, guidance=args.guidance, trace=False)

    def batched():
        return wdc.rollout_batch(ctxs, zs, conds, outs, **kw)[0]

    def sequential():
        return [wdc.rollout_batch([ctxs[0]], [zs[b]], [conds[b]], [outs[b]], **kw)[0][0] for b in range(B)]

    res = {}
    for name, fn in [("batched", batched), ("sequential", sequential)]:
        decs = fn()                                   # warm-up (and the decisions)
        torch.cuda.synchronize()
        ts = []
        for _ in range(args.reps):
            t0 = time.perf_counter()
            fn()
            torch.cuda.synchronize()
            ts.append(time.perf_counter() - t0)
        sec = statistics.median(ts)
        res[name] = {"s": sec, "samples_per_s": B / sec, "steps_per_s": B * T / sec,
                     "exact_steps": [T - sum(d) for d in decs]}
    res["batched"]["exact_batches"] = sum(1 for k in range(T) if any(d[k] == 0 for d in decs))
    print(json.dumps({"op": "batch", "workload": args.workload, "B": B, "cfg": bool(args.cfg),
                      "guidance": args.guidance if args.cfg else None, **res,
                      "speedup": res["sequential"]["s"] / res["batched"]["s"]}))


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="wdc", choices=["wdc", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-extra-rollouts", action="store_true",
                    help="skip the other full-size workload's and the 2-layer model's rollouts")
    ap.add_argument("--no-components", action="store_true",
                    help="print the rollout line without the component measurements (for launch-list captures)")
    ap.add_argument("--ablation", choices=sorted(ABLATIONS),
                    help="run the timed rollout under one ablation variant (Tables 3-4) and report its "
                         "final latent against the uncached rollout")
    ap.add_argument("--op", choices=["attention", "gemm", "gemms", "block", "skip", "secant", "skip_sweep", "control",
                                     "batch"],
                    help="time one operator at its 5B-scale shape (profiler captures); batch: the batched "
                         "cached rollout against one-at-a-time rollouts")
    ap.add_argument("--batch", type=int, default=2, help="--op batch: samples per batch")
    ap.add_argument("--n", type=int, default=SKIP_SWEEP_N, help="--op skip / secant: latent elements")
    ap.add_argument("--bank", type=int, default=4, help="--op skip: bank records K")
    ap.add_argument("--cfg", action="store_true", help="--op batch: classifier-free guidance on every exact step")
    ap.add_argument("--guidance", type=float, default=5.0, help="--op batch: guidance scale with --cfg")
    ap.add_argument("--reps", type=int, default=3)
    ap.add_argument("--workload", choices=sorted(WORKLOADS), default="5b",
                    help="rollout / --op shape (5b: 42 layers, 48x64 heads, L=17776; 13b: 60 dual-stream layers, "
                         "24x128 heads, L=13568)")
    args = ap.parse_args()
    if args.op:
        return run_op(args)
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        return run_reference(args, rank, world)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    run_gpu(args, rank, world, local_rank)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
