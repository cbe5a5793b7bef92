"""Host-side arithmetic of bench.py (no GPU): workload shapes, the algorithmic
work the roofline divides by, and the rule that a recorded DRAM-traffic
figure is only reported for the kernel source it was captured on."""
import json
import os

import bench

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_workload_token_counts():
    assert bench.tokens(bench.WORKLOADS["5b"]) == 226 + 13 * 30 * 45 == 17776
    assert bench.tokens(bench.WORKLOADS["13b"]) == 256 + 13 * 32 * 32 == 13568


def test_block_flops_match_the_hand_count():
    w = bench.WORKLOADS["5b"]
    L, D, M, H, d = 17776, 3072, 12288, 48, 64
    gemm = 2 * L * D * (3 * D + D + 2 * M)
    attn = 4 * H * L * L * d
    parts = bench.block_flops(w)
    assert parts[1] == attn == 4 * 48 * 17776 ** 2 * 64
    assert abs(sum(parts) - (gemm + attn)) <= 1e-9 * (gemm + attn)
    assert abs(sum(parts) - 7.909e12) < 0.001e12


def test_traffic_is_reported_only_for_the_captured_source():
    rec = json.load(open(os.path.join(ROOT, "profiles", "traffic.json")))
    for fname, e in rec.items():
        path = os.path.join(ROOT, "paper_2608_01845_gb300", "csrc", fname)
        got = bench.traffic_for(path, e["bench_workload"])
        if bench.kernel_hash(path) == e["source_sha256_16"]:
            assert got == e["dram_bytes_per_launch"]
        else:
            assert got is None
        other = "13b" if e["bench_workload"] == "5b" else "5b"
        assert bench.traffic_for(path, other) is None


def test_surrogate_reading_names_each_observation():
    assert bench.surrogate_reading(0).startswith("Eq. 5 as printed")
    assert bench.surrogate_reading(0x02).startswith("native latent secant")
    assert bench.surrogate_reading(0x100).startswith("residual reading")
    assert bench.surrogate_reading(0x40).startswith("linear observation")
    # every ablation the bench offers maps to one reading
    for v in bench.ABLATIONS.values():
        assert bench.surrogate_reading(v["flags"])


def test_oracle_step_rates_are_reported_per_host():
    n, K = 4096, 2
    r = bench.oracle_step_gbps(n, K)
    assert r["kind"] == "oracle" and r["cores"] == os.cpu_count()
    assert 0 < r["skip_gbps"] < 1e4 and 0 < r["anchor_gbps"] < 1e4


def test_paper_speedups_sit_beside_the_right_workloads():
    assert bench.WORKLOADS["5b"]["paper_speedup"] == 2.15     # Aether-5B, 47% exact calls
    assert bench.WORKLOADS["13b"]["paper_speedup"] == 4.92    # HunyuanVoyager-13B, 20% exact calls
    assert bench.WORKLOADS["5b"]["target_exact"] == 23 and bench.WORKLOADS["13b"]["target_exact"] == 10
