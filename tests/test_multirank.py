"""The N > 1 host path of bench.py on CPU: two gloo ranks (127.0.0.1).

The rollout does not shard (one trajectory is sequential in its steps), so
N GPUs run N independent replicas: each rank draws its own latent, times its
own rollouts, and the only cross-rank traffic is the barrier and the max of
the ranks' times.  This checks that reduction, the whole-job throughput built
from it, that replicas draw different inputs, and that only rank 0 of the
reference arm prints."""
import io
import os
import socket
import sys
from contextlib import redirect_stdout

import multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    import hashlib
    import types

    import torch.distributed as dist

    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        own_ms = [12.5, 30.0][rank]
        ms = bench.max_over_ranks(own_ms, world, "cpu")
        value = bench.job_steps_per_s(world, 50, 3, ms * 1e-3)
        w = dict(bench.WORKLOADS["5b"], in_ch=4, frames=2, height=8, width=8, cond_tokens=4, cond_dim=16)
        zT, ct, _ = bench.inputs(w, rank)
        printed = ""
        if rank == 1:
            buf = io.StringIO()
            with redirect_stdout(buf):
                bench.run_reference(types.SimpleNamespace(workload="5b", warmup=3, steps=2, gpus=world), rank, world)
            printed = buf.getvalue()
        dist.barrier()
        q.put((rank, ms, value, hashlib.sha256(zT.tobytes()).hexdigest(), hashlib.sha256(ct.tobytes()).hexdigest(),
               printed))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_replicas():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in range(2))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, ms0, v0, z0, c0, out0), (r1, ms1, v1, z1, c1, out1) = res
    assert ms0 == ms1 == 30.0                      # the slowest rank's time, on every rank
    assert v0 == v1 == 2 * 50 * 3 / 0.030          # all ranks' steps over that time
    assert z0 != z1 and c0 == c1                   # own latent per replica, shared condition
    assert out1 == ""                              # reference arm: rank 1 does no work and prints nothing


def test_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(7.0, 1, "cpu") == 7.0
    assert bench.job_steps_per_s(1, 50, 2, 4.0) == 25.0
