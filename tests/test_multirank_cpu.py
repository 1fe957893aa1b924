"""The multi-rank host logic of bench.py on two CPU ranks (gloo): with N GPUs every rank runs an
independent replica, the job's time is the slowest rank's, the job's value counts all ranks'
tokens, and the reference arm runs on rank 0 alone. No GPU is used."""
import io
import json
import multiprocessing as mp
import os
import socket
import sys
from contextlib import redirect_stdout

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import torch.distributed as dist
    import bench
    from paper_2604_11947_gb300 import synth
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        local_ms = 10.0 + 5.0 * rank                     # rank 1 is the slower one
        ms = bench.max_over_ranks(local_ms, dist, "cpu")
        value = bench.job_throughput(512, world, 3, ms)
        args = type("A", (), dict(steps=1, warmup=0, gpus=world))()
        buf = io.StringIO()
        with redirect_stdout(buf):
            bench.run_reference(args, synth.CONFIGS["tiny_f32"], rank)
        q.put((rank, ms, value, buf.getvalue()))
    finally:
        dist.destroy_process_group()


def test_two_cpu_ranks_time_value_and_reference_arm():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = {}
    for _ in procs:
        rank, ms, value, out = q.get(timeout=300)
        res[rank] = (ms, value, out)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank in (0, 1):
        ms, value, _ = res[rank]
        assert ms == 15.0                                # the slowest rank's time on every rank
        assert abs(value - 512 * 2 * 3 / 0.015) < 1e-6   # all ranks' tokens over that time
    lines = [ln for ln in res[0][2].splitlines() if ln.strip()]
    assert len(lines) == 1
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["n_gpus"] == 2 and line["value"] > 0
    assert line["cpu_baseline"]["kind"] == "oracle"
    assert res[1][2].strip() == ""                       # rank 1 prints nothing
