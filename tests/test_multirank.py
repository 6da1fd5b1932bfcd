"""The N-GPU bench path on CPU: two ranks over gloo (127.0.0.1), as torchrun would
start them. The path has no data-path collective (every rank decodes its own
replica), so what runs across ranks is the timing logic: the job's step time is
the slowest rank's, the whole-job value counts every rank's tokens, and the
reference arm prints from rank 0 only."""
import io
import json
import os
import socket
from contextlib import redirect_stdout

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank: int, world: int, port: int, results):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ws, r, local = bench.dist_env()
        local_ms = 0.1 + 0.05 * rank               # rank 1 is the slower one
        ms = bench.max_over_ranks(local_ms, dist, "cpu")
        value = bench.whole_job_value(ws, 1000.0, ms)
        # the reference arm: rank 0 alone runs the oracle and prints one line
        args = bench.parse(["--impl", "reference", "--workload", "tiny_b1_h16_l256_int4", "--steps", "1",
                            "--warmup", "0"])
        buf = io.StringIO()
        with redirect_stdout(buf):
            bench.run_reference(args, ws, r)
        dist.barrier()
        results[rank] = {"ws": ws, "rank": r, "local": local, "ms": ms, "value": value, "out": buf.getvalue()}
    finally:
        dist.destroy_process_group()


@pytest.mark.timeout(300)
def test_two_ranks_gloo():
    world = 2
    with mp.Manager() as m:
        results = m.dict()
        mp.spawn(_rank_main, args=(world, _free_port(), results), nprocs=world, join=True)
        res = dict(results)
    assert sorted(res) == [0, 1]
    for rank, r in res.items():
        assert (r["ws"], r["rank"], r["local"]) == (2, rank, rank)
        assert r["ms"] == pytest.approx(0.15)                 # the slowest rank's time on every rank
        assert r["value"] == pytest.approx(2 * 1000.0 / 0.15e-3)
    assert res[1]["out"] == ""
    line = json.loads(res[0]["out"].strip())
    assert line["impl"] == "reference" and line["n_gpus"] == 2 and line["unit"] == "KV-tokens/s"
    assert line["cpu_baseline"]["kind"] == "oracle" and line["e2e"]["h2d_bytes_per_step"] == 0


def test_single_process_helpers():
    assert bench.max_over_ranks(0.25, None, "cpu") == 0.25
    assert bench.whole_job_value(1, 500.0, 0.5) == pytest.approx(1e6)

