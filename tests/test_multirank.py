"""The multi-rank host logic of bench.py on CPU: world_size-2 gloo ranks.

Sequences are independent, so ranks are replicas that each run their own shard of
the batch; they meet only at the barriers around the timed region and in one
max-reduction of the elapsed time.  These tests run that plumbing in two real
processes (gloo backend, 127.0.0.1) without a GPU."""
import json
import os
import socket
import sys

import numpy as np
import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, outdir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import bench
    import workloads as wl
    import torch.distributed as dist

    ws, r, local = bench.dist_init()
    assert (ws, r, local) == (world, rank, rank) and dist.get_backend() == "gloo"
    bench.barrier(ws)
    elapsed_ms = 3.0 + 2.0 * rank                       # this rank's device time over its steps
    worst = bench.max_over_ranks(elapsed_ms, ws)
    w = wl.CONFIGS["decode_loop_b128_ctx32k"].replace(B=2, prompt_len=64, out_len=32)
    tok, _ = wl.token_streams(w, w.T, bench.shard_seed(w.seed, rank))
    bench.barrier(ws)
    with open(os.path.join(outdir, f"rank{rank}.json"), "w") as f:
        json.dump({"worst": worst, "value": bench.steps_per_second(ws, 10, worst),
                   "tokens": tok.tolist()}, f)
    dist.destroy_process_group()


def test_two_gloo_ranks_shard_and_take_the_slowest(tmp_path):
    world = 2
    mp.start_processes(_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world,
                       start_method="spawn", join=True)
    res = [json.load(open(tmp_path / f"rank{r}.json")) for r in range(world)]
    # both ranks agree on the slowest rank's time and on the aggregate
    assert res[0]["worst"] == res[1]["worst"] == 5.0
    assert res[0]["value"] == res[1]["value"] == pytest.approx(2 * 10 / 5.0e-3)
    # the shards are different batches of sequences
    assert not np.array_equal(np.array(res[0]["tokens"]), np.array(res[1]["tokens"]))


def test_single_rank_needs_no_process_group(monkeypatch):
    sys.path.insert(0, ROOT)
    import bench
    for k in ("WORLD_SIZE", "RANK", "LOCAL_RANK"):
        monkeypatch.delenv(k, raising=False)
    ws, r, local = bench.dist_init()
    assert (ws, r, local) == (1, 0, 0)
    assert bench.max_over_ranks(4.5, 1) == 4.5
    assert bench.steps_per_second(1, 256, 23.04) == pytest.approx(256 / 0.02304)
    assert bench.shard_seed(1005, 0) == 1005 and bench.shard_seed(1005, 1) != 1005
