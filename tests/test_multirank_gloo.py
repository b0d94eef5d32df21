"""The N > 1 path on CPU: two gloo ranks run the host logic bench.py uses
under torchrun (per-rank inputs, barrier, slowest-rank timing, whole-job
throughput); heads are independent, so the only collective is the timing
reduction. CPU only."""
import json
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2607_20214_gb300 import multirank
from paper_2607_20214_gb300.workloads import Workload, make_inputs


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out_dir):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        wl = Workload(name="tiny", B=1, H=2, N=128, d_h=32, dtype="fp32",
                      block=32, race_tables=2, recipe="plain",
                      temperature=1.0, seed=3, plane_seed=1003)
        wl_r = multirank.rank_workload(wl, rank)
        x = make_inputs(wl_r)
        multirank.barrier()
        # each rank's "step time": the job waits for the slowest rank
        slowest = multirank.max_over_ranks(10.0 + rank)
        tput = multirank.job_throughput(multirank.world_size(), wl.tokens,
                                        slowest)
        # per-rank work is independent: each rank's own oracle output
        from oracle import oracle as orc
        p = orc.params_from_workload(wl_r)
        r = orc.forward(x, p, heads=[(0, 0)], threads=1)[(0, 0)]
        rec = {"rank": rank, "seed": wl_r.seed,
               "q_sum": float(x["q"].double().sum()),
               "slowest": slowest, "tput": tput,
               "o_sum": float(np.asarray(r["O"]).sum()),
               "world": multirank.world_size()}
        with open(os.path.join(out_dir, "rank%d.json" % rank), "w") as f:
            json.dump(rec, f)
        multirank.barrier()
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks(tmp_path):
    world = 2
    mp.spawn(_rank_main, args=(world, _free_port(), str(tmp_path)),
             nprocs=world, join=True)
    recs = [json.load(open(tmp_path / ("rank%d.json" % r)))
            for r in range(world)]
    assert [r["world"] for r in recs] == [2, 2]
    # distinct inputs per rank, independent results
    assert recs[0]["seed"] != recs[1]["seed"]
    assert recs[0]["q_sum"] != recs[1]["q_sum"]
    assert recs[0]["o_sum"] != recs[1]["o_sum"]
    # the slowest rank's time, seen by every rank
    assert recs[0]["slowest"] == recs[1]["slowest"] == 11.0
    tokens = 1 * 128  # B * N (tokens, not heads x tokens)
    assert recs[0]["tput"] == pytest.approx(2 * tokens / 11.0e-3)


def test_single_process_helpers_are_identity():
    assert multirank.world_size() == 1
    assert multirank.max_over_ranks(3.5) == 3.5
    assert multirank.job_throughput(1, 1000, 2.0) == pytest.approx(5e5)
