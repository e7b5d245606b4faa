"""Host logic of the multi-rank benchmark on CPU: two gloo ranks (no GPU).

bench.py under torchrun runs one rank per GPU, each on its own batch of independent
sequences (heads and sequences never interact), with collectives only on timings: a
barrier around the timed region and a max over ranks of the step time.  These tests run
that logic as two CPU processes with the gloo backend."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out_dir):
    os.environ.update({"MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port), "RANK": str(rank),
                       "WORLD_SIZE": str(world), "LOCAL_RANK": str(rank)})
    import bench
    from paper_2609_36529_gb300 import inputs
    torch.distributed.init_process_group("gloo", rank=rank, world_size=world)
    ws_n, r, local = bench.dist_env()
    barrier, max_over_ranks = bench.rank_ops(ws_n, torch.device("cpu"))
    barrier()
    slowest = max_over_ranks(10.0 + rank)          # each rank reports its own step time
    # each rank draws its own sequences (seed = rank): no data is exchanged by the benchmark,
    # so compare a checksum here only to show the batches differ
    x = inputs.chunk_inputs(1, 65, 2, 16, 16, 2, dtype="bf16", with_beta=True, backward=True,
                            device="cpu", seed=r)
    mine = torch.tensor([float(x["q"].float().sum()), float(x["v"].float().sum())], dtype=torch.float64)
    every = [torch.zeros_like(mine) for _ in range(world)]
    torch.distributed.all_gather(every, mine)
    res = {"env": [ws_n, r, local], "slowest": slowest,
           "value": bench.job_tokens_per_s(ws_n, 65536, slowest),
           "sums": [t.tolist() for t in every]}
    with open(os.path.join(out_dir, f"rank{rank}.json"), "w") as f:
        json.dump(res, f)
    barrier()
    torch.distributed.destroy_process_group()


def test_two_gloo_ranks_timing_and_independent_batches(tmp_path):
    port = _free_port()
    mp.start_processes(_rank_main, args=(2, port, str(tmp_path)), nprocs=2, join=True,
                       start_method="spawn")
    res = [json.load(open(tmp_path / f"rank{r}.json")) for r in range(2)]
    for r, x in enumerate(res):
        assert x["env"] == [2, r, r]
        assert x["slowest"] == 11.0                   # the max over ranks, seen by both
        assert x["value"] == pytest.approx(2 * 65536 / 0.011)   # whole-job tokens/s
    assert res[0]["sums"] == res[1]["sums"]           # both ranks see the same gathered list
    assert res[0]["sums"][0] != res[0]["sums"][1]     # and the two ranks' batches differ


def test_reference_arm_prints_on_rank_zero_only(tmp_path):
    """Under torchrun only rank 0 runs and prints the reference arm's line; the others exit 0."""
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1", MASTER_ADDR="127.0.0.1",
               MASTER_PORT=str(_free_port()))
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--gpus", "2", "--steps", "1", "--warmup", "0", "--ref-tokens", "64"],
                       env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    assert r.stdout.strip() == ""
