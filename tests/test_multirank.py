"""The multi-process path of bench.py on CPU (gloo, world size 2).

The path shards by sequences with no data-path collective (replicas): each
rank embeds its own sub-streams of the query stream, and the only
collectives are the timing barrier and the max over ranks of the step time.
These tests run the ranks as processes on the CPU.
"""

import json
import os
import socket
import subprocess
import sys

import numpy as np
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out_dir):
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank),
                      MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    sys.path.insert(0, ROOT)
    import bench
    import synth
    import torch.distributed as dist

    w_, r_, l_ = bench.dist_setup()
    assert (w_, r_) == (world, rank)
    bench.barrier(world)
    m = bench.max_over_ranks(10.0 * rank + 1.0, world)
    w = synth.WORKLOADS["tiny"]
    seqs = [list(range((rank * bench.N_BATCHES + k) * w.B, (rank * bench.N_BATCHES + k + 1) * w.B))
            for k in range(bench.N_BATCHES)]
    first = synth.query_tokens(w, range(seqs[0][0], seqs[0][-1] + 1))
    np.save(os.path.join(out_dir, f"rank{rank}.npy"), first)
    with open(os.path.join(out_dir, f"rank{rank}.json"), "w") as f:
        json.dump({"max": m, "seqs": sorted(s for b in seqs for s in b)}, f)
    dist.destroy_process_group()


def test_two_ranks_barrier_max_and_disjoint_sequences(tmp_path):
    port = free_port()
    mp.start_processes(_rank_main, args=(2, port, str(tmp_path)), nprocs=2, start_method="spawn")
    r0 = json.load(open(tmp_path / "rank0.json"))
    r1 = json.load(open(tmp_path / "rank1.json"))
    assert r0["max"] == r1["max"] == 11.0
    assert not set(r0["seqs"]) & set(r1["seqs"])          # weak scaling: own sequences
    a, b = np.load(tmp_path / "rank0.npy"), np.load(tmp_path / "rank1.npy")
    assert a.shape == b.shape and not np.array_equal(a, b)


def test_reference_arm_under_torchrun_prints_once():
    port = free_port()
    r = subprocess.run([sys.executable, "-m", "torch.distributed.run", "--nnodes=1",
                        "--nproc-per-node", "2", "--master-addr", "127.0.0.1", "--master-port",
                        str(port), "bench.py", "--impl", "reference", "--workload", "tiny",
                        "--gpus", "2", "--steps", "2", "--warmup", "3"],
                       cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["value"] > 0 and d["cpu_baseline"]["kind"] == "oracle"
