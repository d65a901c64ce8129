"""Host logic of bench.py's multi-GPU mode, on two gloo ranks on the CPU.

The path shards by independent units (streams / layers / KV heads), so N GPUs
run N replicas with no data-path collective; the only cross-rank operations
are a barrier and the max-over-ranks of the timed region.
"""
import json
import os
import subprocess
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import bench

    w, r, local = bench.dist_setup()
    assert (w, r, local) == (world, rank, rank)
    assert dist.get_backend() == "gloo"
    bench.barrier(w)
    t = bench.max_over_ranks(10.0 + rank, w, torch.device("cpu"))
    q.put((rank, t))
    dist.destroy_process_group()


def _free_port():
    import socket

    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


@pytest.mark.skipif(torch.cuda.is_available(), reason="exercises the CPU (gloo) path")
def test_two_ranks_agree_on_the_max_time():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    got = dict(q.get(timeout=10) for _ in range(2))
    assert got == {0: 11.0, 1: 11.0}


@pytest.mark.skipif(torch.cuda.is_available(), reason="exercises the CPU (gloo) path")
def test_reference_arm_prints_once_under_two_ranks():
    """--impl reference under torchrun: rank 0 times the oracle and prints one
    JSON line; rank 1 exits 0 without work."""
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node=2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), "bench.py",
           "--impl", "reference", "--gpus", "2", "--steps", "3", "--warmup", "3",
           "--workload", "toy"]
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["value"] > 0 and line["n_gpus"] == 2
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["cpu_baseline"]["kind"] == "oracle"


def test_workload_of_the_bench_is_the_7b_stack():
    sys.path.insert(0, ROOT)
    import bench
    from paper_2605_31598_gb300.inputs import WORKLOADS

    assert bench.DEFAULT_WORKLOAD == "qwen7b_stack"
    s = WORKLOADS[bench.DEFAULT_WORKLOAD]
    assert (s.num_layers, s.num_q_heads, s.num_kv_heads, s.head_dim, s.tokens_per_frame,
            s.state_capacity, s.max_frames) == (28, 28, 4, 128, 196, 2048, 256)
    # algorithmic FLOPs of one steady-state layer-frame: 4 d Hq (T B + T (T+1)/2)
    assert abs(bench.attn_flops(s, 2048) - 6.031e9) / 6.031e9 < 1e-3
