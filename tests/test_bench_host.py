"""Host logic of bench.py: algorithmic work counts and the multi-rank timing
reduction (two gloo ranks on the CPU stand in for two GPUs)."""
import os
import socket

import pytest
import torch
import torch.multiprocessing as mp

import bench
from paper_2608_02032_gb300.workloads import WORKLOADS, Workload


def test_sma_pair_and_flop_counts_of_the_l16k_workload():
    w = WORKLOADS["prefill_l16k"]
    # token t sees t // S memories: 1 x 32 heads x 256 tokens x (0 + 1 + ... + 63)
    assert bench.sma_pairs(w) == 32 * 256 * (64 * 63 // 2) == 16_515_072
    assert bench.sma_flops(w) == pytest.approx(16_515_072 * 4 * 128 * 64)
    # brute-force pair count on a small case
    s = Workload("s", 2, 3, 40, 8, 4, 8)
    assert bench.sma_pairs(s) == sum((t // 8) for _ in range(2 * 3) for t in range(40))


def test_decode_bytes_of_the_b64_workload():
    w = WORKLOADS["decode_b64"]
    n = bench.decode_bytes(w, w.mem + 1)
    cache = 64 * 64 * 32 * 128 * 64 * 2  # 2 GiB of bf16 memories
    state = 2 * 64 * 32 * 128 * 64 * 4   # state read + write
    part = 64 * 32 * 128 * 64 * 4        # partial written (chunk start: not read)
    assert cache == 2 ** 31
    assert cache + state + part < n < cache + state + part + 2 ** 20


def test_scan_bytes_of_the_l16k_workload():
    """The forward scan's algorithmic HBM bytes: bf16 X, B, C and fp32 dt in;
    fp32 Y_ssd, memories and their inverse RMS out (64 chunks)."""
    w = WORKLOADS["prefill_l16k"]
    T = 16384
    reads = T * 32 * 64 * 2 + 2 * T * 128 * 2 + T * 32 * 4
    writes = T * 32 * 64 * 4 + 64 * 32 * 128 * 64 * 4 + 64 * 32 * 128 * 4
    assert bench.scan_bytes(w) == reads + writes
    assert 279e6 < bench.scan_bytes(w) < 281e6


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import torch.distributed as dist

    dist.init_process_group("gloo", rank=rank, world_size=world)
    v = bench.max_over_ranks(1.5 + rank, world, torch.device("cpu"))
    bench.barrier(world)
    out[rank] = v
    dist.destroy_process_group()


def test_max_over_ranks_with_two_gloo_ranks():
    world = 2
    out = mp.Manager().dict()
    mp.spawn(_rank_main, args=(world, _free_port(), out), nprocs=world, join=True)
    assert dict(out) == {0: 2.5, 1: 2.5}


def test_oracle_sample_runs_on_a_tiny_workload():
    from paper_2608_02032_gb300.workloads import prefill_inputs

    w = Workload("tiny", 1, 2, 64, 8, 4, 16, dtype="f32", seed=3)
    secs, threads = bench.oracle_sample(w, prefill_inputs(w), 1)
    assert secs > 0 and threads >= 1
