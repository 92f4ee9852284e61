"""Multi-rank plumbing of the replicas-only multi-GPU mode, on CPU: the
token-balanced sequence split and the host-level reductions, with two gloo
ranks (127.0.0.1)."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2607_14557_gb300 import replicas as R


def test_shard_sequences_covers_disjointly_and_balances():
    rng = np.random.default_rng(0)
    tokens = list(rng.integers(100, 4000, 37))
    for world in (1, 2, 3, 8):
        parts = R.shard_sequences(tokens, world)
        flat = sorted(i for p in parts for i in p)
        assert flat == list(range(len(tokens)))
        loads = [sum(tokens[i] for i in p) for p in parts]
        # greedy longest-first: no rank exceeds the mean by more than the longest sequence
        assert max(loads) - sum(loads) / world <= max(tokens)


def test_shard_sequences_hand_case():
    # longest first onto the least-loaded rank: 9 -> r0, 7 -> r1, 5 -> r1 (7 < 9),
    # 4 -> r0 (9 < 12), 3 -> r1 (12 < 13)
    assert R.shard_sequences([5, 9, 3, 7, 4], 2) == [[1, 4], [0, 2, 3]]


def test_reductions_without_a_group_are_identity():
    assert R.max_over_ranks(3.5) == 3.5
    assert R.sum_over_ranks(2.0) == 2.0
    R.barrier()


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        R.barrier()
        out[rank, 0] = R.max_over_ranks(10.0 + rank)
        out[rank, 1] = R.sum_over_ranks(1000.0 * (rank + 1))
        parts = R.shard_sequences([300, 200, 100, 50], world)
        out[rank, 2] = sum([300, 200, 100, 50][i] for i in parts[rank])
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_reduce_on_the_host():
    world = 2
    out = torch.zeros((world, 3), dtype=torch.float64).share_memory_()
    mp.start_processes(_worker, args=(world, _free_port(), out), nprocs=world, join=True, start_method="spawn")
    assert out[:, 0].tolist() == [11.0, 11.0]
    assert out[:, 1].tolist() == [3000.0, 3000.0]
    assert out[:, 2].tolist() == [350.0, 300.0]    # 300 + 50 on rank 0, 200 + 100 on rank 1
