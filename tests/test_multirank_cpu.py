"""Multi-rank host logic on the CPU (gloo, world size 2).

Algorithm 1 of the paper exchanges exactly two things between data-parallel
ranks: the summed [E,256] high-byte counts (step 2) and the summed low-byte
counts inside the selected bins (step 5).  These tests shard a batch across
two processes the way bench.py does under torchrun (contiguous token ranges,
global target rank), all-reduce the per-rank counts with torch.distributed,
and check that both ranks recover the single-process quantile and bias.
The sums go through bench.py's own all-reduce helper.  The per-rank counts
come from the oracle (no GPU here)."""
import os
import socket
import sys

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def shard_bounds(T, world, rank):
    """Contiguous shard of T tokens for `rank` (sizes differ by at most one)."""
    return (T * rank) // world, (T * (rank + 1)) // world


def _worker(rank, world, port, T, E, K, seed, out_q):
    sys.path.insert(0, ROOT)
    sys.path.insert(0, os.path.join(ROOT, "tests"))
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import brute
        import oracle
        from bench import allreduce_
        rng = np.random.default_rng(seed)
        z = brute.bf16_bits_from_f32(rng.standard_normal((T, E)).astype(np.float32))
        b = (rng.standard_normal(E) * 0.2).astype(np.float32)
        a, c = shard_bounds(T, world, rank)
        zl = z[a:c]
        _, tau, _ = oracle.route(zl, b, K)
        r = oracle.target_rank(T, E, K)          # global rank, as in Algorithm 1
        H = torch.from_numpy(oracle.hist_hi(zl, tau))
        allreduce_(H)                             # step 2
        u, rho = oracle.select_hi(H.numpy(), r)   # step 3
        L = torch.from_numpy(oracle.hist_lo(zl, tau, u))
        allreduce_(L)                             # step 5
        q = oracle.select_lo(L.numpy(), u, rho)   # steps 5-6
        out_q.put((rank, q.tolist(), oracle.bias_update(q).view(np.uint32).tolist()))
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("T", [4000, 4001])
def test_two_rank_histogram_allreduce_recovers_global_quantile(T):
    sys.path.insert(0, os.path.join(ROOT, "tests"))
    import brute
    import oracle
    E, K, seed, world = 16, 3, 11, 2
    ctx = mp.get_context("spawn")
    q_out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, T, E, K, seed, q_out))
             for r in range(world)]
    for p in procs:
        p.start()
    res = [q_out.get(timeout=300) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    rng = np.random.default_rng(seed)
    z = brute.bf16_bits_from_f32(rng.standard_normal((T, E)).astype(np.float32))
    b = (rng.standard_normal(E) * 0.2).astype(np.float32)
    ref = oracle.eqb_step(z, b, K)
    for rank, q, bn in res:
        assert q == ref["qhat"].tolist(), f"rank {rank} quantile differs"
        assert bn == ref["b_next"].view(np.uint32).tolist()


def test_shard_bounds_cover_batch():
    for T in (1, 7, 4096, 65537):
        for world in (1, 2, 3, 8):
            spans = [shard_bounds(T, world, r) for r in range(world)]
            assert spans[0][0] == 0 and spans[-1][1] == T
            assert all(spans[i][1] == spans[i + 1][0] for i in range(world - 1))
