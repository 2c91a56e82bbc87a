"""The comparison estimates of Sec. 2 on the GPU against the oracle, bit for
bit: rank-averaged QB (per-shard exact quantiles, averaged, centered) and the
fixed-resolution histogram (256 equal bins, upper bin edge, centered)."""
import numpy as np
import pytest
import torch

import brute
import oracle
import paper_2609_28053_gb300 as eqb
from eqb_workloads import bits, make_bias, make_logits, ragged_offsets
from gpu_harness import Guarded, to_dev_bf16

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib(cuda_ok):
    eqb.load()


def case(T, E, K, seed):
    rng = np.random.default_rng(seed)
    z = brute.bf16_bits_from_f32((rng.standard_normal((T, E)) + rng.normal(0, 0.5, E)).astype(np.float32))
    b = (0.1 * rng.standard_normal(E)).astype(np.float32)
    _, tau, _ = oracle.route(z, b, K)  # tau from the oracle, so both sides see the same input
    return z, tau


def workspace(E):
    return torch.zeros(eqb.eqb_layer_workspace_bytes(E), dtype=torch.uint8, device="cuda")


@pytest.mark.parametrize("T,E,K,shards", [(4000, 64, 8, [0, 1000, 1000, 2500, 4000]), (3001, 16, 2, [0, 3001]),
                                          (20000, 256, 8, list(range(0, 20001, 2500))), (5000, 128, 6, [0, 7, 5000]),
                                          (3000, 384, 8, [0, 1500, 3000]),
                                          (70000, 256, 8, [0] + sorted(np.random.default_rng(9).integers(0, 70000, 39).tolist()) + [70000])])
def test_rank_averaged_bias_matches_oracle(T, E, K, shards):
    z, tau = case(T, E, K, seed=T + E)
    want_b, want_q = oracle.rank_averaged_bias(z, tau, K, shards)
    P = len(shards) - 1
    B = Guarded((E,), torch.float32)
    Q = Guarded((P, E), torch.bfloat16, canary=-5.0)
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    ws = torch.zeros(eqb.eqb_rank_averaged_workspace_bytes(E, P), dtype=torch.uint8, device="cuda")
    eqb.eqb_rank_averaged_bias(to_dev_bf16(z), torch.from_numpy(tau).cuda(), K, np.array(shards), ws,
                               b_out=B.view, q_shards=Q.view, err_flag=err)
    torch.cuda.synchronize()
    assert B.intact() and Q.intact() and err.item() == 0
    q = Q.view.view(torch.int16).cpu().numpy().view(np.uint16)
    nonempty = [p for p in range(P) if shards[p + 1] > shards[p]]
    assert np.array_equal(q[nonempty], want_q)
    assert np.all(q[[p for p in range(P) if p not in nonempty]] == 0)
    assert np.array_equal(B.view.cpu().numpy().view(np.uint32), want_b.view(np.uint32))


@pytest.mark.parametrize("T,E,K,lo,width", [(4000, 64, 8, -4.0, 1.0 / 32), (3001, 16, 2, -1.0, 0.01),
                                            (20000, 256, 8, -8.0, 0.0625), (5000, 128, 6, 0.5, 0.1),
                                            (3000, 1024, 8, -6.0, 0.05)])
def test_fixed_hist_bias_matches_oracle(T, E, K, lo, width):
    """Includes ranges that clamp many margins into the edge bins."""
    z, tau = case(T, E, K, seed=T * 3 + E)
    want_b, want_est = oracle.fixed_hist_bias(z, tau, K, lo, width)
    B = Guarded((E,), torch.float32)
    X = Guarded((E,), torch.float64, canary=-5.0)
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    eqb.eqb_fixed_hist_bias(to_dev_bf16(z), torch.from_numpy(tau).cuda(), K, lo, width, workspace(E),
                            b_out=B.view, estimate=X.view, err_flag=err)
    torch.cuda.synchronize()
    assert B.intact() and X.intact() and err.item() == 0
    assert np.array_equal(X.view.cpu().numpy(), want_est)
    assert np.array_equal(B.view.cpu().numpy().view(np.uint32), want_b.view(np.uint32))


def test_partition_invariance_eqb_vs_rank_average():
    """Sec. 3: EQB's bias does not depend on how tokens are sharded, the
    rank-averaged one does (global workload distribution, 65,536 tokens)."""
    T, E, K = 65536, 256, 8
    z = bits(make_logits("global", T=T))
    b = make_bias("global").numpy()
    _, tau, _ = oracle.route(z, b, K)
    zd, td = to_dev_bf16(z), torch.from_numpy(tau).cuda()
    outs = []
    for shards in ([0, T], list(range(0, T + 1, 8192)), [0, 5000, 30000, 30000, T]):
        ws = torch.zeros(eqb.eqb_rank_averaged_workspace_bytes(E, len(shards) - 1), dtype=torch.uint8,
                         device="cuda")
        bq, _ = eqb.eqb_rank_averaged_bias(zd, td, K, np.array(shards), ws)
        outs.append(bq.cpu().numpy())
    torch.cuda.synchronize()
    # one shard is EQB itself
    assert np.array_equal(outs[0], oracle.eqb_step(z, b, K)["b_next"])
    assert not np.array_equal(outs[0], outs[1]) and not np.array_equal(outs[1], outs[2])
