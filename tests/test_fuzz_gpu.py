"""Seeded random shapes through the one-call step against the oracle: T from
1 to 400,000, E a multiple of 8 up to 1024, K up to min(E-1, 15), ragged and
empty microbatches (sometimes more microbatches than the LEI coefficient table
holds, which runs LEI as its own pass), random eta and c (c <= 0 is
unnormalised LEI), logits of mixed scales with ties.  Routing, loads, the next
bias bit for bit; LEI within |d| <= 1e-7 + 1e-5 |g_ref|."""
import numpy as np
import pytest
import torch

import brute
import oracle
import paper_2609_28053_gb300 as eqb
from eqb_workloads import ragged_offsets
from gpu_harness import Guarded, bits_f32, oracle_forward, to_dev_bf16

pytestmark = pytest.mark.gpu

LEI_ATOL, LEI_RTOL = 1e-7, 1e-5


@pytest.fixture(scope="module", autouse=True)
def _lib(cuda_ok):
    eqb.load()


def draw_case(seed):
    rng = np.random.default_rng(10_000 + seed)
    E = int(rng.choice([8, 16, 24, 64, 128, 136, 256, 264, 512, 1024]))
    K = int(rng.integers(1, min(E - 1, 15) + 1))
    kindT = rng.integers(0, 4)
    if kindT == 0:  # smaller than a warp round, a histogram block or a LEI chunk
        T = int(rng.choice([1, 2, 31, 33, 257]))
    elif kindT == 3 and E <= 256:  # several histogram flush intervals per block
        T = int(rng.integers(100_000, 400_000))
    else:
        T = int(rng.integers(1, 40_000))
    if E >= 512:
        T = min(T, 6000)
    M = int(rng.choice([1, 2, 3, 7, 64, 300]))
    M = max(1, min(M, T)) if T > 1 else 1
    kind = rng.integers(0, 3)
    if kind == 0:  # plain normal logits
        v = rng.standard_normal((T, E))
    elif kind == 1:  # coarse grid: many exact ties
        v = rng.integers(-3, 4, size=(T, E)) * 0.5
    else:  # per-expert offsets, small spread (tie-heavy config shape)
        v = 0.05 * rng.standard_normal((T, E)) + rng.normal(0, 0.5, E)
    z = brute.bf16_bits_from_f32(v.astype(np.float32))
    b = (rng.standard_normal(E) * float(rng.choice([0.0, 0.1, 0.5]))).astype(np.float32)
    off = ragged_offsets(T, M, seed=seed)
    eta = float(rng.choice([2e-5, 0.25, 1.0]))
    c = float(rng.choice([0.0, 0.5, 1.0, 4.0]))
    return T, E, K, M, z, b, off, eta, c


@pytest.mark.parametrize("seed", range(100))
def test_random_layer_step(seed):
    T, E, K, M, z, b, off, eta, c = draw_case(seed)
    rng = np.random.default_rng(seed)
    g = (rng.standard_normal((T, E)) * 0.1).astype(np.float32)
    o = oracle_forward(z, b, K, off)
    g_ref, _ = oracle.lei(g, o["loads"], off, K, eta, c)

    idx = Guarded((T, K), torch.int32)
    tau = Guarded((T,), torch.float32)
    loads = Guarded((M, E), torch.int32, fill=3)
    bn = Guarded((E,), torch.float32)
    G = Guarded((T, E), torch.float32)
    G.view.copy_(torch.from_numpy(g))
    ws = torch.zeros(eqb.eqb_layer_workspace_bytes(E), dtype=torch.uint8, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    eqb.eqb_layer_step(to_dev_bf16(z), torch.from_numpy(b).cuda(), K, torch.from_numpy(off).cuda(), loads.view,
                       bn.view, ws, tau=tau.view, topk_idx=idx.view, grad_s=G.view, eta=eta, c=c,
                       mb_offsets_host=off, err_flag=err)
    torch.cuda.synchronize()
    for buf in (idx, tau, loads, bn, G):
        assert buf.intact()
    assert err.item() == 0
    assert np.array_equal(idx.view.cpu().numpy(), o["idx"])
    assert np.array_equal(bits_f32(tau.view.cpu().numpy()), bits_f32(o["tau"]))
    assert np.array_equal(loads.view.cpu().numpy(), o["loads"])
    assert np.array_equal(bits_f32(bn.view.cpu().numpy()), bits_f32(o["b_next"]))
    got = G.view.cpu().numpy().astype(np.float64)
    assert np.all(np.abs(got - g_ref) <= LEI_ATOL + LEI_RTOL * np.abs(g_ref))
