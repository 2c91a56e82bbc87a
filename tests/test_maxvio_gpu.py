"""MaxVio (Sec. 5 metrics, App. E) on the GPU against the oracle, bit for bit
(both evaluate the same fp64 expressions in the same order)."""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_28053_gb300 as eqb
from eqb_workloads import ragged_offsets
from gpu_harness import Guarded

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib(cuda_ok):
    eqb.load()


def run(loads, off, K):
    M, E = loads.shape
    out = Guarded((2,), torch.float64, canary=-9.0)
    per = Guarded((M,), torch.float64, canary=-9.0)
    eqb.eqb_maxvio(torch.from_numpy(loads).cuda(), torch.from_numpy(off).cuda(), K, out=out.view,
                   per_mb=per.view)
    torch.cuda.synchronize()
    assert out.intact() and per.intact()
    return out.view.cpu().numpy(), per.view.cpu().numpy()


@pytest.mark.parametrize("M,E,K,T", [(1, 8, 2, 100), (5, 64, 8, 1000), (64, 256, 8, 2097152),
                                     (7, 40, 31, 333), (8000, 16, 2, 64000)])
def test_maxvio_matches_oracle(M, E, K, T):
    rng = np.random.default_rng(M + E + K)
    off = ragged_offsets(T, M, seed=M) if M > 1 else np.array([0, T], np.int64)
    if M > 2:
        off[2] = off[1]  # an empty microbatch
    loads = np.zeros((M, E), np.int32)
    n = np.diff(off)
    for l in range(M):
        # K * n_l selections spread over the experts with a random skew
        p = rng.dirichlet(np.ones(E) * 0.5)
        loads[l] = rng.multinomial(K * int(n[l]), p)
    (g, loc), per = run(loads, off, K)
    wg, wl, wper = oracle.maxvio(loads, off, K)
    assert g == wg and loc == wl
    assert np.array_equal(per, wper)


def test_maxvio_of_routed_loads():
    """MaxVio of the loads the routing kernel counted on a skewed batch
    equals the oracle's MaxVio of the oracle's loads."""
    from gpu_harness import gpu_forward
    rng = np.random.default_rng(3)
    T, E, K = 20000, 64, 6
    z = (rng.standard_normal((T, E)) + np.linspace(0, 2, E)).astype(np.float32)
    import brute
    zb = brute.bf16_bits_from_f32(z)
    b = np.zeros(E, np.float32)
    off = ragged_offsets(T, 6, seed=1)
    gf = gpu_forward(zb, b, K, off)
    _, _, loads_or = oracle.route(zb, b, K, off)
    (g, loc), _ = run(gf["loads"], off, K)
    wg, wl, _ = oracle.maxvio(loads_or, off, K)
    assert g == wg and loc == wl
    assert g > 0.5  # the skew is visible
