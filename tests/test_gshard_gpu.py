"""GShard auxiliary-loss gradient (App. D, Eq. gshard-grad) on the GPU
against the oracle's fp64 evaluation.

Tolerance, derived from the kernel's fp32 arithmetic: sigmoid through expf
(a few ulp), sums of E terms for d_t and for sum_e s_e R_e (at most (E+4)
rounding errors of 2^-24 relative to the sum of magnitudes), two divisions,
R_j and alpha/n rounded from fp64, one product and the final add.  With
scale_t = alpha / (n_l d_t) this gives
  |g - g_ref| <= 2^-23 |g_ref| + 1e-12 + scale_t (4E + 32) 2^-24 (max_e |R_e| + |R_j - m_t|),
m_t = sum_e p_e R_e."""
import numpy as np
import pytest
import torch

import brute
import oracle
import paper_2609_28053_gb300 as eqb
from eqb_workloads import ragged_offsets
from gpu_harness import Guarded, to_dev_bf16

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib(cuda_ok):
    eqb.load()


def bound(z_bits, loads, off, K, alpha, g_ref):
    T, E = z_bits.shape
    s = 1.0 / (1.0 + np.exp(-brute.f32_from_bf16_bits(z_bits).astype(np.float64)))
    d = s.sum(1)
    n = np.diff(off)
    mb = np.searchsorted(off, np.arange(T), side="right") - 1
    R = loads / (K * np.maximum(n, 1))[:, None] - 1.0 / E
    Rt = R[mb]
    m = (s / d[:, None] * Rt).sum(1)
    scale = alpha / (n[mb] * d)
    return (2.0 ** -23 * np.abs(g_ref) + 1e-12
            + (scale * (4 * E + 32) * 2.0 ** -24)[:, None] * (np.abs(Rt).max(1)[:, None] + np.abs(Rt - m[:, None])))


@pytest.mark.parametrize("T,E,K,M", [(1, 8, 2, 1), (1000, 64, 8, 5), (777, 24, 3, 3), (4099, 256, 8, 7),
                                     (3000, 128, 6, 4), (500, 40, 4, 2), (777, 512, 8, 3), (300, 1024, 6, 2),
                                     (400, 264, 4, 2)])
@pytest.mark.parametrize("alpha", [1e-2, 3.0])
def test_gshard_matches_oracle(T, E, K, M, alpha):
    rng = np.random.default_rng(T + E + K)
    z = brute.bf16_bits_from_f32((rng.standard_normal((T, E)) + np.linspace(-1, 1, E)).astype(np.float32))
    off = ragged_offsets(T, M, seed=T) if M > 1 else np.array([0, T], np.int64)
    if M > 2:
        off[2] = off[1]
    _, _, loads = oracle.route(z, np.zeros(E, np.float32), K, off)
    g = (0.1 * rng.standard_normal((T, E))).astype(np.float32)
    want = oracle.gshard(g, z, loads, off, K, alpha)
    G = Guarded((T, E), torch.float32)
    G.view.copy_(torch.from_numpy(g))
    eqb.gshard_inject_grad(G.view, to_dev_bf16(z), torch.from_numpy(loads).cuda(), torch.from_numpy(off).cuda(),
                           K, alpha)
    torch.cuda.synchronize()
    assert G.intact()
    got = G.view.cpu().numpy().astype(np.float64)
    tol = bound(z, loads, off, K, alpha, want.astype(np.float64))
    err = np.abs(got - want)
    assert np.all(err <= tol), f"max excess {np.max(err - tol)}"
    assert np.any(got != g)  # the term is not lost


def test_gshard_balanced_loads_leave_gradient_unchanged():
    T, E, K = 512, 64, 8
    rng = np.random.default_rng(1)
    z = brute.bf16_bits_from_f32(rng.standard_normal((T, E)).astype(np.float32))
    off = np.array([0, 256, 512], np.int64)
    loads = np.full((2, E), K * 256 // E, np.int32)
    g = (0.1 * rng.standard_normal((T, E))).astype(np.float32)
    gd = torch.from_numpy(g).cuda()
    eqb.gshard_inject_grad(gd, to_dev_bf16(z), torch.from_numpy(loads).cuda(), torch.from_numpy(off).cuda(), K, 5.0)
    torch.cuda.synchronize()
    assert torch.equal(gd.cpu(), torch.from_numpy(g))
