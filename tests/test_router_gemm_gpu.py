"""Router logits on the tensor cores (Sec. 2, z_t = W_r x_t) against the
oracle's fp64 dot products.

Tolerance, derived from the arithmetic: the kernel forms each product of two
bf16 values exactly, accumulates d of them in fp32 (error at most
d * 2^-24 * sum_k |x_k w_k|) and rounds once to bf16 (at most half a bf16
ulp).  So |z - z_exact| <= ulp_bf16/2 + d * 2^-24 * S, S = sum_k |x_k w_k|.
Most entries must equal the exactly rounded value."""
import numpy as np
import pytest
import torch

import brute
import oracle
import paper_2609_28053_gb300 as eqb
from eqb_workloads import SHAPES, make_router_inputs
from gpu_harness import Guarded, to_dev_bf16

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib(cuda_ok):
    eqb.load()


def ulp_bf16(v):
    a = np.abs(v).astype(np.float64)
    e = np.floor(np.log2(np.maximum(a, 2.0 ** -126)))
    return 2.0 ** (e - 7)


def check_rows(z_gpu_bits, x_bits, W_bits, rows):
    d = x_bits.shape[1]
    ref, S = oracle.router_logits(x_bits, W_bits, rows)
    got = brute.f32_from_bf16_bits(z_gpu_bits[rows]).astype(np.float64)
    tol = 0.5 * ulp_bf16(np.maximum(np.abs(ref), np.abs(got))) + d * 2.0 ** -24 * S
    assert np.all(np.abs(got - ref) <= tol), f"max excess {np.max(np.abs(got - ref) - tol)}"
    exact = brute.bf16_bits_from_f32(ref.astype(np.float32))
    agree = np.mean(exact == z_gpu_bits[rows])
    assert agree > 0.95, f"only {agree:.3f} of entries equal the exactly rounded value"
    return agree


@pytest.mark.parametrize("T,d,E", [(1, 64, 16), (127, 64, 128), (128, 128, 64), (129, 4096, 128),
                                   (1000, 256, 256), (4099, 512, 128), (300, 4096, 16), (70000, 128, 128)])
def test_router_logits_matches_oracle(T, d, E):
    rng = np.random.default_rng(T + d + E)
    x = brute.bf16_bits_from_f32(rng.standard_normal((T, d)).astype(np.float32))
    W = brute.bf16_bits_from_f32((rng.standard_normal((E, d)) / np.sqrt(d)).astype(np.float32))
    Z = Guarded((T, E), torch.bfloat16, canary=-7.0)
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    eqb.eqb_router_logits(to_dev_bf16(x), to_dev_bf16(W), Z.view, err)
    torch.cuda.synchronize()
    assert Z.intact() and err.item() == 0
    zb = Z.view.view(torch.int16).cpu().numpy().view(np.uint16)
    rows = np.arange(T) if T <= 1024 else np.sort(rng.choice(T, 1024, replace=False))
    check_rows(zb, x, W, rows)


def test_router_logits_full_size_sampled():
    """Router configuration: T = 1,048,576, d = 4096, E = 128, sampled rows
    (including the first and the last tile)."""
    sh = SHAPES["router"]
    x, W = make_router_inputs(device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    z = eqb.eqb_router_logits(x, W, err_flag=err)
    torch.cuda.synchronize()
    assert err.item() == 0
    rng = np.random.default_rng(4)
    rows = np.unique(np.concatenate([np.arange(128), np.arange(sh.T - 128, sh.T),
                                     rng.choice(sh.T, 768, replace=False)]))
    xb = x[torch.from_numpy(rows).cuda()].view(torch.int16).cpu().numpy().view(np.uint16)
    Wb = W.view(torch.int16).cpu().numpy().view(np.uint16)
    zb = z[torch.from_numpy(rows).cuda()].view(torch.int16).cpu().numpy().view(np.uint16)
    check_rows(zb, xb, Wb, np.arange(len(rows)))


def test_router_logits_repeatable():
    """Two calls give identical bits (fixed accumulation order)."""
    x, W = make_router_inputs(T=5000, device="cuda")
    a = eqb.eqb_router_logits(x, W)
    b = eqb.eqb_router_logits(x, W)
    torch.cuda.synchronize()
    assert torch.equal(a.view(torch.int16), b.view(torch.int16))
