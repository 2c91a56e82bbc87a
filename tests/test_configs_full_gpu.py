"""Full-size parity of two of the five workload configurations as they are
defined, through the library's one-call entry points:

* router: x bf16 [1,048,576, 4096], W_r bf16 [128, 4096], K = 8, 16
  microbatches, three steps with fresh activations and the bias iterated
  from b^(0) = 0 (Eq. 2: b^(q+1) routes step q+1).  Each step runs
  eqb_router_layer_step, projection included; the oracle gets the bytes of
  the z the library wrote (tensor-core accumulation order differs from the
  CPU's, so EQB parity is defined on the GPU's logits) and the GPU's bias of
  the previous step, which the bit-for-bit check of that step equates with
  its own.  Routing, loads and b^(q+1) bit for bit, 4,096 sampled gradient
  rows within the LEI tolerance.
* mid: T = 524,288, E = 128, K = 8, 32 microbatches of 16,384 tokens, 16 hot
  experts, the bias from one update on an independent prior batch, LEI on
  the configuration's own gradients: routing, loads and the next bias bit for
  bit, every gradient row within the LEI tolerance."""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_28053_gb300 as eqb
from eqb_workloads import (SHAPES, bits, even_offsets, make_grad, make_logits, make_router_inputs,
                           prior_batch_logits)
from gpu_harness import bits_f32, oracle_forward

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

LEI_ATOL, LEI_RTOL = 1e-7, 1e-5


@pytest.fixture(scope="module", autouse=True)
def _lib(cuda_ok):
    eqb.load()


def test_router_config_three_steps_on_library_logits():
    sh = SHAPES["router"]
    T, E, K, M = sh.T, sh.E, sh.K, sh.M
    eta, c = 2e-5, 1.0
    off = even_offsets(T, M)
    offd = torch.from_numpy(off).cuda()
    rows = np.sort(np.random.default_rng(11).choice(T, 4096, replace=False))
    rows_d = torch.from_numpy(rows).cuda()
    mb = np.searchsorted(off, rows, side="right") - 1
    b = torch.zeros(E, dtype=torch.float32, device="cuda")
    ws = torch.zeros(eqb.eqb_layer_workspace_bytes(E), dtype=torch.uint8, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    z = torch.empty((T, E), dtype=torch.bfloat16, device="cuda")
    idx = torch.empty((T, K), dtype=torch.int32, device="cuda")
    tau = torch.empty(T, dtype=torch.float32, device="cuda")
    loads = torch.zeros((M, E), dtype=torch.int32, device="cuda")
    bn = torch.empty(E, dtype=torch.float32, device="cuda")
    for step in range(3):
        x, W = make_router_inputs(T=T, step=step, device="cuda")
        G = make_grad("router", T=T, seed=SHAPES["router"].seed + 7 * step, device="cuda")
        g_rows = G[rows_d].cpu().numpy()
        b_host = b.cpu().numpy()
        eqb.eqb_router_layer_step(x, W, b, K, offd, loads, bn, ws, z=z, tau=tau, topk_idx=idx, grad_s=G,
                                  eta=eta, c=c, mb_offsets_host=off, err_flag=err)
        torch.cuda.synchronize()
        assert err.item() == 0, f"step {step}"
        del x
        o = oracle_forward(bits(z), b_host, K, off, experts=np.arange(E))
        assert np.array_equal(idx.cpu().numpy(), o["idx"]), f"step {step}"
        assert np.array_equal(bits_f32(tau.cpu().numpy()), bits_f32(o["tau"])), f"step {step}"
        assert np.array_equal(loads.cpu().numpy(), o["loads"]), f"step {step}"
        assert np.array_equal(bits_f32(bn.cpu().numpy()), bits_f32(oracle.bias_update(o["q"]))), f"step {step}"
        _, a = oracle.lei(None, o["loads"], off, K, eta, c)
        want = g_rows.astype(np.float64) + a[mb]
        got = G[rows_d].cpu().numpy().astype(np.float64)
        assert np.all(np.abs(got - want) <= LEI_ATOL + LEI_RTOL * np.abs(want)), f"step {step}"
        del G
        b.copy_(bn)  # b^(q+1) routes step q+1


def test_mid_config_step_with_lei():
    name = "mid"
    sh = SHAPES[name]
    T, E, K, M = sh.T, sh.E, sh.K, sh.M
    eta, c = 0.25, 1.0
    zt = make_logits(name, device="cuda")
    z = bits(zt)
    b = oracle.eqb_step(bits(prior_batch_logits(name)), np.zeros(E, np.float32), K)["b_next"]
    off = even_offsets(T, M)
    g = make_grad(name).numpy()
    G = torch.from_numpy(g).cuda()
    idx = torch.empty((T, K), dtype=torch.int32, device="cuda")
    tau = torch.empty(T, dtype=torch.float32, device="cuda")
    loads = torch.zeros((M, E), dtype=torch.int32, device="cuda")
    bn = torch.empty(E, dtype=torch.float32, device="cuda")
    ws = torch.zeros(eqb.eqb_layer_workspace_bytes(E), dtype=torch.uint8, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    eqb.eqb_layer_step(zt, torch.from_numpy(b).cuda(), K, torch.from_numpy(off).cuda(), loads, bn, ws, tau=tau,
                       topk_idx=idx, grad_s=G, eta=eta, c=c, mb_offsets_host=off, err_flag=err)
    torch.cuda.synchronize()
    assert err.item() == 0
    o = oracle_forward(z, b, K, off)
    assert np.array_equal(idx.cpu().numpy(), o["idx"])
    assert np.array_equal(bits_f32(tau.cpu().numpy()), bits_f32(o["tau"]))
    assert np.array_equal(loads.cpu().numpy(), o["loads"])
    assert np.array_equal(bits_f32(bn.cpu().numpy()), bits_f32(o["b_next"]))
    g_ref, _ = oracle.lei(g, o["loads"], off, K, eta, c)
    got = G.cpu().numpy().astype(np.float64)
    assert np.all(np.abs(got - g_ref) <= LEI_ATOL + LEI_RTOL * np.abs(g_ref))
