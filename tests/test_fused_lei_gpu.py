"""GPU parity of the LEI coefficient table (lei_coefficients) and of the
histogram passes that stream the injection beside their counting
(eqb_margin_hist_lei), against the oracle: histograms bit-exact, injected
gradients within |d| <= 1e-7 + 1e-5 |g_ref| on the requested token range and
bit-identical (untouched) outside it; the one-call step both with the fused
passes and with the coefficient table too large for them."""
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


def case(T, E, K, M, seed):
    rng = np.random.default_rng(seed)
    z = brute.bf16_bits_from_f32(rng.standard_normal((T, E)).astype(np.float32))
    b = (rng.standard_normal(E) * 0.3).astype(np.float32)
    off = ragged_offsets(T, M, seed=seed)
    if M >= 3:
        off[1] = off[2]  # an empty microbatch
    _, tau, loads = oracle.route(z, b, K, off)
    g = (rng.standard_normal((T, E)) * 0.1).astype(np.float32)
    return z, off, tau, loads, g


def within(got, want):
    got = np.asarray(got, np.float64)
    return bool(np.all(np.abs(got - want) <= LEI_ATOL + LEI_RTOL * np.abs(want)))


@pytest.mark.parametrize("M,E,K", [(1, 8, 2), (5, 64, 8), (64, 256, 8), (3, 1024, 8), (7, 24, 3)])
@pytest.mark.parametrize("eta,c", [(1.0, 0.5), (2e-5, 1.0), (0.02, 0.0)])
def test_lei_coefficients_match_oracle(M, E, K, eta, c):
    T = max(37 * M, 200)
    z, off, tau, loads, g = case(T, E, K, M, seed=M + E)
    _, a = oracle.lei(None, loads, off, K, eta, c)
    C = Guarded((M, E), torch.float32, fill=7)
    eqb.lei_coefficients(torch.from_numpy(loads).cuda(), torch.from_numpy(off).cuda(), K, eta, c, coef=C.view)
    torch.cuda.synchronize()
    assert C.intact()
    got = C.view.cpu().numpy()
    assert within(got, a)
    if M >= 3:
        assert np.all(got[1] == 0)  # the empty microbatch


# Shapes covering every expert tiling of the counting kernel (8 experts per
# lane up to 256 per block; 512- and 1024-thread blocks), ragged microbatches.
SHAPES = [(5000, 256, 8, 5), (4097, 128, 6, 3), (3001, 64, 8, 4), (2500, 24, 3, 7), (1500, 512, 8, 2),
          (777, 8, 2, 3)]


@pytest.mark.parametrize("T,E,K,M", SHAPES)
@pytest.mark.parametrize("pass_", [1, 2])
@pytest.mark.parametrize("span", ["half", "all", "none", "ragged"])
def test_fused_pass_matches_oracle(T, E, K, M, pass_, span):
    z, off, tau, loads, g = case(T, E, K, M, seed=T + E + pass_)
    t0, t1 = {"half": (0, T // 2) if pass_ == 1 else (T // 2, T), "all": (0, T),
              "none": (T // 3, T // 3), "ragged": (17, T - 5)}[span]
    eta, c = 0.5, 1.0
    H = oracle.hist_hi(z, tau)
    u, _ = oracle.select_hi(H, oracle.target_rank(T, E, K))
    want_hist = H if pass_ == 1 else oracle.hist_lo(z, tau, u)
    g_ref, _ = oracle.lei(g, loads, off, K, eta, c)

    offd = torch.from_numpy(off).cuda()
    coef = eqb.lei_coefficients(torch.from_numpy(loads).cuda(), offd, K, eta, c)
    hist = Guarded((E, 256), torch.int32)
    G = Guarded((T, E), torch.float32)
    G.view.copy_(torch.from_numpy(g))
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    eqb.eqb_margin_hist_lei(to_dev_bf16(z), torch.from_numpy(tau).cuda(), pass_, hist.view, G.view, coef, offd,
                            t0, t1, u=torch.from_numpy(u).cuda() if pass_ == 2 else None, err_flag=err)
    torch.cuda.synchronize()
    assert hist.intact() and G.intact()
    assert err.item() == 0
    assert np.array_equal(hist.view.cpu().numpy(), want_hist)
    got = G.view.cpu().numpy()
    assert np.array_equal(bits_f32(got[:t0]), bits_f32(g[:t0]))
    assert np.array_equal(bits_f32(got[t1:]), bits_f32(g[t1:]))
    assert within(got[t0:t1], g_ref[t0:t1])


def test_fused_pass_rejects_bad_ranges():
    T, E = 64, 8
    z = torch.zeros((T, E), dtype=torch.bfloat16, device="cuda")
    tau = torch.zeros(T, device="cuda")
    hist = torch.zeros((E, 256), dtype=torch.int32, device="cuda")
    g = torch.zeros((T, E), device="cuda")
    off = torch.tensor([0, T], dtype=torch.int64, device="cuda")
    coef = torch.zeros((1, E), device="cuda")
    for t0, t1 in [(-1, 4), (5, 4), (0, T + 1)]:
        with pytest.raises(eqb.EqbError):
            eqb.eqb_margin_hist_lei(z, tau, 1, hist, g, coef, off, t0, t1)
    with pytest.raises(eqb.EqbError):
        eqb.eqb_margin_hist_lei(z, tau, 3, hist, g, coef, off, 0, T)
    with pytest.raises(eqb.EqbError):
        eqb.eqb_margin_hist_lei(z, tau, 2, hist, g, coef, off, 0, T)  # pass 2 without u


@pytest.mark.parametrize("T,E,K,M", [(20000, 1024, 8, 64), (20000, 1024, 8, 65), (30000, 256, 8, 300),
                                     (20000, 128, 8, 4)])
def test_layer_step_at_and_past_the_coefficient_table(T, E, K, M):
    """M * E = 65,536 runs the fused passes; one microbatch more (or many
    small ones) runs LEI last.  Both reproduce the oracle, and both give the
    bits of the separate LEI launch."""
    rng = np.random.default_rng(T + M)
    z = brute.bf16_bits_from_f32(rng.standard_normal((T, E)).astype(np.float32))
    b = (rng.standard_normal(E) * 0.3).astype(np.float32)
    off = ragged_offsets(T, M, seed=M)
    g = (rng.standard_normal((T, E)) * 0.1).astype(np.float32)
    eta, c = 0.25, 1.0
    o = oracle_forward(z, b, K, off)
    g_ref, _ = oracle.lei(g, o["loads"], off, K, eta, c)
    loads = torch.zeros((M, E), dtype=torch.int32, device="cuda")
    bn = torch.empty(E, device="cuda")
    tau = torch.empty(T, device="cuda")
    G = Guarded((T, E), torch.float32)
    G.view.copy_(torch.from_numpy(g))
    ws = torch.zeros(eqb.eqb_layer_workspace_bytes(E), dtype=torch.uint8, device="cuda")
    eqb.eqb_layer_step(to_dev_bf16(z), torch.from_numpy(b).cuda(), K, torch.from_numpy(off).cuda(), loads, bn, ws,
                       tau=tau, grad_s=G.view, eta=eta, c=c, mb_offsets_host=off)
    torch.cuda.synchronize()
    assert G.intact()
    assert np.array_equal(loads.cpu().numpy(), o["loads"])
    assert np.array_equal(bits_f32(bn.cpu().numpy()), bits_f32(o["b_next"]))
    assert within(G.view.cpu().numpy(), g_ref)
    G2 = torch.from_numpy(g).cuda()
    eqb.lei_inject_grad(G2, torch.from_numpy(o["loads"]).cuda(), torch.from_numpy(off).cuda(), K, eta, c)
    torch.cuda.synchronize()
    assert np.array_equal(bits_f32(G.view.cpu().numpy()), bits_f32(G2.cpu().numpy()))


@pytest.mark.parametrize("T", [1, 2, 3, 31, 33, 1025])
@pytest.mark.parametrize("E,K", [(8, 2), (64, 8), (256, 8)])
def test_layer_step_tiny_batches_with_lei(T, E, K):
    """Batches smaller than a warp round, a histogram block or a LEI chunk
    (an empty first half at T = 1) through the fused step."""
    rng = np.random.default_rng(T * 1000 + E)
    z = brute.bf16_bits_from_f32(rng.standard_normal((T, E)).astype(np.float32))
    b = (rng.standard_normal(E) * 0.3).astype(np.float32)
    off = np.array([0, T // 2, T], np.int64) if T >= 2 else np.array([0, T], np.int64)
    M = len(off) - 1
    g = (rng.standard_normal((T, E)) * 0.1).astype(np.float32)
    eta, c = 0.5, 2.0
    o = oracle_forward(z, b, K, off)
    g_ref, _ = oracle.lei(g, o["loads"], off, K, eta, c)
    idx = Guarded((T, K), torch.int32)
    tau = Guarded((T,), torch.float32)
    loads = Guarded((M, E), torch.int32, fill=5)
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
    assert np.array_equal(loads.view.cpu().numpy(), o["loads"])
    assert np.array_equal(bits_f32(bn.view.cpu().numpy()), bits_f32(o["b_next"]))
    assert within(G.view.cpu().numpy(), g_ref)
