"""Router logits with routing from the accumulator (eqb_router_route): the
projection of Sec. 2 (Eq. 1) and the top-K / cutoff / loads step of the same
section in one kernel.

Parity against the oracle uses integer-valued inputs: x in {-3..3} and W_r in
{-1, 0, 1} keep every partial sum an integer below 2^24, so the fp32
accumulation is exact in any order and z = bf16_rne(exact dot product) on both
sides (the fp64 -> fp32 step is exact for these values).  Integer logits also
make ties common, which exercises the lower-index rule.  Random real-valued
inputs are checked against the two separate library calls (eqb_router_logits
then eqb_route_topk), which the other parity tests pin to the oracle."""
import numpy as np
import pytest
import torch

import brute
import oracle
import paper_2609_28053_gb300 as eqb
from eqb_workloads import SHAPES, make_router_inputs, ragged_offsets
from gpu_harness import Guarded, to_dev_bf16

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib(cuda_ok):
    eqb.load()


def integer_inputs(T, d, E, seed):
    rng = np.random.default_rng(seed)
    x = rng.integers(-3, 4, size=(T, d)).astype(np.float32)
    W = rng.choice(np.array([-1.0, 0.0, 1.0], np.float32), size=(E, d), p=[0.2, 0.6, 0.2])
    # a few biases repeat, so that equal scores from equal logits occur
    b = rng.choice(np.array([0.0, 0.5, -0.25, 1.0, -1.5], np.float32), size=E)
    return brute.bf16_bits_from_f32(x), brute.bf16_bits_from_f32(W), b.astype(np.float32)


def run_fused(x_bits, W_bits, b, K, offsets):
    T, _ = x_bits.shape
    E = W_bits.shape[0]
    M = len(offsets) - 1
    Z = Guarded((T, E), torch.bfloat16, canary=-7.0)
    idx = Guarded((T, K), torch.int32, fill=-7)
    tau = Guarded((T,), torch.float32, fill=-7.0)
    loads = Guarded((M, E), torch.int32)
    H = Guarded((E, 256), torch.int32)
    err = Guarded((1,), torch.int32)
    off = torch.from_numpy(np.ascontiguousarray(offsets, np.int64)).cuda()
    eqb.eqb_router_route(to_dev_bf16(x_bits), to_dev_bf16(W_bits), torch.from_numpy(b).cuda(), K, off,
                         z=Z.view, topk_idx=idx.view, tau=tau.view, loads=loads.view, hist_hi=H.view,
                         err_flag=err.view)
    torch.cuda.synchronize()
    for g in (Z, idx, tau, loads, H, err):
        assert g.intact(), "write outside an output buffer"
    run_fused.last_hist = H.view.cpu().numpy()
    return (Z.view.view(torch.int16).cpu().numpy().view(np.uint16), idx.view.cpu().numpy(),
            tau.view.cpu().numpy(), loads.view.cpu().numpy(), int(err.view.item()))


@pytest.mark.parametrize("T,d,E,K", [(1, 64, 64, 1), (127, 64, 128, 8), (129, 128, 64, 2),
                                     (1000, 256, 128, 8), (4099, 512, 64, 6), (70000, 128, 128, 8),
                                     (300, 4096, 128, 7), (513, 256, 64, 3)])
def test_router_route_matches_oracle(T, d, E, K):
    x, W, b = integer_inputs(T, d, E, seed=T * 7 + d + E + K)
    offsets = ragged_offsets(T, 5, seed=T + K) if T >= 5 else np.array([0, T], np.int64)
    z, idx, tau, loads, err = run_fused(x, W, b, K, offsets)
    assert err == 0
    zref, _ = oracle.router_logits(x, W, np.arange(T))
    assert np.all(np.abs(zref) < 2 ** 24) and np.all(zref == np.round(zref))
    z_or = brute.bf16_bits_from_f32(zref.astype(np.float32))
    np.testing.assert_array_equal(z, z_or)
    i_or, t_or, l_or = oracle.route(z_or, b, K, offsets)
    np.testing.assert_array_equal(idx, i_or)
    np.testing.assert_array_equal(tau.view(np.uint32), t_or.view(np.uint32))
    np.testing.assert_array_equal(loads, l_or)
    # the coarse histogram counted in the epilogue (Algorithm 1 step 1)
    np.testing.assert_array_equal(run_fused.last_hist, oracle.hist_hi(z_or, t_or))


def two_calls(x, W, b, K, off, M):
    T = x.shape[0]
    E = W.shape[0]
    z = eqb.eqb_router_logits(x, W)
    idx = torch.empty((T, K), dtype=torch.int32, device="cuda")
    tau = torch.empty(T, dtype=torch.float32, device="cuda")
    loads = torch.zeros((M, E), dtype=torch.int32, device="cuda")
    H = torch.zeros((E, 256), dtype=torch.int32, device="cuda")
    eqb.eqb_route_topk(z, b, K, off, topk_idx=idx, tau=tau, loads=loads, hist_hi=H)
    return z, idx, tau, loads, H


def fused(x, W, b, K, off, M):
    T = x.shape[0]
    E = W.shape[0]
    idx = torch.empty((T, K), dtype=torch.int32, device="cuda")
    loads = torch.zeros((M, E), dtype=torch.int32, device="cuda")
    H = torch.zeros((E, 256), dtype=torch.int32, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    z, idx, tau = eqb.eqb_router_route(x, W, b, K, off, topk_idx=idx, loads=loads, hist_hi=H, err_flag=err)
    return z, idx, tau, loads, err, H


@pytest.mark.parametrize("T,d,E,K", [(5000, 4096, 128, 8), (3001, 1024, 64, 8), (777, 512, 128, 2)])
def test_router_route_equals_two_calls(T, d, E, K):
    x, W = make_router_inputs(T=T, d_model=d, device="cuda", E=E)
    g = torch.Generator(device="cpu").manual_seed(T + E)
    b = (0.05 * torch.randn(E, generator=g)).float().cuda()
    off = torch.from_numpy(ragged_offsets(T, 4, seed=3)).cuda()
    a = two_calls(x, W, b, K, off, 4)
    f = fused(x, W, b, K, off, 4)
    torch.cuda.synchronize()
    assert f[4].item() == 0
    assert torch.equal(a[0].view(torch.int16), f[0].view(torch.int16))
    assert torch.equal(a[1], f[1])
    assert torch.equal(a[2].view(torch.int32), f[2].view(torch.int32))
    assert torch.equal(a[3], f[3])
    assert torch.equal(a[4], f[5])


def test_router_route_full_size_equals_two_calls():
    """Router configuration at full size (T = 1,048,576, d = 4096, E = 128,
    K = 8, 16 microbatches): every output equals the separate calls'."""
    sh = SHAPES["router"]
    x, W = make_router_inputs(device="cuda")
    g = torch.Generator(device="cpu").manual_seed(11)
    b = (0.05 * torch.randn(sh.E, generator=g)).float().cuda()
    off = torch.arange(0, sh.T + 1, sh.T // sh.M, dtype=torch.int64).cuda()
    a = two_calls(x, W, b, sh.K, off, sh.M)
    f = fused(x, W, b, sh.K, off, sh.M)
    torch.cuda.synchronize()
    assert f[4].item() == 0
    assert torch.equal(a[0].view(torch.int16), f[0].view(torch.int16))
    assert torch.equal(a[1], f[1])
    assert torch.equal(a[2].view(torch.int32), f[2].view(torch.int32))
    assert torch.equal(a[3], f[3])
    assert torch.equal(a[4], f[5])
    assert int(f[3].sum()) == sh.T * sh.K
    assert torch.all(f[5].sum(1) == sh.T)


@pytest.mark.slow
def test_router_route_epilogue_counters_at_their_limit():
    """The largest T whose coarse histogram is still counted in the
    epilogue: every block takes 511 tiles (65,408 tokens), so each 16-bit
    window counter climbs to 65,408 when all tokens agree.  Constant
    integer rows make every token's logits, top-K, cutoff and margins the
    same (b = 0), so H = T x the histogram of one row (Algorithm 1 step 1)
    and each microbatch's loads are its size on the row's top-K."""
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    T, d, E, K = 511 * sms * 128, 64, 128, 8
    xr, W, _ = integer_inputs(1, d, E, seed=21)
    b = np.zeros(E, np.float32)
    offsets = ragged_offsets(T, 3, seed=4)
    x = to_dev_bf16(xr).expand(T, d).contiguous()
    idx = torch.empty((T, K), dtype=torch.int32, device="cuda")
    loads = torch.zeros((3, E), dtype=torch.int32, device="cuda")
    H = torch.zeros((E, 256), dtype=torch.int32, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    z, idx, tau = eqb.eqb_router_route(x, to_dev_bf16(W), torch.from_numpy(b).cuda(), K,
                                       torch.from_numpy(offsets).cuda(), topk_idx=idx, loads=loads,
                                       hist_hi=H, err_flag=err)
    torch.cuda.synchronize()
    assert err.item() == 0
    del x
    zr, _ = oracle.router_logits(xr, W, np.arange(1))
    z_row = brute.bf16_bits_from_f32(zr.astype(np.float32))
    i_row, t_row, _ = oracle.route(z_row, b, K, np.array([0, 1], np.int64))
    assert torch.equal(z[0].view(torch.int16).cpu(), torch.from_numpy(z_row[0].view(np.int16)))
    assert bool((idx == torch.from_numpy(i_row[0]).cuda()).all())
    assert bool((tau.view(torch.int32) == int(t_row.view(np.int32)[0])).all())
    np.testing.assert_array_equal(H.cpu().numpy(), T * oracle.hist_hi(z_row, t_row).astype(np.int64))
    want = np.zeros((3, E), np.int64)
    want[:, i_row[0]] = np.diff(offsets)[:, None]
    np.testing.assert_array_equal(loads.cpu().numpy(), want)


@pytest.mark.slow
def test_router_route_coarse_pass_beyond_the_epilogue_limit():
    """T = 10,000,000 with d = 64: more than 65,535 tokens for some block, so
    the coarse histogram comes from the coarse pass over z after the
    projection; it equals the separate calls' (and so does everything
    else)."""
    T, d, E, K, M = 10_000_000, 64, 128, 8, 5
    x, W = make_router_inputs(T=T, d_model=d, device="cuda", E=E)
    b = torch.zeros(E, dtype=torch.float32, device="cuda")
    off = torch.from_numpy(ragged_offsets(T, M, seed=9)).cuda()
    a = two_calls(x, W, b, K, off, M)
    f = fused(x, W, b, K, off, M)
    torch.cuda.synchronize()
    assert f[4].item() == 0
    assert torch.equal(a[1], f[1])
    assert torch.equal(a[3], f[3])
    assert torch.equal(a[4], f[5])
    assert torch.all(f[5].sum(1) == T)


def test_router_route_nonfinite_bias_flagged():
    x, W, b = integer_inputs(200, 64, 64, seed=5)
    b[17] = np.inf
    *_, err = run_fused(x, W, b, 4, np.array([0, 200], np.int64))
    assert err == 4  # EQB_ERR_NONFINITE


def test_router_route_optional_outputs():
    """Without topk_idx and loads only z and tau are written."""
    x, W, b = integer_inputs(300, 128, 128, seed=9)
    xd, Wd, bd = to_dev_bf16(x), to_dev_bf16(W), torch.from_numpy(b).cuda()
    z, idx, tau = eqb.eqb_router_route(xd, Wd, bd, 8)
    torch.cuda.synchronize()
    assert idx is None
    zref, _ = oracle.router_logits(x, W, np.arange(300))
    z_or = brute.bf16_bits_from_f32(zref.astype(np.float32))
    _, t_or, _ = oracle.route(z_or, b, 8)
    np.testing.assert_array_equal(tau.cpu().numpy().view(np.uint32), t_or.view(np.uint32))


LEI_ATOL, LEI_RTOL = 1e-7, 1e-5


@pytest.mark.parametrize("T,d,E,K,M", [(3000, 256, 128, 8, 4), (2049, 128, 64, 2, 3),
                                       (1500, 128, 256, 8, 2), (777, 192, 96, 5, 3)])
def test_router_layer_step_matches_oracle(T, d, E, K, M):
    """eqb_router_layer_step from x: projection, routing, both EQB passes,
    the bias update (bit for bit) and LEI (within tolerance) on the oracle's
    integer-valued case.  E = 256 and E = 96 take the unfused routing."""
    x, W, b = integer_inputs(T, d, E, seed=T + d + E)
    off = ragged_offsets(T, M, seed=M + 1)
    g = (np.random.default_rng(T).standard_normal((T, E)) * 0.1).astype(np.float32)
    eta, c = 0.25, 1.0
    zref, _ = oracle.router_logits(x, W, np.arange(T))
    z_or = brute.bf16_bits_from_f32(zref.astype(np.float32))
    o = oracle.eqb_step(z_or, b, K, off)
    g_ref, _ = oracle.lei(g, o["loads"], off, K, eta, c)

    Z = Guarded((T, E), torch.bfloat16, canary=-7.0)
    idx = Guarded((T, K), torch.int32)
    tau = Guarded((T,), torch.float32)
    loads = Guarded((M, E), torch.int32, fill=99)
    bn = Guarded((E,), torch.float32)
    G = Guarded((T, E), torch.float32)
    G.view.copy_(torch.from_numpy(g))
    ws = torch.zeros(eqb.eqb_layer_workspace_bytes(E), dtype=torch.uint8, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    eqb.eqb_router_layer_step(to_dev_bf16(x), to_dev_bf16(W), torch.from_numpy(b).cuda(), K,
                              torch.from_numpy(off).cuda(), loads.view, bn.view, ws, z=Z.view,
                              tau=tau.view, topk_idx=idx.view, grad_s=G.view, eta=eta, c=c,
                              mb_offsets_host=off, err_flag=err)
    torch.cuda.synchronize()
    for buf in (Z, idx, tau, loads, bn, G):
        assert buf.intact()
    assert err.item() == 0
    np.testing.assert_array_equal(Z.view.view(torch.int16).cpu().numpy().view(np.uint16), z_or)
    np.testing.assert_array_equal(idx.view.cpu().numpy(), o["idx"])
    np.testing.assert_array_equal(tau.view.cpu().numpy().view(np.uint32), o["tau"].view(np.uint32))
    np.testing.assert_array_equal(loads.view.cpu().numpy(), o["loads"])
    np.testing.assert_array_equal(bn.view.cpu().numpy().view(np.uint32), o["b_next"].view(np.uint32))
    got = G.view.cpu().numpy().astype(np.float64)
    assert np.all(np.abs(got - g_ref) <= LEI_ATOL + LEI_RTOL * np.abs(g_ref))


def test_router_route_loads_long_run():
    """Enough tiles per block (over 2047 at up to 160 SMs) that the kernel's
    16-bit shared-memory load counters must be flushed on the way: one
    microbatch, and a bias that puts expert 5 in every token's top-K, so its
    counter climbs as fast as it can.  Loads must equal the histogram of
    topk_idx."""
    T = 2100 * 160 * 128 + 77
    d, E, K = 64, 64, 2
    x, W = make_router_inputs(T=T, d_model=d, device="cuda", E=E)
    b = torch.zeros(E, dtype=torch.float32, device="cuda")
    b[5] = 1.0e4
    off = torch.tensor([0, T], dtype=torch.int64, device="cuda")
    idx = torch.empty((T, K), dtype=torch.int32, device="cuda")
    loads = torch.zeros((1, E), dtype=torch.int32, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    z, idx, tau = eqb.eqb_router_route(x, W, b, K, off, topk_idx=idx, loads=loads, err_flag=err)
    torch.cuda.synchronize()
    assert err.item() == 0
    assert int(loads[0, 5]) == T
    hist = torch.bincount(idx.flatten().long(), minlength=E).to(torch.int32)
    assert torch.equal(loads[0], hist)
    del x, z
