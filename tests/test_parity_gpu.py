"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle on the
same seeded inputs.  Bit-exact for top-K indices, cutoffs, loads, both
histograms, u, rho, the quantiles and the bias; LEI gradients within
|d| <= 1e-7 + 1e-5 |g_ref|."""
import numpy as np
import pytest
import torch

import brute
import oracle
import paper_2609_28053_gb300 as eqb
from eqb_workloads import (SHAPES, bits, even_offsets, make_bias, make_grad, make_logits,
                           prior_batch_logits, ragged_offsets)
from gpu_harness import Guarded, bits_f32, gpu_forward, oracle_forward, to_dev_bf16

pytestmark = pytest.mark.gpu

LEI_ATOL, LEI_RTOL = 1e-7, 1e-5


@pytest.fixture(scope="module", autouse=True)
def _lib(cuda_ok):
    eqb.load()


def assert_forward_equal(g, o, check_hist=True):
    assert np.array_equal(g["idx"], o["idx"]), "top-K indices differ"
    assert np.array_equal(bits_f32(g["tau"]), bits_f32(o["tau"])), "tau differs"
    assert np.array_equal(g["loads"], o["loads"]), "loads differ"
    if check_hist:
        assert np.array_equal(g["H"], o["H"]), "coarse histogram differs"
        assert np.array_equal(g["u"], o["u"]) and np.array_equal(g["rho"], o["rho"])
        assert np.array_equal(g["L"], o["L"]), "fine histogram differs"
    assert np.array_equal(g["q"], o["q"]), "quantile differs"
    assert np.array_equal(bits_f32(g["b_next"]), bits_f32(o["b_next"])), "bias update differs"
    assert g["err"][0] == 0


def rand_case(T, E, seed, scale=1.0, bias_scale=0.3, ties=False):
    rng = np.random.default_rng(seed)
    if ties:
        v = rng.integers(-2, 3, size=(T, E)).astype(np.float32) * 0.25
        b = np.zeros(E, np.float32)
    else:
        v = (rng.standard_normal((T, E)) * scale).astype(np.float32)
        b = (rng.standard_normal(E) * bias_scale).astype(np.float32)
    return brute.bf16_bits_from_f32(v), b


# ------------------------------------------------------------- edge shapes

@pytest.mark.parametrize("T", [1, 31, 32, 33, 1000, 4099])
@pytest.mark.parametrize("E,K", [(8, 1), (8, 2), (8, 7), (16, 3), (24, 5), (64, 6), (64, 8),
                                 (128, 8), (256, 6), (256, 8), (256, 15), (256, 31), (40, 31)])
def test_forward_small_shapes(T, E, K):
    z, b = rand_case(T, E, seed=T * 1000 + E * 10 + K)
    off = ragged_offsets(T, 3, seed=T + E) if T > 3 else np.array([0, T], np.int64)
    assert_forward_equal(gpu_forward(z, b, K, off), oracle_forward(z, b, K, off))


@pytest.mark.parametrize("T", [33, 1000])
@pytest.mark.parametrize("E,K", [(264, 8), (384, 8), (512, 6), (1024, 8), (1024, 31)])
def test_forward_many_experts(T, E, K):
    """E above 256: the compile-time-width routing kernel (E = 384, 512 with
    K + 1 <= 16) and the runtime-width one (E = 264, 1024, and K = 31),
    histograms tiled over experts, selection and the bias update on up to
    1024 experts."""
    z, b = rand_case(T, E, seed=T + E + K)
    off = ragged_offsets(T, 3, seed=E)
    assert_forward_equal(gpu_forward(z, b, K, off), oracle_forward(z, b, K, off))


@pytest.mark.parametrize("E,K", [(8, 2), (64, 8), (128, 2), (128, 8), (256, 8), (256, 15), (256, 20)])
def test_forward_exact_ties(E, K):
    """Integer-valued logits with b = 0: most scores tie, so the candidate
    lists overflow and the exact fallback decides by lower index."""
    z, b = rand_case(517, E, seed=E + K, ties=True)
    off = np.array([0, 200, 200, 517], np.int64)  # includes an empty microbatch
    assert_forward_equal(gpu_forward(z, b, K, off), oracle_forward(z, b, K, off))


@pytest.mark.parametrize("E", [64, 128, 256])
def test_forward_constant_rows(E):
    T, K = 300, 8
    z = np.full((T, E), brute.bf16_bits_from_f32(np.float32([0.75]))[0], np.uint16)
    z[::7] = brute.bf16_bits_from_f32(np.float32([-1.5]))[0]
    b = np.zeros(E, np.float32)
    off = np.array([0, T], np.int64)
    assert_forward_equal(gpu_forward(z, b, K, off), oracle_forward(z, b, K, off))


@pytest.mark.parametrize("E", [64, 128, 256])
def test_forward_signed_zero_subnormal_and_large_values(E):
    rng = np.random.default_rng(5 + E)
    T, K = 777, 8
    v = (rng.standard_normal((T, E))).astype(np.float32)
    v[rng.random((T, E)) < 0.1] = 0.0
    v[rng.random((T, E)) < 0.1] = -0.0
    v[rng.random((T, E)) < 0.05] = (rng.standard_normal(1) * 1e-39).astype(np.float32)[0]
    v[rng.random((T, E)) < 0.02] = 1e30
    v[rng.random((T, E)) < 0.02] = -1e30
    z = brute.bf16_bits_from_f32(v)
    b = (rng.standard_normal(E) * 1e-38).astype(np.float32)
    b[::5] = -0.0
    off = np.array([0, 400, T], np.int64)
    assert_forward_equal(gpu_forward(z, b, K, off), oracle_forward(z, b, K, off))


# ------------------------------------------------------------- configs

def config_inputs(name, T=None):
    sh = SHAPES[name]
    T = sh.T if T is None else T
    z = bits(make_logits(name, T=T))
    if name == "mid":
        zp = bits(prior_batch_logits(name, T=T))
        b = oracle.eqb_step(zp, np.zeros(sh.E, np.float32), sh.K)["b_next"]
    else:
        b = make_bias(name).numpy()
    return z, b, even_offsets(T, sh.M), sh.K


@pytest.mark.parametrize("name", ["tiny", "tie", "mid"])
def test_config_forward(name):
    z, b, off, K = config_inputs(name)
    assert_forward_equal(gpu_forward(z, b, K, off), oracle_forward(z, b, K, off))


def test_tie_config_repartitioned():
    """Tie-heavy config: the quantile is the same for P = 8, 1, 3, 13 and 64
    uneven partitions and for a token permutation: histograms of
    per-partition calls accumulate into the same device buffers."""
    z, b, off, K = config_inputs("tie")
    T, E = z.shape
    ref = oracle_forward(z, b, K, off)
    r = ref["r"]
    rng = np.random.default_rng(0)
    for P, perm in [(8, False), (1, False), (3, False), (13, True), (64, True)]:
        order = rng.permutation(T) if perm else np.arange(T)
        zz = z[order]
        cuts = np.sort(rng.choice(np.arange(1, T), size=P - 1, replace=False)) if P > 1 else []
        bounds = np.concatenate([[0], cuts, [T]]).astype(np.int64)
        zd = to_dev_bf16(zz)
        bt = torch.from_numpy(b).cuda()
        tau = torch.empty(T, dtype=torch.float32, device="cuda")
        H = torch.zeros((E, 256), dtype=torch.int32, device="cuda")
        L = torch.zeros_like(H)
        u = torch.zeros(E, dtype=torch.uint8, device="cuda")
        rho = torch.zeros(E, dtype=torch.int32, device="cuda")
        q = torch.zeros(E, dtype=torch.bfloat16, device="cuda")
        err = torch.zeros(1, dtype=torch.int32, device="cuda")
        for p in range(P):
            a, c = int(bounds[p]), int(bounds[p + 1])
            eqb.eqb_route_topk(zd[a:c], bt, K, None, None, tau[a:c], None, H, err)
        eqb.eqb_select_quantile(H, 1, r, u, rho, None, err)
        for p in range(P):
            a, c = int(bounds[p]), int(bounds[p + 1])
            eqb.eqb_margin_hist_pass2(zd[a:c], tau[a:c], u, L)
        eqb.eqb_select_quantile(L, 2, r, u, rho, q, err)
        torch.cuda.synchronize()
        assert np.array_equal(H.cpu().numpy(), ref["H"])
        assert np.array_equal(q.view(torch.int16).cpu().numpy().view(np.uint16), ref["q"])
        assert err.item() == 0


@pytest.mark.slow
def test_global_config_full_size_sampled():
    """Full size (T = 2,097,152, E = 256, K = 8, M = 64): every token's top-K
    and cutoff, all loads, and the exact quantile of 16 sampled experts
    against the oracle; the launch configuration is the benchmark's."""
    name = "global"
    sh = SHAPES[name]
    zt = make_logits(name, device="cuda")
    z = bits(zt)
    b = make_bias(name, device="cuda").cpu().numpy()
    off = even_offsets(sh.T, sh.M)
    g = gpu_forward(z, b, sh.K, off)
    experts = np.random.default_rng(1).choice(sh.E, 16, replace=False)
    o = oracle_forward(z, b, sh.K, off, experts=experts)
    assert np.array_equal(g["idx"], o["idx"])
    assert np.array_equal(bits_f32(g["tau"]), bits_f32(o["tau"]))
    assert np.array_equal(g["loads"], o["loads"])
    assert np.array_equal(g["q"][experts], o["q"])
    # histogram totals: every expert saw all T margins
    assert np.all(g["H"].sum(1) == sh.T)
    assert np.all(g["L"].sum(1) >= g["rho"])
    assert g["err"][0] == 0


@pytest.mark.slow
@pytest.mark.parametrize("name", ["global", "paper", "wide"])
def test_layer_step_full_size(name):
    """The benchmark's timed call at full size (eqb_layer_step on the global
    workload, T = 2,097,152, E = 256, K = 8, M = 64, on the paper's shape,
    T = 9,437,184, K = 6, and on the wide workload, T = 1,048,576, E = 512;
    LEI streamed inside the histogram passes, eta and c of the benchmark):
    every token's top-K and cutoff, all loads and the next bias of every
    expert bit for bit against the oracle (full-sort quantiles), and 4,096
    sampled rows of the injected gradient within the LEI tolerance of the
    oracle's coefficients."""
    sh = SHAPES[name]
    T, E, K, M = sh.T, sh.E, sh.K, sh.M
    eta, c = 2e-5, 1.0
    zt = make_logits(name, device="cuda")
    bt = make_bias(name, device="cuda")
    G = make_grad(name, device="cuda")
    rows = np.sort(np.random.default_rng(5).choice(T, 4096, replace=False))
    rows_d = torch.from_numpy(rows).cuda()
    g_rows = G[rows_d].cpu().numpy()
    off = even_offsets(T, M)
    offd = torch.from_numpy(off).cuda()
    idx = torch.empty((T, K), dtype=torch.int32, device="cuda")
    tau = torch.empty(T, dtype=torch.float32, device="cuda")
    loads = torch.zeros((M, E), dtype=torch.int32, device="cuda")
    bn = torch.empty(E, dtype=torch.float32, device="cuda")
    ws = torch.zeros(eqb.eqb_layer_workspace_bytes(E), dtype=torch.uint8, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    eqb.eqb_layer_step(zt, bt, K, offd, loads, bn, ws, tau=tau, topk_idx=idx, grad_s=G, eta=eta, c=c,
                       mb_offsets_host=off, err_flag=err)
    torch.cuda.synchronize()
    assert err.item() == 0
    got_rows = G[rows_d].cpu().numpy()
    z = bits(zt)
    o = oracle_forward(z, bt.cpu().numpy(), K, off, experts=np.arange(E))
    assert np.array_equal(idx.cpu().numpy(), o["idx"])
    assert np.array_equal(bits_f32(tau.cpu().numpy()), bits_f32(o["tau"]))
    assert np.array_equal(loads.cpu().numpy(), o["loads"])
    assert np.array_equal(bits_f32(bn.cpu().numpy()), bits_f32(oracle.bias_update(o["q"])))
    _, a = oracle.lei(None, o["loads"], off, K, eta, c)
    mb = np.searchsorted(off, rows, side="right") - 1
    want = g_rows.astype(np.float64) + a[mb]
    assert np.all(np.abs(got_rows.astype(np.float64) - want) <= LEI_ATOL + LEI_RTOL * np.abs(want))


@pytest.mark.slow
def test_paper_config_full_size_sampled():
    """The paper's own shape (Sec. 5 / App. E.1: E = 256, K = 6, 147,456 tokens
    on each of 64 ranks, T = 9,437,184): every token's top-K and cutoff, all
    loads, and the exact quantile of 8 sampled experts against the oracle."""
    name = "paper"
    sh = SHAPES[name]
    z = bits(make_logits(name, device="cuda"))
    b = make_bias(name, device="cuda").cpu().numpy()
    off = even_offsets(sh.T, sh.M)
    g = gpu_forward(z, b, sh.K, off)
    experts = np.random.default_rng(2).choice(sh.E, 8, replace=False)
    o = oracle_forward(z, b, sh.K, off, experts=experts)
    assert o["r"] == 221184
    assert np.array_equal(g["idx"], o["idx"])
    assert np.array_equal(bits_f32(g["tau"]), bits_f32(o["tau"]))
    assert np.array_equal(g["loads"], o["loads"])
    assert np.array_equal(g["q"][experts], o["q"])
    assert np.all(g["H"].sum(1) == sh.T)
    assert g["err"][0] == 0


@pytest.mark.slow
def test_router_config_three_steps_on_torch_logits():
    """Router config: z = bf16(x W_r^T) (here from torch's matmul), bias
    iterated for 3 steps from b^(0) = 0 with fresh activations; each step's
    GPU bias feeds the next GPU step and the oracle's feeds the oracle's, so
    bit-exact agreement at every step pins the whole chain.  Reduced T."""
    from eqb_workloads import make_router_inputs
    sh = SHAPES["router"]
    T = 65536
    b_gpu = np.zeros(sh.E, np.float32)
    b_or = np.zeros(sh.E, np.float32)
    off = even_offsets(T, sh.M)
    for step in range(3):
        x, W = make_router_inputs(T=T, step=step, device="cuda")
        z = bits((x.float() @ W.float().t()).to(torch.bfloat16))
        g = gpu_forward(z, b_gpu, sh.K, off)
        o = oracle_forward(z, b_or, sh.K, off)
        assert_forward_equal(g, o)
        b_gpu, b_or = g["b_next"], o["b_next"]


# ------------------------------------------------------------- per-call units

def test_standalone_pass1_matches_oracle_counts():
    z, b = rand_case(3000, 128, seed=11)
    _, tau, _ = oracle.route(z, b, 8)
    H_ref = oracle.hist_hi(z, tau)
    H = Guarded((128, 256), torch.int32)
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    eqb.eqb_margin_hist_pass1(to_dev_bf16(z), torch.from_numpy(tau).cuda(), H.view, err)
    torch.cuda.synchronize()
    assert H.intact() and np.array_equal(H.view.cpu().numpy(), H_ref) and err.item() == 0


def test_select_and_bias_from_oracle_histograms():
    z, b = rand_case(5000, 64, seed=12)
    K = 6
    _, tau, _ = oracle.route(z, b, K)
    r = oracle.target_rank(5000, 64, K)
    H = oracle.hist_hi(z, tau)
    u, rho = oracle.select_hi(H, r)
    L = oracle.hist_lo(z, tau, u)
    q = oracle.select_lo(L, u, rho)
    bn = oracle.bias_update(q)
    ud = torch.zeros(64, dtype=torch.uint8, device="cuda")
    rd = torch.zeros(64, dtype=torch.int32, device="cuda")
    qd = torch.zeros(64, dtype=torch.bfloat16, device="cuda")
    bd = torch.zeros(64, dtype=torch.float32, device="cuda")
    eqb.eqb_select_quantile(torch.from_numpy(H).cuda(), 1, r, ud, rd)
    torch.cuda.synchronize()
    assert np.array_equal(ud.cpu().numpy(), u) and np.array_equal(rd.cpu().numpy(), rho)
    eqb.eqb_select_quantile(torch.from_numpy(L).cuda(), 2, r, torch.from_numpy(u).cuda(),
                            torch.from_numpy(rho).cuda(), qd)
    eqb.eqb_bias_update(torch.from_numpy(q.view(np.int16)).view(torch.bfloat16).cuda(), bd)
    torch.cuda.synchronize()
    assert np.array_equal(qd.view(torch.int16).cpu().numpy().view(np.uint16), q)
    assert np.array_equal(bits_f32(bd.cpu().numpy()), bits_f32(bn))


@pytest.mark.parametrize("T,E,K,M", [(4096, 8, 2, 4), (1001, 64, 8, 5), (65536, 64, 8, 8),
                                     (33, 256, 8, 2), (5000, 24, 3, 7), (2000, 512, 8, 3), (700, 1024, 6, 2)])
@pytest.mark.parametrize("eta,c", [(1.0, 0.5), (0.25, 4.0), (0.02, 0.0), (2e-5, 1.0)])
def test_lei_matches_oracle(T, E, K, M, eta, c):
    z, b = rand_case(T, E, seed=T + E)
    off = ragged_offsets(T, M, seed=E)
    _, _, loads = oracle.route(z, b, K, off)
    g = (np.random.default_rng(T).standard_normal((T, E)) * 0.1).astype(np.float32)
    g_ref, _ = oracle.lei(g, loads, off, K, eta, c)
    G = Guarded((T, E), torch.float32)
    G.view.copy_(torch.from_numpy(g))
    eqb.lei_inject_grad(G.view, torch.from_numpy(loads).cuda(), torch.from_numpy(off).cuda(), K, eta, c)
    torch.cuda.synchronize()
    assert G.intact()
    got = G.view.cpu().numpy()
    assert np.all(np.abs(got.astype(np.float64) - g_ref) <= LEI_ATOL + LEI_RTOL * np.abs(g_ref))


def test_lei_eta_zero_and_balanced_are_identity():
    T, E, K = 2048, 64, 8
    g = (np.random.default_rng(1).standard_normal((T, E)) * 0.1).astype(np.float32)
    off = np.array([0, 1024, 2048], np.int64)
    loads = np.full((2, E), K * 1024 // E, np.int32)  # perfectly balanced
    for eta, ld in [(0.0, np.random.default_rng(2).integers(0, 300, (2, E)).astype(np.int32)),
                    (1.0, loads)]:
        G = torch.from_numpy(g).cuda()
        eqb.lei_inject_grad(G, torch.from_numpy(ld).cuda(), torch.from_numpy(off).cuda(), K, eta, 1.0)
        torch.cuda.synchronize()
        assert np.array_equal(G.cpu().numpy(), g)


def test_lei_global_config_full_size_sampled():
    name = "global"
    sh = SHAPES[name]
    T, E = sh.T, sh.E
    off = even_offsets(T, sh.M)
    rng = np.random.default_rng(3)
    loads = rng.multinomial(sh.K * (T // sh.M), np.ones(E) / E, size=sh.M).astype(np.int32)
    G = make_grad(name, device="cuda")
    g0 = G.clone()
    eqb.lei_inject_grad(G, torch.from_numpy(loads).cuda(), torch.from_numpy(off).cuda(), sh.K, 2e-5, 1.0)
    rows = np.sort(rng.choice(T, 4096, replace=False))
    got = G[torch.from_numpy(rows).cuda()].cpu().numpy()
    g_rows = g0[torch.from_numpy(rows).cuda()].cpu().numpy()
    _, a = oracle.lei(None, loads, off, sh.K, 2e-5, 1.0)
    mb = np.searchsorted(off, rows, side="right") - 1
    want = (g_rows.astype(np.float64) + a[mb]).astype(np.float32)
    assert np.all(np.abs(got.astype(np.float64) - want) <= LEI_ATOL + LEI_RTOL * np.abs(want))


# ------------------------------------------------------------- device-side errors

def test_nonfinite_logit_sets_flag():
    z, b = rand_case(500, 64, seed=3)
    z[123, 7] = 0x7fc0  # NaN
    g = gpu_forward(z, b, 8, np.array([0, 500], np.int64))
    assert g["err"][0] == 4


def test_infinite_logit_sets_flag():
    z, b = rand_case(500, 64, seed=4)
    z[10, 3] = 0xff80  # -inf
    g = gpu_forward(z, b, 8, np.array([0, 500], np.int64))
    assert g["err"][0] == 4


def test_nonfinite_bias_sets_flag():
    z, b = rand_case(100, 64, seed=5)
    b[9] = np.inf
    g = gpu_forward(z, b, 8, np.array([0, 100], np.int64))
    assert g["err"][0] == 4


def test_huge_margin_refused_on_both_sides():
    """A finite margin of magnitude >= 2^127 shares kappa's high byte with
    the non-finite patterns: the kernels flag it (EQB_ERR_NONFINITE) and the
    oracle refuses it, the same reading on both sides."""
    z, b = rand_case(100, 64, seed=6)
    z[5, :] = brute.bf16_bits_from_f32(np.float32([3e38]))[0]
    z[5, 0] = brute.bf16_bits_from_f32(np.float32([-3e38]))[0]
    g = gpu_forward(z, b, 8, np.array([0, 100], np.int64))
    assert g["err"][0] == 4
    _, tau, _ = oracle.route(z, b, 8)
    with pytest.raises(oracle.OracleError):
        oracle.quantile(z, tau, oracle.target_rank(100, 64, 8), experts=[0])


@pytest.mark.parametrize("E", [64, 128, 256])
def test_margins_just_below_the_domain_limit(E):
    """Margins up to the largest bf16 below 2^127 (kappa high byte 0xfe at
    the top, 0x01 at the bottom) are inside the method's domain: no flag,
    and everything bit for bit against the oracle."""
    z, b = rand_case(300, E, seed=8 + E)
    big = brute.bf16_bits_from_f32(np.float32([1.6e38, -1.6e38]))
    z[:, 1] = big[1]           # expert 1: margins near +1.6e38
    z[::3, 2] = big[0]         # expert 2: in the top-K of every third token
    off = np.array([0, 150, 300], np.int64)
    assert_forward_equal(gpu_forward(z, b, 8, off), oracle_forward(z, b, 8, off))


def test_unreachable_rank_sets_flag():
    z, b = rand_case(100, 64, seed=7)
    _, tau, _ = oracle.route(z, b, 8)
    H = oracle.hist_hi(z, tau)
    u = torch.zeros(64, dtype=torch.uint8, device="cuda")
    rho = torch.zeros(64, dtype=torch.int32, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    eqb.eqb_select_quantile(torch.from_numpy(H).cuda(), 1, 101, u, rho, None, err)
    torch.cuda.synchronize()
    assert err.item() == 5


@pytest.mark.parametrize("E", [256, 1024])
@pytest.mark.parametrize("kind", ["narrow", "wide", "subnormal", "zeros"])
def test_bias_update_exact_against_oracle(kind, E):
    """The fixed-order fp64 centering of Eq. (2) reproduces the oracle bit for
    bit both when a tree sum is provably exact (narrow exponent span) and
    when it is not (wide span forces the ascending sequential sum)."""
    rng = np.random.default_rng(sum(map(ord, kind)) + E)
    v = (rng.standard_normal(E) * 3).astype(np.float32)
    if kind == "wide":
        v[::17] *= np.float32(1e30)
        v[5::23] *= np.float32(1e-30)
    elif kind == "subnormal":
        v[::3] = np.float32(1e-39)
    elif kind == "zeros":
        v[:] = 0.0
    q = brute.bf16_bits_from_f32(v)
    want = oracle.bias_update(q)
    bd = torch.zeros(E, dtype=torch.float32, device="cuda")
    eqb.eqb_bias_update(torch.from_numpy(q.view(np.int16)).view(torch.bfloat16).cuda(), bd)
    torch.cuda.synchronize()
    assert np.array_equal(bits_f32(bd.cpu().numpy()), bits_f32(want))


# ------------------------------------------------------------- one-call step

@pytest.mark.parametrize("T,E,K,M", [(300000, 256, 8, 11), (140000, 128, 6, 4), (5000, 64, 8, 3),
                                     (20000, 512, 8, 3)])
def test_layer_step_matches_oracle(T, E, K, M):
    """eqb_layer_step reproduces the oracle: routing, loads and the bias
    update bit for bit, LEI within tolerance."""
    z, b = rand_case(T, E, seed=T + E + K)
    off = ragged_offsets(T, M, seed=M)
    off[1] = off[2]  # one empty microbatch
    g = (np.random.default_rng(T).standard_normal((T, E)) * 0.1).astype(np.float32)
    eta, c = 0.25, 1.0
    o = oracle_forward(z, b, K, off)
    g_ref, _ = oracle.lei(g, o["loads"], off, K, eta, c)

    zd, bd = to_dev_bf16(z), torch.from_numpy(b).cuda()
    offd = torch.from_numpy(off).cuda()
    idx = Guarded((T, K), torch.int32)
    tau = Guarded((T,), torch.float32)
    loads = Guarded((M, E), torch.int32, fill=99)
    bn = Guarded((E,), torch.float32)
    G = Guarded((T, E), torch.float32)
    G.view.copy_(torch.from_numpy(g))
    ws = torch.zeros(eqb.eqb_layer_workspace_bytes(E), dtype=torch.uint8, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    eqb.eqb_layer_step(zd, bd, K, offd, loads.view, bn.view, ws, tau=tau.view, topk_idx=idx.view,
                       grad_s=G.view, eta=eta, c=c, mb_offsets_host=off, err_flag=err)
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


def test_layer_step_unreachable_rank_sets_flag():
    """A target rank above T cannot be reached: the selection that the
    coarse pass's last block runs inside the one-call step raises
    EQB_ERR_RANK, as the separate selection does."""
    T, E, K = 3000, 64, 8
    z, b = rand_case(T, E, seed=11)
    off = np.array([0, T], np.int64)
    loads = torch.zeros((1, E), dtype=torch.int32, device="cuda")
    bn = torch.zeros(E, dtype=torch.float32, device="cuda")
    ws = torch.zeros(eqb.eqb_layer_workspace_bytes(E), dtype=torch.uint8, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    eqb.eqb_layer_step(to_dev_bf16(z), torch.from_numpy(b).cuda(), K, torch.from_numpy(off).cuda(), loads, bn,
                       ws, r=T + 1, mb_offsets_host=off, err_flag=err)
    torch.cuda.synchronize()
    assert err.item() == 5


@pytest.mark.parametrize("T,E,K,M", [(200000, 256, 8, 8), (3000, 64, 8, 3)])
def test_layer_step_reuses_its_workspace(T, E, K, M):
    """Two steps on different inputs through one workspace: the second
    reproduces the oracle on its own inputs (the passes' block counters and
    histograms are cleared for every step, so each pass's last block
    selects again)."""
    ws = torch.full((eqb.eqb_layer_workspace_bytes(E),), 0x5a, dtype=torch.uint8, device="cuda")
    off = ragged_offsets(T, M, seed=M)
    offd = torch.from_numpy(off).cuda()
    for seed in (1, 2):
        z, b = rand_case(T, E, seed=T + seed)
        g = (np.random.default_rng(seed).standard_normal((T, E)) * 0.1).astype(np.float32)
        o = oracle_forward(z, b, K, off)
        g_ref, _ = oracle.lei(g, o["loads"], off, K, 0.5, 1.0)
        loads = torch.zeros((M, E), dtype=torch.int32, device="cuda")
        bn = torch.zeros(E, dtype=torch.float32, device="cuda")
        G = torch.from_numpy(g).cuda()
        err = torch.zeros(1, dtype=torch.int32, device="cuda")
        eqb.eqb_layer_step(to_dev_bf16(z), torch.from_numpy(b).cuda(), K, offd, loads, bn, ws, grad_s=G, eta=0.5,
                           c=1.0, mb_offsets_host=off, err_flag=err)
        torch.cuda.synchronize()
        assert err.item() == 0
        assert np.array_equal(loads.cpu().numpy(), o["loads"])
        assert np.array_equal(bits_f32(bn.cpu().numpy()), bits_f32(o["b_next"]))
        got = G.cpu().numpy().astype(np.float64)
        assert np.all(np.abs(got - g_ref) <= LEI_ATOL + LEI_RTOL * np.abs(g_ref))
