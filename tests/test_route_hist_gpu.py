"""GPU parity of routing with the coarse histogram from one read of z
(eqb_route_hist_fused) through the C ABI, and closed forms past the
65,535-token flush of the 16-bit block counters:

* top-K, cutoffs, loads and the coarse histogram bit for bit against the
  oracle and against eqb_route_topk (two kernels), including margins outside
  the one-read kernel's shared-memory bin window (counted in global memory),
  zero margins (b = 0), ragged and empty microbatches and ragged last tiles;
* T = 10,500,000 > 65,535 x the SM count: every block of the one-read kernel,
  of the coarse pass and of the fine pass counts more than 65,535 tokens, so
  their 16-bit counters are added into the global histograms mid-kernel;
  constant rows make H, the loads, the quantiles and the next bias known in
  closed form."""
import numpy as np
import pytest
import torch

import brute
import oracle
import paper_2609_28053_gb300 as eqb
from eqb_workloads import ragged_offsets
from gpu_harness import Guarded, bits_f32, oracle_forward, to_dev_bf16

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib(cuda_ok):
    eqb.load()


def case(T, E, seed, bias="normal", spread=False):
    rng = np.random.default_rng(seed)
    v = rng.standard_normal((T, E)).astype(np.float32)
    if spread:
        # margins outside [2^-15, 2^17) in both directions: huge logits, and
        # whole rows of tiny ones (tiny cutoffs and margins)
        m = rng.random((T, E))
        v[m < 0.02] *= np.float32(3e5)
        v[(m >= 0.02) & (m < 0.04)] *= np.float32(1e-7)
        v[rng.random(T) < 0.05] *= np.float32(1e-6)
    if bias == "zero":
        b = np.zeros(E, np.float32)
    else:
        b = (rng.standard_normal(E) * 0.3).astype(np.float32)
    return brute.bf16_bits_from_f32(v), b


def run(fn, z, b, K, off):
    T, E = z.shape
    M = len(off) - 1
    zd, bd = to_dev_bf16(z), torch.from_numpy(b).cuda()
    offd = torch.from_numpy(off).cuda()
    out = dict(idx=Guarded((T, K), torch.int32, fill=-7), tau=Guarded((T,), torch.float32),
               loads=Guarded((M, E), torch.int32), H=Guarded((E, 256), torch.int32),
               err=Guarded((1,), torch.int32))
    fn(zd, bd, K, offd, out["idx"].view, out["tau"].view, out["loads"].view, out["H"].view, out["err"].view)
    torch.cuda.synchronize()
    for k, v in out.items():
        assert v.intact(), f"write outside the {k} buffer"
    return {k: v.view.cpu().numpy() for k, v in out.items()}


@pytest.mark.parametrize("T,E,K,M,bias,spread", [
    (1, 128, 8, 1, "normal", False),
    (33, 256, 8, 2, "normal", False),
    (4099, 128, 8, 3, "zero", False),
    (20000, 256, 8, 5, "normal", True),
    (70001, 256, 6, 9, "zero", True),
    (50000, 128, 2, 64, "normal", False),
    (30000, 256, 15, 7, "normal", False),
    (30000, 128, 1, 3, "zero", True),
])
def test_route_hist_fused_matches_oracle(T, E, K, M, bias, spread):
    z, b = case(T, E, seed=T + E + K, bias=bias, spread=spread)
    off = ragged_offsets(T, M, seed=M) if T > M else np.array([0] + [T] * M, np.int64)
    if M > 2:
        off[1] = off[2]  # an empty microbatch
    fused = run(eqb.eqb_route_hist_fused, z, b, K, off)
    two = run(eqb.eqb_route_topk, z, b, K, off)
    o = oracle_forward(z, b, K, off)
    for g in (fused, two):
        assert g["err"][0] == 0
        assert np.array_equal(g["idx"], o["idx"])
        assert np.array_equal(bits_f32(g["tau"]), bits_f32(o["tau"]))
        assert np.array_equal(g["loads"], o["loads"])
        assert np.array_equal(g["H"], o["H"])


def test_route_hist_fused_rejects_other_widths():
    z = torch.zeros((64, 64), dtype=torch.bfloat16, device="cuda")
    b = torch.zeros(64, dtype=torch.float32, device="cuda")
    H = torch.zeros((64, 256), dtype=torch.int32, device="cuda")
    with pytest.raises(eqb.EqbError):
        eqb.eqb_route_hist_fused(z, b, 8, hist_hi=H)


def constant_rows(E):
    """z[t, e] = c_e, distinct bf16 values (c_e = -2 + 4 e / E)."""
    c = (-2.0 + 4.0 * np.arange(E) / E).astype(np.float32)
    row = brute.bf16_bits_from_f32(c)
    assert len(set(row.tolist())) == E
    return row, c


@pytest.mark.slow
@pytest.mark.parametrize("E", [128, 256])
def test_flush_crossing_closed_form(E):
    """T = 10,500,000 > 65,535 x 152: every block of the one-read kernel,
    of the coarse pass and of the fine pass counts more than 65,535 tokens,
    so the 16-bit block counters are added into the global histograms
    mid-kernel.  Constant rows (z[t, e] = c_e distinct, b = 0) have one
    cutoff for all tokens and one margin per expert, so in closed form:
    H[e, kappa(m_e) >> 8] = T, the top-K experts carry every token of every
    microbatch, q_hat_e = m_e and the next bias is the Eq. (2) centering of
    those margins."""
    T, K, M = 10_500_000, 8, 7
    row, c = constant_rows(E)
    zd = torch.from_numpy(row.astype(np.int16)).view(torch.bfloat16).cuda().expand(T, E).contiguous()
    bd = torch.zeros(E, dtype=torch.float32, device="cuda")
    off = np.linspace(0, T, M + 1).astype(np.int64)
    offd = torch.from_numpy(off).cuda()
    # the closed form: tau is the (K+1)-th largest c, margins bf16(tau - c_e)
    top = np.argsort(-c, kind="stable")
    tau = np.float32(c[top[K]])
    m = brute.bf16_bits_from_f32((tau - c).astype(np.float32))
    m = np.where(m == 0x8000, 0, m).astype(np.uint16)
    hb = np.array([oracle.kappa(int(x)) >> 8 for x in m])
    want_H = np.zeros((E, 256), np.int64)
    want_H[np.arange(E), hb] = T
    want_loads = np.zeros((M, E), np.int64)
    want_loads[:, top[:K]] = np.diff(off)[:, None]
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    taus = torch.empty(T, dtype=torch.float32, device="cuda")
    for fn in (eqb.eqb_route_hist_fused, eqb.eqb_route_topk):
        H = torch.zeros((E, 256), dtype=torch.int32, device="cuda")
        loads = torch.zeros((M, E), dtype=torch.int32, device="cuda")
        fn(zd, bd, K, offd, None, taus, loads, H, err)
        torch.cuda.synchronize()
        assert err.item() == 0
        assert np.array_equal(H.cpu().numpy(), want_H)
        assert torch.all(taus == torch.tensor(float(tau), device="cuda")).item()
        assert np.array_equal(loads.cpu().numpy(), want_loads)
        del H
    del taus
    # the whole step (the fine pass included): the quantile of expert e is m_e
    ws = torch.zeros(eqb.eqb_layer_workspace_bytes(E), dtype=torch.uint8, device="cuda")
    bn = torch.empty(E, dtype=torch.float32, device="cuda")
    loads = torch.zeros((M, E), dtype=torch.int32, device="cuda")
    eqb.eqb_layer_step(zd, bd, K, offd, loads, bn, ws, mb_offsets_host=off, err_flag=err)
    torch.cuda.synchronize()
    assert err.item() == 0
    assert np.array_equal(bits_f32(bn.cpu().numpy()), bits_f32(oracle.bias_update(m)))
    assert np.array_equal(loads.cpu().numpy(), want_loads)
