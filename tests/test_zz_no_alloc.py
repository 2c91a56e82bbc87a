"""The allocation-free step entry point (eqb_layer_step_noalloc) gives the
same results as eqb_layer_step with a caller-provided workspace.

It exists for callers that cannot allocate device memory (plugins inside a
framework that owns the device memory pool, code that must not stall on an
allocation); its scratch is an array inside the library shared by all
calls.  Two calls in a row check that a call does not depend on what the
previous call left in that array.  This file is collected last so that a
run stopping at the first failure has run everything else first."""
import numpy as np
import pytest
import torch

import paper_2609_28053_gb300 as eqb
from eqb_workloads import make_bias, make_grad, make_logits, ragged_offsets
from gpu_harness import bits_f32

pytestmark = pytest.mark.gpu

LEI_ATOL, LEI_RTOL = 1e-7, 1e-5


@pytest.fixture(scope="module", autouse=True)
def _lib(cuda_ok):
    eqb.load()


def run_step(fn, z, b, K, off_d, off_h, g, **kw):
    T, E = z.shape
    M = off_d.numel() - 1
    idx = torch.full((T, K), -1, dtype=torch.int32, device="cuda")
    tau = torch.full((T,), -1.0, dtype=torch.float32, device="cuda")
    loads = torch.full((M, E), 7, dtype=torch.int32, device="cuda")
    bn = torch.zeros(E, dtype=torch.float32, device="cuda")
    gg = g.clone()
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    fn(z, b, K, off_d, loads, bn, tau=tau, topk_idx=idx, grad_s=gg, eta=0.25, c=1.0,
       mb_offsets_host=off_h, err_flag=err, **kw)
    torch.cuda.synchronize()
    assert err.item() == 0
    return idx.cpu().numpy(), tau.cpu().numpy(), loads.cpu().numpy(), bn.cpu().numpy(), gg.cpu().numpy()


@pytest.mark.parametrize("name,T", [("global", 200000), ("tie", 65536), ("tiny", 4096)])
def test_noalloc_step_matches_workspace_step_twice(name, T):
    z = make_logits(name, T=T, device="cuda")
    E = z.shape[1]
    K = {"global": 8, "tie": 8, "tiny": 2}[name]
    b = make_bias(name, device="cuda")
    g = make_grad(name, T=T, device="cuda")
    off_h = ragged_offsets(T, 7, seed=T)
    off_d = torch.from_numpy(off_h).cuda()
    ws = torch.zeros(eqb.eqb_layer_workspace_bytes(E), dtype=torch.uint8, device="cuda")
    want = run_step(lambda *a, **k: eqb.eqb_layer_step(*a[:6], ws, **k), z, b, K, off_d, off_h, g)
    for _ in range(2):  # the second call starts from the first call's scratch contents
        got = run_step(eqb.eqb_layer_step_noalloc, z, b, K, off_d, off_h, g)
        assert np.array_equal(got[0], want[0])
        assert np.array_equal(bits_f32(got[1]), bits_f32(want[1]))
        assert np.array_equal(got[2], want[2])
        assert np.array_equal(bits_f32(got[3]), bits_f32(want[3]))
        d = np.abs(got[4].astype(np.float64) - want[4])
        assert np.all(d <= LEI_ATOL + LEI_RTOL * np.abs(want[4]))


def test_noalloc_rejects_too_many_experts():
    z = torch.zeros((4, 264), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(eqb.EqbError):
        eqb.eqb_layer_step_noalloc(z, torch.zeros(264, device="cuda"), 8,
                                   torch.tensor([0, 4], dtype=torch.int64, device="cuda"),
                                   torch.zeros((1, 264), dtype=torch.int32, device="cuda"),
                                   torch.zeros(264, device="cuda"))
