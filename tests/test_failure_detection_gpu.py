"""Failure detection without a GPU fault: a bounded wait that runs out
reports EQB_ERR_CUDA through the error word, and the context keeps working
(the next calls run and match the oracle)."""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_28053_gb300 as eqb
from gpu_harness import gpu_forward, oracle_forward

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib(cuda_ok):
    eqb.load()


def test_stalled_wait_reports_and_context_survives():
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    eqb.eqb_selftest_stalled_wait(err, polls=1 << 14)
    torch.cuda.synchronize()
    assert err.item() == 3  # EQB_ERR_CUDA
    # the context is intact: a full forward statistic still matches the oracle
    rng = np.random.default_rng(0)
    import brute
    z = brute.bf16_bits_from_f32(rng.standard_normal((500, 64)).astype(np.float32))
    b = np.zeros(64, np.float32)
    off = np.array([0, 200, 500], np.int64)
    g = gpu_forward(z, b, 8, off)
    o = oracle_forward(z, b, 8, off)
    assert np.array_equal(g["idx"], o["idx"]) and np.array_equal(g["q"], o["q"])
    assert g["err"][0] == 0


def test_error_word_is_sticky_first_code():
    """A later error does not overwrite the first one (atomic CAS from 0)."""
    err = torch.full((1,), 4, dtype=torch.int32, device="cuda")
    eqb.eqb_selftest_stalled_wait(err, polls=64)
    torch.cuda.synchronize()
    assert err.item() == 4
