"""The C-ABI library builds, loads without a GPU, exports every entry point
that include/eqb.h declares, and rejects invalid calls on the host before
any CUDA call (so these run on a CPU-only machine)."""
import ctypes
import os
import re
import shutil

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "eqb.h")

pytestmark = pytest.mark.skipif(shutil.which("nvcc") is None and not os.path.exists(
    os.path.join(ROOT, "paper_2609_28053_gb300", "libeqb.so")), reason="no nvcc and no prebuilt library")


@pytest.fixture(scope="module")
def lib():
    from paper_2609_28053_gb300 import build, _lib
    build.build()
    return _lib.load()


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    names = re.findall(r"^\s*(?:const\s+)?[A-Za-z_][\w\s\*]*?\b((?:eqb|lei)_\w+)\s*\(", src, re.M)
    return sorted(set(names))


def test_header_declares_the_paper_entry_points():
    names = declared_functions()
    for n in ("eqb_route_topk", "eqb_margin_hist_pass1", "eqb_margin_hist_pass2",
              "eqb_select_quantile", "eqb_bias_update", "lei_inject_grad", "eqb_target_rank"):
        assert n in names


def test_every_declared_symbol_is_exported(lib):
    for n in declared_functions():
        assert hasattr(lib, n), f"{n} declared in eqb.h but not exported"


def test_status_strings_and_version(lib):
    for code, name in [(0, b"EQB_OK"), (1, b"EQB_ERR_INVALID_ARG"), (2, b"EQB_ERR_UNSUPPORTED"),
                       (3, b"EQB_ERR_CUDA"), (4, b"EQB_ERR_NONFINITE"), (5, b"EQB_ERR_RANK")]:
        assert lib.eqb_status_string(code) == name
    assert lib.eqb_version() >= 100


def test_target_rank(lib):
    assert lib.eqb_target_rank(2097152, 256, 8) == 65536
    assert lib.eqb_target_rank(10, 8, 3) == 4
    assert lib.eqb_target_rank(-1, 8, 3) == -1
    assert lib.eqb_target_rank(10, 0, 3) == -1


# A fake, well-aligned address: invalid calls must return before using it.
FAKE = ctypes.c_void_p(0x10000)
MISALIGNED = ctypes.c_void_p(0x10002)
NULL = None
INVALID, UNSUPPORTED = 1, 2


def route(lib, z=FAKE, b=FAKE, T=64, E=64, K=8, off=FAKE, M=1, idx=FAKE, tau=FAKE, loads=FAKE,
          hist=FAKE, err=FAKE):
    return lib.eqb_route_topk(z, b, T, E, K, off, M, idx, tau, loads, hist, err, NULL)


@pytest.mark.parametrize("kw,code", [
    (dict(K=0), INVALID), (dict(K=64), INVALID), (dict(T=-1), INVALID), (dict(E=1), INVALID),
    (dict(E=12), UNSUPPORTED), (dict(E=1032), UNSUPPORTED), (dict(E=64, K=32), UNSUPPORTED),
    (dict(T=1 << 31), UNSUPPORTED), (dict(z=NULL), INVALID), (dict(b=NULL), INVALID),
    (dict(tau=NULL), INVALID), (dict(off=NULL), INVALID), (dict(M=0), INVALID),
    (dict(z=MISALIGNED), INVALID), (dict(tau=MISALIGNED), INVALID),
])
def test_route_rejects(lib, kw, code):
    assert route(lib, **kw) == code


def test_route_zero_tokens_is_a_noop(lib):
    assert route(lib, T=0) == 0


def test_hist_and_select_reject(lib):
    assert lib.eqb_margin_hist_pass1(NULL, FAKE, 10, 64, FAKE, NULL, NULL) == INVALID
    assert lib.eqb_margin_hist_pass1(FAKE, FAKE, 10, 60, FAKE, NULL, NULL) == UNSUPPORTED
    assert lib.eqb_margin_hist_pass1(FAKE, FAKE, 0, 64, FAKE, NULL, NULL) == 0
    assert lib.eqb_margin_hist_pass2(FAKE, FAKE, 10, 64, NULL, FAKE, NULL) == INVALID
    assert lib.eqb_margin_hist_pass2(MISALIGNED, FAKE, 10, 64, FAKE, FAKE, NULL) == INVALID
    assert lib.eqb_select_quantile(FAKE, 64, 3, 5, FAKE, FAKE, FAKE, NULL, NULL) == INVALID
    assert lib.eqb_select_quantile(FAKE, 64, 1, 0, FAKE, FAKE, NULL, NULL, NULL) == INVALID
    assert lib.eqb_select_quantile(FAKE, 64, 2, 5, FAKE, FAKE, NULL, NULL, NULL) == INVALID
    assert lib.eqb_select_quantile(FAKE, 300, 1, 5, FAKE, FAKE, NULL, NULL, NULL) == UNSUPPORTED
    assert lib.eqb_bias_update(FAKE, 0, FAKE, NULL) == INVALID
    assert lib.eqb_bias_update(FAKE, 1025, FAKE, NULL) == UNSUPPORTED


def test_lei_rejects(lib):
    f = lib.lei_inject_grad
    assert f(NULL, FAKE, FAKE, 1, 10, 64, 8, ctypes.c_float(1.0), ctypes.c_float(1.0), NULL) == INVALID
    assert f(FAKE, FAKE, FAKE, 0, 10, 64, 8, ctypes.c_float(1.0), ctypes.c_float(1.0), NULL) == INVALID
    assert f(MISALIGNED, FAKE, FAKE, 1, 10, 64, 8, ctypes.c_float(1.0), ctypes.c_float(1.0), NULL) == INVALID
    assert f(FAKE, FAKE, FAKE, 1, 10, 64, 8, ctypes.c_float(float("nan")), ctypes.c_float(1.0), NULL) == INVALID
    assert f(FAKE, FAKE, FAKE, 1, 0, 64, 8, ctypes.c_float(1.0), ctypes.c_float(1.0), NULL) == 0


def test_lei_coefficients_rejects(lib):
    f = lib.lei_coefficients
    one = ctypes.c_float(1.0)
    assert f(NULL, FAKE, 1, 64, 8, one, one, FAKE, NULL) == INVALID
    assert f(FAKE, FAKE, 0, 64, 8, one, one, FAKE, NULL) == INVALID
    assert f(FAKE, FAKE, 1, 64, 8, one, one, NULL, NULL) == INVALID
    assert f(FAKE, FAKE, 1, 64, 8, one, one, MISALIGNED, NULL) == INVALID
    assert f(FAKE, FAKE, 1, 64, 64, one, one, FAKE, NULL) == INVALID  # K >= E
    assert f(FAKE, FAKE, 1, 64, 8, ctypes.c_float(float("nan")), one, FAKE, NULL) == INVALID
    assert f(FAKE, FAKE, 1, 2048, 8, one, one, FAKE, NULL) == UNSUPPORTED


def test_fused_pass_rejects(lib):
    f = lib.eqb_margin_hist_lei

    def call(T=100, E=64, pass_=1, u=FAKE, grad=FAKE, coef=FAKE, off=FAKE, M=1, t0=0, t1=100, z=FAKE):
        return f(z, FAKE, T, E, pass_, u, FAKE, NULL, grad, coef, off, M, t0, t1, NULL)

    assert call(pass_=3) == INVALID
    assert call(pass_=2, u=NULL) == INVALID
    assert call(grad=NULL) == INVALID
    assert call(coef=NULL) == INVALID
    assert call(off=NULL) == INVALID
    assert call(M=0) == INVALID
    assert call(t0=-1) == INVALID
    assert call(t0=50, t1=40) == INVALID
    assert call(t1=101) == INVALID
    assert call(grad=MISALIGNED) == INVALID
    assert call(coef=MISALIGNED) == INVALID
    assert call(z=MISALIGNED) == INVALID
    assert call(E=12) == UNSUPPORTED
    assert call(T=0, t1=0) == 0


def test_route_hist_fused_rejects(lib):
    """Routing + coarse histogram in one kernel: host-side rejection of bad
    calls, nothing launched."""
    f = lib.eqb_route_hist_fused

    def call(T=100, E=256, K=8, M=2, off=FAKE, loads=FAKE, hist=FAKE, tau=FAKE, z=FAKE):
        return f(z, FAKE, T, E, K, off, M, FAKE, tau, loads, hist, NULL, NULL)

    assert call(E=64) == UNSUPPORTED            # only E = 128 and 256
    assert call(E=384) == UNSUPPORTED
    assert call(K=16) == UNSUPPORTED            # K + 1 > 16
    assert call(hist=NULL) == INVALID
    assert call(tau=NULL) == INVALID
    assert call(off=NULL) == INVALID            # loads given without offsets
    assert call(M=0) == INVALID
    assert call(z=MISALIGNED) == INVALID
    assert call(K=0) == INVALID
    assert call(loads=NULL, off=NULL, M=0, T=0) == 0


def test_binding_fails_loudly_without_library(tmp_path):
    from paper_2609_28053_gb300 import _lib
    with pytest.raises(RuntimeError, match="no CPU fallback"):
        _lib.load(str(tmp_path / "missing.so"))


def test_router_logits_rejects(lib):
    f = lib.eqb_router_logits
    assert f(FAKE, FAKE, 10, 4096, 8, FAKE, NULL, NULL) == UNSUPPORTED     # E not a multiple of 16
    assert f(FAKE, FAKE, 10, 4000, 128, FAKE, NULL, NULL) == UNSUPPORTED   # d not a multiple of 64
    assert f(FAKE, FAKE, 10, 4096, 272, FAKE, NULL, NULL) == UNSUPPORTED   # E > 256
    assert f(NULL, FAKE, 10, 4096, 128, FAKE, NULL, NULL) == INVALID
    assert f(FAKE, FAKE, -1, 4096, 128, FAKE, NULL, NULL) == INVALID
    assert f(MISALIGNED, FAKE, 10, 4096, 128, FAKE, NULL, NULL) == INVALID
    assert f(FAKE, FAKE, 0, 4096, 128, FAKE, NULL, NULL) == 0


def test_router_route_rejects(lib):
    f = lib.eqb_router_route

    def call(x=FAKE, T=10, d=4096, E=128, K=8, b=FAKE, off=FAKE, M=1, z=FAKE, idx=FAKE, tau=FAKE,
             loads=FAKE, hist=NULL):
        return f(x, FAKE, T, d, E, K, b, off, M, z, idx, tau, loads, hist, NULL, NULL)

    assert call(E=256) == UNSUPPORTED       # fused routing only for E in {64, 128}
    assert call(E=96) == UNSUPPORTED
    assert call(K=9) == UNSUPPORTED         # K + 1 <= 9
    assert call(d=4000) == UNSUPPORTED      # d not a multiple of 64
    assert call(K=0) == INVALID
    assert call(E=64, K=64) == INVALID
    assert call(x=NULL) == INVALID
    assert call(b=NULL) == INVALID
    assert call(tau=NULL) == INVALID
    assert call(off=NULL) == INVALID        # loads without offsets
    assert call(M=0) == INVALID
    assert call(x=MISALIGNED) == INVALID
    assert call(hist=MISALIGNED) == INVALID
    assert call(T=-1) == INVALID
    assert call(T=0) == 0
    assert call(T=0, hist=FAKE) == 0
    assert call(T=0, off=NULL, loads=NULL, idx=NULL) == 0


def test_layer_step_workspace_size(lib):
    assert lib.eqb_layer_workspace_bytes(256) >= 2 * 256 * 256 * 4 + 256 * 7
    assert lib.eqb_layer_workspace_bytes(256) % 256 == 0
    assert lib.eqb_layer_workspace_bytes(0) == 0
    # the size the header and the allocation-free entry point state
    assert lib.eqb_layer_workspace_bytes(256) == 788480
    src = open(HEADER).read()
    assert "788,480 bytes" in src


def test_layer_step_rejects(lib):
    import numpy as np
    f = lib.eqb_layer_step
    ws = lib.eqb_layer_workspace_bytes(64)
    good = np.array([0, 40, 100], np.int64)
    bad = np.array([0, 60, 50], np.int64)
    short = np.array([0, 40, 99], np.int64)
    fl = ctypes.c_float(0.0)

    def call(T=100, E=64, K=8, off_h=good, ws_bytes=ws, workspace=FAKE, z=FAKE, M=2):
        hp = None if off_h is None else off_h.ctypes.data_as(ctypes.c_void_p)
        return f(z, FAKE, T, E, K, FAKE, hp, M, 0, FAKE, FAKE, FAKE, FAKE, NULL, fl, fl,
                 workspace, ws_bytes, NULL, NULL)
    assert call(off_h=bad) == INVALID          # decreasing offsets
    assert call(off_h=short) == INVALID        # offsets do not end at T
    assert call(ws_bytes=ws - 1) == INVALID    # workspace too small
    assert call(workspace=NULL) == INVALID
    assert call(workspace=ctypes.c_void_p(0x10010)) == INVALID  # not 256-byte aligned
    assert call(z=NULL) == INVALID
    assert call(T=0) == INVALID
    assert call(E=60) == UNSUPPORTED


def test_router_layer_step_rejects(lib):
    import numpy as np
    f = lib.eqb_router_layer_step
    ws = lib.eqb_layer_workspace_bytes(128)
    good = np.array([0, 40, 100], np.int64)
    bad = np.array([0, 60, 50], np.int64)
    fl = ctypes.c_float(0.0)

    def call(x=FAKE, T=100, d=4096, E=128, K=8, off_h=good, ws_bytes=ws, z=FAKE, M=2):
        hp = None if off_h is None else off_h.ctypes.data_as(ctypes.c_void_p)
        return f(x, FAKE, T, d, E, K, FAKE, FAKE, hp, M, 0, z, FAKE, FAKE, FAKE, FAKE, NULL, fl, fl,
                 FAKE, ws_bytes, NULL, NULL)
    assert call(x=NULL) == INVALID
    assert call(x=MISALIGNED) == INVALID
    assert call(d=4000) == UNSUPPORTED         # d not a multiple of 64
    assert call(E=72) == UNSUPPORTED           # E not a multiple of 16
    assert call(off_h=bad) == INVALID
    assert call(ws_bytes=ws - 1) == INVALID
    assert call(z=NULL) == INVALID
    assert call(K=0) == INVALID


def test_maxvio_rejects(lib):
    f = lib.eqb_maxvio
    assert f(FAKE, FAKE, 0, 8, 2, FAKE, NULL, NULL) == INVALID
    assert f(FAKE, FAKE, 16385, 8, 2, FAKE, NULL, NULL) == UNSUPPORTED
    assert f(NULL, FAKE, 4, 8, 2, FAKE, NULL, NULL) == INVALID
    assert f(FAKE, FAKE, 4, 8, 2, NULL, NULL, NULL) == INVALID
    assert f(FAKE, FAKE, 4, 0, 2, FAKE, NULL, NULL) == INVALID
    assert f(FAKE, FAKE, 4, 8, 2, ctypes.c_void_p(0x10004), NULL, NULL) == INVALID  # maxvio not 8-aligned


def test_gshard_rejects(lib):
    f = lib.gshard_inject_grad
    a = ctypes.c_float(0.01)
    assert f(FAKE, FAKE, FAKE, FAKE, 2, 10, 12, 2, a, NULL) == UNSUPPORTED     # E % 8
    assert f(FAKE, FAKE, FAKE, FAKE, 2, 10, 1032, 2, a, NULL) == UNSUPPORTED   # E > 1024
    assert f(NULL, FAKE, FAKE, FAKE, 2, 10, 64, 2, a, NULL) == INVALID
    assert f(MISALIGNED, FAKE, FAKE, FAKE, 2, 10, 64, 2, a, NULL) == INVALID
    assert f(FAKE, FAKE, FAKE, FAKE, 2, 10, 64, 2, ctypes.c_float(float("nan")), NULL) == INVALID
    assert f(FAKE, FAKE, FAKE, FAKE, 0, 10, 64, 2, a, NULL) == INVALID
    assert f(FAKE, FAKE, FAKE, FAKE, 2, 0, 64, 2, a, NULL) == 0


def test_comparison_statistics_reject(lib):
    import numpy as np
    ws = lib.eqb_rank_averaged_workspace_bytes(64, 2)
    assert ws >= 2 * 2 * 64 * 256 * 4
    good = np.array([0, 40, 100], np.int64)
    bad = np.array([0, 60, 50], np.int64)
    f = lib.eqb_rank_averaged_bias

    def ra(off=good, P=2, q=FAKE, wsb=ws, E=64):
        return f(FAKE, FAKE, 100, E, 8, None if off is None else off.ctypes.data_as(ctypes.c_void_p), P, q,
                 FAKE, FAKE, wsb, NULL, NULL)
    assert ra(off=bad) == INVALID
    assert ra(off=None) == INVALID
    assert ra(q=NULL) == INVALID
    assert ra(wsb=ws - 1) == INVALID
    assert ra(E=1032) == UNSUPPORTED
    ws = lib.eqb_layer_workspace_bytes(64)
    g = lib.eqb_fixed_hist_bias
    fl = ctypes.c_float
    assert g(FAKE, FAKE, 100, 64, 8, fl(-1.0), fl(0.0), FAKE, NULL, FAKE, ws, NULL, NULL) == INVALID
    assert g(FAKE, FAKE, 100, 64, 8, fl(float("nan")), fl(0.1), FAKE, NULL, FAKE, ws, NULL, NULL) == INVALID
    assert g(FAKE, FAKE, 100, 64, 8, fl(-1.0), fl(0.1), FAKE, NULL, FAKE, ws - 1, NULL, NULL) == INVALID
    assert g(FAKE, FAKE, 100, 64, 8, fl(-1.0), fl(0.1), FAKE, ctypes.c_void_p(0x10004), FAKE, ws, NULL,
             NULL) == INVALID


def test_selftest_rejects(lib):
    f = lib.eqb_selftest_stalled_wait
    assert f(NULL, 100, NULL) == INVALID
    assert f(FAKE, 0, NULL) == INVALID
    assert f(FAKE, (1 << 24) + 1, NULL) == INVALID
    assert f(MISALIGNED, 100, NULL) == INVALID


def test_noalloc_wrapper_requires_the_current_device(monkeypatch):
    """eqb_layer_step_noalloc takes its scratch array on the current device,
    so the binding refuses tensors that live on another one (checked before
    any call into the library; a stand-in tensor and a stubbed current
    device, no GPU needed)."""
    import torch
    import paper_2609_28053_gb300 as eqb

    class Dev:
        index = 0

    class Fake:
        device = Dev()

    monkeypatch.setattr(torch.cuda, "current_device", lambda: 1)
    with pytest.raises(ValueError, match="current device"):
        eqb._on_current_device(Fake(), "z")
    monkeypatch.setattr(torch.cuda, "current_device", lambda: 0)
    eqb._on_current_device(Fake(), "z")  # same device: accepted
