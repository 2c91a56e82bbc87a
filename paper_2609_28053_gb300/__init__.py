"""GB300-native EQB + LEI routing-balance path (arXiv 2609.28053).

Thin Python binding over the C ABI of ``libeqb.so`` (include/eqb.h).  Each
function has the C entry point's name, checks dtypes/devices/shapes, and
passes raw device pointers plus the current CUDA stream; every step of the
path runs in the library's CUDA kernels.  PyTorch provides device memory
and streams only.

The routing-balance step of one MoE layer, in the paper's order:

    eqb_route_topk        Sec. 2: top-K of z + b, cutoff tau_t, loads f_e
                          (+ Algorithm 1 step 1, the coarse histogram)
    eqb_select_quantile   Algorithm 1 step 3 (pass 1): u_e, rho_e
    eqb_margin_hist_pass2 Algorithm 1 step 4: fine histogram
    eqb_select_quantile   Algorithm 1 steps 5-6 (pass 2): exact quantile
    eqb_bias_update       Eq. (2): centred bias for the next step
    lei_inject_grad       Sec. 4: Eq. (LEI) with Eq. (norm)

and, for layers whose logits are produced here, eqb_router_logits (Sec. 2,
z_t = W_r x_t) on the tensor cores.
"""
from __future__ import annotations

import ctypes

import torch

from ._lib import STATUS, EqbError, load

__all__ = [
    "EqbError", "STATUS", "load", "eqb_target_rank", "eqb_route_topk", "eqb_margin_hist_pass1",
    "eqb_margin_hist_pass2", "eqb_select_quantile", "eqb_bias_update", "lei_inject_grad",
    "EqbWorkspace", "eqb_layer_forward", "eqb_router_logits", "eqb_layer_workspace_bytes",
    "eqb_layer_step", "eqb_layer_step_noalloc", "eqb_router_route", "eqb_router_layer_step",
    "eqb_maxvio", "gshard_inject_grad", "eqb_rank_averaged_bias", "eqb_fixed_hist_bias",
    "eqb_rank_averaged_workspace_bytes", "eqb_selftest_stalled_wait", "lei_coefficients",
    "eqb_margin_hist_lei",
]


def _p(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _need(t, dtype, name, shape=None):
    if t is None:
        return
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} must have shape {tuple(shape)}, got {tuple(t.shape)}")


def _on_current_device(t, name):
    """The library takes its scratch and streams from the CUDA device that is
    current when it is called: the tensors must live on that device."""
    cur = torch.cuda.current_device()
    if t.device.index != cur:
        raise ValueError(f"{name} is on cuda:{t.device.index} but cuda:{cur} is the current device; "
                         f"call inside torch.cuda.device({t.device})")


def _check(rc, what):
    if rc != 0:
        raise EqbError(rc, what)


def eqb_target_rank(T: int, E: int, K: int) -> int:
    return int(load().eqb_target_rank(T, E, K))


def eqb_route_topk(z, b, K, mb_offsets=None, topk_idx=None, tau=None, loads=None, hist_hi=None,
                   err_flag=None, stream=None):
    """Top-K routing, cutoffs and loads (+ optional coarse histogram).
    z bf16 [T,E]; b fp32 [E]; mb_offsets int64 [M+1]; outputs as in eqb.h.
    loads and hist_hi are accumulated into.  Returns (topk_idx, tau)."""
    T, E = z.shape
    _need(z, torch.bfloat16, "z")
    _need(b, torch.float32, "b", (E,))
    if tau is None:
        tau = torch.empty(T, dtype=torch.float32, device=z.device)
    _need(tau, torch.float32, "tau", (T,))
    _need(topk_idx, torch.int32, "topk_idx", (T, K))
    M = 0
    if mb_offsets is not None:
        _need(mb_offsets, torch.int64, "mb_offsets")
        M = mb_offsets.numel() - 1
    _need(loads, torch.int32, "loads", (M, E) if loads is not None else None)
    _need(hist_hi, torch.int32, "hist_hi", (E, 256))
    _need(err_flag, torch.int32, "err_flag")
    rc = load().eqb_route_topk(_p(z), _p(b), T, E, K, _p(mb_offsets), M, _p(topk_idx), _p(tau),
                               _p(loads), _p(hist_hi), _p(err_flag), _stream(stream))
    _check(rc, "eqb_route_topk")
    return topk_idx, tau


def eqb_route_hist_fused(z, b, K, mb_offsets=None, topk_idx=None, tau=None, loads=None, hist_hi=None,
                         err_flag=None, stream=None):
    """Routing and the coarse histogram from one kernel that reads z once
    (E = 128 or 256): the outputs of eqb_route_topk with hist_hi, bit for
    bit.  Returns tau."""
    T, E = z.shape
    _need(z, torch.bfloat16, "z")
    _need(b, torch.float32, "b", (E,))
    if tau is None:
        tau = torch.empty(T, dtype=torch.float32, device=z.device)
    _need(tau, torch.float32, "tau", (T,))
    _need(topk_idx, torch.int32, "topk_idx", (T, K))
    _need(mb_offsets, torch.int64, "mb_offsets")
    M = 0 if mb_offsets is None else mb_offsets.numel() - 1
    _need(loads, torch.int32, "loads", (M, E) if loads is not None else None)
    _need(hist_hi, torch.int32, "hist_hi", (E, 256))
    if hist_hi is None:
        raise ValueError("hist_hi is required")
    _need(err_flag, torch.int32, "err_flag")
    _check(load().eqb_route_hist_fused(_p(z), _p(b), T, E, int(K), _p(mb_offsets), M, _p(topk_idx), _p(tau),
                                       _p(loads), _p(hist_hi), _p(err_flag), _stream(stream)),
           "eqb_route_hist_fused")
    return tau


def eqb_margin_hist_pass1(z, tau, hist_hi, err_flag=None, stream=None):
    T, E = z.shape
    _need(z, torch.bfloat16, "z")
    _need(tau, torch.float32, "tau", (T,))
    _need(hist_hi, torch.int32, "hist_hi", (E, 256))
    _need(err_flag, torch.int32, "err_flag")
    _check(load().eqb_margin_hist_pass1(_p(z), _p(tau), T, E, _p(hist_hi), _p(err_flag),
                                        _stream(stream)), "eqb_margin_hist_pass1")


def eqb_margin_hist_pass2(z, tau, u, hist_lo, stream=None):
    T, E = z.shape
    _need(z, torch.bfloat16, "z")
    _need(tau, torch.float32, "tau", (T,))
    _need(u, torch.uint8, "u", (E,))
    _need(hist_lo, torch.int32, "hist_lo", (E, 256))
    _check(load().eqb_margin_hist_pass2(_p(z), _p(tau), T, E, _p(u), _p(hist_lo), _stream(stream)),
           "eqb_margin_hist_pass2")


def eqb_select_quantile(hist, pass_, r, u, rho, q_hat=None, err_flag=None, stream=None):
    E = hist.shape[0]
    _need(hist, torch.int32, "hist", (E, 256))
    _need(u, torch.uint8, "u", (E,))
    _need(rho, torch.int32, "rho", (E,))
    _need(q_hat, torch.bfloat16, "q_hat", (E,))
    _need(err_flag, torch.int32, "err_flag")
    _check(load().eqb_select_quantile(_p(hist), E, int(pass_), int(r), _p(u), _p(rho), _p(q_hat),
                                      _p(err_flag), _stream(stream)), "eqb_select_quantile")


def eqb_bias_update(q_hat, b_next, stream=None):
    E = q_hat.shape[0]
    _need(q_hat, torch.bfloat16, "q_hat", (E,))
    _need(b_next, torch.float32, "b_next", (E,))
    _check(load().eqb_bias_update(_p(q_hat), E, _p(b_next), _stream(stream)), "eqb_bias_update")


def lei_inject_grad(grad_s, loads, mb_offsets, K, eta, c, stream=None):
    T, E = grad_s.shape
    _need(grad_s, torch.float32, "grad_s")
    _need(mb_offsets, torch.int64, "mb_offsets")
    M = mb_offsets.numel() - 1
    _need(loads, torch.int32, "loads", (M, E))
    _check(load().lei_inject_grad(_p(grad_s), _p(loads), _p(mb_offsets), M, T, E, K, float(eta),
                                  float(c), _stream(stream)), "lei_inject_grad")


def lei_coefficients(loads, mb_offsets, K, eta, c, coef=None, stream=None):
    """The [M,E] table of LEI coefficients eta * sigma_l * rho_{l,e} (the
    values lei_inject_grad adds).  Returns coef (fp32 [M,E])."""
    M, E = loads.shape
    _need(loads, torch.int32, "loads")
    _need(mb_offsets, torch.int64, "mb_offsets", (M + 1,))
    if coef is None:
        coef = torch.empty((M, E), dtype=torch.float32, device=loads.device)
    _need(coef, torch.float32, "coef", (M, E))
    _check(load().lei_coefficients(_p(loads), _p(mb_offsets), M, E, int(K), float(eta), float(c), _p(coef),
                                   _stream(stream)), "lei_coefficients")
    return coef


def eqb_margin_hist_lei(z, tau, pass_, hist, grad_s, coef, mb_offsets, lei_t0, lei_t1, u=None,
                        err_flag=None, stream=None):
    """A histogram pass (1: coarse, 2: fine, needs u) with grad_s[t] +=
    coef[mb(t)] for t in [lei_t0, lei_t1) streamed beside it, one kernel."""
    T, E = z.shape
    _need(z, torch.bfloat16, "z")
    _need(tau, torch.float32, "tau", (T,))
    _need(hist, torch.int32, "hist", (E, 256))
    _need(u, torch.uint8, "u", (E,))
    _need(err_flag, torch.int32, "err_flag")
    _need(grad_s, torch.float32, "grad_s", (T, E))
    _need(mb_offsets, torch.int64, "mb_offsets")
    M = mb_offsets.numel() - 1
    _need(coef, torch.float32, "coef", (M, E))
    _check(load().eqb_margin_hist_lei(_p(z), _p(tau), T, E, int(pass_), _p(u), _p(hist), _p(err_flag),
                                      _p(grad_s), _p(coef), _p(mb_offsets), M, int(lei_t0), int(lei_t1),
                                      _stream(stream)), "eqb_margin_hist_lei")


def eqb_router_logits(x, W_r, z=None, err_flag=None, stream=None):
    """Router logits z = bf16(x W_r^T), fp32 accumulation on the tensor cores.
    x bf16 [T,d], W_r bf16 [E,d]; returns z bf16 [T,E]."""
    T, d = x.shape
    E = W_r.shape[0]
    _need(x, torch.bfloat16, "x")
    _need(W_r, torch.bfloat16, "W_r", (E, d))
    if z is None:
        z = torch.empty((T, E), dtype=torch.bfloat16, device=x.device)
    _need(z, torch.bfloat16, "z", (T, E))
    _need(err_flag, torch.int32, "err_flag")
    _check(load().eqb_router_logits(_p(x), _p(W_r), T, d, E, _p(z), _p(err_flag), _stream(stream)),
           "eqb_router_logits")
    return z


def eqb_router_route(x, W_r, b, K, mb_offsets=None, z=None, topk_idx=None, tau=None, loads=None,
                     err_flag=None, stream=None, hist_hi=None):
    """Router logits and routing in one kernel (see eqb.h): z = bf16(x W_r^T)
    and, from the same accumulators, eqb_route_topk's topk_idx, tau and loads
    (accumulated into); with hist_hi [E,256] also the coarse histogram
    (accumulated into).  E in {64, 128}, K <= 8.  Returns (z, topk_idx, tau)."""
    T, d = x.shape
    E = W_r.shape[0]
    _need(x, torch.bfloat16, "x")
    _need(W_r, torch.bfloat16, "W_r", (E, d))
    _need(b, torch.float32, "b", (E,))
    if z is None:
        z = torch.empty((T, E), dtype=torch.bfloat16, device=x.device)
    if tau is None:
        tau = torch.empty(T, dtype=torch.float32, device=x.device)
    _need(z, torch.bfloat16, "z", (T, E))
    _need(tau, torch.float32, "tau", (T,))
    _need(topk_idx, torch.int32, "topk_idx", (T, K))
    M = 0
    if mb_offsets is not None:
        _need(mb_offsets, torch.int64, "mb_offsets")
        M = mb_offsets.numel() - 1
    _need(loads, torch.int32, "loads", (M, E) if loads is not None else None)
    _need(hist_hi, torch.int32, "hist_hi", (E, 256) if hist_hi is not None else None)
    _need(err_flag, torch.int32, "err_flag")
    _check(load().eqb_router_route(_p(x), _p(W_r), T, d, E, K, _p(b), _p(mb_offsets), M, _p(z),
                                   _p(topk_idx), _p(tau), _p(loads), _p(hist_hi), _p(err_flag), _stream(stream)),
           "eqb_router_route")
    return z, topk_idx, tau


def gshard_inject_grad(grad_s, z, loads, mb_offsets, K, alpha, stream=None):
    """GShard auxiliary-loss gradient added to grad_s in place (see eqb.h):
    grad_s fp32 [T,E], z bf16 [T,E], loads int32 [M,E], mb_offsets int64."""
    T, E = z.shape
    _need(grad_s, torch.float32, "grad_s", (T, E))
    _need(z, torch.bfloat16, "z")
    _need(mb_offsets, torch.int64, "mb_offsets")
    M = mb_offsets.numel() - 1
    _need(loads, torch.int32, "loads", (M, E))
    _check(load().gshard_inject_grad(_p(grad_s), _p(z), _p(loads), _p(mb_offsets), M, T, E, K,
                                     float(alpha), _stream(stream)), "gshard_inject_grad")
    return grad_s


def eqb_rank_averaged_workspace_bytes(E: int, P: int) -> int:
    return int(load().eqb_rank_averaged_workspace_bytes(E, P))


def eqb_rank_averaged_bias(z, tau, K, shard_offsets_host, workspace, b_out=None, q_shards=None,
                           err_flag=None, stream=None):
    """Rank-averaged QB (Sec. 2): each shard's own K/E margin quantile,
    averaged over the non-empty shards and centered.  shard_offsets_host: int64
    host array [P+1]; workspace: uint8 CUDA tensor of
    eqb_rank_averaged_workspace_bytes(E, P) bytes.  Returns (b fp32 [E],
    q_shards bf16 [P,E], row p = shard p)."""
    import numpy as np
    T, E = z.shape
    _need(z, torch.bfloat16, "z")
    _need(tau, torch.float32, "tau", (T,))
    off = np.ascontiguousarray(np.asarray(shard_offsets_host), dtype=np.int64)
    P = len(off) - 1
    if b_out is None:
        b_out = torch.empty(E, dtype=torch.float32, device=z.device)
    if q_shards is None:
        q_shards = torch.zeros((P, E), dtype=torch.bfloat16, device=z.device)
    _need(b_out, torch.float32, "b_out", (E,))
    _need(q_shards, torch.bfloat16, "q_shards", (P, E))
    _need(workspace, torch.uint8, "workspace")
    _need(err_flag, torch.int32, "err_flag")
    _check(load().eqb_rank_averaged_bias(_p(z), _p(tau), T, E, K, off.ctypes.data_as(ctypes.c_void_p), P,
                                         _p(q_shards), _p(b_out), _p(workspace), workspace.numel(),
                                         _p(err_flag), _stream(stream)), "eqb_rank_averaged_bias")
    return b_out, q_shards


def eqb_fixed_hist_bias(z, tau, K, lo, width, workspace, b_out=None, estimate=None, err_flag=None,
                        stream=None):
    """Fixed-resolution (256 equal bins) histogram estimate of the K/E margin
    quantile (Sec. 2), centered.  Returns (b fp32 [E], estimate fp64 [E])."""
    T, E = z.shape
    _need(z, torch.bfloat16, "z")
    _need(tau, torch.float32, "tau", (T,))
    if b_out is None:
        b_out = torch.empty(E, dtype=torch.float32, device=z.device)
    if estimate is None:
        estimate = torch.empty(E, dtype=torch.float64, device=z.device)
    _need(b_out, torch.float32, "b_out", (E,))
    _need(estimate, torch.float64, "estimate", (E,))
    _need(workspace, torch.uint8, "workspace")
    _need(err_flag, torch.int32, "err_flag")
    _check(load().eqb_fixed_hist_bias(_p(z), _p(tau), T, E, K, float(lo), float(width), _p(b_out),
                                      _p(estimate), _p(workspace), workspace.numel(), _p(err_flag),
                                      _stream(stream)), "eqb_fixed_hist_bias")
    return b_out, estimate


def eqb_selftest_stalled_wait(err_flag, polls=1 << 16, stream=None):
    """Run the bounded-wait failure path on purpose (see eqb.h): afterwards
    err_flag holds EQB_ERR_CUDA and the context is still usable."""
    _need(err_flag, torch.int32, "err_flag")
    _check(load().eqb_selftest_stalled_wait(_p(err_flag), int(polls), _stream(stream)),
           "eqb_selftest_stalled_wait")


def eqb_maxvio(loads, mb_offsets, K, out=None, per_mb=None, stream=None):
    """Global and Local MaxVio (Sec. 5 metrics) of int32 loads [M,E] over the
    microbatches given by mb_offsets; returns a float64 CUDA tensor [2]
    (global, local)."""
    M, E = loads.shape
    _need(loads, torch.int32, "loads")
    _need(mb_offsets, torch.int64, "mb_offsets", (M + 1,))
    if out is None:
        out = torch.empty(2, dtype=torch.float64, device=loads.device)
    _need(out, torch.float64, "out", (2,))
    _need(per_mb, torch.float64, "per_mb", (M,) if per_mb is not None else None)
    _check(load().eqb_maxvio(_p(loads), _p(mb_offsets), M, E, K, _p(out), _p(per_mb), _stream(stream)),
           "eqb_maxvio")
    return out


def eqb_layer_workspace_bytes(E: int) -> int:
    return int(load().eqb_layer_workspace_bytes(E))


def eqb_layer_step(z, b, K, mb_offsets, loads, b_next, workspace, tau=None, topk_idx=None,
                   grad_s=None, eta=0.0, c=0.0, mb_offsets_host=None, r=0, err_flag=None,
                   stream=None):
    """The whole routing-balance step of one layer in one library call (see
    eqb.h).  workspace: uint8 CUDA tensor of eqb_layer_workspace_bytes(E)
    bytes.  mb_offsets_host: optional int64 host copy of the offsets, checked
    by the library before anything is launched."""
    T, E = z.shape
    _need(z, torch.bfloat16, "z")
    _need(b, torch.float32, "b", (E,))
    _need(mb_offsets, torch.int64, "mb_offsets")
    M = mb_offsets.numel() - 1
    _need(loads, torch.int32, "loads", (M, E))
    _need(b_next, torch.float32, "b_next", (E,))
    _need(workspace, torch.uint8, "workspace")
    if tau is None:
        tau = torch.empty(T, dtype=torch.float32, device=z.device)
    _need(tau, torch.float32, "tau", (T,))
    _need(topk_idx, torch.int32, "topk_idx", (T, K))
    _need(grad_s, torch.float32, "grad_s", (T, E) if grad_s is not None else None)
    _need(err_flag, torch.int32, "err_flag")
    host = None
    if mb_offsets_host is not None:
        import numpy as np
        host = np.ascontiguousarray(np.asarray(mb_offsets_host), dtype=np.int64)
        if host.shape != (M + 1,):
            raise ValueError("mb_offsets_host must have M+1 entries")
    hp = None if host is None else host.ctypes.data_as(ctypes.c_void_p)
    rc = load().eqb_layer_step(_p(z), _p(b), T, E, K, _p(mb_offsets), hp, M, int(r), _p(topk_idx),
                               _p(tau), _p(loads), _p(b_next), _p(grad_s), float(eta), float(c),
                               _p(workspace), workspace.numel(), _p(err_flag), _stream(stream))
    _check(rc, "eqb_layer_step")
    return tau


def eqb_router_layer_step(x, W_r, b, K, mb_offsets, loads, b_next, workspace, z=None, tau=None,
                          topk_idx=None, grad_s=None, eta=0.0, c=0.0, mb_offsets_host=None, r=0,
                          err_flag=None, stream=None):
    """The routing-balance step of one layer from the router input x (see
    eqb.h): the projection z = bf16(x W_r^T), routed from its accumulators
    where the shape allows, then everything eqb_layer_step does.  Returns
    (z, tau)."""
    T, d = x.shape
    E = W_r.shape[0]
    _need(x, torch.bfloat16, "x")
    _need(W_r, torch.bfloat16, "W_r", (E, d))
    _need(b, torch.float32, "b", (E,))
    _need(mb_offsets, torch.int64, "mb_offsets")
    M = mb_offsets.numel() - 1
    _need(loads, torch.int32, "loads", (M, E))
    _need(b_next, torch.float32, "b_next", (E,))
    _need(workspace, torch.uint8, "workspace")
    if z is None:
        z = torch.empty((T, E), dtype=torch.bfloat16, device=x.device)
    if tau is None:
        tau = torch.empty(T, dtype=torch.float32, device=x.device)
    _need(z, torch.bfloat16, "z", (T, E))
    _need(tau, torch.float32, "tau", (T,))
    _need(topk_idx, torch.int32, "topk_idx", (T, K))
    _need(grad_s, torch.float32, "grad_s", (T, E) if grad_s is not None else None)
    _need(err_flag, torch.int32, "err_flag")
    host = None
    if mb_offsets_host is not None:
        import numpy as np
        host = np.ascontiguousarray(np.asarray(mb_offsets_host), dtype=np.int64)
        if host.shape != (M + 1,):
            raise ValueError("mb_offsets_host must have M+1 entries")
    hp = None if host is None else host.ctypes.data_as(ctypes.c_void_p)
    rc = load().eqb_router_layer_step(_p(x), _p(W_r), T, d, E, K, _p(b), _p(mb_offsets), hp, M, int(r),
                                      _p(z), _p(topk_idx), _p(tau), _p(loads), _p(b_next), _p(grad_s),
                                      float(eta), float(c), _p(workspace), workspace.numel(),
                                      _p(err_flag), _stream(stream))
    _check(rc, "eqb_router_layer_step")
    return z, tau


def eqb_layer_step_noalloc(z, b, K, mb_offsets, loads, b_next, tau=None, topk_idx=None,
                           grad_s=None, eta=0.0, c=0.0, mb_offsets_host=None, r=0, err_flag=None,
                           stream=None):
    """eqb_layer_step without a workspace argument, for callers that cannot
    allocate device memory: the step's scratch is an array inside the
    library (E <= 256).  Calls that overlap on the GPU share that array and
    race; the first call on a device should come before any stream capture.
    z (and every other tensor) must be on the current CUDA device: the
    library looks the scratch array up on that device."""
    T, E = z.shape
    _need(z, torch.bfloat16, "z")
    _on_current_device(z, "z")
    _need(b, torch.float32, "b", (E,))
    _need(mb_offsets, torch.int64, "mb_offsets")
    M = mb_offsets.numel() - 1
    _need(loads, torch.int32, "loads", (M, E))
    _need(b_next, torch.float32, "b_next", (E,))
    if tau is None:
        tau = torch.empty(T, dtype=torch.float32, device=z.device)
    _need(tau, torch.float32, "tau", (T,))
    _need(topk_idx, torch.int32, "topk_idx", (T, K))
    _need(grad_s, torch.float32, "grad_s", (T, E) if grad_s is not None else None)
    _need(err_flag, torch.int32, "err_flag")
    hp = None
    if mb_offsets_host is not None:
        import numpy as np
        host = np.ascontiguousarray(np.asarray(mb_offsets_host), dtype=np.int64)
        if host.shape != (M + 1,):
            raise ValueError("mb_offsets_host must have M+1 entries")
        hp = host.ctypes.data_as(ctypes.c_void_p)
    rc = load().eqb_layer_step_noalloc(_p(z), _p(b), T, E, K, _p(mb_offsets), hp, M, int(r),
                                       _p(topk_idx), _p(tau), _p(loads), _p(b_next), _p(grad_s),
                                       float(eta), float(c), _p(err_flag), _stream(stream))
    _check(rc, "eqb_layer_step_noalloc")
    return tau


class EqbWorkspace:
    """Device buffers of one layer's EQB statistic: the two [E,256] int32
    histograms, u, rho, q_hat and the error word.  Allocated once by the
    caller (through torch), reused every step."""

    def __init__(self, E: int, device="cuda"):
        self.E = E
        self.hist_hi = torch.zeros((E, 256), dtype=torch.int32, device=device)
        self.hist_lo = torch.zeros((E, 256), dtype=torch.int32, device=device)
        self.u = torch.zeros(E, dtype=torch.uint8, device=device)
        self.rho = torch.zeros(E, dtype=torch.int32, device=device)
        self.q_hat = torch.zeros(E, dtype=torch.bfloat16, device=device)
        self.err = torch.zeros(1, dtype=torch.int32, device=device)

    def zero_(self):
        self.hist_hi.zero_()
        self.hist_lo.zero_()
        self.err.zero_()


def eqb_layer_forward(z, b, K, mb_offsets, ws: EqbWorkspace, topk_idx, tau, loads, b_next,
                      r=None, stream=None):
    """One layer's forward routing-balance statistic, in the paper's order:
    routing + coarse pass, select 1, fine pass, select 2, bias update.
    `loads` must be zeroed by the caller (it is accumulated into); the
    workspace histograms are zeroed here.  All steps run on `stream`."""
    T, E = z.shape
    if r is None:
        r = eqb_target_rank(T, E, K)
    ws.zero_()
    eqb_route_topk(z, b, K, mb_offsets, topk_idx, tau, loads, ws.hist_hi, ws.err, stream)
    eqb_select_quantile(ws.hist_hi, 1, r, ws.u, ws.rho, None, ws.err, stream)
    eqb_margin_hist_pass2(z, tau, ws.u, ws.hist_lo, stream)
    eqb_select_quantile(ws.hist_lo, 2, r, ws.u, ws.rho, ws.q_hat, ws.err, stream)
    eqb_bias_update(ws.q_hat, b_next, stream)
