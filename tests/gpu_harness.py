"""Shared helpers for the GPU parity tests: run the CUDA path through the C
ABI, run the oracle on the same bytes, and guard-band output buffers."""
from __future__ import annotations

from concurrent.futures import ThreadPoolExecutor

import numpy as np
import torch

import oracle
import paper_2609_28053_gb300 as eqb

GUARD = 64  # elements of canary on each side of an output buffer


class Guarded:
    """A 1-D device buffer with canaries on both sides; `.view` is the
    contiguous middle of the requested shape."""

    def __init__(self, shape, dtype, fill=0, canary=None):
        n = int(np.prod(shape))
        self.n = n
        self.buf = torch.empty(n + 2 * GUARD, dtype=dtype, device="cuda")
        if canary is None:
            canary = -12345 if not dtype.is_floating_point else -1234.5
        self.canary = canary
        self.buf.fill_(canary)
        self.view = self.buf[GUARD:GUARD + n].view(*shape)
        self.view.fill_(fill)

    def intact(self) -> bool:
        head = self.buf[:GUARD]
        tail = self.buf[GUARD + self.n:]
        c = torch.full_like(head, self.canary)
        return bool(torch.equal(head, c) and torch.equal(tail, c))


def to_dev_bf16(bits: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).cuda()


def gpu_forward(z_bits, b, K, offsets, guard=True):
    """The forward statistic on the GPU through the C ABI, every output
    guard-banded.  Returns host numpy arrays."""
    z = to_dev_bf16(z_bits)
    T, E = z.shape
    M = len(offsets) - 1
    bt = torch.from_numpy(np.ascontiguousarray(b, np.float32)).cuda()
    off = torch.from_numpy(np.ascontiguousarray(offsets, np.int64)).cuda()
    g = dict(
        idx=Guarded((T, K), torch.int32, fill=-7),
        tau=Guarded((T,), torch.float32, fill=-7.0),
        loads=Guarded((M, E), torch.int32),
        H=Guarded((E, 256), torch.int32),
        L=Guarded((E, 256), torch.int32),
        u=Guarded((E,), torch.uint8, canary=77),
        rho=Guarded((E,), torch.int32),
        q=Guarded((E,), torch.bfloat16, canary=-3.0),
        b_next=Guarded((E,), torch.float32),
        err=Guarded((1,), torch.int32),
    )
    r = eqb.eqb_target_rank(T, E, K)
    eqb.eqb_route_topk(z, bt, K, off, g["idx"].view, g["tau"].view, g["loads"].view, g["H"].view,
                       g["err"].view)
    eqb.eqb_select_quantile(g["H"].view, 1, r, g["u"].view, g["rho"].view, None, g["err"].view)
    eqb.eqb_margin_hist_pass2(z, g["tau"].view, g["u"].view, g["L"].view)
    eqb.eqb_select_quantile(g["L"].view, 2, r, g["u"].view, g["rho"].view, g["q"].view, g["err"].view)
    eqb.eqb_bias_update(g["q"].view, g["b_next"].view)
    torch.cuda.synchronize()
    for k, v in g.items():
        assert v.intact(), f"write outside the {k} buffer"
    out = {k: v.view.cpu() for k, v in g.items()}
    out["q"] = out["q"].view(torch.int16).numpy().view(np.uint16)
    for k in list(out):
        if isinstance(out[k], torch.Tensor):
            out[k] = out[k].numpy()
    out["r"] = r
    return out


def oracle_route_parallel(z_bits, b, K, offsets, threads=16):
    """Oracle routing over token chunks in parallel threads (each call is
    the single-threaded oracle; ctypes releases the GIL).  Loads are the
    per-microbatch counts of the oracle's index lists."""
    T, E = z_bits.shape
    chunks = np.linspace(0, T, min(threads * 4, max(T // 1024, 1)) + 1).astype(np.int64)

    def one(i):
        a, c = chunks[i], chunks[i + 1]
        return oracle.route(z_bits[a:c], b, K)[:2]

    with ThreadPoolExecutor(threads) as ex:
        parts = list(ex.map(one, range(len(chunks) - 1)))
    idx = np.concatenate([p[0] for p in parts])
    tau = np.concatenate([p[1] for p in parts])
    M = len(offsets) - 1
    loads = np.zeros((M, E), np.int32)
    for l in range(M):
        loads[l] = np.bincount(idx[offsets[l]:offsets[l + 1]].ravel(), minlength=E)
    return idx, tau, loads


def oracle_forward(z_bits, b, K, offsets, experts=None, threads=16):
    """The oracle's forward statistic.  `experts` restricts the full-sort
    quantile to a sample (at full size); histograms are per sampled expert."""
    T, E = z_bits.shape
    if T * E <= (1 << 24):
        idx, tau, loads = oracle.route(z_bits, b, K, offsets)
    else:
        idx, tau, loads = oracle_route_parallel(z_bits, b, K, offsets, threads)
    r = oracle.target_rank(T, E, K)
    out = dict(idx=idx, tau=tau, loads=loads, r=r)
    if experts is None:
        H = oracle.hist_hi(z_bits, tau)
        u, rho = oracle.select_hi(H, r)
        L = oracle.hist_lo(z_bits, tau, u)
        q_steps = oracle.select_lo(L, u, rho)
        q = oracle.quantile(z_bits, tau, r)
        assert np.array_equal(q, q_steps)  # the oracle's own radix = sort invariant
        out.update(H=H, u=u, rho=rho, L=L, q=q, b_next=oracle.bias_update(q))
    else:
        ex = np.asarray(experts, np.int32)
        with ThreadPoolExecutor(threads) as pool:
            qs = list(pool.map(lambda e: oracle.quantile(z_bits, tau, r, experts=[e])[0], ex))
        out.update(experts=ex, q=np.array(qs, np.uint16))
    return out


def bits_f32(x):
    return np.ascontiguousarray(x, np.float32).view(np.uint32)
