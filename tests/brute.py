"""Brute-force statements of the paper's definitions for tiny inputs.

Used only to pin the C oracle to something other than itself.  Each function
follows a different route from the oracle's code:

* top-(K+1) by repeated maximum extraction with an explicit tie rule
  (the oracle sorts);
* the quantile as the smallest minimiser of the piecewise-linear objective
  of App. B (the oracle sorts);
* the cutoff as the lower-endpoint minimiser of the threshold identity
  (App. B, TopKSum_K(x) = min_a {K a + sum_e [x_e - a]_+});
* Algorithm 1 (two-pass radix selection) run literally on Python ints;
* bf16 rounding through torch's own conversion (a library routine).

Arithmetic on scores is done with numpy float32 scalars, so every add and
subtract is one IEEE single-precision operation.
"""
from __future__ import annotations

from fractions import Fraction

import numpy as np
import torch


def bf16_bits_from_f32(x) -> np.ndarray:
    """Round-to-nearest-even fp32 -> bf16 via torch (library routine)."""
    t = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32))
    return t.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def f32_from_bf16_bits(bits) -> np.ndarray:
    b = np.ascontiguousarray(bits, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32)


def topk_by_extraction(s_row, K):
    """Pick the largest remaining score K+1 times; among equal scores the
    lower expert index wins.  Returns (top-K list, value of the (K+1)th)."""
    s_row = [np.float32(v) for v in s_row]
    taken = set()
    order = []
    for _ in range(K + 1):
        best = None
        for e, v in enumerate(s_row):
            if e in taken:
                continue
            if best is None or v > s_row[best]:  # strict: earlier index kept on ties
                best = e
        taken.add(best)
        order.append(best)
    return order[:K], s_row[order[K]]


def scores(z_bits_row, b):
    zf = f32_from_bf16_bits(z_bits_row)
    return [np.float32(zf[e]) + np.float32(b[e]) for e in range(len(zf))]


def cutoff_by_threshold_identity(x, K):
    """App. B: TopKSum_K(x) = min_a {K a + sum_e [x_e - a]_+}; the cutoff is
    the smallest minimiser over the candidate set {x_e} (exact rationals)."""
    xs = [Fraction(float(v)) for v in x]

    def D(a):
        return K * a + sum(max(v - a, 0) for v in xs)

    vals = sorted(set(xs))
    best = min(D(a) for a in vals)
    return min(a for a in vals if D(a) == best), best


def quantile_by_objective(m_values, r):
    """App. B: for fixed cutoffs the bias minimises
    sum_t [b - m_t]_+ - r b; its smallest minimiser over {m_t} is the r-th
    smallest margin.  Exact rational arithmetic."""
    ms = [Fraction(float(v)) for v in m_values]

    def G(bb):
        return sum(max(bb - m, 0) for m in ms) - r * bb

    cands = sorted(set(ms))
    best = min(G(c) for c in cands)
    return min(c for c in cands if G(c) == best)


def kappa_py(x: int) -> int:
    """Order-preserving key: negative patterns flipped entirely, positive
    patterns get the sign bit set."""
    return (~x) & 0xFFFF if x & 0x8000 else x | 0x8000


def kappa_inv_py(k: int) -> int:
    return k & 0x7FFF if k & 0x8000 else (~k) & 0xFFFF


def radix_select_alg1(margin_bits_per_rank, r):
    """Algorithm 1 run literally: per-rank 256-bin counts of the high byte,
    summed across ranks, prefix to the rank; then low-byte counts inside the
    selected bin.  `margin_bits_per_rank` is a list (ranks) of lists of bf16
    bit patterns for ONE expert.  Returns the bf16 bits of kappa^{-1}(u, v)
    with zero as +0."""
    H = [0] * 256
    for rank in margin_bits_per_rank:
        local = [0] * 256
        for x in rank:
            local[kappa_py(int(x)) >> 8] += 1
        H = [a + b for a, b in zip(H, local)]
    acc = 0
    for u in range(256):
        if acc + H[u] >= r:
            break
        acc += H[u]
    rho = r - acc
    Lc = [0] * 256
    for rank in margin_bits_per_rank:
        for x in rank:
            k = kappa_py(int(x))
            if (k >> 8) == u:
                Lc[k & 0xFF] += 1
    acc = 0
    for v in range(256):
        acc += Lc[v]
        if acc >= rho:
            break
    q = kappa_inv_py((u << 8) | v)
    return 0 if q == 0x8000 else q
