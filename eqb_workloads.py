"""Seeded synthetic inputs for the EQB + LEI routing-balance path.

This module only draws random numbers and lays them out; it contains none of
the method's arithmetic, so both the CUDA path and the CPU oracle consume its
output unchanged.  It stands in for router logits of the paper's 7.5B MoE
(Sec. 5 / App. E.1), whose weights and data are not available.

Shapes (token count T, experts E, experts per token K, microbatches M):

  tiny    T=4,096      E=8    K=2  M=4  x 1,024   z ~ N(0,1), b = 0
  tie     T=65,536     E=64   K=8  M=8  x 8,192   z = bf16(0.05 N(0,1) + mu_e),
                                                   mu_e ~ N(0, 0.5^2),
                                                   b ~ U(-0.1, 0.1)
  mid     T=524,288    E=128  K=8  M=32 x 16,384  z ~ N(0,1) + 1.0 on 16 hot
                                                   experts; b from one QB
                                                   update on an independent
                                                   prior batch (the caller
                                                   computes it)
  global  T=2,097,152  E=256  K=8  M=64 x 32,768  z per element: 0.9 N(0,1),
                                                   0.1 2*StudentT(3); b ~ N(0, 0.2^2)
  router  T=1,048,576  d=4096 E=128 K=8 M=16 x 65,536  x ~ N(0,1), W ~ N(0,1/d),
                                                   b^(0) = 0, 3 steps
  paper   T=9,437,184  E=256  K=6  M=64 x 147,456 z ~ N(0,1); b ~ N(0, 0.2^2)
          (the paper's own setting, Sec. 5 / App. E.1: 256 experts, top-6,
          147,456 tokens per data-parallel rank, 64 ranks)
  wide    T=1,048,576  E=512  K=8  M=32 x 32,768  z ~ N(0,1); b ~ N(0, 0.2^2)
          (more experts than one histogram block holds)

Upstream router-score gradients g ~ N(0, 0.1^2) fp32 (variance 1e-2) for
every config.  Logits are rounded to bf16 round-to-nearest-even by torch.

Two generators are provided: numpy PCG64 on the host (bit-stable across
machines and library versions; used for test sizes) and torch's Philox on a
CUDA device (fast; used at full size, where the host copy is taken from the
device so both sides still see identical bytes).
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np
import torch

CONFIG_NAMES = ("tiny", "tie", "mid", "global", "router", "paper", "wide")


@dataclass(frozen=True)
class Shape:
    name: str
    T: int
    E: int
    K: int
    M: int
    d: int = 0
    steps: int = 1
    seed: int = 0
    extra: dict = field(default_factory=dict)


SHAPES = {
    "tiny": Shape("tiny", 4096, 8, 2, 4, seed=1000),
    "tie": Shape("tie", 65536, 64, 8, 8, seed=1001),
    "mid": Shape("mid", 524288, 128, 8, 32, seed=1002),
    "global": Shape("global", 2097152, 256, 8, 64, seed=1003),
    "router": Shape("router", 1048576, 128, 8, 16, d=4096, steps=3, seed=1004),
    "paper": Shape("paper", 9437184, 256, 6, 64, seed=1005),
    # more experts than one histogram block holds (expert-tiled passes)
    "wide": Shape("wide", 1048576, 512, 8, 32, seed=1006),
}


def even_offsets(T: int, M: int) -> np.ndarray:
    """Microbatch boundaries [M+1] splitting T tokens into M contiguous,
    near-equal ranges (sizes differ by at most one)."""
    return np.array([(T * l) // M for l in range(M + 1)], dtype=np.int64)


def ragged_offsets(T: int, M: int, seed: int) -> np.ndarray:
    """M contiguous ranges of random, uneven sizes (some may be empty)."""
    rng = np.random.default_rng(seed)
    cuts = np.sort(rng.integers(0, T + 1, size=M - 1))
    return np.concatenate([[0], cuts, [T]]).astype(np.int64)


class _Draw:
    """Uniform interface over numpy (host) and torch (device) generators."""

    def __init__(self, seed: int, device: str):
        self.device = device
        if device == "cpu":
            self.rng = np.random.default_rng(seed)
        else:
            self.gen = torch.Generator(device=device)
            self.gen.manual_seed(seed)

    def normal(self, shape):
        if self.device == "cpu":
            return torch.from_numpy(self.rng.standard_normal(shape, dtype=np.float32))
        return torch.randn(shape, generator=self.gen, device=self.device, dtype=torch.float32)

    def uniform(self, shape, lo, hi):
        if self.device == "cpu":
            return torch.from_numpy(self.rng.uniform(lo, hi, size=shape).astype(np.float32))
        u = torch.rand(shape, generator=self.gen, device=self.device, dtype=torch.float32)
        return u * (hi - lo) + lo

    def bernoulli_mask(self, shape, p):
        if self.device == "cpu":
            return torch.from_numpy(self.rng.random(shape, dtype=np.float32) < p)
        return torch.rand(shape, generator=self.gen, device=self.device) < p

    def permutation(self, n):
        if self.device == "cpu":
            return torch.from_numpy(self.rng.permutation(n))
        return torch.randperm(n, generator=self.gen, device=self.device)


def _bf16(x: torch.Tensor) -> torch.Tensor:
    return x.to(torch.bfloat16)


def make_logits(name: str, T: int | None = None, seed: int | None = None,
                device: str = "cpu") -> torch.Tensor:
    """bf16 router logits z [T,E] following the config's recipe."""
    sh = SHAPES[name]
    T = sh.T if T is None else T
    seed = sh.seed if seed is None else seed
    E = sh.E
    d = _Draw(seed, device)
    if name in ("tiny", "router", "paper", "wide"):
        return _bf16(d.normal((T, E)))
    if name == "tie":
        mu = d.normal((E,)) * 0.5
        return _bf16(d.normal((T, E)) * 0.05 + mu)
    if name == "mid":
        hot = d.permutation(E)[:16]
        shift = torch.zeros(E, dtype=torch.float32, device=device)
        shift[hot.to(shift.device)] = 1.0
        return _bf16(d.normal((T, E)) + shift)
    if name == "global":
        base = d.normal((T, E))
        # Student-t(3) = N / sqrt(chi2_3 / 3), chi2_3 a sum of three squared normals
        n = d.normal((T, E))
        chi = d.normal((T, E)) ** 2 + d.normal((T, E)) ** 2 + d.normal((T, E)) ** 2
        t3 = n / torch.sqrt(chi / 3.0)
        mask = d.bernoulli_mask((T, E), 0.1)
        return _bf16(torch.where(mask, 2.0 * t3, base))
    raise KeyError(name)


def make_bias(name: str, seed: int | None = None, device: str = "cpu") -> torch.Tensor:
    """fp32 expert bias b [E] for configs whose bias is drawn directly.  The
    'mid' config's bias comes from a QB update on `prior_batch_logits`, which
    the caller computes; this returns zeros for it (and for tiny / router)."""
    sh = SHAPES[name]
    seed = (sh.seed if seed is None else seed) + 7
    d = _Draw(seed, device)
    if name == "tie":
        return d.uniform((sh.E,), -0.1, 0.1)
    if name in ("global", "paper", "wide"):
        return d.normal((sh.E,)) * 0.2
    return torch.zeros(sh.E, dtype=torch.float32, device=device)


def prior_batch_logits(name: str, T: int | None = None, device: str = "cpu") -> torch.Tensor:
    """An independent batch of the same distribution (seed + 100) from which
    the 'mid' config derives its prior-step bias."""
    return make_logits(name, T=T, seed=SHAPES[name].seed + 100, device=device)


def make_grad(name: str, T: int | None = None, seed: int | None = None,
              device: str = "cpu") -> torch.Tensor:
    """Upstream router-score gradient dL/ds fp32 [T,E] ~ N(0, 0.1^2)."""
    sh = SHAPES[name]
    T = sh.T if T is None else T
    seed = (sh.seed if seed is None else seed) + 13
    return _Draw(seed, device).normal((T, sh.E)) * 0.1


def make_router_inputs(T: int | None = None, d_model: int | None = None, step: int = 0,
                       device: str = "cpu", E: int | None = None):
    """Router config: activations x bf16 [T,d] ~ N(0,1) with a fresh seed per
    step, and the projection W_r bf16 [E,d] ~ N(0, 1/d) with a fixed seed."""
    sh = SHAPES["router"]
    T = sh.T if T is None else T
    d_model = sh.d if d_model is None else d_model
    E = sh.E if E is None else E
    x = _bf16(_Draw(sh.seed + 31 * (step + 1), device).normal((T, d_model)))
    W = _bf16(_Draw(sh.seed + 5, device).normal((E, d_model)) * (1.0 / np.sqrt(d_model)))
    return x, W


def bits(t: torch.Tensor) -> np.ndarray:
    """Host numpy view of a bf16 tensor's raw 16-bit patterns."""
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)
