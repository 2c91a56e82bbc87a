"""CPU oracle for the EQB + LEI routing-balance path (test infrastructure).

Only the test suite, ``__graft_entry__.smoke()`` and the benchmark's CPU
baseline leg may import this package.  It wraps ``eqb_oracle.c`` (plain,
single-threaded C, compiled with ``-ffp-contract=off`` and no fast-math) with
ctypes and numpy.  It shares no code with the CUDA path.

Every wrapper cites the passage of arXiv 2609.28053 it follows:

* :func:`route`            -- Sec. 2, Eq. (1) and the QB paragraph (top-K of
                              z + b, cutoff tau_t = (K+1)st largest, loads f_e).
* :func:`quantile`         -- Eq. (2): r-th smallest margin by a full sort.
* :func:`hist_hi`,
  :func:`hist_lo`          -- Algorithm 1, steps 1 and 4 (plain counting).
* :func:`select_hi`,
  :func:`select_lo`        -- Algorithm 1, steps 3, 5 and 6.
* :func:`bias_update`      -- Eq. (2) centering.
* :func:`lei`              -- Sec. 4, Eq. (LEI) with Eq. (norm).
* :func:`router_logits`    -- Sec. 2, z_t = W_r x_t, dot products in fp64.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "eqb_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

OK, ERR_ARG, ERR_NONFINITE, ERR_NOMEM = 0, 1, 4, 5


def build(force: bool = False) -> str:
    """Compile ``liboracle.so`` next to its source with gcc (no fast-math,
    no FMA contraction).  Returns the library path."""
    if (not force and os.path.exists(_LIB)
            and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC)):
        return _LIB
    tmp = _LIB + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off",
           "-fno-fast-math", "-Wall", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            # EQB_ORACLE_LIB lets the mutation test load a deliberately broken
            # build of this same source; nothing else sets it.
            lib = ctypes.CDLL(os.environ.get("EQB_ORACLE_LIB") or build())
            P = ctypes.c_void_p
            i64, i32, f32 = ctypes.c_int64, ctypes.c_int32, ctypes.c_float
            sig = {
                "oracle_route": [P, P, i64, i32, i32, P, i32, P, i64, P, P, P],
                "oracle_margins": [P, P, i64, i32, i32, P],
                "oracle_quantile": [P, P, i64, i32, i64, P, i32, P],
                "oracle_hist_hi": [P, P, i64, i64, i32, P],
                "oracle_hist_lo": [P, P, i64, i64, i32, P, P],
                "oracle_select_hi": [P, i32, i64, P, P],
                "oracle_select_lo": [P, i32, P, P, P],
                "oracle_bias_update": [P, i32, P],
                "oracle_lei": [P, P, P, i32, i64, i32, i32, f32, f32, P, P],
                "oracle_router_logits": [P, P, i64, i32, i32, P, i64, P, P],
                "oracle_maxvio": [P, P, i32, i32, i32, P, P, P],
                "oracle_gshard": [P, P, P, P, i32, i64, i32, i32, f32, P],
            }
            for name, args in sig.items():
                fn = getattr(lib, name)
                fn.argtypes = args
                fn.restype = ctypes.c_int
            lib.oracle_target_rank.argtypes = [i64, i32, i32]
            lib.oracle_target_rank.restype = i64
            lib.oracle_f32_to_bf16.argtypes = [ctypes.c_float]
            lib.oracle_f32_to_bf16.restype = ctypes.c_uint16
            lib.oracle_kappa.argtypes = [ctypes.c_uint16]
            lib.oracle_kappa.restype = ctypes.c_uint16
            lib.oracle_kappa_inv.argtypes = [ctypes.c_uint16]
            lib.oracle_kappa_inv.restype = ctypes.c_uint16
            _lib = lib
    return _lib


class OracleError(RuntimeError):
    pass


def _check(rc: int, what: str):
    if rc != OK:
        raise OracleError(f"{what} failed with status {rc}")


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def target_rank(T: int, E: int, K: int) -> int:
    """r = ceil(T K / E): Sec. 3 (r = TK/E), rounded up when not integral."""
    return int(_load().oracle_target_rank(T, E, K))


def f32_to_bf16_bits(x: float) -> int:
    return int(_load().oracle_f32_to_bf16(float(x)))


def kappa(x: int) -> int:
    """Algorithm 1's order-preserving 16-bit key of a bf16 bit pattern."""
    return int(_load().oracle_kappa(int(x)))


def kappa_inv(k: int) -> int:
    return int(_load().oracle_kappa_inv(int(k)))


def route(z_bits, b, K, offsets=None, rows=None):
    """Sec. 2: top-K of s = fp32(z) + b (ties to the lower index), tau_t = the
    (K+1)st largest s, and per-microbatch loads f_e.

    z_bits: uint16 [T,E] bf16 bit patterns; b: float32 [E];
    offsets: int64 [M+1] microbatch boundaries (default: one microbatch).
    rows: optional int64 token subset (then loads are not computed).
    Returns (idx int32 [n,K], tau float32 [n], loads int32 [M,E] or None)."""
    z_bits = _c(z_bits, np.uint16)
    T, E = z_bits.shape
    b = _c(b, np.float32)
    if offsets is None:
        offsets = np.array([0, T], dtype=np.int64)
    offsets = _c(offsets, np.int64)
    M = len(offsets) - 1
    if rows is not None:
        rows = _c(rows, np.int64)
        n = len(rows)
    else:
        n = T
    idx = np.zeros((n, K), dtype=np.int32)
    tau = np.zeros(n, dtype=np.float32)
    loads = None if rows is not None else np.zeros((M, E), dtype=np.int32)
    rc = _load().oracle_route(_ptr(z_bits), _ptr(b), T, E, K, _ptr(offsets), M,
                              _ptr(rows), n, _ptr(idx), _ptr(tau), _ptr(loads))
    _check(rc, "oracle_route")
    return idx, tau, loads


def margins(z_bits, tau, e):
    """m_{t,e} = bf16_rne(tau_t - fp32(z_{t,e})) for one expert, as bits."""
    z_bits = _c(z_bits, np.uint16)
    T, E = z_bits.shape
    tau = _c(tau, np.float32)
    m = np.zeros(T, dtype=np.uint16)
    _check(_load().oracle_margins(_ptr(z_bits), _ptr(tau), T, E, int(e), _ptr(m)),
           "oracle_margins")
    return m


def quantile(z_bits, tau, r, experts=None):
    """Eq. (2): b_hat_e = r-th smallest margin of expert e over all T tokens,
    by a full sort.  Returns bf16 bit patterns (uint16), zero as +0."""
    z_bits = _c(z_bits, np.uint16)
    T, E = z_bits.shape
    tau = _c(tau, np.float32)
    ex = None if experts is None else _c(experts, np.int32)
    n = E if ex is None else len(ex)
    q = np.zeros(n, dtype=np.uint16)
    rc = _load().oracle_quantile(_ptr(z_bits), _ptr(tau), T, E, int(r), _ptr(ex), n,
                                 _ptr(q))
    _check(rc, "oracle_quantile")
    return q


def hist_hi(z_bits, tau, t0=0, t1=None):
    """Algorithm 1 step 1: H[e,u] counts over tokens [t0, t1)."""
    z_bits = _c(z_bits, np.uint16)
    T, E = z_bits.shape
    t1 = T if t1 is None else t1
    tau = _c(tau, np.float32)
    H = np.zeros((E, 256), dtype=np.int32)
    _check(_load().oracle_hist_hi(_ptr(z_bits), _ptr(tau), t0, t1, E, _ptr(H)),
           "oracle_hist_hi")
    return H


def hist_lo(z_bits, tau, u, t0=0, t1=None):
    """Algorithm 1 step 4: L[e,v] counts inside the selected high byte u_e."""
    z_bits = _c(z_bits, np.uint16)
    T, E = z_bits.shape
    t1 = T if t1 is None else t1
    tau = _c(tau, np.float32)
    u = _c(u, np.uint8)
    L = np.zeros((E, 256), dtype=np.int32)
    _check(_load().oracle_hist_lo(_ptr(z_bits), _ptr(tau), t0, t1, E, _ptr(u), _ptr(L)),
           "oracle_hist_lo")
    return L


def select_hi(H, r):
    """Algorithm 1 step 3: (u_e, rho_e) from the summed high-byte counts."""
    H = _c(H, np.int32)
    E = H.shape[0]
    u = np.zeros(E, dtype=np.uint8)
    rho = np.zeros(E, dtype=np.int32)
    _check(_load().oracle_select_hi(_ptr(H), E, int(r), _ptr(u), _ptr(rho)),
           "oracle_select_hi")
    return u, rho


def select_lo(L, u, rho):
    """Algorithm 1 steps 5-6: v_e and b_hat_e = kappa^{-1}(u_e, v_e)."""
    L = _c(L, np.int32)
    E = L.shape[0]
    q = np.zeros(E, dtype=np.uint16)
    _check(_load().oracle_select_lo(_ptr(L), E, _ptr(_c(u, np.uint8)),
                                    _ptr(_c(rho, np.int32)), _ptr(q)),
           "oracle_select_lo")
    return q


def bias_update(qhat_bits):
    """Eq. (2): b = b_hat - mean(b_hat), fp64 mean in ascending expert order."""
    q = _c(qhat_bits, np.uint16)
    out = np.zeros(len(q), dtype=np.float32)
    _check(_load().oracle_bias_update(_ptr(q), len(q), _ptr(out)), "oracle_bias_update")
    return out


def lei(g, loads, offsets, K, eta, c):
    """Sec. 4 Eq. (LEI) and Eq. (norm): g + eta * rho~_e on every (t, e) of
    each microbatch.  Returns (g_out float32 [T,E], a float64 [M,E])."""
    loads = _c(loads, np.int32)
    offsets = _c(offsets, np.int64)
    M, E = loads.shape
    T = int(offsets[-1])
    gp = None
    g_out = None
    if g is not None:
        gp = _c(g, np.float32)
        g_out = np.zeros_like(gp)
    a = np.zeros((M, E), dtype=np.float64)
    rc = _load().oracle_lei(_ptr(gp), _ptr(loads), _ptr(offsets), M, T, E, K,
                            float(eta), float(c), _ptr(g_out), _ptr(a))
    _check(rc, "oracle_lei")
    return g_out, a


def router_logits(x_bits, W_bits, rows):
    """Sec. 2: z_t = W_r x_t for the listed rows, in fp64.  Returns
    (z float64 [n,E], sum of |products| float64 [n,E])."""
    x_bits = _c(x_bits, np.uint16)
    W_bits = _c(W_bits, np.uint16)
    T, d = x_bits.shape
    E = W_bits.shape[0]
    rows = _c(rows, np.int64)
    out = np.zeros((len(rows), E), np.float64)
    ab = np.zeros((len(rows), E), np.float64)
    _check(_load().oracle_router_logits(_ptr(x_bits), _ptr(W_bits), T, d, E, _ptr(rows), len(rows),
                                        _ptr(out), _ptr(ab)), "oracle_router_logits")
    return out, ab


def maxvio(loads, offsets, K):
    """Sec. 5 / App. E: MaxVio = max_e [f_e / fbar - 1], fbar = K|B|/E, for the
    loads summed over the step (global) and per non-empty microbatch, then
    averaged (local).  Returns (global, local, per_microbatch float64 [M])."""
    loads = _c(loads, np.int32)
    M, E = loads.shape
    offsets = _c(offsets, np.int64)
    g = ctypes.c_double(0.0)
    lo = ctypes.c_double(0.0)
    per = np.zeros(M, np.float64)
    _check(_load().oracle_maxvio(_ptr(loads), _ptr(offsets), M, E, K, ctypes.byref(g),
                                 ctypes.byref(lo), _ptr(per)), "oracle_maxvio")
    return g.value, lo.value, per


def gshard(g, z_bits, loads, offsets, K, alpha):
    """App. D, Eq. (gshard-grad): g + alpha * d/ds sum_e F_e P^G_e per local
    batch, with s = sigmoid(z), F stop-gradient.  Returns float32 [T,E]."""
    g = _c(g, np.float32)
    z_bits = _c(z_bits, np.uint16)
    T, E = z_bits.shape
    loads = _c(loads, np.int32)
    offsets = _c(offsets, np.int64)
    M = len(offsets) - 1
    out = g.copy()
    _check(_load().oracle_gshard(_ptr(g), _ptr(z_bits), _ptr(loads), _ptr(offsets), M, T, E, K,
                                 float(alpha), _ptr(out)), "oracle_gshard")
    return out


def _f32_of_bf16(bits):
    return (np.asarray(bits, np.uint16).astype(np.uint32) << 16).view(np.float32)


def _center_f64(v):
    """Eq. (2) centering of fp64 values: mean summed sequentially in ascending
    expert order, b_e = fp32(v_e - mean)."""
    acc = 0.0
    for x in v:
        acc += float(x)
    mean = acc / len(v)
    return np.array([np.float32(float(x) - mean) for x in v], np.float32)


def rank_averaged_bias(z_bits, tau, K, shard_offsets):
    """The rank-averaged QB estimate that Sec. 2 contrasts with the global
    quantile: every data-parallel shard p takes its own K/E quantile of the
    margins tau_t - z_{t,e} (the r_p-th smallest, r_p = ceil(n_p K / E)), the
    shards' quantiles are averaged in fp64 (ascending p; an empty shard has
    no quantile and is left out), and the average is centered as in Eq. (2).
    Returns (b float32 [E], per-shard quantiles uint16 [P', E])."""
    z_bits = _c(z_bits, np.uint16)
    T, E = z_bits.shape
    tau = _c(tau, np.float32)
    off = np.asarray(shard_offsets, np.int64)
    qs = []
    for p in range(len(off) - 1):
        a, b = int(off[p]), int(off[p + 1])
        if b == a:
            continue
        qs.append(quantile(z_bits[a:b], tau[a:b], target_rank(b - a, E, K)))
    qs = np.array(qs, np.uint16)
    avg = np.zeros(E, np.float64)
    for e in range(E):
        acc = 0.0
        for p in range(len(qs)):
            acc += float(_f32_of_bf16(qs[p, e]))
        avg[e] = acc / len(qs)
    return _center_f64(avg), qs


def fixed_hist_bias(z_bits, tau, K, lo, width, nbins=256):
    """The fixed-resolution histogram estimate of Sec. 2 (histogram counts of
    the margins summed over ranks): margin m falls in bin
    j = floor(fp32(fp32(m - lo) * fp32(1 / width))) clamped to [0, nbins - 1];
    the estimate of expert e is the upper edge lo + (j + 1) * width (fp64) of
    the first bin whose cumulative count reaches r = ceil(T K / E), centered
    as in Eq. (2).  Returns (b float32 [E], estimates float64 [E])."""
    z_bits = _c(z_bits, np.uint16)
    T, E = z_bits.shape
    tau = _c(tau, np.float32)
    r = target_rank(T, E, K)
    lo32, inv_w = np.float32(lo), np.float32(np.float32(1.0) / np.float32(width))
    est = np.zeros(E, np.float64)
    for e in range(E):
        m = _f32_of_bf16(margins(z_bits, tau, e))
        x = (m - lo32) * inv_w  # float32 arithmetic, round to nearest
        j = np.clip(np.floor(x), 0, nbins - 1).astype(np.int64)
        counts = np.bincount(j, minlength=nbins)
        jr = int(np.argmax(np.cumsum(counts) >= r))
        est[e] = float(np.float32(lo)) + (jr + 1) * float(np.float32(width))
    return _center_f64(est), est


def eqb_step(z_bits, b, K, offsets=None):
    """The whole forward statistic of one layer on the oracle: routing, the
    exact quantile of every expert by full sort, and the centered bias."""
    idx, tau, loads = route(z_bits, b, K, offsets)
    T, E = np.asarray(z_bits).shape
    r = target_rank(T, E, K)
    qhat = quantile(z_bits, tau, r)
    return dict(idx=idx, tau=tau, loads=loads, qhat=qhat, b_next=bias_update(qhat), r=r)
