"""Pins for the CPU oracle, each against something other than the oracle:
brute force with a different algorithm, closed forms from App. B, invariants
the paper states, and library routines.  CPU only."""
import json
import os

import numpy as np
import pytest
import torch

import brute
import oracle
from eqb_workloads import even_offsets, ragged_offsets

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def rand_bits(rng, T, E, scale=1.0, ties=False):
    if ties:
        # integer-valued logits in a tiny range: many exact ties in s = z + 0
        v = rng.integers(-3, 4, size=(T, E)).astype(np.float32) * 0.5
    else:
        v = (rng.standard_normal((T, E)) * scale).astype(np.float32)
    return brute.bf16_bits_from_f32(v)


# ---------------------------------------------------------------- encodings

def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(1)
    x = np.concatenate([
        rng.standard_normal(20000).astype(np.float32),
        (rng.standard_normal(2000) * 1e-39).astype(np.float32),   # fp32 subnormals
        np.array([0.0, -0.0, 1.0 + 2**-8, 1.0 + 3 * 2**-8, -(1.0 + 2**-8), 2**-133,
                  2**-134, 2**-135, -(2**-134), 3.0e38, -3.0e38, 1.7e38], dtype=np.float32),
        rng.integers(0, 2**32, 20000, dtype=np.uint64).astype(np.uint32).view(np.float32),
    ])
    x = x[np.isfinite(x)]
    want = brute.bf16_bits_from_f32(x)
    got = np.array([oracle.f32_to_bf16_bits(v) for v in x], dtype=np.uint16)
    # torch may saturate differently only for values that round past bf16 max
    fin = np.isfinite(brute.f32_from_bf16_bits(want))
    assert np.array_equal(got[fin], want[fin])


def test_kappa_is_order_preserving_and_invertible():
    allb = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    vals = brute.f32_from_bf16_bits(allb)
    fin = np.isfinite(vals)
    keys = np.array([oracle.kappa(int(x)) for x in allb])
    assert len(set(keys.tolist())) == 65536
    assert all(oracle.kappa_inv(int(k)) == int(x) for k, x in zip(keys, allb))
    fk, fv = keys[fin], vals[fin]
    order = np.argsort(fk, kind="stable")
    sv = fv[order]
    assert np.all(sv[1:] >= sv[:-1])  # keys sort values ascending (-0 just below +0)


# ---------------------------------------------------------------- routing

@pytest.mark.parametrize("E", [2, 3, 8])
@pytest.mark.parametrize("ties", [False, True])
def test_route_matches_repeated_extraction(E, ties):
    rng = np.random.default_rng(10 + E + 100 * ties)
    T = 40
    z = rand_bits(rng, T, E, ties=ties)
    b = np.zeros(E, np.float32) if ties else (rng.standard_normal(E) * 0.3).astype(np.float32)
    for K in range(1, E):
        idx, tau, loads = oracle.route(z, b, K)
        for t in range(T):
            want_idx, want_tau = brute.topk_by_extraction(brute.scores(z[t], b), K)
            assert list(idx[t]) == want_idx
            assert np.float32(tau[t]).tobytes() == np.float32(want_tau).tobytes()


def test_cutoff_is_lower_endpoint_of_threshold_identity():
    rng = np.random.default_rng(3)
    E = 8
    z = rand_bits(rng, 24, E)
    b = (rng.standard_normal(E) * 0.5).astype(np.float32)
    for K in (1, 2, 5, 7):
        _, tau, _ = oracle.route(z, b, K)
        for t in range(24):
            s = brute.scores(z[t], b)
            alpha, value = brute.cutoff_by_threshold_identity(s, K)
            assert float(tau[t]) == float(alpha)
            topk_sum = sum(sorted(s, reverse=True)[:K])
            assert abs(float(value) - float(topk_sum)) < 1e-5


def test_loads_sum_to_K_times_tokens():
    rng = np.random.default_rng(4)
    T, E = 999, 16
    z = rand_bits(rng, T, E)
    b = (rng.standard_normal(E) * 0.2).astype(np.float32)
    for off in (even_offsets(T, 7), ragged_offsets(T, 9, 5)):
        for K in (1, 4, 15):
            idx, _, loads = oracle.route(z, b, K, off)
            n = np.diff(off)
            assert np.array_equal(loads.sum(1), K * n)
            assert loads.sum() == K * T
            # each token's list is K distinct experts
            assert all(len(set(r)) == K for r in idx)
            # loads are exactly the per-microbatch counts of the index lists
            for l in range(len(n)):
                cnt = np.bincount(idx[off[l]:off[l + 1]].ravel(), minlength=E)
                assert np.array_equal(cnt, loads[l])


# ---------------------------------------------------------------- quantile

def test_quantile_is_smallest_minimiser_of_app_b_objective():
    rng = np.random.default_rng(6)
    for ties in (False, True):
        T, E = 30, 6
        z = rand_bits(rng, T, E, ties=ties)
        b = np.zeros(E, np.float32)
        for K in (1, 2, 5):
            _, tau, _ = oracle.route(z, b, K)
            r = oracle.target_rank(T, E, K)
            q = oracle.quantile(z, tau, r)
            for e in range(E):
                m = brute.f32_from_bf16_bits(oracle.margins(z, tau, e))
                want = brute.quantile_by_objective(m, r)
                assert float(brute.f32_from_bf16_bits(q[e:e + 1])[0]) == float(want)


def test_quantile_counting_invariant():
    rng = np.random.default_rng(7)
    T, E, K = 5000, 32, 4
    z = rand_bits(rng, T, E)
    b = (rng.standard_normal(E) * 0.3).astype(np.float32)
    _, tau, _ = oracle.route(z, b, K)
    r = oracle.target_rank(T, E, K)
    q = brute.f32_from_bf16_bits(oracle.quantile(z, tau, r))
    for e in range(E):
        m = brute.f32_from_bf16_bits(oracle.margins(z, tau, e))
        assert np.sum(m < q[e]) < r <= np.sum(m <= q[e])


@pytest.mark.parametrize("parts", [[1], [3, 5, 8], [64]])
def test_radix_selection_equals_full_sort(parts):
    """Algorithm 1 run literally (brute, Python) over any partition of the
    tokens into ranks returns the full-sort quantile, and so do the oracle's
    own step functions; the summed per-rank counts equal the whole-batch
    counts (P:111 partition invariance)."""
    rng = np.random.default_rng(8)
    T, E, K = 600, 8, 2
    z = rand_bits(rng, T, E, scale=0.7)
    b = (rng.standard_normal(E) * 0.2).astype(np.float32)
    _, tau, _ = oracle.route(z, b, K)
    r = oracle.target_rank(T, E, K)
    q_sort = oracle.quantile(z, tau, r)
    H_all = oracle.hist_hi(z, tau)
    u, rho = oracle.select_hi(H_all, r)
    q_steps = oracle.select_lo(oracle.hist_lo(z, tau, u), u, rho)
    assert np.array_equal(q_steps, q_sort)
    for P in parts:
        perm = rng.permutation(T)
        cuts = np.sort(rng.choice(np.arange(1, T), size=P - 1, replace=False)) if P > 1 else []
        bounds = np.concatenate([[0], cuts, [T]]).astype(int)
        zp, taup = z[perm], tau[perm]
        H_sum = sum(oracle.hist_hi(zp, taup, bounds[p], bounds[p + 1]) for p in range(P))
        assert np.array_equal(H_sum, H_all)
        L_sum = sum(oracle.hist_lo(zp, taup, u, bounds[p], bounds[p + 1]) for p in range(P))
        assert np.array_equal(oracle.select_lo(L_sum, u, rho), q_sort)
        for e in range(E):
            m = oracle.margins(zp, taup, e)
            ranks = [m[bounds[p]:bounds[p + 1]] for p in range(P)]
            assert brute.radix_select_alg1(ranks, r) == int(q_sort[e])


def test_token_permutation_changes_no_quantile_or_global_load():
    rng = np.random.default_rng(9)
    T, E, K = 1000, 16, 3
    z = rand_bits(rng, T, E)
    b = (rng.standard_normal(E) * 0.2).astype(np.float32)
    a = oracle.eqb_step(z, b, K)
    perm = rng.permutation(T)
    p = oracle.eqb_step(z[perm], b, K)
    assert np.array_equal(a["qhat"], p["qhat"])
    assert np.array_equal(a["loads"].sum(0), p["loads"].sum(0))
    assert np.array_equal(a["tau"][perm], p["tau"])


# ---------------------------------------------------------------- closed forms

def cyclic_logits(T, E, K):
    """App. B: enumerate the TK slots cyclically over the E experts;
    token t owns slots tK .. tK+K-1.  z = 1 on owned experts, else 0."""
    z = np.zeros((T, E), np.float32)
    for t in range(T):
        for j in range(K):
            z[t, (t * K + j) % E] = 1.0
    return brute.bf16_bits_from_f32(z)


def test_cyclic_balanced_assignment_golden():
    with open(os.path.join(GOLDEN, "cyclic_balanced.json")) as f:
        cases = json.load(f)["cases"]
    for c in cases:
        T, E, K, M = c["T"], c["E"], c["K"], c["M"]
        z = cyclic_logits(T, E, K)
        b = np.zeros(E, np.float32)
        off = even_offsets(T, M)
        st = oracle.eqb_step(z, b, K, off)
        assert st["r"] == c["r"]
        assert np.all(st["loads"].sum(0) == c["r"])
        assert np.all(st["loads"] == c["load_per_microbatch"])
        assert np.all(st["tau"] == c["tau"])
        assert np.all(brute.f32_from_bf16_bits(st["qhat"]) == c["qhat"])
        assert np.all(st["b_next"] == c["b_next"])
        g = np.random.default_rng(2).standard_normal((T, E)).astype(np.float32)
        g_out, a = oracle.lei(g, st["loads"], off, K, eta=0.5, c=1.0)
        assert np.all(a == c["lei_coefficient"])
        assert np.array_equal(g_out, g)
        mg, ml, _ = oracle.maxvio(st["loads"], off, K)
        assert (mg, ml) == (c["maxvio_global"], c["maxvio_local"])


def test_constant_columns_closed_form():
    """z_{t,e} = c_e for all t, b = 0: every token has the same top-K and
    cutoff tau = c_(K+1); every margin of expert e equals bf16(tau - c_e), so
    b_hat_e = that value; loads are n_l on the top-K experts and 0 elsewhere,
    giving rho = E/K - 1 or -1 and the LEI coefficient of Eq. (norm)."""
    E, K, T = 8, 3, 120
    cvals = np.array([0.5, -1.25, 2.0, 0.75, -0.5, 1.5, 0.25, -2.0], np.float32)
    z = np.tile(brute.bf16_bits_from_f32(cvals), (T, 1))
    b = np.zeros(E, np.float32)
    off = np.array([0, 50, 120], np.int64)
    st = oracle.eqb_step(z, b, K, off)
    order = sorted(range(E), key=lambda e: (-cvals[e], e))
    assert all(list(r) == order[:K] for r in st["idx"])
    tau = cvals[order[K]]
    assert np.all(st["tau"] == tau)
    want_q = brute.bf16_bits_from_f32(np.float32(tau) - cvals)
    want_q[want_q == 0x8000] = 0
    assert np.array_equal(st["qhat"], want_q)
    eta, c = 0.01, 1.5
    _, a = oracle.lei(None, st["loads"], off, K, eta, c)
    rho = np.where(np.isin(np.arange(E), order[:K]), E / K - 1.0, -1.0)
    xi = np.abs(rho).max() / c
    eta_f = float(np.float32(eta))  # the interface takes eta and c as fp32
    xi = np.abs(rho).max() / float(np.float32(c))
    assert np.allclose(a, eta_f * np.tanh(xi) / xi * rho[None, :], rtol=1e-13, atol=0)


def test_margin_domain_boundary():
    """The margins the method accepts are finite with |m| < 2^127: kappa's
    high bytes 0x00 and 0xff hold both |m| >= 2^127 and the non-finite
    patterns.  Constant columns (one cutoff, one margin per expert) put
    expert 0's margin at the largest bf16 below 2^127 (accepted: its
    quantile is that value, high byte 0xfe) or at 2^127 itself (refused by
    the quantile and by the coarse histogram)."""
    E, K, T = 8, 2, 10
    base = np.array([0.0, 1.0, 2.0, 3.0, -1.0, -2.0, 0.5, 1.5], np.float32)
    for z0, ok in [(np.float32(-1.6e38), True), (np.float32(-2.0 ** 127), False)]:
        cols = base.copy()
        cols[0] = z0
        z = np.tile(brute.bf16_bits_from_f32(cols), (T, 1))
        b = np.zeros(E, np.float32)
        _, tau, _ = oracle.route(z, b, K)
        m0 = brute.bf16_bits_from_f32(np.float32(tau[0]) - brute.f32_from_bf16_bits(z[0, :1]))[0]
        assert (oracle.kappa(int(m0)) >> 8) == (0xFE if ok else 0xFF)
        r = oracle.target_rank(T, E, K)
        if ok:
            q = oracle.quantile(z, tau, r, experts=[0])
            assert q[0] == m0
            assert oracle.hist_hi(z, tau)[0, 0xFE] == T
        else:
            with pytest.raises(oracle.OracleError):
                oracle.quantile(z, tau, r, experts=[0])
            with pytest.raises(oracle.OracleError):
                oracle.hist_hi(z, tau)


# ---------------------------------------------------------------- LEI

def test_lei_invariants():
    rng = np.random.default_rng(12)
    T, E, K = 3000, 32, 4
    z = rand_bits(rng, T, E)
    b = (rng.standard_normal(E) * 0.3).astype(np.float32)
    off = ragged_offsets(T, 6, 3)
    _, _, loads = oracle.route(z, b, K, off)
    g = (rng.standard_normal((T, E)) * 0.1).astype(np.float32)
    n = np.diff(off)
    for c in (0.5, 1.0, 4.0, 0.0):
        eta = float(np.float32(0.7))  # the interface takes eta as fp32
        g_out, a = oracle.lei(g, loads, off, K, eta, c)
        for l in range(len(n)):
            if n[l] == 0:
                assert np.all(a[l] == 0)
                continue
            fbar = K * n[l] / E
            rho = loads[l] / fbar - 1.0
            assert abs(rho.sum()) < 1e-9                                  # zero-centred
            assert np.all(np.sign(a[l]) == np.sign(loads[l] - fbar))      # direction
            rt = a[l] / eta
            if c > 0:
                xi = np.abs(rho).max() / c
                assert np.isclose(np.abs(rt).max(), c * np.tanh(xi), rtol=1e-12)
                assert np.abs(rt).max() < c                               # bounded (Eq. norm)
                assert np.allclose(rt / rho, np.tanh(xi) / xi, rtol=1e-12)  # one shared scale
            else:
                assert np.allclose(rt, rho, rtol=1e-12)                   # unnormalised Eq. (LEI)
            seg = slice(off[l], off[l + 1])
            want = (g[seg].astype(np.float64) + a[l][None, :]).astype(np.float32)
            assert np.array_equal(g_out[seg], want)
    g0, a0 = oracle.lei(g, loads, off, K, 0.0, 1.0)
    assert np.array_equal(g0, g) and np.all(a0 == 0)


def test_lei_scale_limit_at_zero():
    """tanh(xi)/xi -> 1 as xi -> 0: a perfectly balanced microbatch has a = 0,
    and a tiny imbalance with large c gives a ~= eta * rho."""
    E, K = 4, 1
    off = np.array([0, 4000], np.int64)
    loads = np.array([[1000, 1000, 1000, 1000]], np.int32)
    _, a = oracle.lei(None, loads, off, K, 2.0, 1.0)
    assert np.all(a == 0)
    loads = np.array([[1001, 999, 1000, 1000]], np.int32)
    _, a = oracle.lei(None, loads, off, K, 2.0, 1e6)
    rho = loads[0] / 1000.0 - 1.0
    assert np.allclose(a[0], 2.0 * rho, rtol=1e-9)


# ---------------------------------------------------------------- bias update

def test_bias_update_centering():
    rng = np.random.default_rng(13)
    q = brute.bf16_bits_from_f32((rng.standard_normal(256) * 2).astype(np.float32))
    bn = oracle.bias_update(q)
    qv = brute.f32_from_bf16_bits(q).astype(np.float64)
    mean = qv.sum() / 256  # exact here: all partial sums fit in fp64
    assert np.array_equal(bn, (qv - mean).astype(np.float32))
    assert abs(bn.astype(np.float64).sum()) < 256 * 2**-22
    # a common shift of b_hat leaves the update unchanged when exact
    shifted = brute.bf16_bits_from_f32(brute.f32_from_bf16_bits(q).astype(np.float32))
    assert np.array_equal(oracle.bias_update(shifted), bn)


def test_target_rank():
    assert oracle.target_rank(4096, 8, 2) == 1024
    assert oracle.target_rank(65536, 64, 8) == 8192
    assert oracle.target_rank(524288, 128, 8) == 32768
    assert oracle.target_rank(2097152, 256, 8) == 65536
    assert oracle.target_rank(1048576, 128, 8) == 65536
    assert oracle.target_rank(10, 8, 3) == 4  # ceil(30/8)


# ---------------------------------------------------------------- router projection

def test_router_logits_matches_float64_matmul_and_one_hot():
    """Sec. 2: z_t = W_r x_t.  Pinned against numpy's float64 matmul (a
    library routine) and the one-hot closed form (x = e_k picks column k)."""
    rng = np.random.default_rng(21)
    T, d, E = 37, 192, 24
    x = brute.bf16_bits_from_f32(rng.standard_normal((T, d)).astype(np.float32))
    W = brute.bf16_bits_from_f32((rng.standard_normal((E, d)) / np.sqrt(d)).astype(np.float32))
    rows = np.arange(T)
    z, ab = oracle.router_logits(x, W, rows)
    xf = brute.f32_from_bf16_bits(x).astype(np.float64)
    Wf = brute.f32_from_bf16_bits(W).astype(np.float64)
    assert np.allclose(z, xf @ Wf.T, rtol=1e-12, atol=1e-12)
    assert np.allclose(ab, np.abs(xf) @ np.abs(Wf).T, rtol=1e-12, atol=1e-12)
    onehot = np.zeros((d, d), np.float32)
    np.fill_diagonal(onehot, 1.0)
    zo, _ = oracle.router_logits(brute.bf16_bits_from_f32(onehot), W, np.arange(0, d, 7))
    assert np.array_equal(zo, Wf[:, ::7].T)


# ------------------------------------------------------------------ MaxVio

def test_maxvio_paper_example():
    """Sec. 5 / App. E: a Local MaxVio of 5.96 means the most-loaded expert
    receives 6.96 times its uniform load.  E = 100, K = 4, n = 2500 tokens:
    the uniform load is K n / E = 100, so a top load of 696 gives 5.96."""
    E, K, n = 100, 4, 2500
    loads = np.full((1, E), 94, np.int32)
    loads[0, 0] = 696
    loads[0, E - 1] = K * n - 696 - 94 * (E - 2)  # loads sum to K n
    assert loads.sum() == K * n and 0 <= loads.min() and loads[0, 1:].max() < 696
    g, l, per = oracle.maxvio(loads, np.array([0, n]), K)
    assert g == l == per[0] == pytest.approx(5.96, abs=1e-12)


def test_maxvio_all_tokens_on_one_expert():
    """Every token of a microbatch picks expert 3: its load is n = fbar E / K,
    so MaxVio = E/K - 1 for that microbatch."""
    E, K = 16, 4
    off = np.array([0, 40, 40, 100], np.int64)  # the middle microbatch is empty
    loads = np.zeros((3, E), np.int32)
    for l, n in enumerate(np.diff(off)):
        loads[l, 3] = n
        loads[l, 4:4 + K - 1] = n
    g, loc, per = oracle.maxvio(loads, off, K)
    assert per[0] == per[2] == E / K - 1 and per[1] == 0.0
    assert loc == E / K - 1
    assert g == E / K - 1


@pytest.mark.parametrize("seed", range(4))
def test_maxvio_against_exact_rationals(seed):
    """Random loads over uneven (one empty) microbatches: the definition
    evaluated in exact rationals, max over experts of f_e / fbar - 1 with
    fbar = K |B| / E; Local is the plain mean over the non-empty microbatches
    and Global uses the loads summed over the step."""
    from fractions import Fraction
    rng = np.random.default_rng(seed)
    E, K, M = 24, 3, 5
    off = np.sort(np.concatenate([[0], rng.integers(1, 400, M - 1), [400]])).astype(np.int64)
    off[2] = off[1]  # an empty microbatch
    loads = np.zeros((M, E), np.int32)
    for l in range(M):
        n = int(off[l + 1] - off[l])
        for _ in range(n):
            loads[l, rng.choice(E, K, replace=False, p=rng.dirichlet(np.ones(E)))] += 1
    g, loc, per = oracle.maxvio(loads, off, K)
    exact = []
    for l in range(M):
        n = int(off[l + 1] - off[l])
        if n:
            fbar = Fraction(K * n, E)
            exact.append(max(Fraction(int(f)) / fbar - 1 for f in loads[l]))
    want_local = sum(exact, Fraction(0)) / len(exact)
    fbar_g = Fraction(K * int(off[-1]), E)
    want_global = max(Fraction(int(f)) / fbar_g - 1 for f in loads.sum(0))
    assert abs(Fraction(loc) - want_local) <= Fraction(1, 2 ** 48)
    assert abs(Fraction(g) - want_global) <= Fraction(1, 2 ** 48)
    assert per[1] == 0.0


# ------------------------------------------------------------------ GShard STE

def gshard_case(T, E, K, M, seed):
    rng = np.random.default_rng(seed)
    z = brute.bf16_bits_from_f32(rng.standard_normal((T, E)).astype(np.float32))
    off = ragged_offsets(T, M, seed=seed)
    _, _, loads = oracle.route(z, np.zeros(E, np.float32), K, off)
    g = (0.1 * rng.standard_normal((T, E))).astype(np.float32)
    return z, off, loads, g


def test_gshard_is_gradient_of_aux_loss():
    """Finite differences of L = alpha sum_e F_e P^G_e (Sec. 2, the GShard
    loss with F held fixed), P^G_e = |B_l|^-1 sum_t s_{t,e} / sum_j s_{t,j},
    with respect to each score s_{t,j}, against the injected term."""
    T, E, K, M = 6, 5, 2, 2
    z, _, _, g = gshard_case(T, E, K, M, seed=11)
    off = np.array([0, 2, 6], np.int64)  # two local batches, neither the whole step
    _, _, loads = oracle.route(z, np.zeros(E, np.float32), K, off)
    alpha = 0.75
    term = oracle.gshard(np.zeros((T, E), np.float32), z, loads, off, K, alpha).astype(np.float64)
    s0 = 1.0 / (1.0 + np.exp(-brute.f32_from_bf16_bits(z).astype(np.float64)))

    def loss(s):
        total = 0.0
        for l in range(M):
            a, b_ = int(off[l]), int(off[l + 1])
            if b_ == a:
                continue
            F = loads[l] / (K * (b_ - a))
            P = (s[a:b_] / s[a:b_].sum(1, keepdims=True)).mean(0)
            total += alpha * float((F * P).sum())
        return total

    h = 1e-6
    for t in range(T):
        for j in range(E):
            sp, sm = s0.copy(), s0.copy()
            sp[t, j] += h
            sm[t, j] -= h
            fd = (loss(sp) - loss(sm)) / (2 * h)
            assert abs(fd - term[t, j]) <= 1e-7 + 1e-5 * abs(fd), (t, j, fd, term[t, j])


def test_gshard_orthogonal_to_scores_and_zero_when_balanced():
    """The aux loss depends on s_t only through s_t / sum_j s_t,j, so the
    gradient is orthogonal to s_t (sum_j s_tj dL/ds_tj = 0); with loads equal
    to K n / E for every expert (F = Q) the term vanishes and g is unchanged."""
    T, E, K, M = 200, 8, 2, 3
    z, off, loads, g = gshard_case(T, E, K, M, seed=5)
    term = oracle.gshard(np.zeros((T, E), np.float32), z, loads, off, K, 1.0).astype(np.float64)
    s = 1.0 / (1.0 + np.exp(-brute.f32_from_bf16_bits(z).astype(np.float64)))
    assert np.max(np.abs((s * term).sum(1))) < 1e-9
    assert np.max(np.abs(term)) > 1e-6
    off_b = np.array([0, 80, 160, 200], np.int64)  # K n / E integral: n in {80, 80, 40}
    bal = np.repeat((K * np.diff(off_b) // E)[:, None], E, axis=1).astype(np.int32)
    assert np.array_equal(oracle.gshard(g, z, bal, off_b, K, 3.0), g)


# ------------------------------------------- comparison statistics (Sec. 2)

def integer_case(T, E, K, seed):
    """Integer logits (so every score, cutoff and margin is an integer) with
    b = 0; returns z bits and tau."""
    rng = np.random.default_rng(seed)
    z = brute.bf16_bits_from_f32(rng.integers(-8, 9, size=(T, E)).astype(np.float32))
    _, tau, _ = oracle.route(z, np.zeros(E, np.float32), K)
    return z, tau


def pin_rank_avg_single_shard_is_eqb(fn):
    rng = np.random.default_rng(1)
    T, E, K = 300, 16, 2
    z = brute.bf16_bits_from_f32(rng.standard_normal((T, E)).astype(np.float32))
    st = oracle.eqb_step(z, np.zeros(E, np.float32), K)
    b, _ = fn(z, st["tau"], K, [0, T])
    assert np.array_equal(b, st["b_next"])


def pin_rank_avg_against_sorted_shards(fn):
    """Each shard's quantile by numpy's sort of its margins, the average and
    the centering in exact rationals."""
    from fractions import Fraction
    rng = np.random.default_rng(2)
    T, E, K = 240, 8, 3
    z = brute.bf16_bits_from_f32(rng.standard_normal((T, E)).astype(np.float32))
    _, tau, _ = oracle.route(z, np.zeros(E, np.float32), K)
    off = [0, 40, 40, 130, 240]  # includes an empty shard
    b, _ = fn(z, tau, K, off)
    zf = brute.f32_from_bf16_bits(z)
    avg = []
    for e in range(E):
        qs = []
        for p in range(len(off) - 1):
            a, c = off[p], off[p + 1]
            if c == a:
                continue
            m = brute.f32_from_bf16_bits(brute.bf16_bits_from_f32((tau[a:c] - zf[a:c, e]).astype(np.float32)))
            r = -(-(c - a) * K // E)
            qs.append(Fraction(float(np.sort(m)[r - 1])))
        avg.append(sum(qs, Fraction(0)) / len(qs))
    mean = sum(avg, Fraction(0)) / E
    want = np.array([float(a - mean) for a in avg])
    assert np.all(np.abs(b.astype(np.float64) - want) <= 2.0 ** -20 * np.maximum(1.0, np.abs(want)))


def pin_fixed_hist_integer_grid_is_eqb(fn):
    """Integer margins and unit bins centred on the integers: every margin has
    its own bin, the estimate is the r-th smallest margin + 1/2, and the shift
    cancels in the centering (E a power of two keeps the mean exact)."""
    T, E, K = 400, 16, 2
    z, tau = integer_case(T, E, K, seed=3)
    st = oracle.eqb_step(z, np.zeros(E, np.float32), K)
    b, est = fn(z, tau, K, -64.5, 1.0)
    assert np.array_equal(est, brute.f32_from_bf16_bits(st["qhat"]).astype(np.float64) + 0.5)
    assert np.array_equal(b, st["b_next"])


def pin_fixed_hist_is_bin_of_rth_margin(fn):
    """The first bin whose cumulative count reaches r is the bin that holds
    the r-th smallest margin (order statistic from numpy's sort)."""
    rng = np.random.default_rng(4)
    T, E, K = 300, 8, 2
    z = brute.bf16_bits_from_f32(rng.standard_normal((T, E)).astype(np.float32))
    _, tau, _ = oracle.route(z, np.zeros(E, np.float32), K)
    lo, w = -2.0, 0.0625
    _, est = fn(z, tau, K, lo, w, nbins=64)
    zf = brute.f32_from_bf16_bits(z)
    r = -(-T * K // E)
    inv = np.float32(np.float32(1.0) / np.float32(w))
    for e in range(E):
        m = np.sort(brute.f32_from_bf16_bits(brute.bf16_bits_from_f32((tau - zf[:, e]).astype(np.float32))))[r - 1]
        j = int(min(max(np.floor((np.float32(m) - np.float32(lo)) * inv), 0), 63))
        assert est[e] == lo + (j + 1) * w


COMPARISON_PINS = {
    "rank_avg": [pin_rank_avg_single_shard_is_eqb, pin_rank_avg_against_sorted_shards],
    "fixed_hist": [pin_fixed_hist_integer_grid_is_eqb, pin_fixed_hist_is_bin_of_rth_margin],
}


@pytest.mark.parametrize("pin", COMPARISON_PINS["rank_avg"], ids=lambda f: f.__name__)
def test_rank_averaged_bias_pins(pin):
    pin(oracle.rank_averaged_bias)


@pytest.mark.parametrize("pin", COMPARISON_PINS["fixed_hist"], ids=lambda f: f.__name__)
def test_fixed_hist_bias_pins(pin):
    pin(oracle.fixed_hist_bias)


def _rank_avg_size_weighted(z_bits, tau, K, off):
    """A plausible mistake: shards weighted by their token counts."""
    T, E = z_bits.shape
    num = np.zeros(E)
    for p in range(len(off) - 1):
        a, c = off[p], off[p + 1]
        if c > a:
            q = oracle.quantile(z_bits[a:c], tau[a:c], oracle.target_rank(c - a, E, K))
            num += (c - a) * brute.f32_from_bf16_bits(q)
    avg = num / T
    return (avg - avg.mean()).astype(np.float32), None


def _rank_avg_global_rank(z_bits, tau, K, off):
    """A plausible mistake: every shard uses the global rank r = ceil(TK/E)."""
    T, E = z_bits.shape
    qs = []
    for p in range(len(off) - 1):
        a, c = off[p], off[p + 1]
        if c > a:
            qs.append(brute.f32_from_bf16_bits(oracle.quantile(z_bits[a:c], tau[a:c],
                                                               min(c - a, oracle.target_rank(T, E, K)))))
    avg = np.mean(qs, axis=0).astype(np.float64)
    return (avg - avg.mean()).astype(np.float32), None


def _fixed_hist_lower_edge(z_bits, tau, K, lo, w, nbins=256):
    """A plausible mistake: the lower bin edge as the estimate."""
    b, est = oracle.fixed_hist_bias(z_bits, tau, K, lo, w, nbins)
    est = est - w
    return (est - est.mean()).astype(np.float32), est


@pytest.mark.parametrize("kind,wrong", [("rank_avg", _rank_avg_size_weighted),
                                        ("rank_avg", _rank_avg_global_rank),
                                        ("fixed_hist", _fixed_hist_lower_edge)],
                         ids=["size_weighted", "global_rank", "lower_edge"])
def test_comparison_pins_reject_planted_mistakes(kind, wrong):
    failed = 0
    for pin in COMPARISON_PINS[kind]:
        try:
            pin(wrong)
        except AssertionError:
            failed += 1
    assert failed > 0
