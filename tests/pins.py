"""Pins for the fp64 oracle: facts fixed by the paper and by mathematics.

Each ``check_*`` takes an ``oracle.Oracle`` (the real one, or a mutant built
by ``test_oracle_planted.py``) and raises ``AssertionError`` when the oracle
disagrees with the fact.  Every check computes its expected side from the
definitions directly (numpy, brute force over tokens or pairs), never from the
oracle's own helpers.
"""
from __future__ import annotations

import ast
import json
import math
import operator
import os

import numpy as np

import oracle

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


# --------------------------------------------------------------------------
# small input builders (bf16 bit patterns, exact by construction)
# --------------------------------------------------------------------------
def gauss_cache(rng, n, d, offset=1.5, outliers=True):
    """Rows m + r z with a per-cache offset m and log-normal per-row scale."""
    m = rng.normal(size=d) * offset
    r = np.exp(rng.normal(scale=0.5, size=(n, 1)))
    if outliers:
        r[rng.random(n) < 0.1] *= 8.0
    return oracle.bf16_bits(m + r * rng.normal(size=(n, d)))


def int_cache(rng, n, d, lo=-8, hi=8):
    """Small integers: exact in bf16, and still exact after integer shifts."""
    return oracle.bf16_bits(rng.integers(lo, hi + 1, size=(n, d)).astype(np.float32))


def as_float(v):
    return oracle.bits_to_float(v)


# --------------------------------------------------------------------------
# golden fixtures (hand-derived closed forms)
# --------------------------------------------------------------------------
_OPS = {ast.Add: operator.add, ast.Sub: operator.sub, ast.Mult: operator.mul,
        ast.Div: operator.truediv, ast.USub: operator.neg}


def closed_form(expr: str) -> float:
    """Evaluate a fixture value such as '1 - 1/sqrt(2)' (numbers, + - * /,
    sqrt only)."""
    def ev(node):
        if isinstance(node, ast.Expression):
            return ev(node.body)
        if isinstance(node, ast.Constant) and isinstance(node.value, (int, float)):
            return float(node.value)
        if isinstance(node, ast.BinOp) and type(node.op) in _OPS:
            return _OPS[type(node.op)](ev(node.left), ev(node.right))
        if isinstance(node, ast.UnaryOp) and type(node.op) in _OPS:
            return _OPS[type(node.op)](ev(node.operand))
        if (isinstance(node, ast.Call) and isinstance(node.func, ast.Name)
                and node.func.id == "sqrt" and len(node.args) == 1):
            return math.sqrt(ev(node.args[0]))
        raise ValueError(f"unsupported fixture expression: {expr!r}")
    return ev(ast.parse(expr, mode="eval"))


def golden_cases():
    out = []
    for name in sorted(os.listdir(GOLDEN)):
        if name.endswith(".json"):
            with open(os.path.join(GOLDEN, name)) as f:
                out.append((name, json.load(f)))
    return out


def check_golden(orc, case):
    if "dispersion" in case:
        x = oracle.bf16_bits(np.asarray(case["x"], np.float32))
        assert math.isclose(orc.dispersion(x), closed_form(case["dispersion"]), rel_tol=1e-12,
                            abs_tol=1e-15)
        return
    if "weights" in case:
        v = oracle.bf16_bits(np.asarray(case["v"], np.float32))
        s = orc.scores_weighted(v, np.asarray(case["weights"], np.float64), oracle.L2)
        want = np.array([closed_form(x) for x in case["weighted_scores"]])
        assert np.allclose(s, want, rtol=1e-12, atol=1e-12), (s, want)
        assert orc.select_top_n(s, case["N"]).tolist() == case["kept"]
        return
    if "v_stream" in case:
        d_vs = np.asarray(case["v_stream"], np.float32).reshape(-1, 1)
        d_ks = np.asarray(case["k_stream"], np.float32).reshape(-1, 1)
        kc, vc, events = orc.block_process(oracle.bf16_bits(d_ks), oracle.bf16_bits(d_vs),
                                           case["B"], case["N"], oracle.L2)
        got = [None if e is None else e.tolist() for e in events]
        assert got == case["events_kept"], (got, case["events_kept"])
        assert as_float(vc).ravel().tolist() == case["final_v"]
        assert as_float(kc).ravel().tolist() == case["final_k"]
        return
    v = oracle.bf16_bits(np.asarray(case["v"], np.float32))
    assert np.allclose(orc.mean(v), [closed_form(x) for x in case["mean"]], rtol=0, atol=1e-12)
    for name, expected in case["scores"].items():
        var = oracle.VARIANTS[name]
        s = orc.scores(v, var)
        want = np.array([closed_form(x) for x in expected])
        assert np.allclose(s, want, rtol=1e-12, atol=1e-12), (name, s, want)
        kept = orc.select_top_n(s, case["N"])
        assert kept.tolist() == case["kept"][name], (name, kept, case["kept"][name])
        k = v[::-1].copy()
        k2, v2, kept2, _ = orc.evict_unit(k, v, case["N"], var)
        assert kept2.tolist() == case["kept"][name]
        assert np.array_equal(v2, v[kept2]) and np.array_equal(k2, k[kept2])


# --------------------------------------------------------------------------
# Eq. (decomp): s^2 = |v|^2 - 2 |v| |mean| cos + |mean|^2, tying L2, Dir, Norm
# --------------------------------------------------------------------------
def check_decomp(orc, v):
    x = as_float(v)
    mu = x.mean(axis=0)                      # independent of the oracle
    mn = np.linalg.norm(mu)
    s_l2 = orc.scores(v, oracle.L2)
    s_dir = orc.scores(v, oracle.DIR)
    s_norm = orc.scores(v, oracle.NORM)
    assert np.allclose(s_norm, np.linalg.norm(x, axis=1), rtol=1e-13, atol=0)
    ok = s_norm > 0
    lhs = s_l2[ok] ** 2
    rhs = s_norm[ok] ** 2 - 2 * s_norm[ok] * mn * (1.0 - s_dir[ok]) + mn ** 2
    scale = s_norm[ok] ** 2 + mn ** 2
    assert np.all(np.abs(lhs - rhs) <= 1e-12 * scale), np.max(np.abs(lhs - rhs) / scale)


# --------------------------------------------------------------------------
# Eq. (uniform_outputs) / (recon_error) and the Proposition of Sec. 3.3
# --------------------------------------------------------------------------
def check_recon_error(orc, v):
    x = as_float(v)
    n = x.shape[0]
    s = orc.scores(v, oracle.L2)
    o_star = x.sum(axis=0) / n
    disturb = np.empty(n)
    for j in range(n):                        # brute force: drop token j, re-average
        o_minus_j = np.delete(x, j, axis=0).sum(axis=0) / (n - 1)
        disturb[j] = np.sum((o_star - o_minus_j) ** 2)
    lhs = disturb * (n - 1) ** 2
    assert np.allclose(lhs, s ** 2, rtol=1e-10, atol=1e-12 * np.max(s ** 2)), (lhs, s ** 2)
    # the minimal-disturbance token is the ValueDiff argmin
    assert np.argmin(disturb) == np.argmin(s) or np.isclose(disturb.min(), disturb[np.argmin(s)])
    # and the full ranking agrees
    order_d = np.argsort(disturb, kind="stable")
    order_s = np.argsort(s, kind="stable")
    assert np.allclose(disturb[order_s], disturb[order_d], rtol=1e-9)


# --------------------------------------------------------------------------
# App. A: Dirichlet(1,...,1) expectation and its exact intermediate identities
# --------------------------------------------------------------------------
def check_dirichlet_identities(orc, v):
    x = as_float(v)
    n = x.shape[0]
    s = orc.scores(v, oracle.L2)
    mu = x.mean(axis=0)
    S2 = np.sum(x * x)
    const = S2 - n * np.dot(mu, mu)
    for j in range(n):
        dvec = x[j] - np.delete(x, j, axis=0)           # d_i = v_j - v_i, i != j
        sum_d = dvec.sum(axis=0)
        sum_d2 = np.sum(dvec * dvec)
        # Eq. (app_sum_d)
        assert math.isclose(np.dot(sum_d, sum_d), n * n * s[j] ** 2,
                            rel_tol=1e-10, abs_tol=1e-10 * (1 + S2))
        # Eq. (app_sum_d2)
        assert math.isclose(sum_d2, n * s[j] ** 2 + const, rel_tol=1e-10, abs_tol=1e-10 * (1 + S2))
        # Eq. (app_dirichlet_quad) -> Eq. (app_second_factor)
        quad = (sum_d2 + np.dot(sum_d, sum_d)) / ((n - 1) * n)
        want = (n + 1) / (n - 1) * s[j] ** 2 + const / ((n - 1) * n)
        assert math.isclose(quad, want, rel_tol=1e-10, abs_tol=1e-10 * (1 + S2))


def check_dirichlet_mc(orc, v, rng, draws=400_000, z=4.5):
    """Eq. (app_claim) by Monte Carlo: E[(a_j/(1-a_j))^2 |v_j - o(a)|^2] with
    a ~ Dirichlet(1,...,1) equals 2 s_j^2 / (n(n-1)) + C(n)."""
    x = as_float(v)
    n = x.shape[0]
    s = orc.scores(v, oracle.L2)
    mu = x.mean(axis=0)
    S2 = np.sum(x * x)
    C = 2.0 * (S2 - n * np.dot(mu, mu)) / (n * n * (n - 1) * (n + 1))
    e = rng.exponential(size=(draws, n))
    a = e / e.sum(axis=1, keepdims=True)                  # Dirichlet(1,...,1)
    o = a @ x
    w = (a / (1.0 - a)) ** 2
    for j in range(n):
        g = w[:, j] * np.sum((x[j] - o) ** 2, axis=1)
        mean, se = g.mean(), g.std(ddof=1) / math.sqrt(draws)
        want = 2.0 * s[j] ** 2 / (n * (n - 1)) + C
        assert abs(mean - want) <= z * se + 1e-12, (j, mean, want, se)


# --------------------------------------------------------------------------
# App. B, Eq. (app_eviction_bound): distance from the symmetric limit
# --------------------------------------------------------------------------
def check_distance_bound(orc, v, rng, trials=200):
    x = as_float(v)
    n = x.shape[0]
    s = orc.scores(v, oracle.L2)
    diam = max(np.linalg.norm(x[i] - x[k]) for i in range(n) for k in range(n))
    checked = 0
    for _ in range(trials):
        conc = rng.choice([0.3, 3.0, 30.0, 300.0])
        a = rng.dirichlet(np.full(n, conc))
        delta = np.abs(a - 1.0 / n).sum()
        if 1.0 - 1.0 / n - delta <= 0:
            continue
        phi = (1.0 / n + delta) / (1.0 - 1.0 / n - delta)
        o = a @ x
        for j in range(n):
            e_j = a[j] / (1.0 - a[j]) * np.linalg.norm(x[j] - o)
            assert e_j <= phi * (s[j] + 0.5 * delta * diam) * (1 + 1e-12) + 1e-12
            checked += 1
    assert checked > 0


# --------------------------------------------------------------------------
# invariances that follow from Eq. (vd)
# --------------------------------------------------------------------------
def check_translation(orc, v_int, shift):
    """L2 is unchanged by v_i + c (exact for small integers); Dir and Norm are
    not translation invariant and must move."""
    x = as_float(v_int)
    v2 = oracle.bf16_bits((x + shift).astype(np.float32))
    assert np.array_equal(as_float(v2), x + shift), "shift must be exact in bf16"
    a, b = orc.scores(v_int, oracle.L2), orc.scores(v2, oracle.L2)
    assert np.allclose(a, b, rtol=1e-12, atol=1e-12)
    assert not np.allclose(orc.scores(v_int, oracle.NORM), orc.scores(v2, oracle.NORM))
    assert not np.allclose(orc.scores(v_int, oracle.DIR), orc.scores(v2, oracle.DIR))


def check_homogeneity(orc, v, power, N):
    """Scaling every v by 2^k (exact in bf16 and fp64) scales L2 and Norm by
    2^k and leaves Dir and every kept set unchanged."""
    x = as_float(v)
    v2 = oracle.bf16_bits((x * 2.0 ** power).astype(np.float32))
    assert np.array_equal(as_float(v2), x * 2.0 ** power)
    for var, factor in ((oracle.L2, 2.0 ** power), (oracle.NORM, 2.0 ** power), (oracle.DIR, 1.0)):
        a, b = orc.scores(v, var), orc.scores(v2, var)
        assert np.allclose(b, a * factor, rtol=1e-12, atol=1e-300), var
        assert np.array_equal(orc.select_top_n(a, N), orc.select_top_n(b, N)), var


def check_permutation(orc, v, perm, N):
    """Permuting tokens permutes scores; the kept set maps through the
    permutation (inputs with distinct scores)."""
    for var in (oracle.L2, oracle.DIR, oracle.NORM):
        a = orc.scores(v, var)
        b = orc.scores(v[perm], var)
        assert np.allclose(b, a[perm], rtol=1e-12, atol=1e-13), var
        kept_a = set(orc.select_top_n(a, N).tolist())
        kept_b = set(perm[orc.select_top_n(b, N)].tolist())
        assert kept_a == kept_b, var


# --------------------------------------------------------------------------
# Eq. (eviction): top-N against a brute-force O(n^2) ranking
# --------------------------------------------------------------------------
def brute_force_kept(s, N):
    n = len(s)
    keep = []
    for j in range(n):
        rank = sum(1 for i in range(n) if s[i] > s[j]) + sum(1 for i in range(j) if s[i] == s[j])
        if rank < N:
            keep.append(j)
    return keep


def check_top_n(orc, s, N):
    got = orc.select_top_n(np.asarray(s, np.float64), N).tolist()
    assert got == brute_force_kept(list(s), N), (got, brute_force_kept(list(s), N))


def check_gather(orc, rng, n, d, N, var):
    """pi_N gathers K and V by the same ascending kept list (out-of-place
    numpy gather as the reference); the cache length becomes min(n, N)."""
    v = gauss_cache(rng, n, d)
    k = gauss_cache(rng, n, d)
    k2, v2, kept, s = orc.evict_unit(k, v, N, var)
    assert len(kept) == min(n, N)
    assert np.all(np.diff(kept) > 0)
    assert np.array_equal(v2, v[kept]) and np.array_equal(k2, k[kept])
    if n > N:
        assert kept.tolist() == brute_force_kept(list(orc.scores(v, var)), N)


def check_special_cases(orc, rng):
    d = 4
    # n <= N: identity, nothing moves
    v = gauss_cache(rng, 6, d)
    k2, v2, kept, s = orc.evict_unit(v.copy(), v, 6, oracle.L2)
    assert kept.tolist() == list(range(6)) and s is None and np.array_equal(v2, v)
    # all equal: every L2 score is zero, keep the first N
    v = np.repeat(oracle.bf16_bits(rng.normal(size=(1, d))), 9, axis=0)
    assert np.all(orc.scores(v, oracle.L2) == 0)
    assert orc.evict_unit(v, v, 4, oracle.L2)[2].tolist() == [0, 1, 2, 3]
    # symmetric set {v, -v}: zero mean, L2 ranking = Norm ranking
    h = as_float(gauss_cache(rng, 5, d))
    v = oracle.bf16_bits(np.concatenate([h, -h]).astype(np.float32))
    assert np.allclose(orc.scores(v, oracle.L2), orc.scores(v, oracle.NORM), rtol=1e-14)
    # n = N + 1: evict the argmin; among tied minima the highest index goes
    v = int_cache(rng, 12, d, -2, 2)
    s = orc.scores(v, oracle.L2)
    kept = orc.select_top_n(s, 11)
    evicted = sorted(set(range(12)) - set(kept.tolist()))
    assert len(evicted) == 1
    lowest = np.flatnonzero(s == s.min())
    assert evicted[0] == lowest.max()


def check_block_equivalences(orc, rng):
    """Sec. 2.2: B = T is standard (one-shot) eviction; B = 1 is the per-token
    (decode) loop that evicts at most one token per step."""
    T, d, N = 40, 8, 12
    ks, vs = gauss_cache(rng, T, d), gauss_cache(rng, T, d)
    kc, vc, ev = orc.block_process(ks, vs, T, N)
    k1, v1, kept1, _ = orc.evict_unit(ks, vs, N)
    assert np.array_equal(vc, v1) and np.array_equal(kc, k1) and ev[0].tolist() == kept1.tolist()
    kc, vc, ev = orc.block_process(ks, vs, 1, N)
    kk, vv = ks[:0], vs[:0]
    for t in range(T):
        kk = np.concatenate([kk, ks[t:t + 1]])
        vv = np.concatenate([vv, vs[t:t + 1]])
        kk, vv, kept, _ = orc.evict_unit(kk, vv, N)
        assert len(kept) == min(t + 1, N)
    assert np.array_equal(vc, vv) and np.array_equal(kc, kk)


# --------------------------------------------------------------------------
# App. A, Eq. (app_fastcaote) and (recon_error): the weighted score at the
# uniform attention vector is the brute-force output disturbance
# --------------------------------------------------------------------------
def check_fastcaote_uniform(orc, v):
    x = as_float(v)
    n = x.shape[0]
    w = orc.scores_weighted(v, np.full(n, 1.0 / n), oracle.L2)
    o_star = x.mean(axis=0)
    for j in range(n):                       # drop token j, renormalise uniformly
        o_minus_j = np.delete(x, j, axis=0).mean(axis=0)
        assert math.isclose(w[j], np.linalg.norm(o_star - o_minus_j), rel_tol=1e-10,
                            abs_tol=1e-12)
    # zero attention weight -> zero score; the uniform ranking is ValueDiff's
    z = np.full(n, 1.0 / n)
    z[0] = 0.0
    assert orc.scores_weighted(v, z, oracle.L2)[0] == 0.0
    assert np.array_equal(orc.select_top_n(w, n // 2),
                          orc.select_top_n(orc.scores(v, oracle.L2), n // 2))


# --------------------------------------------------------------------------
# Sec. 3.1: sigma = std over tokens of the distance from the cache mean
# --------------------------------------------------------------------------
def check_dispersion(orc, x_bits):
    x = as_float(x_bits)
    dist = np.linalg.norm(x - x.mean(axis=0), axis=1)
    assert math.isclose(orc.dispersion(x_bits), float(np.std(dist)), rel_tol=1e-10, abs_tol=1e-12)
    same = np.repeat(x_bits[:1], 5, axis=0)
    assert orc.dispersion(same) == 0.0


def all_checks(orc, seed=0):
    """Every pin at a small size; returns the list of (name, error) failures."""
    rng = np.random.default_rng(seed)
    failures = []

    def run(name, fn, *args):
        try:
            fn(*args)
        except AssertionError as e:   # collect, so a mutant report names every pin it breaks
            failures.append((name, repr(e)[:200]))

    for name, case in golden_cases():
        run(f"golden:{name}", check_golden, orc, case)
    run("decomp", check_decomp, orc, gauss_cache(rng, 48, 16))
    run("recon_error", check_recon_error, orc, gauss_cache(rng, 11, 6))
    run("dirichlet_identities", check_dirichlet_identities, orc, gauss_cache(rng, 9, 5))
    run("dirichlet_mc", check_dirichlet_mc, orc, gauss_cache(rng, 6, 4, outliers=False),
        np.random.default_rng(seed + 1))
    run("distance_bound", check_distance_bound, orc, gauss_cache(rng, 7, 5), rng)
    run("translation", check_translation, orc, int_cache(rng, 30, 8), 5.0)
    run("homogeneity", check_homogeneity, orc, gauss_cache(rng, 40, 8), 3, 17)
    run("permutation", check_permutation, orc, gauss_cache(rng, 33, 8),
        rng.permutation(33), 10)
    s = rng.integers(0, 6, size=25).astype(np.float64)
    run("top_n_ties", check_top_n, orc, s, 9)
    run("top_n_distinct", check_top_n, orc, rng.normal(size=40), 13)
    for var in (oracle.L2, oracle.DIR, oracle.NORM):
        run(f"gather:{var}", check_gather, orc, rng, 37, 8, 20, var)
    run("special_cases", check_special_cases, orc, rng)
    run("fastcaote_uniform", check_fastcaote_uniform, orc, gauss_cache(rng, 9, 6))
    run("dispersion", check_dispersion, orc, gauss_cache(rng, 40, 8))
    run("block_equivalences", check_block_equivalences, orc, rng)
    return failures
