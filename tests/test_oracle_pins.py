"""The fp64 oracle against what the paper and mathematics fix (CPU only)."""
import numpy as np
import pytest

import oracle
import pins


@pytest.mark.parametrize("name,case", pins.golden_cases(), ids=[n for n, _ in pins.golden_cases()])
def test_golden(orc, name, case):
    pins.check_golden(orc, case)


@pytest.mark.parametrize("n,d", [(2, 1), (5, 3), (64, 16), (300, 64)])
def test_decomp_identity(orc, n, d):
    pins.check_decomp(orc, pins.gauss_cache(np.random.default_rng(n * d), n, d))


@pytest.mark.parametrize("n,d", [(2, 3), (3, 1), (9, 4), (12, 8)])
def test_uniform_attention_reconstruction(orc, n, d):
    pins.check_recon_error(orc, pins.gauss_cache(np.random.default_rng(n + d), n, d))


@pytest.mark.parametrize("n,d", [(3, 2), (8, 6)])
def test_dirichlet_identities(orc, n, d):
    pins.check_dirichlet_identities(orc, pins.gauss_cache(np.random.default_rng(7 * n), n, d))


@pytest.mark.parametrize("n", [3, 5, 8])
def test_dirichlet_expectation_monte_carlo(orc, n):
    rng = np.random.default_rng(100 + n)
    pins.check_dirichlet_mc(orc, pins.gauss_cache(rng, n, 4, outliers=False), rng)


def test_distance_from_symmetric_limit(orc):
    rng = np.random.default_rng(5)
    for n in (4, 6, 9):
        pins.check_distance_bound(orc, pins.gauss_cache(rng, n, 5), rng)


@pytest.mark.parametrize("shift", [1.0, -7.0, 32.0])
def test_translation_invariance(orc, shift):
    pins.check_translation(orc, pins.int_cache(np.random.default_rng(3), 50, 8), shift)


@pytest.mark.parametrize("power", [-4, 1, 6])
def test_positive_homogeneity(orc, power):
    pins.check_homogeneity(orc, pins.gauss_cache(np.random.default_rng(4), 64, 16), power, 20)


def test_permutation_equivariance(orc):
    rng = np.random.default_rng(6)
    for n in (10, 47):
        pins.check_permutation(orc, pins.gauss_cache(rng, n, 8), rng.permutation(n), n // 3)


@pytest.mark.parametrize("seed", range(6))
def test_top_n_brute_force(orc, seed):
    rng = np.random.default_rng(seed)
    n = int(rng.integers(1, 60))
    s = rng.integers(0, 5, size=n).astype(np.float64) if seed % 2 else rng.normal(size=n)
    for N in sorted({1, max(1, n // 2), max(1, n - 1), n, n + 3}):
        pins.check_top_n(orc, s, N)


@pytest.mark.parametrize("var", [oracle.L2, oracle.DIR, oracle.NORM])
def test_gather_matches_out_of_place(orc, var):
    rng = np.random.default_rng(8)
    for n, N in ((1, 1), (20, 19), (33, 5), (64, 64), (80, 100)):
        pins.check_gather(orc, rng, n, 8, N, var)


def test_special_cases(orc):
    pins.check_special_cases(orc, np.random.default_rng(9))


def test_block_equivalences(orc):
    pins.check_block_equivalences(orc, np.random.default_rng(10))


def test_batched_units_match_single_units(orc):
    """The threaded many-unit entry point (the CPU baseline) is the per-unit
    eviction applied to each unit with that unit's sequence length and budget."""
    rng = np.random.default_rng(11)
    n_seq, per_seq, cap, d = 3, 4, 40, 8
    U = n_seq * per_seq
    k = np.stack([pins.gauss_cache(rng, cap, d) for _ in range(U)])
    v = np.stack([pins.gauss_cache(rng, cap, d) for _ in range(U)])
    lens = np.array([40, 17, 30], np.int32)
    Ns = np.array([25, 20, 29], np.int32)
    k1, v1 = k.copy(), v.copy()
    kept = orc.evict_units(k1, v1, lens, Ns, per_seq, oracle.DIR, nthreads=4, kept_stride=29)
    for u in range(U):
        s = u // per_seq
        n = lens[s]
        k2, v2, kp, _ = orc.evict_unit(k[u, :n], v[u, :n], int(Ns[s]), oracle.DIR)
        m = len(kp)
        assert np.array_equal(kept[u, :m], kp) and np.all(kept[u, m:] == -1)
        assert np.array_equal(v1[u, :m], v2) and np.array_equal(k1[u, :m], k2)
        assert np.array_equal(v1[u, m:], v[u, m:])   # slots past the new length untouched


def test_sum_rows_is_exact_for_bf16(orc):
    """fp64 sums of bf16 rows of moderate range are exact: the compensated sum
    equals an exact rational sum."""
    from fractions import Fraction
    rng = np.random.default_rng(12)
    v = pins.gauss_cache(rng, 500, 4)
    x = pins.as_float(v)
    got = orc.sum_rows(v)
    for c in range(4):
        exact = sum(Fraction(float(t)) for t in x[:, c])
        assert got[c] == float(exact)


@pytest.mark.parametrize("n,d", [(2, 3), (7, 5), (16, 8)])
def test_fastcaote_at_uniform_attention(orc, n, d):
    pins.check_fastcaote_uniform(orc, pins.gauss_cache(np.random.default_rng(n * 31 + d), n, d))


@pytest.mark.parametrize("n,d", [(3, 1), (50, 16), (400, 64)])
def test_dispersion_definition(orc, n, d):
    pins.check_dispersion(orc, pins.gauss_cache(np.random.default_rng(n + 2 * d), n, d))


def test_weights_outside_unit_interval_give_nan(orc):
    v = pins.gauss_cache(np.random.default_rng(1), 4, 4)
    s = orc.scores_weighted(v, np.array([0.2, 1.0, -0.1, 0.0]), oracle.L2)
    assert np.isnan(s[1]) and np.isnan(s[2]) and s[3] == 0.0 and s[0] > 0


def test_nan_ranks_below_zero_and_negative_zero_equals_zero(orc):
    """Reading where the paper is silent: a NaN score (only an invalid input
    makes one) is evicted before any number, including a zero score at a
    higher slot; -0 ties with +0 and the lower slot wins.  Checked against the
    brute-force rank with NaN mapped below every number."""
    s = np.array([np.nan, 0.0, -0.0, 3.0, np.nan, 0.0, 2.0])
    assert list(orc.select_top_n(s, 3)) == [1, 3, 6]
    assert list(orc.select_top_n(s, 5)) == [1, 2, 3, 5, 6]
    assert list(orc.select_top_n(s, 6)) == [0, 1, 2, 3, 5, 6]
    key = np.where(np.isnan(s), -np.inf, s)
    for N in range(1, len(s)):
        assert np.array_equal(orc.select_top_n(s, N), pins.brute_force_kept(key, N))
    # a weight of -0 gives a score of -0, which ranks with the zeros
    v = pins.gauss_cache(np.random.default_rng(3), 4, 4)
    w = orc.scores_weighted(v, np.array([0.5, -0.0, 0.0, 1.0]), oracle.L2)
    assert w[1] == 0.0 and w[2] == 0.0 and np.isnan(w[3])
    assert list(orc.select_top_n(w, 3)) == [0, 1, 2]
