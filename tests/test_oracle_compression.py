"""Pins for the oracle's compression side: SVD (Eq. 3), spectral information
(Eq. 5), greedy rank allocation (Eq. 6-7), compression ratio (Eq. 4) and the
dense footprint (Eq. 2)."""
import itertools
import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


@pytest.mark.parametrize("shape", [(12, 5), (5, 12), (7, 7), (64, 16), (1, 4), (4, 1), (33, 8)])
def test_svd_matches_numpy_and_is_orthonormal(oracle, shape):
    rng = np.random.default_rng(shape[0] * 31 + shape[1])
    X = rng.standard_normal(shape) * np.exp(rng.standard_normal(shape[1]))
    sigma, C, P = oracle.svd(X)
    ref = np.linalg.svd(X, compute_uv=False)
    np.testing.assert_allclose(sigma, ref, rtol=1e-12, atol=1e-13 * ref[0])
    assert np.all(np.diff(sigma) <= 0)
    k = min(shape)
    np.testing.assert_allclose(P @ P.T, np.eye(k), atol=1e-13)
    np.testing.assert_allclose(C @ P, X, atol=1e-12 * max(1.0, ref[0]))
    # columns of C are orthogonal with norms sigma
    np.testing.assert_allclose(C.T @ C, np.diag(sigma ** 2), atol=1e-11 * ref[0] ** 2)


def test_svd_rank_deficient(oracle):
    rng = np.random.default_rng(3)
    X = rng.standard_normal((10, 3)) @ rng.standard_normal((3, 6))  # rank 3
    sigma, C, P = oracle.svd(X)
    assert sigma[3:].max() < 1e-12 * sigma[0]
    np.testing.assert_allclose(C @ P, X, atol=1e-12)


@pytest.mark.parametrize("r", [0, 1, 3, 5])
def test_eckart_young_truncation_error(oracle, r):
    """||X - C[:, :r] P[:r]||_F^2 = sum_{j > r} sigma_j^2."""
    rng = np.random.default_rng(4)
    X = rng.standard_normal((20, 6))
    sigma, C, P = oracle.svd(X)
    err = np.linalg.norm(X - C[:, :r] @ P[:r]) ** 2
    np.testing.assert_allclose(err, (sigma[r:] ** 2).sum(), rtol=1e-11, atol=1e-12)


def test_spectral_information_closed_forms(oracle):
    eps = 0.5
    sigma = np.array([eps, eps * math.sqrt(3), 0.0])
    # log(1 + 1) + log(1 + 3) + log(1 + 0)
    assert oracle.spectral_information(sigma, 0, eps) == 0.0
    np.testing.assert_allclose(oracle.spectral_information(sigma, 1, eps), math.log(2), rtol=1e-15)
    np.testing.assert_allclose(oracle.spectral_information(sigma, 3, eps), math.log(8), rtol=1e-15)
    # marginal gain of Eq. 7 is the increment of Eq. 5
    s = np.array([3.0, 1.0, 0.25])
    for r in range(2):
        gain = oracle.spectral_information(s, r + 1, 0.1) - oracle.spectral_information(s, r, 0.1)
        np.testing.assert_allclose(gain, math.log(1 + s[r] ** 2 / 0.01), rtol=1e-13)


def test_greedy_hand_example(oracle):
    gold = json.load(open(os.path.join(GOLDEN, "greedy_hand_example.json")))
    r = oracle.allocate_ranks([np.array(s) for s in gold["sigmas"]], gold["r_min"],
                              gold["r_max"], gold["R_tot"], gold["eps"])
    assert list(r) == gold["expected_ranks"]


def _objective(sigmas, ranks, eps):
    return sum(sum(math.log1p(s[j] ** 2 / eps ** 2) for j in range(r)) for s, r in zip(sigmas, ranks))


@pytest.mark.parametrize("seed", range(12))
def test_greedy_equals_exhaustive_optimum(oracle, seed):
    """On tiny problems the greedy result attains the Eq. 6 optimum found by
    enumerating every feasible rank vector."""
    rng = np.random.default_rng(seed)
    nb = int(rng.integers(1, 5))
    d = int(rng.integers(2, 7))
    avail = [int(min(rng.integers(1, 9), d)) for _ in range(nb)]
    sigmas = [np.sort(rng.exponential(1.0, a))[::-1] for a in avail]
    r_min = int(rng.integers(0, 2))
    r_max = int(rng.integers(max(r_min, 1), d + 1))
    start = sum(min(r_min, a) for a in avail)
    R_tot = start + int(rng.integers(0, sum(avail) + 2))
    eps = float(rng.uniform(0.05, 2.0))
    got = oracle.allocate_ranks(sigmas, r_min, r_max, R_tot, eps)
    best = -1.0
    for ranks in itertools.product(*[range(min(r_min, a), min(r_max, a) + 1) for a in avail]):
        if sum(ranks) <= R_tot:
            best = max(best, _objective(sigmas, ranks, eps))
    np.testing.assert_allclose(_objective(sigmas, got, eps), best, rtol=1e-12)
    caps = [min(r_max, a) for a in avail]
    assert all(min(r_min, a) <= r <= c for r, a, c in zip(got, avail, caps))
    assert sum(got) == min(R_tot, sum(caps))   # budget met exactly unless every cap binds


@pytest.mark.parametrize("seed", range(6))
def test_greedy_equals_top_singular_values(oracle, seed):
    """Closed form: r_min per block plus the largest remaining singular values
    (subject to r_max) -- the gain is increasing in sigma, for any eps."""
    rng = np.random.default_rng(100 + seed)
    nb, d = 9, 16
    sigmas = [np.sort(rng.exponential(1.0, d))[::-1] for _ in range(nb)]
    r_min, r_max = 2, 11
    U = 40
    R_tot = nb * r_min + U
    cand = [(s[j], -b, b) for b, s in enumerate(sigmas) for j in range(r_min, r_max)]
    cand.sort(reverse=True)
    expect = np.full(nb, r_min)
    for _, _, b in cand[:U]:
        expect[b] += 1
    for eps in (1e-6, 0.3, 10.0):
        got = oracle.allocate_ranks(sigmas, r_min, r_max, R_tot, eps)
        np.testing.assert_array_equal(got, expect)


def test_greedy_ties_go_to_lowest_index_and_zero_gain_flag(oracle):
    s = [np.array([1.0, 0.5, 0.0]), np.array([1.0, 0.5, 0.0])]
    assert list(oracle.allocate_ranks(s, 0, 3, 1, 1.0)) == [1, 0]
    assert list(oracle.allocate_ranks(s, 0, 3, 3, 1.0)) == [2, 1]
    # zero singular values still take budget unless the stop flag is set
    assert list(oracle.allocate_ranks(s, 0, 3, 6, 1.0)) == [3, 3]
    assert list(oracle.allocate_ranks(s, 0, 3, 6, 1.0, stop_at_zero_gain=True)) == [2, 2]
    with pytest.raises(RuntimeError):
        oracle.allocate_ranks(s, 2, 3, 3, 1.0)   # r_min alone exceeds R_tot


def test_compression_ratio_hand_example(oracle):
    gold = json.load(open(os.path.join(GOLDEN, "compression_ratio_example.json")))
    n = len(gold["rank_k"])
    rho = oracle.compression_ratio([gold["B"]] * n, gold["rank_k"], gold["rank_v"], gold["d"])
    assert rho == Fraction(*gold["expected_num_den"])
    half = oracle.compression_ratio([gold["B"]] * 3, [64] * 3, [64] * 3, gold["d"])
    assert half == Fraction(*gold["uniform_half_rank_expected"])


def test_compression_ratio_counts_stored_numbers(oracle):
    """rho = (numbers stored by the factors) / (numbers in the dense K and V)."""
    rng = np.random.default_rng(5)
    d = 16
    bl = rng.integers(4, 40, size=7)
    rk = np.minimum(rng.integers(0, 17, size=7), bl)
    rv = np.minimum(rng.integers(0, 17, size=7), bl)
    stored = sum(int(k) * (int(n) + d) + int(v) * (int(n) + d) for n, k, v in zip(bl, rk, rv))
    dense = sum(2 * int(n) * d for n in bl)
    assert oracle.compression_ratio(bl, rk, rv, d) == Fraction(stored, dense)


def test_kv_cache_bytes_matches_dense_tensors(oracle):
    import torch
    N, L, H, d = 37, 3, 2, 8
    kv = [torch.zeros((N, H, d), dtype=torch.float16) for _ in range(2 * L)]
    assert oracle.kv_cache_bytes(N, L, H, d) == sum(t.numel() * t.element_size() for t in kv)


def test_compress_then_truncate_keeps_budget(oracle):
    """Alg. 1 Stage 1 composition: stored ranks obey the budget and the stored
    factors are the leading singular triplets."""
    rng = np.random.default_rng(6)
    d = 8
    K = [rng.standard_normal((n, d)) * np.linspace(2, 0.1, d) for n in (12, 20, 9)]
    V = [rng.standard_normal((n, d)) for n in (12, 20, 9)]
    comp = oracle.compress_blocks(K, V, R_tot_k=12, R_tot_v=9, r_min=1, r_max=6)
    assert comp["rank_k"].sum() == 12 and comp["rank_v"].sum() == 9
    for b, Kb in enumerate(K):
        r = int(comp["rank_k"][b])
        C = comp["arena"][comp["off_ck"][b]:comp["off_ck"][b] + Kb.shape[0] * r].reshape(-1, r)
        P = comp["arena"][comp["off_pk"][b]:comp["off_pk"][b] + r * d].reshape(r, d)
        err = np.linalg.norm(Kb - C @ P) ** 2
        s = np.linalg.svd(Kb, compute_uv=False)
        np.testing.assert_allclose(err, (s[r:] ** 2).sum(), rtol=1e-10, atol=1e-12)
