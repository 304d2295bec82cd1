"""Pins for the verification oracle (Sec. 3.1: the unmodified speculative-sampling
rule of Leviathan et al.).  None of these re-types the oracle's formulas: they
check it against the losslessness theorem, exact brute-force integration,
library softmax, and special cases with known answers."""
import json
import os

import numpy as np
import pytest
from scipy.special import softmax as sp_softmax

from oracle import verify as ov
from oracle.drafter import inverse_cdf

GOLD = os.path.join(os.path.dirname(__file__), "golden", "hand_cases.json")


def _dyadic(perm_seed: int):
    g = json.load(open(GOLD))["dyadic_verify"]
    rng = np.random.default_rng(perm_seed)
    perm = rng.permutation(16)
    q = np.asarray(g["q_counts"], float)[perm] / g["denominator"]
    p = np.asarray(g["p_counts"], float)[perm] / g["denominator"]
    return p, q


def _rand_rows(rng, n, V, zero_frac=0.0):
    z = rng.standard_normal((n, V)) * 2.0
    if zero_frac:
        z[rng.random((n, V)) < zero_frac] = -np.inf
        z[:, 0] = 0.0
    return sp_softmax(z, axis=-1)


def test_softmax_t_matches_scipy():
    rng = np.random.default_rng(0)
    z = rng.standard_normal((3, 50)) * 4
    for T in (0.5, 1.0, 1.7):
        np.testing.assert_allclose(ov.softmax_t(z, T), sp_softmax(z / T, axis=-1), rtol=1e-13)


@pytest.mark.parametrize("K", [1, 2, 3])
@pytest.mark.parametrize("seed", [0, 1, 2])
def test_emission_distribution_is_lossless(K, seed):
    """Leviathan et al. Theorem: the emitted token at every reached position is
    distributed as p; acceptance at i is sum_y min(p_i, q_i)."""
    rng = np.random.default_rng(seed)
    p = _rand_rows(rng, K + 1, 16, zero_frac=0.2 if seed == 2 else 0.0)
    q = _rand_rows(rng, K, 16, zero_frac=0.2 if seed == 1 else 0.0)
    e = ov.emission_distribution(p, q)
    np.testing.assert_allclose(e["D"], p, atol=1e-12)
    np.testing.assert_allclose(e["accept"], np.minimum(p[:K], q).sum(-1), atol=1e-12)
    # expected emitted tokens per verify: sum_k prod_{i<k} alpha_i
    alpha = np.minimum(p[:K], q).sum(-1)
    closed = sum(np.prod(alpha[:k]) for k in range(K + 1))
    assert abs(e["reach"].sum() - closed) < 1e-12


def _logits_of(prob, T):
    return (T * np.log(prob)).astype(np.float64)


@pytest.mark.parametrize("T", [1.0, 0.7])
def test_bruteforce_position0_exact(T):
    """Integrate verify() over x0 ~ q0 and 64-point midpoint grids of u_accept and
    u_sample.  With the dyadic rows every boundary sits on a grid edge, so the
    empirical emission distribution must equal p_0 to rounding."""
    p0, q0 = _dyadic(3)
    p1, _ = _dyadic(4)
    N = 64
    grid = (np.arange(N) + 0.5) / N
    X, UA, US = np.meshgrid(np.arange(16), grid, grid, indexing="ij")
    X, UA, US = X.ravel(), UA.ravel(), US.ravel()
    B = X.size
    zp = np.broadcast_to(np.stack([_logits_of(p0, T), _logits_of(p1, T)]), (B, 2, 16))
    zq = np.broadcast_to(_logits_of(q0, T)[None, None], (B, 1, 16))
    r = ov.verify(zp, zq, X[:, None], T, UA[:, None], np.stack([US, US], 1))
    w = q0[X] / (N * N)
    emitted0 = r["out_tokens"][:, 0]
    dist = np.bincount(emitted0, weights=w, minlength=16)
    np.testing.assert_allclose(dist, p0, atol=1e-12)
    # accepted fraction = sum_y min(p, q)
    assert abs((w * r["n_accepted"]).sum() - np.minimum(p0, q0).sum()) < 1e-12
    # bonus after acceptance is distributed as p_1
    acc = r["n_accepted"] == 1
    bonus = np.bincount(r["out_tokens"][acc, 1], weights=w[acc], minlength=16)
    np.testing.assert_allclose(bonus / w[acc].sum(), p1, atol=1e-12)


def test_bruteforce_position1_and_expected_length():
    """K=2: the token emitted at position 1, given position 0 accepted, is
    distributed as p_1; E[n_accepted + 1] = 1 + a0 + a0*a1 exactly."""
    p0, q0 = _dyadic(5)
    p1, q1 = _dyadic(6)
    p2, _ = _dyadic(7)
    zp = np.stack([np.log(p0), np.log(p1), np.log(p2)])
    zq = np.stack([np.log(q0), np.log(q1)])
    N = 64
    grid = (np.arange(N) + 0.5) / N
    # position 1 given acceptance at 0 (u_accept[0] = 0 accepts any ratio > 0)
    X1, UA, US = [a.ravel() for a in np.meshgrid(np.arange(16), grid, grid, indexing="ij")]
    B = X1.size
    x = np.stack([np.zeros(B, int), X1], 1)
    r = ov.verify(np.broadcast_to(zp, (B, 3, 16)), np.broadcast_to(zq, (B, 2, 16)), x, 1.0,
                  np.stack([np.zeros(B), UA], 1), np.stack([US, US, US], 1))
    assert (r["n_accepted"] >= 1).all()
    w = q1[X1] / (N * N)
    dist = np.bincount(r["out_tokens"][:, 1], weights=w, minlength=16)
    np.testing.assert_allclose(dist, p1, atol=1e-12)
    # expected emitted length over x0, x1 ~ q and both acceptance uniforms
    X0, X1, U0, U1 = [a.ravel() for a in np.meshgrid(np.arange(16), np.arange(16), grid, grid,
                                                      indexing="ij")]
    B = X0.size
    r = ov.verify(np.broadcast_to(zp, (B, 3, 16)), np.broadcast_to(zq, (B, 2, 16)),
                  np.stack([X0, X1], 1), 1.0, np.stack([U0, U1], 1), np.full((B, 3), 0.5))
    w = q0[X0] * q1[X1] / (N * N)
    a0, a1 = np.minimum(p0, q0).sum(), np.minimum(p1, q1).sum()
    assert abs((w * (r["n_accepted"] + 1)).sum() - (1 + a0 + a0 * a1)) < 1e-12


def test_identical_drafter_accepts_all():
    """p = q row for row (the same bytes): every draft is accepted (ratio 1 > u)
    and the bonus is the inverse CDF of p_K at u_sample[K]."""
    rng = np.random.default_rng(11)
    B, K, V = 4, 5, 4096
    zq = rng.standard_normal((B, K, V)).astype(np.float32) * 3
    zp = np.concatenate([zq, rng.standard_normal((B, 1, V)).astype(np.float32)], 1)
    x = rng.integers(0, V, (B, K))
    ua = rng.random((B, K)).astype(np.float32)
    us = rng.random((B, K + 1)).astype(np.float32)
    r = ov.verify(zp, zq, x, 1.0, ua, us)
    assert (r["n_accepted"] == K).all()
    np.testing.assert_array_equal(r["out_tokens"][:, :K], x)
    for b in range(B):
        p = sp_softmax(zp[b, K].astype(np.float64))
        C = np.cumsum(p)
        expect = int(np.argmax(C > us[b, K] * C[-1]))
        assert r["out_tokens"][b, K] == expect


def test_greedy_is_textbook_argmax():
    rng = np.random.default_rng(12)
    B, K, V = 3, 4, 1000
    zp = rng.standard_normal((B, K + 1, V)).astype(np.float32)
    am = zp.argmax(-1)
    x = am[:, :K].copy()
    x[1, 2] = (x[1, 2] + 1) % V          # reject at position 2 of sequence 1
    x[2, 0] = (x[2, 0] + 5) % V          # reject at position 0 of sequence 2
    r = ov.verify(zp, None, x, 0.0, np.zeros((B, K), np.float32), np.zeros((B, K + 1), np.float32))
    assert list(r["n_accepted"]) == [K, 2, 0]
    assert list(r["out_tokens"][0]) == list(am[0])
    assert list(r["out_tokens"][1]) == list(am[1, :3]) + [-1, -1]
    assert list(r["out_tokens"][2]) == [am[2, 0], -1, -1, -1, -1]
    # ties go to the lowest id
    zt = np.zeros((1, 2, 8), np.float32)
    zt[0, 0, [3, 5]] = 1.0
    r = ov.verify(zt, None, np.array([[5]]), 0.0, np.zeros((1, 1)), np.zeros((1, 2)))
    assert r["n_accepted"][0] == 0 and r["out_tokens"][0, 0] == 3


def test_temperature_is_logit_scaling():
    rng = np.random.default_rng(13)
    B, K, V = 8, 3, 300
    zq = rng.standard_normal((B, K, V)) * 2
    zp = np.concatenate([zq + 0.5 * rng.standard_normal((B, K, V)),
                         rng.standard_normal((B, 1, V))], 1)
    x = rng.integers(0, V, (B, K))
    ua, us = rng.random((B, K)), rng.random((B, K + 1))
    T = 0.7
    a = ov.verify(zp, zq, x, T, ua, us)
    b = ov.verify(zp / T, zq / T, x, 1.0, ua, us)
    np.testing.assert_array_equal(a["out_tokens"], b["out_tokens"])
    np.testing.assert_allclose(a["p_x"], b["p_x"], rtol=1e-12)


def test_inverse_cdf_special_cases():
    w = np.zeros(16)
    w[9] = 1.0
    for u in (0.0, 0.3, 0.999):
        assert inverse_cdf(w, u)[0] == 9
    flat = np.ones(16)
    for u in np.linspace(0.01, 0.98, 37):
        if abs(16 * u - round(16 * u)) > 1e-6:
            assert inverse_cdf(flat, u)[0] == int(np.floor(16 * u))
    # zero-weight ids are never chosen
    w = np.array([0.0, 1.0, 0.0, 0.0, 2.0, 0.0])
    picks = {inverse_cdf(w, u)[0] for u in np.linspace(0, 0.999, 200)}
    assert picks == {1, 4}


def test_flags_mark_boundaries():
    # ratio exactly equal to u: flag bit 0 set
    V = 8
    p = np.full(V, 1 / V)
    q = p.copy()
    q[0], q[1] = 2 / V, 0.0 + 1e-9
    q /= q.sum()
    zp = np.log(np.stack([p, p]))[None]
    zq = np.log(q)[None, None]
    ratio = p[0] / q[0]
    r = ov.verify(zp, zq, np.array([[0]]), 1.0, np.array([[ratio]]), np.array([[0.3, 0.3]]))
    assert r["flags"][0, 0] & ov.FLAG_RATIO
    # inverse-CDF point on a bin edge: flag bit 1 set
    zp2 = np.log(np.stack([np.full(4, 0.25)] * 2))[None]
    r = ov.verify(zp2, zp2[:, :1], np.array([[2]]), 1.0, np.array([[0.1]]), np.array([[0.5, 0.5]]))
    assert r["n_accepted"][0] == 1 and r["flags"][0, 1] & ov.FLAG_CDF


def test_acceptance_threshold_is_strict_and_exact():
    """Accept iff u < p(x)/q(x): measured on a 10^5-point midpoint grid the accepted
    share is N*min(1, p/q) to within one point, and u equal to the ratio rejects."""
    rng = np.random.default_rng(21)
    V = 50
    zq = rng.standard_normal(V) * 2
    zp = zq + 0.8 * rng.standard_normal(V)
    p, q = sp_softmax(zp), sp_softmax(zq)
    x = int(np.argmax(q / p))          # a token with ratio < 1
    ratio = p[x] / q[x]
    N = 100_000
    u = (np.arange(N) + 0.5) / N
    B = N
    r = ov.verify(np.broadcast_to(np.stack([zp, zp]), (B, 2, V)), np.broadcast_to(zq, (B, 1, V)),
                  np.full((B, 1), x), 1.0, u[:, None], np.full((B, 2), 0.5))
    assert abs(r["n_accepted"].sum() - N * ratio) <= 1.0
    # exact tie: p/q = 1/2 with u = 1/2 rejects
    zq2 = np.log(np.array([0.5, 0.25, 0.25]))
    zp2 = np.log(np.array([0.25, 0.5, 0.25]))
    r = ov.verify(np.stack([zp2, zp2])[None], zq2[None, None], np.array([[0]]), 1.0,
                  np.array([[0.5]]), np.array([[0.1, 0.1]]))
    assert r["n_accepted"][0] == 0 and r["out_tokens"][0, 0] == 1


def test_inverse_cdf_point_on_edge_takes_next_bin():
    """u*S equal to C_j selects j+1 (smallest j with u*S < C_j)."""
    zp2 = np.log(np.stack([np.full(4, 0.25)] * 2))[None]
    r = ov.verify(zp2, zp2[:, :1], np.array([[2]]), 1.0, np.array([[0.1]]), np.array([[0.5, 0.5]]))
    assert r["out_tokens"][0, 1] == 2
    r = ov.verify(zp2, zp2[:, :1], np.array([[2]]), 1.0, np.array([[0.1]]), np.array([[0.5, 0.25]]))
    assert r["out_tokens"][0, 1] == 1


def test_emitted_tokens_pass_chi_square():
    """Monte Carlo on a 16-token vocabulary: draft tokens x_i ~ q_i, random
    uniforms; the first emitted token follows p_0 and, among the sequences that
    accepted position 0, the second follows p_1 (Pearson chi-square).  The same
    counts reject q_0, so the test can tell the two apart."""
    from scipy.stats import chisquare
    rng = np.random.default_rng(11)
    V, K, N = 16, 3, 40000
    zp = (rng.standard_normal((K + 1, V)) * 1.5).astype(np.float32)
    zq = (zp[:K] + rng.standard_normal((K, V)).astype(np.float32)).astype(np.float32)
    p = sp_softmax(zp.astype(np.float64), axis=-1)
    q = sp_softmax(zq.astype(np.float64), axis=-1)
    ud = rng.random((N, K))
    cq = np.cumsum(q, axis=-1)
    x = np.stack([np.minimum(np.searchsorted(cq[i], ud[:, i] * cq[i, -1], side="right"), V - 1)
                  for i in range(K)], 1).astype(np.int32)
    o = ov.verify(np.broadcast_to(zp, (N, K + 1, V)).copy(), np.broadcast_to(zq, (N, K, V)).copy(), x, 1.0,
                  rng.random((N, K), dtype=np.float32), rng.random((N, K + 1), dtype=np.float32))
    first = np.bincount(o["out_tokens"][:, 0], minlength=V)
    assert chisquare(first, N * p[0]).pvalue > 1e-3
    assert chisquare(first, N * q[0]).pvalue < 1e-6
    reached = o["n_accepted"] >= 1
    second = np.bincount(o["out_tokens"][reached, 1], minlength=V)
    assert chisquare(second, reached.sum() * p[1]).pvalue > 1e-3
