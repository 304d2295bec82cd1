"""Pins for the tree-verification oracle (the multi-candidate form of the
Sec. 3.1 rule for drafts with topk > 1).

* k = 1 is the chain rule: identical outputs to oracle.verify.verify (itself
  pinned by brute force and the Leviathan theorem).
* Losslessness by exact enumeration on a 16-token vocabulary: integrating
  ``depth_emission`` over every tuple of k independent candidates from q gives
  the target row p to 1e-12 (k = 1, 2, 3; rows with zeros).
* The uniform-driven rule ``verify_tree`` against ``depth_emission`` for fixed
  candidates, and the emitted tokens of whole two-depth walks against p, by
  Pearson chi-square over seeded trials.
* An identical drafter accepts the whole chain; greedy hand cases."""
import itertools

import numpy as np
import pytest
from scipy import stats

from oracle import tree as ot
from oracle import verify as ov
from oracle.verify import softmax_t


def _rows(rng, n, V, zeros=0):
    z = 2.0 * rng.standard_normal((n, V))
    if zeros:
        for r in range(n):
            z[r, rng.choice(V, zeros, replace=False)] = -np.inf
    return z


@pytest.mark.parametrize("T", [1.0, 0.7, 0.0])
def test_k1_is_the_chain_rule(T):
    rng = np.random.default_rng(5)
    B, K, V = 40, 4, 64
    zq = _rows(rng, B * K, V).reshape(B, K, V).astype(np.float32)
    zp = (np.concatenate([zq, _rows(rng, B, V)[:, None]], 1) + 0.8 * rng.standard_normal((B, K + 1, V))
          ).astype(np.float32)
    x = np.array([[rng.choice(V, p=softmax_t(zq[b, i], T if T > 0 else 1.0)) for i in range(K)] for b in range(B)])
    ua = rng.random((B, K)).astype(np.float32)
    us = rng.random((B, K + 1)).astype(np.float32)
    chain = ov.verify(zp, zq if T > 0 else None, x, T, ua, us)
    # a k = 1 tree's rows: root, then node (i, 0) = chain position i + 1
    tree = ot.verify_tree(zp, zq if T > 0 else None, x[..., None], T, ua[..., None], us)
    np.testing.assert_array_equal(tree["out_tokens"], chain["out_tokens"])
    np.testing.assert_array_equal(tree["n_accepted"], chain["n_accepted"])
    np.testing.assert_array_equal(tree["flags"], chain["flags"])
    np.testing.assert_array_equal(tree["branch"], np.where(chain["n_accepted"] > 0, 0, -1))


@pytest.mark.parametrize("k,zeros", [(1, 0), (2, 0), (2, 3), (3, 0), (3, 4)])
def test_depth_emission_is_p_by_enumeration(k, zeros):
    rng = np.random.default_rng(10 + k + zeros)
    V = 16
    for trial in range(4):
        p = softmax_t(_rows(rng, 1, V, zeros)[0], 1.0)
        q = softmax_t(_rows(rng, 1, V, zeros)[0], 1.0)
        total = np.zeros(V)
        acc_any = 0.0
        for cands in itertools.product(range(V), repeat=k):
            w = np.prod([q[c] for c in cands])
            if w == 0.0:
                continue
            e = ot.depth_emission(p, q, cands)
            total += w * e["D"]
            acc_any += w * e["acc"].sum()
        np.testing.assert_allclose(total, p, atol=1e-12)
        # the chance that some candidate is accepted grows with k, from sum min(p, q) at k = 1
        if k == 1:
            assert abs(acc_any - np.minimum(p, q).sum()) < 1e-12


def _first_draw(zp, zq, cands, T, n, seed):
    """The token emitted at depth 0 of a one-depth tree (root row zp, node rows
    random: they only feed the token after an accepted candidate)."""
    rng = np.random.default_rng(seed)
    B = n
    k = len(cands)
    rows = np.concatenate([zp[None], _rows(rng, k, len(zp))], 0)
    out = ot.verify_tree(np.repeat(rows[None], B, 0), np.repeat(zq[None, None], B, 0),
                         np.tile(np.asarray(cands)[None, None], (B, 1, 1)), T,
                         rng.random((B, 1, k)), rng.random((B, 2)))
    return out["out_tokens"][:, 0]


@pytest.mark.parametrize("cands", [(3, 3), (1, 5), (5, 2, 0)])
def test_rule_matches_depth_emission_chi_square(cands):
    rng = np.random.default_rng(21)
    V, T = 8, 1.0
    zp = _rows(rng, 1, V)[0]
    zq = zp.copy()
    zq[list(cands)] += 2.5            # a drafter over-confident on its candidates: rejections are frequent
    D = ot.depth_emission(softmax_t(zp, T), softmax_t(zq, T), cands)["D"]
    tok = _first_draw(zp, zq, cands, T, 40000, 3)
    obs = np.bincount(tok, minlength=V)
    keep = D > 1e-3
    chi = stats.chisquare(obs[keep], D[keep] / D[keep].sum() * obs[keep].sum())
    assert chi.pvalue > 1e-4, (obs, D * len(tok))
    # a planted mistake - the residual kept at p after a rejection - is rejected by the same test
    p, q = softmax_t(zp, T), softmax_t(zq, T)
    wrong = np.zeros(V)
    reach = 1.0
    for c in cands:
        a = min(1.0, p[c] / q[c])
        wrong[c] += reach * a
        reach *= 1 - a
    wrong += reach * p
    if np.abs(wrong - D).max() > 0.02:
        assert stats.chisquare(obs[keep], wrong[keep] / wrong[keep].sum() * obs[keep].sum()).pvalue < 1e-4


def test_whole_walk_emits_the_target_distribution():
    """Two depths, k = 2 candidates drawn from q at each depth: the first
    emitted token follows p_root, and the second (given the walk descended
    through candidate 0 = y) follows p of node (0, 0) - for every y."""
    rng = np.random.default_rng(33)
    V, K, k, T, n = 6, 2, 2, 1.0, 60000
    zq = _rows(rng, K, V)
    zroot = _rows(rng, 1, V)[0]
    # node rows: (0, 0) and (0, 1) at depth 0; (1, j) at depth 1
    znodes = _rows(rng, K * k, V)
    zp = np.concatenate([zroot[None], znodes], 0)
    q = softmax_t(zq, T)
    cand = np.stack([np.stack([rng.choice(V, size=n, p=q[i]) for _ in range(k)], -1) for i in range(K)], 1)
    # the target rows of depth-1 nodes depend on the path (the chain token at depth 0): a different row per y
    zp_b = np.repeat(zp[None], n, 0)
    per_y = _rows(rng, V, V)
    for y in range(V):
        sel = cand[:, 0, 0] == y
        zp_b[sel, ot.tree_rows(0, 0, k)] = per_y[y]
    out = ot.verify_tree(zp_b.astype(np.float32), np.repeat(zq[None], n, 0).astype(np.float32), cand, T,
                         rng.random((n, K, k)), rng.random((n, K + 1)))
    first = out["out_tokens"][:, 0]
    p0 = softmax_t(zroot, T)
    assert stats.chisquare(np.bincount(first, minlength=V), p0 * n).pvalue > 1e-4
    for y in range(V):
        sel = (out["branch"] >= 0) & (cand[:, 0, 0] == y) & (first == y) & (out["n_accepted"] >= 1)
        sel &= ~((out["n_accepted"] == 1) & (out["branch"] == 1) & (cand[:, 0, 1] == y))   # descended via j = 0
        second = out["out_tokens"][sel, 1]
        if len(second) < 2000:
            continue
        py = softmax_t(per_y[y], T)
        keep = py * len(second) > 5
        obs = np.bincount(second, minlength=V)
        assert stats.chisquare(obs[keep], py[keep] / py[keep].sum() * obs[keep].sum()).pvalue > 1e-4


def test_identical_drafter_accepts_the_chain():
    rng = np.random.default_rng(41)
    B, K, k, V = 16, 5, 3, 50
    zq = _rows(rng, B * K, V).reshape(B, K, V)
    zp = _rows(rng, B * (1 + K * k), V).reshape(B, 1 + K * k, V)
    zp[:, 0] = zq[:, 0]
    for i in range(1, K):
        zp[:, ot.tree_rows(i - 1, 0, k)] = zq[:, i]             # the chain node's row is the next draft row
    cand = rng.integers(0, V, (B, K, k))
    out = ot.verify_tree(zp.astype(np.float32), zq.astype(np.float32), cand, 1.0, rng.random((B, K, k)),
                         rng.random((B, K + 1)))
    assert (out["n_accepted"] == K).all() and (out["branch"] == 0).all()
    np.testing.assert_array_equal(out["out_tokens"][:, :K], cand[:, :, 0])


def test_greedy_hand_cases():
    V, k = 8, 3
    zp = np.full((1, 1 + 2 * k, V), -5.0, np.float32)
    zp[0, 0, 4] = 1.0                         # root argmax 4
    zp[0, ot.tree_rows(0, 1, k), 6] = 2.0     # node (0, 1) argmax 6
    cand = np.array([[[2, 4, 7], [1, 1, 1]]])
    out = ot.verify_tree(zp, None, cand, 0.0, np.zeros((1, 2, k)), np.zeros((1, 3)))
    # argmax 4 is candidate 1 (a leaf): accepted, then the leaf's argmax 6
    np.testing.assert_array_equal(out["out_tokens"][0], [4, 6, -1])
    assert out["n_accepted"][0] == 1 and out["branch"][0] == 1
    cand[0, 0] = [0, 1, 2]                    # no candidate matches: emit the argmax, accept none
    out = ot.verify_tree(zp, None, cand, 0.0, np.zeros((1, 2, k)), np.zeros((1, 3)))
    np.testing.assert_array_equal(out["out_tokens"][0], [4, -1, -1])
    assert out["n_accepted"][0] == 0 and out["branch"][0] == -1


def test_accepted_leaf_ends_the_walk():
    """Candidate 0 rejected, candidate 1 (a leaf) accepted at depth 0 of a
    two-depth tree: the next token is drawn from the leaf's row and the walk
    stops, even though depth 1's candidates would all be accepted."""
    V, K, k = 8, 2, 2
    zq = np.zeros((1, K, V), np.float32)
    zp = np.zeros((1, 1 + K * k, V), np.float32)
    zp[0, ot.tree_rows(0, 1, k), 5] = 30.0         # the leaf's row puts all its mass on id 5
    cand = np.array([[[2, 3], [1, 1]]])
    ua = np.array([[[0.9999, 0.0], [0.0, 0.0]]])   # p/q = 1 everywhere: accept iff u < 1
    ua[0, 0, 0] = 1.0                              # u = p/q = 1 rejects candidate 0
    out = ot.verify_tree(zp, zq, cand, 1.0, ua, np.full((1, K + 1), 0.5))
    np.testing.assert_array_equal(out["out_tokens"][0], [3, 5, -1])
    assert out["n_accepted"][0] == 1 and out["branch"][0] == 1


def test_strict_threshold_grid_count():
    """Accept iff u < r(x)/q(x): over a midpoint grid of N uniforms for
    candidate 0 the count of acceptances is N min(1, ratio) up to one grid
    point, and u equal to the ratio rejects."""
    V, k, N = 8, 2, 20000
    rng = np.random.default_rng(51)
    zp = _rows(rng, 1, V)[0]
    zq = zp.copy()
    zq[3] += 1.0
    p, q = softmax_t(zp, 1.0), softmax_t(zq, 1.0)
    ratio = p[3] / q[3]
    rows = np.concatenate([zp[None], _rows(rng, k, V)], 0)
    u = (np.arange(N) + 0.5) / N
    ua = np.stack([u, np.full(N, 0.99999)], -1)[:, None, :]
    out = ot.verify_tree(np.repeat(rows[None], N, 0), np.repeat(zq[None, None], N, 0),
                         np.tile(np.array([3, 6])[None, None], (N, 1, 1)), 1.0, ua, np.full((N, 2), 0.5))
    hits = int(((out["n_accepted"] == 1) & (out["branch"] == 0)).sum())
    assert abs(hits - N * ratio) <= 1.0
    one = ot.verify_tree(rows[None], zq[None, None], np.array([[[3, 6]]]), 1.0,
                         np.array([[[ratio, 0.99999]]]), np.full((1, 2), 0.5), ratio_band=0.0)
    assert not (one["n_accepted"][0] == 1 and one["branch"][0] == 0)


def test_greedy_first_matching_candidate():
    """A greedy candidate list with a repeated id: the first match (the chain
    candidate) is the accepted one and the walk descends."""
    V, k = 8, 2
    zp = np.full((1, 1 + 2 * k, V), -5.0, np.float32)
    zp[0, 0, 4] = 1.0
    zp[0, ot.tree_rows(0, 0, k), 1] = 1.0
    out = ot.verify_tree(zp, None, np.array([[[4, 4], [1, 0]]]), 0.0, np.zeros((1, 2, k)), np.zeros((1, 3)))
    assert out["branch"][0] == 0 and out["n_accepted"][0] == 2
