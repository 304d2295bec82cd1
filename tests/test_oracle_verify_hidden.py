"""Pins for the logits-free form of sampled verification: the draft rows q_i
come from the drafter's final RMSNorm and LM head applied to the last-layer
state g_i it kept (Sec. 3.3-3.4), not from stored draft logits.

The LM head here is a scaled permutation and every kept state has entries
+-a with a a power of two, so each logit has a closed form by index:
z_{i,j} = c_j * gamma_{pi(j)} * s_{i,pi(j)} (times a / sqrt(a^2 + eps) when
eps > 0).  A transposed head, a dropped gain or norm, eps in the wrong place,
a missing temperature or the wrong row's state all change these values."""
import numpy as np
import pytest

from oracle import verify as ov
from oracle.drafter import inverse_cdf

V = 16


def _case(seed, B=3, K=3):
    rng = np.random.default_rng(seed)
    pi = rng.permutation(V)
    while np.array_equal(pi[pi], np.arange(V)):      # not an involution: W and W^T differ
        pi = rng.permutation(V)
    c = rng.choice([0.5, 1.0, 2.0, 3.0], V)
    W = np.zeros((V, V))
    W[np.arange(V), pi] = c
    gamma = rng.choice([0.5, 1.0, 1.5, 2.0], V)
    s = rng.choice([-1.0, 1.0], (B, K, V))
    a = rng.choice([0.25, 1.0, 4.0], (B, K, 1))
    g = (a * s).astype(np.float32)                     # exact in float32
    return pi, c, W, gamma, s, a, g


def _closed_form(pi, c, gamma, s, a, eps):
    scale = a / np.sqrt(a * a + eps)
    return scale * (c * gamma[pi])[None, None, :] * s[:, :, pi]


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_logits_from_hidden_closed_form(seed):
    pi, c, W, gamma, s, a, g = _case(seed)
    z = ov.draft_logits_from_hidden(g, W, gamma, 0.0)
    np.testing.assert_array_equal(z, _closed_form(pi, c, gamma, s, a, 0.0))
    z = ov.draft_logits_from_hidden(g, W, gamma, 1e-2)
    np.testing.assert_allclose(z, _closed_form(pi, c, gamma, s, a, 1e-2), rtol=1e-14, atol=0)


def test_logits_from_hidden_take_bf16_bits():
    """bf16 bit patterns of the head and gain widen to the same values."""
    pi, c, W, gamma, s, a, g = _case(3)
    bits = lambda x: (np.asarray(x, np.float32).view(np.uint32) >> 16).astype(np.uint16)
    z = ov.draft_logits_from_hidden(g, bits(W), bits(gamma), 0.0)
    np.testing.assert_array_equal(z, _closed_form(pi, c, gamma, s, a, 0.0))


@pytest.mark.parametrize("T", [0.7, 1.0, 1.6])
def test_verify_hidden_matches_rule_on_closed_form_rows(T):
    """Same outcomes as the rule fed the closed-form draft logits, over a grid of
    uniforms; tokens drawn from the closed-form q."""
    pi, c, W, gamma, s, a, g = _case(4, B=64, K=3)
    B, K = g.shape[:2]
    rng = np.random.default_rng(9)
    zq = _closed_form(pi, c, gamma, s, a, 1e-6)
    zp = zq[:, :, :] + rng.standard_normal((B, K, V))
    zp = np.concatenate([zp, rng.standard_normal((B, 1, V)) * 2], axis=1)
    q = ov.softmax_t(zq, T)
    x = np.array([[inverse_cdf(q[b, i], rng.random())[0] for i in range(K)] for b in range(B)])
    ua = rng.random((B, K)).astype(np.float32)
    us = rng.random((B, K + 1)).astype(np.float32)
    got = ov.verify_hidden(zp, g, W, gamma, 1e-6, x, T, ua, us)
    ref = ov.verify(zp, zq, x, T, ua, us)
    for k in ("out_tokens", "n_accepted", "flags"):
        np.testing.assert_array_equal(got[k], ref[k])
    np.testing.assert_allclose(got["q_x"], q[np.arange(B)[:, None], np.arange(K)[None], x], rtol=1e-12)
    assert 0 < (got["n_accepted"] < K).sum() < B       # both residual draws and bonus draws happen


def test_state_scale_does_not_change_outcomes():
    """RMSNorm makes the rows invariant to a positive scale of each kept state
    (exactly, with eps = 0 and power-of-two scales)."""
    pi, c, W, gamma, s, a, g = _case(5, B=32, K=2)
    rng = np.random.default_rng(1)
    zp = rng.standard_normal((32, 3, V))
    x = rng.integers(0, V, (32, 2))
    ua = rng.random((32, 2)).astype(np.float32)
    us = rng.random((32, 3)).astype(np.float32)
    r0 = ov.verify_hidden(zp, g, W, gamma, 0.0, x, 1.0, ua, us)
    r1 = ov.verify_hidden(zp, g * np.float32(8.0), W, gamma, 0.0, x, 1.0, ua, us)
    for k in ("out_tokens", "n_accepted", "flags", "p_x", "q_x"):
        np.testing.assert_array_equal(r0[k], r1[k])


def test_target_equal_to_drafter_accepts_all():
    """Target rows i < K equal to the drafter's own rows: p_i = q_i, every draft
    is accepted and the bonus is the inverse CDF of p_K."""
    pi, c, W, gamma, s, a, g = _case(6, B=16, K=3)
    rng = np.random.default_rng(2)
    zq = _closed_form(pi, c, gamma, s, a, 0.0)
    zb = rng.standard_normal((16, 1, V))
    zp = np.concatenate([zq, zb], axis=1)
    q = ov.softmax_t(zq, 1.0)
    x = np.array([[inverse_cdf(q[b, i], rng.random())[0] for i in range(3)] for b in range(16)])
    ua = rng.random((16, 3)).astype(np.float32)
    us = rng.random((16, 4)).astype(np.float32)
    r = ov.verify_hidden(zp, g, W, gamma, 0.0, x, 1.0, ua, us)
    assert (r["n_accepted"] == 3).all()
    pK = ov.softmax_t(zb[:, 0], 1.0)
    np.testing.assert_array_equal(r["out_tokens"][:, :3], x)
    assert [int(t) for t in r["out_tokens"][:, 3]] == [inverse_cdf(pK[b], float(us[b, 3]))[0] for b in range(16)]
