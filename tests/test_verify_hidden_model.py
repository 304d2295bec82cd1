"""Model of the logits-free verify's flow, on the CPU.

The CUDA path decides every sequence from the target rows and the draft step's
q(x) (Sec. 3.1), then, per group of up to 80 sequences, gathers the kept state
of each decision row r < K, recomputes that row's draft logits through the
final RMSNorm and the LM head (Sec. 3.3-3.4), normalises them with the draft
step's (M, log S) and draws from the residual.  This model follows that order
in float64, with groups smaller than the batch, and must give the oracle's
outcome wherever the oracle flags no near-tie.
"""
import numpy as np
import pytest

from oracle import verify as ov
from oracle.drafter import inverse_cdf


def emulate(zp, hidden, W, gamma, eps, x, T, ua, us, qx, stats, group=80):
    """Decisions for all sequences, then the decision-row draw group by group."""
    B, K1, V = zp.shape
    K = K1 - 1
    out = np.full((B, K1), -1)
    nacc = np.zeros(B, int)
    dec = []
    for b in range(B):
        y = zp[b] / T
        Mp = y.max(-1)
        Sp = np.exp(y - Mp[:, None]).sum(-1)
        r = K
        for i in range(K):
            px = np.exp(y[i, x[b, i]] - Mp[i]) / Sp[i]
            if not (ua[b, i] < px / qx[b, i]):
                r = i
                break
            out[b, i] = x[b, i]
        nacc[b] = r
        # the draft row's normaliser is the draft step's (M, log S)
        dec.append((r, Mp[r], Sp[r], stats[b, r, 0] if r < K else 0, np.exp(stats[b, r, 1]) if r < K else 1))
    for b0 in range(0, B, group):
        n = min(group, B - b0)
        rows = np.zeros((n, hidden.shape[-1]))
        for j in range(n):
            r = dec[b0 + j][0]
            if r < K:
                rows[j] = hidden[b0 + j, r]
        nrm = rows / np.sqrt((rows * rows).mean(-1, keepdims=True) + eps) * gamma
        z = nrm @ W.T
        for j in range(n):
            b = b0 + j
            r, Mp, Sp, Mq, Sq = dec[b]
            p = np.exp(zp[b, r] / T - Mp) / Sp
            w = np.maximum(0, p - np.exp(z[j] / T - Mq) / Sq) if r < K else p
            if w.sum() <= 0:
                w = p
            out[b, r] = inverse_cdf(w, us[b, r])[0]
    return out, nacc


@pytest.mark.parametrize("B,group", [(170, 80), (9, 4), (1, 80)])
def test_grouped_flow_matches_oracle(B, group):
    rng = np.random.default_rng(B)
    V, d, K, T = 512, 64, 3, 0.8
    W = rng.standard_normal((V, d)) * 0.3
    gamma = 1 + 0.1 * rng.standard_normal(d)
    hidden = rng.standard_normal((B, K, d)).astype(np.float32)
    zq = ov.draft_logits_from_hidden(hidden, W, gamma, 1e-6)
    y = zq / T
    M = y.max(-1)
    e = np.exp(y - M[..., None])
    S = e.sum(-1)
    x = np.array([[inverse_cdf(e[b, i], rng.random())[0] for i in range(K)] for b in range(B)])
    qx = np.take_along_axis(e, x[..., None], -1)[..., 0] / S
    stats = np.stack([M, np.log(S)], -1)
    zp = np.concatenate([zq + 0.7 * rng.standard_normal(zq.shape), rng.standard_normal((B, 1, V))], 1)
    ua, us = rng.random((B, K)), rng.random((B, K + 1))
    o = ov.verify_hidden(zp, hidden, W, gamma, 1e-6, x, T, ua, us)
    out, nacc = emulate(zp, hidden, W, gamma, 1e-6, x, T, ua, us, qx, stats, group=group)
    ok = (o["flags"] == 0).all(1)
    assert ok.sum() >= B - 1
    np.testing.assert_array_equal(nacc[ok], o["n_accepted"][ok])
    np.testing.assert_array_equal(out[ok], o["out_tokens"][ok])
    if B > 100:
        assert 0 < (o["n_accepted"] < K).sum() < B   # residual draws and bonus draws both occur
