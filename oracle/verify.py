"""Oracle speculative-sampling verification, float64.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

Sec. 3.1: the target verifies the K draft tokens in one forward pass with the
standard speculative-decoding rule (Leviathan et al.), which Osprey leaves
unmodified.  Written out, for one sequence with target rows p_0..p_K and draft
rows q_0..q_{K-1} (p_i = softmax(z^p_i / T), q_i = softmax(z^q_i / T)):

1. for i = 0, 1, ...: accept draft token x_i when u_i < p_i(x_i) / q_i(x_i);
2. r = the first rejected position, or K when all K are accepted;
3. emit x_0..x_{r-1}, then one more token: for r < K drawn from the residual
   norm(max(0, p_r - q_r)); for r = K (the bonus) drawn from p_K.

Greedy verification (T = 0) accepts while argmax p_i = x_i and emits argmax p_r.

Readings where the rule leaves a choice: accept iff u < p/q (so p >= q always
accepts); every draw is an inverse CDF over token ids in ascending order
(smallest j with u*S < C_j); the emission at r uses u_sample[r] whether it is a
residual or a bonus draw; argmax ties go to the lowest id; a residual whose
mass is zero (impossible after a real rejection) falls back to p_r with flag
bit 3.  Flags mark decisions whose outcome sits within a stated distance of a
boundary, where a run in another precision may legitimately decide otherwise:
bit 0 |u - p/q| < ratio_band at a tested position, bit 1 the inverse-CDF point
within cdf_band * S of an edge of the chosen bin, bit 3 residual fallback.
"""
from __future__ import annotations

import numpy as np

from .bf16 import widen

FLAG_RATIO = 1
FLAG_CDF = 2
FLAG_GREEDY_GAP = 4
FLAG_FALLBACK = 8


def softmax_t(z: np.ndarray, temperature: float) -> np.ndarray:
    """softmax(z / T) over the last axis, float64."""
    y = np.asarray(z, np.float64) / temperature
    e = np.exp(y - y.max(axis=-1, keepdims=True))
    return e / e.sum(axis=-1, keepdims=True)


def _inverse_cdf_rows(w: np.ndarray, u: np.ndarray):
    """Row-wise inverse CDF: smallest j with u*S < C_j.  Returns (j, margin/S)."""
    C = np.cumsum(w, axis=-1)
    S = C[:, -1]
    t = u * S
    j = (C <= t[:, None]).sum(axis=-1)
    j = np.minimum(j, w.shape[-1] - 1)
    rows = np.arange(w.shape[0])
    hi = C[rows, j]
    lo = np.where(j > 0, C[rows, np.maximum(j - 1, 0)], 0.0)
    with np.errstate(invalid="ignore", divide="ignore"):
        margin = np.minimum(t - lo, hi - t) / S
    return j, margin


def verify(target_logits: np.ndarray, draft_logits: np.ndarray | None, draft_tokens: np.ndarray,
           temperature: float, u_accept: np.ndarray, u_sample: np.ndarray,
           ratio_band: float = 1e-5, cdf_band: float = 1e-5) -> dict:
    """Verify a batch.  target [B, K+1, V], draft [B, K, V] (f32 or bf16 bits),
    draft_tokens [B, K], u_accept [B, K], u_sample [B, K+1].

    Returns out_tokens [B, K+1] (-1 after the emitted ones), n_accepted [B],
    flags [B, K+1] (uint8), p_x / q_x [B, K] = p_i(x_i), q_i(x_i).
    """
    zp = widen(target_logits)
    B, K1, V = zp.shape
    K = K1 - 1
    x = np.asarray(draft_tokens, np.int64)
    rows = np.arange(B)
    out = np.full((B, K + 1), -1, np.int64)
    flags = np.zeros((B, K + 1), np.uint8)
    n_acc = np.zeros(B, np.int64)
    p_x = np.zeros((B, K))
    q_x = np.zeros((B, K))

    if temperature == 0.0:
        # greedy: accept while the target's argmax equals the draft token
        alive = np.ones(B, bool)
        for i in range(K + 1):
            a = np.argmax(zp[:, i], axis=-1)
            if i < K:
                acc = alive & (a == x[:, i])
                emit_here = alive & ~acc
                out[emit_here, i] = a[emit_here]
                out[acc, i] = x[acc, i]
                n_acc[acc] += 1
                alive = acc
            else:
                out[alive, K] = a[alive]
        return {"out_tokens": out, "n_accepted": n_acc, "flags": flags, "p_x": p_x, "q_x": q_x}

    zq = widen(draft_logits)
    alive = np.ones(B, bool)
    for i in range(K + 1):
        p = softmax_t(zp[:, i], temperature)
        if i < K:
            q = softmax_t(zq[:, i], temperature)
            px, qx = p[rows, x[:, i]], q[rows, x[:, i]]
            p_x[:, i], q_x[:, i] = px, qx
            ratio = px / qx
            ua = u_accept[:, i].astype(np.float64)
            near = alive & (np.abs(ua - ratio) < ratio_band)
            flags[near, i] |= FLAG_RATIO
            acc = alive & (ua < ratio)
            rej = alive & ~acc
            out[acc, i] = x[acc, i]
            n_acc[acc] += 1
            w = np.maximum(0.0, p - q)
        else:
            rej = alive
            w = p
        if rej.any():
            wr = w[rej]
            fb = wr.sum(axis=-1) <= 0.0
            if fb.any():
                wr[fb] = p[rej][fb]
            j, margin = _inverse_cdf_rows(wr, u_sample[rej, i].astype(np.float64))
            out[rej, i] = j
            idx = np.nonzero(rej)[0]
            flags[idx[margin < cdf_band], i] |= FLAG_CDF
            flags[idx[fb], i] |= FLAG_FALLBACK
        if i < K:
            alive = acc
    return {"out_tokens": out, "n_accepted": n_acc, "flags": flags, "p_x": p_x, "q_x": q_x}


def draft_logits_from_hidden(hidden: np.ndarray, lm_head: np.ndarray, final_norm: np.ndarray,
                             eps: float) -> np.ndarray:
    """Draft logits of the rows a drafter chain produced, from the state it kept.

    Sec. 3.3-3.4: draft token i is sampled from q_i = softmax(z^q_i / T) with
    z^q_i = W_lm (RMSNorm(g_i) * gamma_f), g_i being the last layer's residual
    output (before the final norm) of the row that drafted it.  hidden [B, K, d]
    holds the g_i; lm_head [V, d] and final_norm [d] are bf16 bits or floats.
    Returns z^q [B, K, V] in float64.
    """
    g = np.asarray(hidden, np.float64)
    n = g / np.sqrt(np.mean(g * g, axis=-1, keepdims=True) + eps) * widen(final_norm)
    return n @ widen(lm_head).T


def verify_hidden(target_logits: np.ndarray, hidden: np.ndarray, lm_head: np.ndarray, final_norm: np.ndarray,
                  eps: float, draft_tokens: np.ndarray, temperature: float, u_accept: np.ndarray,
                  u_sample: np.ndarray, ratio_band: float = 1e-5, cdf_band: float = 1e-5) -> dict:
    """The sampled rule of ``verify`` with the draft rows q_i defined by the
    drafter's final norm and LM head applied to the kept states g_i instead of
    stored draft logits (same outputs as ``verify``).  temperature > 0."""
    assert temperature > 0.0, "the draft rows matter only for sampled verification"
    zq = draft_logits_from_hidden(hidden, lm_head, final_norm, eps)
    return verify(target_logits, zq, draft_tokens, temperature, u_accept, u_sample,
                  ratio_band=ratio_band, cdf_band=cdf_band)


def emission_distribution(p: np.ndarray, q: np.ndarray) -> dict:
    """The rule integrated over its uniforms, for one sequence.

    p [K+1, V], q [K, V] probability rows.  Draft token x_i is drawn from q_i.
    Position i is reached when every earlier draft was accepted.  Given that,
    the token emitted at i is x_i with probability min(1, p_i/q_i) (the measure
    of u < p/q), else a draw from the normalised residual.  Returns D [K+1, V]
    (distribution of the token emitted at i given i is reached), accept [K]
    (acceptance probability at i) and reach [K+1].
    """
    K = q.shape[0]
    V = p.shape[1]
    D = np.zeros((K + 1, V))
    accept = np.zeros(K)
    for i in range(K):
        for xi in range(V):
            if q[i, xi] == 0.0:
                continue
            a = min(1.0, p[i, xi] / q[i, xi])
            D[i, xi] += q[i, xi] * a
            accept[i] += q[i, xi] * a
            res = np.maximum(0.0, p[i] - q[i])
            if res.sum() > 0.0 and a < 1.0:
                D[i] += q[i, xi] * (1.0 - a) * res / res.sum()
    D[K] = p[K]
    reach = np.concatenate([[1.0], np.cumprod(accept)])
    return {"D": D, "accept": accept, "reach": reach}
