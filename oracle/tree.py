"""Oracle verification of a draft tree (topk > 1), float64.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

The paper serves its drafters with chain drafting, topk = 1 (Sec. 4,
inference settings), and verifies with the unmodified rule of Leviathan et al.
(Sec. 3.1).  For topk = k > 1 the paper is silent; this oracle follows the
reading stated in the design notes, the multi-candidate form of the same rule:

* The tree is a branching chain.  At depth i = 0..K-1 the drafter's
  distribution q_i (after the verified prefix and the chain tokens of the
  depths before i) yields k candidates x_{i,0..k-1}, independent draws from
  q_i (the inverse CDF at each candidate's own uniform; at T = 0 the k highest
  logits, ties to the lowest id).  Candidate 0 continues the chain; the
  others are leaves.
* The target scores every node in one pass: row 0 is the distribution after
  the prefix (the root, for depth 0) and row 1 + i*k + j the distribution after
  the path ending in x_{i,j}.
* The walk starts at the root.  At depth i, with p the current node's target
  distribution and q = q_i, the residual starts at r = p and the candidates
  are tried in order: x_{i,j} is accepted iff u_accept[i, j] < r(x)/q(x); after a
  rejection r becomes norm(max(0, r - q)).  The first accepted candidate is
  emitted.  If it is candidate 0 and i < K - 1 the walk moves to depth i + 1
  with p = the row of x_{i,0}; otherwise one more token is drawn from the row of
  the accepted node at u_sample[i + 1] and the walk ends.  If all k candidates
  are rejected, a token is drawn from the last residual at u_sample[i] and the
  walk ends.  Every draw is the inverse CDF over ids in ascending order.
* Greedy (T = 0): at depth i the target's argmax y of the current node is
  accepted if it equals a candidate (the first such j); the walk continues
  from candidate 0 as above, a leaf or the last depth emits the argmax of its
  node's row, and no match emits y.
* With k = 1 this is exactly ``oracle.verify.verify``.

Outputs per sequence: the emitted tokens (accepted candidates, then the
drawn one), n_accepted, and the branch j of the candidate accepted at the last
accepted depth (-1 when none).  Flags as ``oracle.verify``: bit 0 a tested
ratio within ratio_band of its uniform, bit 1 the draw within cdf_band * S of a
bin edge, bit 3 a draw from p after a residual without mass.
"""
from __future__ import annotations

import numpy as np

from .bf16 import widen
from .verify import FLAG_CDF, FLAG_FALLBACK, FLAG_RATIO, softmax_t


def _draw(w: np.ndarray, u: float):
    """Inverse CDF over ascending ids: smallest j with u*S < C_j.  Returns (j, margin / S)."""
    C = np.cumsum(w)
    S = C[-1]
    t = float(u) * S
    j = min(int(np.searchsorted(C, t, side="right")), len(w) - 1)
    lo = C[j - 1] if j > 0 else 0.0
    return j, min(t - lo, C[j] - t) / S


def tree_rows(i: int, j: int, k: int) -> int:
    """Target row of node (depth i, candidate j): 1 + i*k + j (row 0 is the root)."""
    return 1 + i * k + j


def verify_tree(target_logits: np.ndarray, draft_logits: np.ndarray | None, cand: np.ndarray, temperature: float,
                u_accept: np.ndarray, u_sample: np.ndarray, ratio_band: float = 1e-5,
                cdf_band: float = 1e-5) -> dict:
    """target [B, 1 + K*k, V], draft [B, K, V] (f32 or bf16 bits; None at T = 0),
    cand [B, K, k] int, u_accept [B, K, k], u_sample [B, K + 1].

    Returns out_tokens [B, K + 1] (-1 after the emitted ones), n_accepted [B],
    branch [B], flags [B, K + 1] (uint8)."""
    zp = widen(target_logits)
    B, _, V = zp.shape
    K, k = cand.shape[1], cand.shape[2]
    out = np.full((B, K + 1), -1, np.int64)
    n_acc = np.zeros(B, np.int64)
    branch = np.full(B, -1, np.int64)
    flags = np.zeros((B, K + 1), np.uint8)
    zq = widen(draft_logits) if temperature > 0.0 else None
    for b in range(B):
        row = 0                                    # the current node's target row
        for i in range(K):
            c = [int(x) for x in cand[b, i]]
            if temperature == 0.0:
                y = int(np.argmax(zp[b, row]))
                j = next((jj for jj in range(k) if c[jj] == y), -1)
                if j < 0:
                    out[b, i] = y
                    break
                out[b, i] = y
                n_acc[b] += 1
                branch[b] = j
                row = tree_rows(i, j, k)
                if j > 0 or i == K - 1:
                    out[b, i + 1] = int(np.argmax(zp[b, row]))
                    break
                continue
            p = softmax_t(zp[b, row], temperature)
            q = softmax_t(zq[b, i], temperature)
            r = p.copy()
            acc = -1
            for jj in range(k):
                ratio = r[c[jj]] / q[c[jj]]
                if abs(float(u_accept[b, i, jj]) - ratio) < ratio_band:
                    flags[b, i] |= FLAG_RATIO
                if float(u_accept[b, i, jj]) < ratio:
                    acc = jj
                    break
                res = np.maximum(0.0, r - q)
                if res.sum() > 0.0:
                    r = res / res.sum()
                else:                              # no residual mass: sample p instead
                    flags[b, i] |= FLAG_FALLBACK
                    r = p.copy()
            if acc < 0:                            # every candidate rejected: draw from the residual
                t, margin = _draw(r, u_sample[b, i])
                out[b, i] = t
                if margin < cdf_band:
                    flags[b, i] |= FLAG_CDF
                break
            out[b, i] = c[acc]
            n_acc[b] += 1
            branch[b] = acc
            row = tree_rows(i, acc, k)
            if acc > 0 or i == K - 1:              # a leaf or the last depth: the next token from its row
                t, margin = _draw(softmax_t(zp[b, row], temperature), u_sample[b, i + 1])
                out[b, i + 1] = t
                if margin < cdf_band:
                    flags[b, i + 1] |= FLAG_CDF
                break
    return {"out_tokens": out, "n_accepted": n_acc, "branch": branch, "flags": flags}


def depth_emission(p: np.ndarray, q: np.ndarray, cands) -> dict:
    """One depth of the walk integrated over its uniforms, for given candidates.

    p, q [V] probability rows; cands: the k candidate ids.  Returns D [V] (the
    distribution of the token emitted at this depth) and acc [k] (the
    probability that candidate j is the accepted one)."""
    V = p.shape[0]
    D = np.zeros(V)
    acc = np.zeros(len(cands))
    r = p.copy()
    reach = 1.0                                    # probability that candidate j is tried
    for j, x in enumerate(cands):
        a = min(1.0, r[x] / q[x]) if q[x] > 0.0 else 0.0
        acc[j] = reach * a
        D[x] += reach * a
        reach *= 1.0 - a
        res = np.maximum(0.0, r - q)
        r = res / res.sum() if res.sum() > 0.0 else p.copy()
    D += reach * r
    return {"D": D, "acc": acc}
