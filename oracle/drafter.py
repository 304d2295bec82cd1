"""Oracle drafter forward and K-token chain, float64.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

What it computes, in the paper's order and notation:

* Eq. 1 (Sec. 3.3): c_t = W_c [h_low; h_mid; h_high], one linear map with no
  bias, and the same c feeds every drafter layer.
* Eq. 2-3 (Sec. 3.3): every layer's QKV projection reads [c_{t-1}; z_t] through
  W~_qkv = [W_ctx  W_qkv] (the context columns first, zero at conversion), so
  with zero context columns the layer computes W_qkv z_t exactly.
* Sec. 3.4: inside a chain the drafter's own hidden state takes the place of
  the target feature at the next step; the state used is the last layer's
  residual output before the final norm.
* The rest is the pruned backbone the paper transfers unchanged (Sec. 3.2-3.3):
  pre-norm blocks with RMSNorm, rotary position embedding (rotate-half
  convention), grouped-query attention, SwiGLU MLP, a final RMSNorm and the LM
  head; layer 0's residual stream starts from the token embedding E[x_t].
* The drafter's KV cache holds bf16 values (paged serving cache, Sec. 4
  inference settings): each new K/V row is rounded to bf16 when it is cached,
  and attention reads the cached values.
* Sampling of each draft token from q = softmax(logits / T) by inverse CDF
  over token ids in ascending order, or argmax (lowest id on ties) when T = 0;
  the chain is drafted with topk = 1 (Sec. 4, inference settings).

Readings where the paper is silent are listed in the design notes: no norm on
c, RMSNorm eps 1e-6, rotate-half RoPE, 1/sqrt(hd) attention scale, no QK-norm.
"""
from __future__ import annotations

import numpy as np

from .bf16 import round_to_bf16, widen


# --------------------------------------------------------------------------
# building blocks

def rmsnorm(x: np.ndarray, gain: np.ndarray, eps: float) -> np.ndarray:
    """x / sqrt(mean(x^2) + eps) * gain over the last axis."""
    x = np.asarray(x, np.float64)
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * gain


def rope_angles(pos: int, head_dim: int, theta: float) -> np.ndarray:
    """Angle pos * theta^(-2i/hd) for each rotated pair i = 0..hd/2-1."""
    i = np.arange(head_dim // 2, dtype=np.float64)
    return float(pos) * theta ** (-2.0 * i / head_dim)


def rope(x: np.ndarray, pos: int, theta: float) -> np.ndarray:
    """Rotate-half RoPE on [..., hd]: pair (i, i + hd/2) turned by angle_i."""
    hd = x.shape[-1]
    a = rope_angles(pos, hd, theta)
    c, s = np.cos(a), np.sin(a)
    x1, x2 = x[..., : hd // 2], x[..., hd // 2:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


def silu(x: np.ndarray) -> np.ndarray:
    return x / (1.0 + np.exp(-x))


def gqa_attention(q: np.ndarray, keys: np.ndarray, values: np.ndarray) -> np.ndarray:
    """Decode attention for one query row.

    q [Hq, hd]; keys, values [n, Hkv, hd] (every cached position the row may
    see).  Query head h reads KV head h // (Hq/Hkv).  Returns [Hq, hd].
    """
    Hq, hd = q.shape
    Hkv = keys.shape[1]
    g = Hq // Hkv
    out = np.empty_like(q)
    for h in range(Hq):
        kh = keys[:, h // g, :]
        vh = values[:, h // g, :]
        scores = kh @ q[h] / np.sqrt(hd)
        w = np.exp(scores - scores.max())
        out[h] = (w / w.sum()) @ vh
    return out


def gather_pages(pages: np.ndarray, page_table_row: np.ndarray, n: int) -> np.ndarray:
    """Read positions 0..n-1 of one sequence out of a paged cache.

    pages [n_pages, Hkv, P, hd]; position t lives in page page_table_row[t // P]
    at slot t % P.  Returns [n, Hkv, hd].
    """
    P = pages.shape[2]
    t = np.arange(n)
    return pages[page_table_row[t // P], :, t % P, :]


# --------------------------------------------------------------------------
# weights

def widen_weights(w: dict) -> dict:
    """bf16 bit patterns -> float64 arrays (exact)."""
    out = {}
    for k, v in w.items():
        out[k] = [widen(a) for a in v] if isinstance(v, list) else widen(v)
    return out


def feature_projection(W_c: np.ndarray, feat: np.ndarray) -> np.ndarray:
    """Eq. 1: c = W_c [h_low; h_mid; h_high] (feat is the 3H concatenation)."""
    return W_c @ feat


def expanded_qkv(W_qkv_tilde: np.ndarray, s: np.ndarray, z: np.ndarray) -> np.ndarray:
    """Eq. 2-3: W~_qkv [s; z] with the context slot s read by the first columns."""
    return W_qkv_tilde @ np.concatenate([s, z])


# --------------------------------------------------------------------------
# one drafter row and the chain

class _SeqCache:
    """Keys/values of one sequence, in position order, per layer (float64)."""

    def __init__(self, k_prefix: list, v_prefix: list):
        self.k = [list(k) for k in k_prefix]
        self.v = [list(v) for v in v_prefix]

    def length(self, layer: int) -> int:
        return len(self.k[layer])


def forward_row(W: dict, shape, cache: _SeqCache, token: int, s: np.ndarray, pos: int,
                new_k: list, new_v: list, forced=None, new_mag: list | None = None) -> np.ndarray:
    """One drafter position through every layer; returns x_L (pre final norm).

    new_k/new_v receive the rows this computation produces.  With ``forced`` =
    (k [L, Hkv, hd], v [L, Hkv, hd]) the cache holds those rows instead (another
    run's cached values at this position), so attention reads the same cache
    state as that run.  ``new_mag`` (optional, per layer a list) receives for
    each new row the pair (k_mag, v_mag): sum_j |W~_ij| |u_j| of the projection
    that made each element (for a rotated key, summed over the two elements
    of its rotation pair), the scale of a rounding error in that element."""
    Hq, Hkv, hd = shape.n_q_heads, shape.n_kv_heads, shape.head_dim
    eps, theta = shape.rms_eps, shape.rope_theta
    x = W["embed"][token].copy()
    for l in range(shape.n_layers):
        z = rmsnorm(x, W["attn_norm"][l], eps)
        qkv = expanded_qkv(W["W_qkv"][l], s, z)
        q = qkv[: Hq * hd].reshape(Hq, hd)
        k = qkv[Hq * hd: (Hq + Hkv) * hd].reshape(Hkv, hd)
        v = qkv[(Hq + Hkv) * hd:].reshape(Hkv, hd)
        if new_mag is not None:
            mag = np.abs(W["W_qkv"][l]) @ np.abs(np.concatenate([s, z]))
            km = mag[Hq * hd: (Hq + Hkv) * hd].reshape(Hkv, hd)
            pair = km[:, : hd // 2] + km[:, hd // 2:]
            new_mag[l].append((np.concatenate([pair, pair], axis=-1), mag[(Hq + Hkv) * hd:].reshape(Hkv, hd)))
        q, k = rope(q, pos, theta), round_to_bf16(rope(k, pos, theta))
        v = round_to_bf16(v)
        assert cache.length(l) == pos, "positions must be contiguous"
        cache.k[l].append(k if forced is None else np.asarray(forced[0][l], dtype=np.float64))
        cache.v[l].append(v if forced is None else np.asarray(forced[1][l], dtype=np.float64))
        new_k[l].append(k)
        new_v[l].append(v)
        attn = gqa_attention(q, np.asarray(cache.k[l]), np.asarray(cache.v[l]))
        x = x + W["W_o"][l] @ attn.reshape(-1)
        n = rmsnorm(x, W["ffn_norm"][l], eps)
        x = x + W["W_down"][l] @ (silu(W["W_gate"][l] @ n) * (W["W_up"][l] @ n))
    return x


def inverse_cdf(w: np.ndarray, u: float):
    """Smallest id j with u*S < C_j, C the inclusive cumulative sum of w over ids
    in ascending order and S = C_{V-1}.  Returns (j, margin) where margin is the
    distance of u*S to the nearer edge of j's bin, divided by S."""
    C = np.cumsum(w)
    S = C[-1]
    t = float(u) * S
    j = int(np.searchsorted(C, t, side="right"))
    j = min(j, len(w) - 1)
    lo = C[j - 1] if j > 0 else 0.0
    return j, min(t - lo, C[j] - t) / S


def sample(z: np.ndarray, temperature: float, u: float) -> dict:
    """Draft token from logits z: q = softmax(z / T), inverse CDF at u; argmax at T = 0.

    Returns token, q(token), stats (M, log S) of z/T (of z when T = 0) and the
    margin used to flag near-ties (bin-edge distance / S, or top-2 logit gap).
    """
    if temperature == 0.0:
        tok = int(np.argmax(z))
        m = float(z[tok])
        top2 = np.partition(z, -2)[-2] if z.size > 1 else -np.inf
        return {"token": tok, "qx": 1.0, "M": m, "logS": float(np.log(np.exp(z - m).sum())),
                "margin": float(m - top2)}
    y = z / temperature
    M = float(y.max())
    e = np.exp(y - M)
    tok, margin = inverse_cdf(e, u)
    S = float(e.sum())
    return {"token": tok, "qx": float(e[tok] / S), "M": M, "logS": float(np.log(S)),
            "margin": float(margin)}


def draft_step(weights: dict, shape, prefix_k: np.ndarray, prefix_v: np.ndarray,
               ctx_lens: np.ndarray, tokens: np.ndarray, feats: np.ndarray,
               n_new: np.ndarray, K: int, temperature: float, u_draft: np.ndarray,
               forced_tokens: np.ndarray | None = None, widened: dict | None = None,
               forced_kv: list | None = None) -> dict:
    """One draft call for a batch of sequences.

    prefix_k/prefix_v: [L, sum(ctx), Hkv, hd] bf16 bits, sequence b owning rows
    [sum(ctx[:b]), sum(ctx[:b+1])).  tokens [B, max_new], feats [B, max_new, 3H]:
    extend row j of sequence b is token tokens[b, j] at position ctx[b] + j paired
    with the projected feature of the previous position (Eq. 2).  The last extend
    row's output gives draft token 1; chain steps 2..K feed the sampled token
    (or ``forced_tokens[b, k-1]`` when given, to follow another run's chain) and
    the previous row's x_L in the context slot (Sec. 3.4).

    forced_kv (optional): per sequence b a pair (k, v) of [L, n_new + K - 1, Hkv,
    hd] arrays, another run's cached rows at the positions this call writes.  The
    cache then holds those rows, as the chain follows forced_tokens: each step
    is computed from the same cache state as that run, while new_k/new_v still
    report the rows this computation produces.  (Cached rows are bf16, so a
    difference of one rounding step in a row would otherwise propagate along the
    chain.)

    Returns logits [B, K, V], tokens/qx [B, K], stats [B, K, 2], margins [B, K],
    new_k/new_v: per sequence [L, n_new + K - 1, Hkv, hd] (with new_k_mag /
    new_v_mag of the same shape: the error scale of each element, see
    forward_row), and g [B, d] (the last row's x_L).
    """
    W = widened if widened is not None else widen_weights(weights)
    B, V, L = len(ctx_lens), shape.vocab, shape.n_layers
    offs = np.concatenate([[0], np.cumsum(ctx_lens)]).astype(np.int64)
    out = {
        "logits": np.zeros((B, K, V)), "tokens": np.zeros((B, K), np.int64),
        "qx": np.zeros((B, K)), "stats": np.zeros((B, K, 2)), "margins": np.zeros((B, K)),
        "new_k": [], "new_v": [], "new_k_mag": [], "new_v_mag": [], "g": np.zeros((B, shape.d_model)),
    }
    for b in range(B):
        L0 = int(ctx_lens[b])
        cache = _SeqCache([widen(prefix_k[l, offs[b]:offs[b + 1]]) for l in range(L)],
                          [widen(prefix_v[l, offs[b]:offs[b + 1]]) for l in range(L)])
        new_k = [[] for _ in range(L)]
        new_v = [[] for _ in range(L)]
        new_mag = [[] for _ in range(L)]
        nb = int(n_new[b])
        fk = None if forced_kv is None else forced_kv[b]

        def fr(i):
            return None if fk is None else (fk[0][:, i], fk[1][:, i])

        for j in range(nb):
            c = feature_projection(W["W_c"], widen(feats[b, j]))
            g = forward_row(W, shape, cache, int(tokens[b, j]), c, L0 + j, new_k, new_v, fr(j), new_mag)
        for k in range(K):
            h = rmsnorm(g, W["final_norm"], shape.rms_eps)
            z = W["lm_head"] @ h
            smp = sample(z, temperature, float(u_draft[b, k]))
            out["logits"][b, k] = z
            out["tokens"][b, k] = smp["token"]
            out["qx"][b, k] = smp["qx"]
            out["stats"][b, k] = (smp["M"], smp["logS"])
            out["margins"][b, k] = smp["margin"]
            if k == K - 1:
                break
            nxt = int(forced_tokens[b, k]) if forced_tokens is not None else smp["token"]
            g = forward_row(W, shape, cache, nxt, g, L0 + nb + k, new_k, new_v, fr(nb + k), new_mag)
        out["g"][b] = g
        out["new_k"].append(np.asarray(new_k))
        out["new_v"].append(np.asarray(new_v))
        out["new_k_mag"].append(np.asarray([[m[0] for m in ml] for ml in new_mag]))
        out["new_v_mag"].append(np.asarray([[m[1] for m in ml] for ml in new_mag]))
    return out
