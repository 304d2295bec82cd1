"""Seeded synthetic inputs for the draft step and for verification.

This module only draws random numbers and lays them out; it holds none of the
method's arithmetic.  Both the CUDA path and the CPU oracle consume the arrays
it returns, byte for byte:

* bf16 tensors are returned as ``uint16`` bit patterns (rounded to nearest
  even from float32 draws);
* uniforms are float32 in [0, 1) from ``numpy.random.default_rng``;
* logits are float32 (a bf16 variant is the same values rounded).

Recipe (stand-in for the paper's chat/code/math prompts and trained drafters,
which are not available): drafter matrices and the embedding ~ N(0, 0.02^2);
RMSNorm gains 1 + N(0, 0.02^2); target features ~ N(0, 1); prefix K/V ~ N(0, 1)
(post-RoPE keys); draft logits = -3.3 ln(rank) over a seeded permutation of
the vocabulary plus N(0, 1) per row (a Zipf s=1.1 shape scaled by 3); target
logits = draft logits + N(0, sigma_p^2); the bonus target row draws its own
draft-shaped base.  Draft tokens for the verify-only inputs are drawn from the
draft distribution with the Gumbel-max trick (argmax for greedy).
"""
from __future__ import annotations

import numpy as np

from .workloads import DrafterShape, Workload

_CHUNK = 1 << 20   # elements per pass; buffers of a few MB are reused, not re-faulted


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """float32 -> bf16 bit pattern (uint16), round to nearest even."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    out = np.empty(x.shape, dtype=np.uint16)
    xf, of = x.reshape(-1), out.reshape(-1)
    t = np.empty(min(_CHUNK, xf.size), dtype=np.uint32)
    r = np.empty_like(t)
    for s in range(0, xf.size, _CHUNK):
        n = min(_CHUNK, xf.size - s)
        u, tn, rn = xf[s:s + n].view(np.uint32), t[:n], r[:n]
        np.right_shift(u, 16, out=rn)
        np.bitwise_and(rn, 1, out=rn)
        np.add(rn, np.uint32(0x7FFF), out=rn)
        np.add(u, rn, out=tn)            # wraps like uint32 arithmetic
        np.right_shift(tn, 16, out=tn)
        of[s:s + n] = tn
    return out


def _normal_bf16(rng: np.random.Generator, shape, std: float = 1.0, mean: float = 0.0) -> np.ndarray:
    out = np.empty(shape, dtype=np.uint16)
    of = out.reshape(-1)
    v = np.empty(min(_CHUNK, of.size), dtype=np.float32)
    for s in range(0, of.size, _CHUNK):
        n = min(_CHUNK, of.size - s)
        vn = v[:n]
        rng.standard_normal(n, dtype=np.float32, out=vn)
        if std != 1.0:
            vn *= np.float32(std)
        if mean != 0.0:
            vn += np.float32(mean)
        of[s:s + n] = bf16_bits(vn)
    return out


def make_weights(shape: DrafterShape, seed: int, zero_expansion: bool = False,
                 peaked_vocab: bool = False) -> dict:
    """Drafter weights as bf16 bit patterns.

    ``W_qkv[l]`` is the expanded projection [(Hq+2Hkv)*hd, 2d] with the columns
    that read the target-feature slot first (Eq. 2); ``zero_expansion`` sets
    that half to zero, as at conversion time.  ``peaked_vocab`` makes one hidden
    coordinate dominate the residual stream and stores a Zipf-shaped column in
    the LM head, so the draft distribution is peaked (used to check sampled
    draft tokens, which a random LM head spreads almost uniformly).
    """
    rng = np.random.default_rng(seed)
    d, L = shape.d_model, shape.n_layers
    a = shape.n_q_heads * shape.head_dim
    w = {
        "W_c": _normal_bf16(rng, (d, shape.feat_dim), 0.02),
        "embed": _normal_bf16(rng, (shape.vocab, d), 0.02),
        "final_norm": _normal_bf16(rng, (d,), 0.02, 1.0),
        "lm_head": _normal_bf16(rng, (shape.vocab, d), 0.02),
        "attn_norm": [], "W_qkv": [], "W_o": [], "ffn_norm": [],
        "W_gate": [], "W_up": [], "W_down": [],
    }
    for _ in range(L):
        w["attn_norm"].append(_normal_bf16(rng, (d,), 0.02, 1.0))
        qkv = _normal_bf16(rng, (shape.qkv_rows, 2 * d), 0.02)
        if zero_expansion:
            qkv[:, :d] = 0
        w["W_qkv"].append(qkv)
        w["W_o"].append(_normal_bf16(rng, (d, a), 0.02))
        w["ffn_norm"].append(_normal_bf16(rng, (d,), 0.02, 1.0))
        w["W_gate"].append(_normal_bf16(rng, (shape.ffn_dim, d), 0.02))
        w["W_up"].append(_normal_bf16(rng, (shape.ffn_dim, d), 0.02))
        w["W_down"].append(_normal_bf16(rng, (d, shape.ffn_dim), 0.02))
    if peaked_vocab:
        j0 = d // 3
        w["embed"][:, j0] = bf16_bits(np.full(shape.vocab, 64.0, np.float32))
        base = _zipf_base(rng, shape.vocab) / np.float32(np.sqrt(d))
        w["lm_head"][:, j0] = bf16_bits(base)
    return w


def _zipf_base(rng: np.random.Generator, V: int) -> np.ndarray:
    ranks = np.arange(1, V + 1, dtype=np.float64)
    base = (-3.3 * np.log(ranks)).astype(np.float32)
    out = np.empty(V, np.float32)
    out[rng.permutation(V)] = base
    return out


def make_contexts(w: Workload, seed: int | None = None) -> np.ndarray:
    rng = np.random.default_rng(w.seed + 17 if seed is None else seed)
    return rng.integers(w.ctx_lo, w.ctx_hi + 1, size=w.batch).astype(np.int32)


def make_kv_prefix(shape: DrafterShape, ctx_lens: np.ndarray, reserve: int, seed: int,
                   spare_pages: int = 0) -> dict:
    """Paged prefix cache contents and a randomly permuted page table.

    ``reserve`` extra positions per sequence are given pages (room for the
    extend rows and the chain).  Returns ``k_rows``/``v_rows`` [L, sum(ctx), Hkv,
    hd] bf16 bits (to be scattered by the append call), ``page_table`` [B,
    max_pages] int32 and ``n_pages``.
    """
    rng = np.random.default_rng(seed)
    P = shape.page_size
    B = len(ctx_lens)
    max_pages = int(-(-(int(ctx_lens.max(initial=0)) + reserve) // P))
    n_pages = B * max_pages + spare_pages
    page_table = rng.permutation(n_pages)[: B * max_pages].reshape(B, max_pages).astype(np.int32)
    total = int(ctx_lens.sum())
    L, H, hd = shape.n_layers, shape.n_kv_heads, shape.head_dim
    return {
        "k_rows": _normal_bf16(rng, (L, total, H, hd)),
        "v_rows": _normal_bf16(rng, (L, total, H, hd)),
        "page_table": page_table,
        "n_pages": n_pages,
        "max_pages": max_pages,
    }


def make_draft_inputs(shape: DrafterShape, batch: int, n_new: int, K: int, seed: int) -> dict:
    """Extend-row tokens, their (previous-position) target features and u_draft."""
    rng = np.random.default_rng(seed)
    return {
        "tokens": rng.integers(0, shape.vocab, size=(batch, n_new)).astype(np.int32),
        "feats": _normal_bf16(rng, (batch, n_new, shape.feat_dim)),
        "u_draft": rng.random((batch, K), dtype=np.float32),
        "n_new": np.full(batch, n_new, np.int32),
    }


def make_verify_inputs(V: int, batch: int, K: int, temperature: float, sigma_p: float,
                       seed: int, base_seed: int | None = None) -> dict:
    """Draft/target logits, draft tokens and the two uniform arrays for verify."""
    rng = np.random.default_rng(seed)
    base = _zipf_base(np.random.default_rng(seed + 7 if base_seed is None else base_seed), V)
    zq = np.empty((batch, K, V), np.float32)
    zp = np.empty((batch, K + 1, V), np.float32)
    tokens = np.empty((batch, K), np.int32)
    for b in range(batch):
        for i in range(K + 1):
            q = base + rng.standard_normal(V, dtype=np.float32)
            zp[b, i] = q + np.float32(sigma_p) * rng.standard_normal(V, dtype=np.float32)
            if i < K:
                zq[b, i] = q
                if temperature > 0:
                    g = -np.log(-np.log(rng.random(V) + 1e-300))
                    tokens[b, i] = int(np.argmax(q.astype(np.float64) / temperature + g))
                else:
                    tokens[b, i] = int(np.argmax(q))
    return {
        "draft_logits": zq,
        "target_logits": zp,
        "draft_tokens": tokens,
        "u_accept": rng.random((batch, K), dtype=np.float32),
        "u_sample": rng.random((batch, K + 1), dtype=np.float32),
    }


def make_tree_inputs(V: int, batch: int, K: int, k: int, temperature: float, sigma_p: float, seed: int) -> dict:
    """Draft and target logits of a branching-chain draft tree, its candidates
    and the uniforms.

    Draft row i of a sequence: the Zipf-shaped base + N(0, 1).  Candidates:
    k independent draws from softmax(row / T) by the Gumbel-max trick (the k
    highest logits when greedy).  Target rows (row 0 the root, row 1 + i*k + j
    the node (i, j)): the root is draft row 0 + N(0, sigma^2); a chain node
    (i, 0) with i < K - 1 is draft row i + 1 + N(0, sigma^2) (the target after
    the chain token the drafter continued from); the other nodes draw their
    own base-shaped rows."""
    rng = np.random.default_rng(seed)
    base = _zipf_base(np.random.default_rng(seed + 7), V)
    zq = np.empty((batch, K, V), np.float32)
    zp = np.empty((batch, 1 + K * k, V), np.float32)
    cand = np.empty((batch, K, k), np.int32)
    for b in range(batch):
        for i in range(K):
            zq[b, i] = base + rng.standard_normal(V, dtype=np.float32)
            if temperature > 0:
                for j in range(k):
                    g = -np.log(-np.log(rng.random(V) + 1e-300))
                    cand[b, i, j] = int(np.argmax(zq[b, i].astype(np.float64) / temperature + g))
            else:
                order = np.lexsort((np.arange(V), -zq[b, i]))
                cand[b, i] = order[:k]
        zp[b, 0] = zq[b, 0] + np.float32(sigma_p) * rng.standard_normal(V, dtype=np.float32)
        for i in range(K):
            for j in range(k):
                r = 1 + i * k + j
                if j == 0 and i < K - 1:
                    zp[b, r] = zq[b, i + 1] + np.float32(sigma_p) * rng.standard_normal(V, dtype=np.float32)
                else:
                    zp[b, r] = base + rng.standard_normal(V, dtype=np.float32)
    return {"draft_logits": zq, "target_logits": zp, "cand": cand,
            "u_accept": rng.random((batch, K, k), dtype=np.float32),
            "u_sample": rng.random((batch, K + 1), dtype=np.float32)}
