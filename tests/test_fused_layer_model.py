"""Model of the fused batch-1 layer kernel's partitioned data flow, on the CPU.

The kernel splits one layer of one chain row over a grid of blocks: pair units
(rows i and i + hd/2 of a head) of the expanded QKV projection with RoPE applied
inside the unit and the K/V rows written to their page slot, key ranges of
each KV head for attention merged across ranges, and row / unit ranges of the
O-proj, gate/up and down projections.  This model follows that partition in
float64 and must give the oracle's layer output (Sec. 3.3 Eq. 2-3 and the
transferred block); a wrong pair, slot, range or merge would not.
"""
from dataclasses import replace

import numpy as np
import pytest

from oracle import drafter as od
from oracle.bf16 import round_to_bf16, widen
from paper_2609_09338_gb300 import synthetic as syn
from paper_2609_09338_gb300.workloads import QWEN3_8B_DRAFTER, TINY


def attn_splits(R, Hkv, max_ctx, sms):
    """Key ranges per (row, KV head) the draft step allots (about four blocks
    per SM, 64 to 1024 keys a range); the fused layer takes at most sms / Hkv."""
    cdiv = lambda x, y: -(-x // y)
    s = max(cdiv(4 * sms, R * Hkv), cdiv(max_ctx, 1024))
    s = min(s, cdiv(max_ctx, 64), 128)
    return max(s, 1)


def emulate(sh, W, pages_k, pages_v, ptab, x, s, pos, grid=152):
    """One layer of one row, block by block; returns the new residual and q."""
    d, F, Hq, Hkv, hd = sh.d_model, sh.ffn_dim, sh.n_q_heads, sh.n_kv_heads, sh.head_dim
    half, G, P = hd // 2, Hq // Hkv, sh.page_size
    nu = (Hq + 2 * Hkv) * half
    inv_freq = sh.rope_theta ** (-2.0 * np.arange(half) / hd)
    q = np.zeros(Hq * hd)
    # A: pair units of W~_qkv [s; RMSNorm(x)], RoPE inside the unit, K/V rows to their page slot
    z = x / np.sqrt(np.mean(x * x) + sh.rms_eps) * W["attn_norm"][0]
    u = np.concatenate([s, z])
    Wq = W["W_qkv"][0]
    for c in range(grid):
        u0, u1 = nu * c // grid, nu * (c + 1) // grid
        for unit in range(u0, u1):
            h, i = divmod(unit, half)
            y1, y2 = Wq[h * hd + i] @ u, Wq[h * hd + half + i] @ u
            x1, x2 = y1, y2
            if h < Hq + Hkv:
                ang = pos * inv_freq[i]
                x1, x2 = y1 * np.cos(ang) - y2 * np.sin(ang), y2 * np.cos(ang) + y1 * np.sin(ang)
            if h < Hq:
                q[h * hd + i], q[h * hd + i + half] = x1, x2
            else:
                is_k = h < Hq + Hkv
                kvh = h - Hq if is_k else h - Hq - Hkv
                page = ptab[pos // P]
                dst = pages_k if is_k else pages_v
                dst[page, kvh, pos % P, i] = round_to_bf16(np.array(x1))
                dst[page, kvh, pos % P, i + half] = round_to_bf16(np.array(x2))
    # B: key ranges per KV head, then the merge across ranges
    max_ctx = len(ptab) * P
    ns = min(grid // Hkv, attn_splits(1, Hkv, max_ctx, grid))
    sl = -(-max_ctx // ns)
    sl = -(-sl // 16) * 16
    part = np.zeros((Hq, ns, hd + 2))
    attn = np.zeros(Hq * hd)
    for c in range(min(grid, Hkv * ns)):
        kvh, split = divmod(c, ns)
        kb, ke = split * sl, min(pos + 1, split * sl + sl)
        for g in range(G):
            hq = kvh * G + g
            if ke <= kb:
                part[hq, split, 0], part[hq, split, 1] = -np.inf, 0.0
                continue
            t = np.arange(kb, ke)
            keys = pages_k[ptab[t // P], kvh, t % P]
            vals = pages_v[ptab[t // P], kvh, t % P]
            sc = keys @ q[hq * hd:(hq + 1) * hd] / np.sqrt(hd)
            M = sc.max()
            e = np.exp(sc - M)
            part[hq, split] = np.concatenate([[M, e.sum()], e @ vals])
    for hq in range(Hq):
        M = part[hq, :, 0].max()
        f = np.where(part[hq, :, 0] == -np.inf, 0.0, np.exp(part[hq, :, 0] - M))
        attn[hq * hd:(hq + 1) * hd] = (f @ part[hq, :, 2:]) / (f @ part[hq, :, 1])
    # C: O-proj rows
    x = x.copy()
    for c in range(grid):
        o0, o1 = d * c // grid, d * (c + 1) // grid
        x[o0:o1] += W["W_o"][0][o0:o1] @ attn
    # D: RMSNorm, gate/up units and SwiGLU
    n = x / np.sqrt(np.mean(x * x) + sh.rms_eps) * W["ffn_norm"][0]
    h = np.zeros(F)
    for c in range(grid):
        f0, f1 = F * c // grid, F * (c + 1) // grid
        gg, uu = W["W_gate"][0][f0:f1] @ n, W["W_up"][0][f0:f1] @ n
        h[f0:f1] = gg / (1 + np.exp(-gg)) * uu
    # E: down rows
    for c in range(grid):
        o0, o1 = d * c // grid, d * (c + 1) // grid
        x[o0:o1] += W["W_down"][0][o0:o1] @ h
    return x, q


def run(sh, ctx_len, seed):
    """Token 3 at position ctx_len after a ctx_len-position paged prefix: the
    block-by-block model and the oracle's forward_row give the same residual."""
    sh = replace(sh, n_layers=1)
    wb = syn.make_weights(sh, seed)
    W = od.widen_weights(wb)
    kv = syn.make_kv_prefix(sh, np.array([ctx_len]), 8, seed + 1)
    ptab = kv["page_table"][0]
    P, Hkv, hd = sh.page_size, sh.n_kv_heads, sh.head_dim
    pages_k = np.zeros((kv["n_pages"], Hkv, P, hd))
    pages_v = np.zeros_like(pages_k)
    t = np.arange(ctx_len)
    pages_k[ptab[t // P], :, t % P] = widen(kv["k_rows"][0])
    pages_v[ptab[t // P], :, t % P] = widen(kv["v_rows"][0])
    rng = np.random.default_rng(seed + 5)
    x = widen(wb["embed"][3])
    s = rng.standard_normal(sh.d_model)
    pos = ctx_len
    xe, _ = emulate(sh, W, pages_k, pages_v, ptab, x, s, pos)
    cache = od._SeqCache([widen(kv["k_rows"][0])], [widen(kv["v_rows"][0])])
    nk, nv = [[]], [[]]
    xo = od.forward_row(W, sh, cache, 3, s, pos, nk, nv)
    err = np.abs(xe - xo).max()
    assert err < 1e-9


@pytest.mark.parametrize("which,ctx_len,seed", [("tiny", 77, 3), ("tiny", 130, 4), ("qwen3", 2048, 5)])
def test_partitioned_layer_matches_oracle(which, ctx_len, seed):
    # the vocabulary plays no part in a layer: the Qwen3-8B-shaped case keeps 4096 tokens
    run(TINY if which == "tiny" else replace(QWEN3_8B_DRAFTER, vocab=4096), ctx_len, seed)
