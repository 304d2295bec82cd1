"""Pins for the drafter oracle (Sec. 3.3 Eq. 1-3, Sec. 3.4).

Each building block is checked against a hand-derived value and a library
routine (torch CPU, float64); the assembled forward is checked against the
invariants the paper states (Eq. 3: zero context columns leave the drafter
independent of the target features) and against closed forms of special
cases (zeroed residual branches, a single cached position, causal extend)."""
import json
import os
from dataclasses import replace

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import drafter as od
from oracle.bf16 import widen
from paper_2609_09338_gb300 import synthetic as syn
from paper_2609_09338_gb300.workloads import TINY

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "hand_cases.json")))


def test_rmsnorm_hand_and_library():
    g = GOLD["rmsnorm"]
    np.testing.assert_allclose(od.rmsnorm(np.array(g["x"], float), 1.0, g["eps"]), g["y"], rtol=1e-15)
    rng = np.random.default_rng(0)
    x, w = rng.standard_normal((5, 64)), rng.standard_normal(64)
    ref = F.rms_norm(torch.from_numpy(x), (64,), torch.from_numpy(w), eps=1e-6).numpy()
    np.testing.assert_allclose(od.rmsnorm(x, w, 1e-6), ref, rtol=1e-13)


def test_rope_hand_and_properties():
    g = GOLD["rope"]
    np.testing.assert_allclose(od.rope(np.array(g["x"], float), g["pos"], g["theta"]), g["y"],
                               atol=1e-15)
    rng = np.random.default_rng(1)
    hd, theta = 128, 1e6
    q, k = rng.standard_normal(hd), rng.standard_normal(hd)
    np.testing.assert_array_equal(od.rope(q, 0, theta), q)           # position 0 is identity
    assert abs(np.linalg.norm(od.rope(q, 777, theta)) - np.linalg.norm(q)) < 1e-12
    # scores depend on the offset only: <R(m)q, R(n)k> = <R(m-n)q, k>
    for m, n in [(5, 3), (4000, 17), (16383, 16000)]:
        a = od.rope(q, m, theta) @ od.rope(k, n, theta)
        b = od.rope(q, m - n, theta) @ k
        assert abs(a - b) < 1e-9 * max(1.0, abs(a))
    # complex-number form: (x_i + j x_{i+hd/2}) * exp(j * pos * theta^(-2i/hd))
    pos = 1234
    z = (q[: hd // 2] + 1j * q[hd // 2:]) * np.exp(1j * pos * theta ** (-np.arange(hd // 2) * 2 / hd))
    np.testing.assert_allclose(od.rope(q, pos, theta), np.concatenate([z.real, z.imag]), atol=1e-12)


def test_silu_hand_and_library():
    g = GOLD["silu"]
    np.testing.assert_allclose(od.silu(np.array(g["x"])), g["y"], rtol=1e-15)
    x = np.linspace(-30, 30, 101)
    np.testing.assert_allclose(od.silu(x), F.silu(torch.from_numpy(x)).numpy(), rtol=1e-13, atol=1e-300)


@pytest.mark.parametrize("Hq,Hkv,n", [(4, 2, 1), (4, 2, 37), (16, 4, 300), (16, 16, 5)])
def test_gqa_attention_vs_torch_sdpa(Hq, Hkv, n):
    rng = np.random.default_rng(Hq * 100 + n)
    hd = 64
    q = rng.standard_normal((Hq, hd))
    k = rng.standard_normal((n, Hkv, hd))
    v = rng.standard_normal((n, Hkv, hd))
    out = od.gqa_attention(q, k, v)
    ref = F.scaled_dot_product_attention(
        torch.from_numpy(q)[None, :, None, :], torch.from_numpy(k).permute(1, 0, 2)[None],
        torch.from_numpy(v).permute(1, 0, 2)[None], enable_gqa=True)[0, :, 0, :].numpy()
    np.testing.assert_allclose(out, ref, rtol=1e-12, atol=1e-12)
    if n == 1:   # a single key returns its value for every query head of the group
        np.testing.assert_array_equal(out, np.repeat(v[0], Hq // Hkv, axis=0))


def test_gather_pages_equals_contiguous():
    rng = np.random.default_rng(3)
    P, H, hd, n = 16, 2, 8, 75
    contig = rng.standard_normal((n, H, hd))
    n_pages = 9
    table = rng.permutation(n_pages)[:5]
    pages = np.full((n_pages, H, P, hd), np.nan)
    for t in range(n):
        pages[table[t // P], :, t % P, :] = contig[t]
    np.testing.assert_array_equal(od.gather_pages(pages, table, n), contig)


# ---------------------------------------------------------------------------
# assembled drafter

SMALL = replace(TINY, vocab=512)
SMALL2 = replace(TINY, vocab=512, n_layers=2)


def _inputs(shape, seed, ctx=(20, 9), n_new=1, K=3, zero=False, **wkw):
    w = syn.make_weights(shape, seed, zero_expansion=zero, **wkw)
    ctx = np.asarray(ctx, np.int32)
    kv = syn.make_kv_prefix(shape, ctx, n_new + K, seed + 1)
    di = syn.make_draft_inputs(shape, len(ctx), n_new, K, seed + 2)
    return w, ctx, kv, di


def _run(shape, w, ctx, kv, di, K=3, T=1.0, **kw):
    return od.draft_step(w, shape, kv["k_rows"], kv["v_rows"], ctx, di["tokens"], di["feats"],
                         di["n_new"], K, T, di["u_draft"], **kw)


@pytest.mark.parametrize("shape", [SMALL, SMALL2])
def test_zero_expansion_is_feature_independent(shape):
    """Eq. 3: with the context columns of W~_qkv zero the drafter computes
    W_qkv z_t, so logits, tokens and new K/V cannot depend on the target
    feature (extend rows) nor on the fed-back hidden state (chain rows)."""
    w, ctx, kv, di = _inputs(shape, 40, zero=True)
    a = _run(shape, w, ctx, kv, di, T=0.0)
    di2 = dict(di, feats=syn.make_draft_inputs(shape, 2, 1, 3, 99)["feats"])
    b = _run(shape, w, ctx, kv, di2, T=0.0)
    np.testing.assert_array_equal(a["logits"], b["logits"])
    np.testing.assert_array_equal(a["tokens"], b["tokens"])
    for x, y in zip(a["new_k"], b["new_k"]):
        np.testing.assert_array_equal(x, y)
    # non-vacuous: with nonzero context columns the features matter
    w, ctx, kv, di = _inputs(shape, 40, zero=False)
    a = _run(shape, w, ctx, kv, di, T=0.0)
    b = _run(shape, w, ctx, kv, di2, T=0.0)
    assert np.abs(a["logits"] - b["logits"]).max() > 1e-3


def test_zeroed_branches_reduce_to_embedding_and_head():
    """With W_o = 0 and W_down = 0 every residual branch vanishes: x_L = E[x] and
    the logits are W_lm RMSNorm(E[x]) for the extend row and every chain row."""
    shape = SMALL2
    w, ctx, kv, di = _inputs(shape, 50)
    for l in range(shape.n_layers):
        w["W_o"][l][:] = 0
        w["W_down"][l][:] = 0
    r = _run(shape, w, ctx, kv, di, T=0.0)
    E, Wlm, gf = (torch.from_numpy(widen(w[k])) for k in ("embed", "lm_head", "final_norm"))
    for b in range(2):
        toks = [int(di["tokens"][b, 0])] + [int(t) for t in r["tokens"][b, :-1]]
        for k, t in enumerate(toks):
            h = F.rms_norm(E[t], (shape.d_model,), gf, eps=shape.rms_eps)
            np.testing.assert_allclose(r["logits"][b, k], F.linear(h, Wlm).numpy(), rtol=1e-10, atol=1e-12)


def test_single_position_attention_copies_value():
    """Empty prefix, one extend row: attention sees only the row's own key, so it
    returns that row's cached (bf16) V (no rotary on V); with W_down = 0 the
    logits follow in closed form from Eq. 1-2 and the GQA head map
    h -> h // (Hq/Hkv)."""
    from oracle.bf16 import round_to_bf16
    shape = SMALL
    w, ctx, kv, di = _inputs(shape, 60, ctx=(0,), K=1)
    w["W_down"][0][:] = 0
    r = _run(shape, w, ctx, kv, di, K=1, T=0.0)
    W = {k: torch.from_numpy(widen(w[k] if not isinstance(w[k], list) else w[k][0]))
         for k in ("embed", "lm_head", "final_norm", "W_c", "W_qkv", "W_o", "attn_norm")}
    d, hd, Hq, Hkv = shape.d_model, shape.head_dim, shape.n_q_heads, shape.n_kv_heads
    x0 = W["embed"][int(di["tokens"][0, 0])]
    c = F.linear(torch.from_numpy(widen(di["feats"][0, 0])), W["W_c"])
    z = F.rms_norm(x0, (d,), W["attn_norm"], eps=shape.rms_eps)
    v = F.linear(torch.cat([c, z]), W["W_qkv"][(Hq + Hkv) * hd:]).reshape(Hkv, hd)
    v = torch.from_numpy(round_to_bf16(v.numpy()))
    attn = v.repeat_interleave(Hq // Hkv, dim=0).reshape(-1)
    x1 = x0 + F.linear(attn, W["W_o"])
    logits = F.linear(F.rms_norm(x1, (d,), W["final_norm"], eps=shape.rms_eps), W["lm_head"])
    np.testing.assert_allclose(r["logits"][0, 0], logits.numpy(), rtol=1e-10, atol=1e-12)


def test_extend_rows_equal_row_by_row_commit():
    """Two extend rows in one call give the same draft as committing the first row
    (appending its K/V to the prefix) and extending with the second."""
    shape = SMALL2
    w, ctx, kv, di = _inputs(shape, 70, ctx=(13,), n_new=2, K=2)
    both = _run(shape, w, ctx, kv, di, K=2, T=0.0)
    first = dict(di, tokens=di["tokens"][:, :1], feats=di["feats"][:, :1], n_new=np.array([1], np.int32))
    r1 = _run(shape, w, ctx, kv, first, K=1, T=0.0)
    # append row 0's K/V (float64, as the oracle keeps it) to the prefix
    k_row = syn.bf16_bits(r1["new_k"][0][:, :1].astype(np.float32))
    v_row = syn.bf16_bits(r1["new_v"][0][:, :1].astype(np.float32))
    kv2 = dict(kv, k_rows=np.concatenate([kv["k_rows"], k_row], 1),
               v_rows=np.concatenate([kv["v_rows"], v_row], 1))
    second = dict(di, tokens=di["tokens"][:, 1:], feats=di["feats"][:, 1:], n_new=np.array([1], np.int32))
    r2 = _run(shape, w, np.array([14], np.int32), kv2, second, K=2, T=0.0)
    # cached rows are bf16 on both paths, so the two computations agree to rounding
    np.testing.assert_allclose(r2["logits"], both["logits"], rtol=1e-9, atol=1e-12)
    np.testing.assert_array_equal(r2["tokens"], both["tokens"])
    # and the two-row call's committed first row is the single-row call's row
    np.testing.assert_array_equal(both["new_k"][0][:, 0], r1["new_k"][0][:, 0])


def test_forced_chain_matches_free_chain():
    shape = SMALL
    w, ctx, kv, di = _inputs(shape, 80)
    free = _run(shape, w, ctx, kv, di, T=1.0)
    forced = _run(shape, w, ctx, kv, di, T=1.0, forced_tokens=free["tokens"])
    np.testing.assert_array_equal(free["logits"], forced["logits"])
    # a different forced token changes the later rows only
    f2 = free["tokens"].copy()
    f2[0, 0] = (f2[0, 0] + 1) % shape.vocab
    alt = _run(shape, w, ctx, kv, di, T=1.0, forced_tokens=f2)
    np.testing.assert_array_equal(alt["logits"][:, 0], free["logits"][:, 0])
    assert np.abs(alt["logits"][0, 1] - free["logits"][0, 1]).max() > 1e-4


def test_forced_cache_rows_match_free_chain():
    """Forcing the cache rows a run wrote reproduces that run exactly; forcing a
    changed row changes the later steps but not the rows this run computes at
    that position."""
    shape = SMALL
    w, ctx, kv, di = _inputs(shape, 81)
    free = _run(shape, w, ctx, kv, di, T=1.0)
    own = [(k, v) for k, v in zip(free["new_k"], free["new_v"])]
    forced = _run(shape, w, ctx, kv, di, T=1.0, forced_tokens=free["tokens"], forced_kv=own)
    np.testing.assert_array_equal(free["logits"], forced["logits"])
    np.testing.assert_array_equal(np.asarray(free["new_k"]), np.asarray(forced["new_k"]))
    alt_k = [k.copy() for k, _ in own]
    alt_k[0][0, 0] += 0.5                       # sequence 0, layer 0, first row written
    alt = _run(shape, w, ctx, kv, di, T=1.0, forced_tokens=free["tokens"],
               forced_kv=[(alt_k[b], own[b][1]) for b in range(len(own))])
    np.testing.assert_array_equal(np.asarray(alt["new_k"])[0][0, 0], np.asarray(free["new_k"])[0][0, 0])
    assert np.abs(alt["logits"][0] - free["logits"][0]).max() > 1e-6


def test_sampling_stats_and_peaked_head():
    """q(token) and (M, log S) describe softmax(z/T); the peaked LM head makes the
    draft distribution concentrated (the sampled-draft parity case)."""
    shape = SMALL
    w, ctx, kv, di = _inputs(shape, 90, peaked_vocab=True)
    r = _run(shape, w, ctx, kv, di, T=1.0)
    for b in range(2):
        for k in range(3):
            z = r["logits"][b, k]
            lse = torch.logsumexp(torch.from_numpy(z), 0).item()
            M, logS = r["stats"][b, k]
            assert abs(M + logS - lse) < 1e-10
            assert abs(r["qx"][b, k] - np.exp(z[r["tokens"][b, k]] - lse)) < 1e-12
            assert np.exp(z.max() - lse) > 0.2      # peaked


def _rope_complex(x, pos, theta):
    """Rotary embedding written as complex multiplication (independent form)."""
    hd = x.shape[-1]
    zc = (x[..., : hd // 2] + 1j * x[..., hd // 2:]) * np.exp(
        1j * pos * theta ** (-np.arange(hd // 2) * 2.0 / hd))
    return np.concatenate([zc.real, zc.imag], -1)


def test_cache_rows_follow_eq2_and_chain_state():
    """W_o = W_down = 0 makes x_L = E[x] at every row, so the K/V each row writes
    has a closed form: K, V = W~_k,v [s; RMSNorm(E[x])] per layer (with that
    layer's weights and gain), rotary on K only at the row's position, and the
    context slot s = W_c feat on the extend row but the previous row's x_L (here
    E[previous token]) on chain rows (Sec. 3.4).  Cached rows are bf16, so the
    comparison allows one bf16 rounding step."""
    shape = SMALL2
    K = 3
    w, ctx, kv, di = _inputs(shape, 110, ctx=(21,), K=K)
    for l in range(shape.n_layers):
        w["W_o"][l][:] = 0
        w["W_down"][l][:] = 0
    r = _run(shape, w, ctx, kv, di, K=K, T=1.0)
    d, hd, Hq, Hkv = shape.d_model, shape.head_dim, shape.n_q_heads, shape.n_kv_heads
    E = torch.from_numpy(widen(w["embed"]))
    toks = [int(di["tokens"][0, 0])] + [int(t) for t in r["tokens"][0, : K - 1]]
    c = F.linear(torch.from_numpy(widen(di["feats"][0, 0])), torch.from_numpy(widen(w["W_c"])))
    for row, t in enumerate(toks):
        s = c if row == 0 else E[toks[row - 1]]
        for l in range(shape.n_layers):
            Wq = torch.from_numpy(widen(w["W_qkv"][l]))
            z = F.rms_norm(E[t], (d,), torch.from_numpy(widen(w["attn_norm"][l])), eps=shape.rms_eps)
            u = torch.cat([s, z])
            k = F.linear(u, Wq[Hq * hd:(Hq + Hkv) * hd]).reshape(Hkv, hd).numpy()
            v = F.linear(u, Wq[(Hq + Hkv) * hd:]).reshape(Hkv, hd).numpy()
            np.testing.assert_allclose(r["new_k"][0][l, row], _rope_complex(k, 21 + row, shape.rope_theta),
                                       rtol=2.0 ** -8, atol=1e-12)
            np.testing.assert_allclose(r["new_v"][0][l, row], v, rtol=2.0 ** -8, atol=1e-12)


def test_mlp_blocks_in_closed_form():
    """W_o = 0 leaves each layer a pre-norm SwiGLU block on the residual stream:
    x <- x + W_down(silu(W_gate n) * W_up n), n = RMSNorm(x) with the layer's
    FFN gain; logits = W_lm RMSNorm(x_L)."""
    shape = SMALL2
    w, ctx, kv, di = _inputs(shape, 120, ctx=(7,), K=1)
    for l in range(shape.n_layers):
        w["W_o"][l][:] = 0
    r = _run(shape, w, ctx, kv, di, K=1, T=0.0)
    T_ = lambda a: torch.from_numpy(widen(a))
    d = shape.d_model
    x = T_(w["embed"])[int(di["tokens"][0, 0])]
    for l in range(shape.n_layers):
        n = F.rms_norm(x, (d,), T_(w["ffn_norm"][l]), eps=shape.rms_eps)
        x = x + F.linear(F.silu(F.linear(n, T_(w["W_gate"][l]))) * F.linear(n, T_(w["W_up"][l])),
                         T_(w["W_down"][l]))
    logits = F.linear(F.rms_norm(x, (d,), T_(w["final_norm"]), eps=shape.rms_eps), T_(w["lm_head"]))
    np.testing.assert_allclose(r["logits"][0, 0], logits.numpy(), rtol=1e-10, atol=1e-12)


def test_round_to_bf16_matches_library_and_keeps_representables():
    from oracle.bf16 import round_to_bf16
    rng = np.random.default_rng(7)
    x = (rng.standard_normal(100_000) * np.exp(rng.uniform(-20, 20, 100_000))).astype(np.float32)
    lib = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(round_to_bf16(x.astype(np.float64)), lib)
    # ties go to even: 1 + 2^-8 lies halfway between 1 and 1 + 2^-7
    assert round_to_bf16(np.array([1 + 2.0 ** -8]))[0] == 1.0
    assert round_to_bf16(np.array([1 + 3 * 2.0 ** -8]))[0] == 1 + 2.0 ** -6
    b = widen(syn.bf16_bits(x[:1000]))
    np.testing.assert_array_equal(round_to_bf16(b), b)
