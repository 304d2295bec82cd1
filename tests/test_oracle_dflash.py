"""Pins for the EAGLE-style DFlash block-drafter oracle (Appendix, "EAGLE-Style
Target Interface for DFlash").

* Zero target-side projections leave a pretrained-only forward: the proposals
  do not depend on the target feature (and do with the columns non-zero).
* The block forward equals a matrix-form causal forward over the whole block,
  written here with torch library routines (RMSNorm, scaled-dot-product
  attention with a causal mask over prefix + block, SiLU): one formulation
  row by row, the other all positions at once.
* A block of size 2 is the chain drafter's first token after one extend row
  with the same feature (oracle.drafter.draft_step, itself pinned).
* Causal attention: computing the last block position changes no proposal,
  and the mask token id moves proposals 1.. but not proposal 0."""
from dataclasses import replace

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import dflash as odf
from oracle import drafter as od
from oracle.bf16 import round_to_bf16, widen
from paper_2609_09338_gb300 import synthetic as syn
from paper_2609_09338_gb300.workloads import TINY

SHAPE = replace(TINY, n_layers=2, n_q_heads=4, n_kv_heads=2, vocab=512)


def _case(seed, B=2, block=5, zero=False, ctx=(37, 5)):
    ctx = np.asarray(ctx[:B], np.int32)
    w = syn.make_weights(SHAPE, seed, zero_expansion=zero)
    kv = syn.make_kv_prefix(SHAPE, ctx, block, seed + 1)
    rng = np.random.default_rng(seed + 2)
    anchors = rng.integers(0, SHAPE.vocab, B)
    feats = syn.make_draft_inputs(SHAPE, B, 1, 1, seed + 3)["feats"][:, 0]
    u = rng.random((B, block - 1), dtype=np.float32)
    return w, kv, ctx, anchors, feats, u


def test_zero_target_projection_is_feature_independent():
    w, kv, ctx, anchors, feats, u = _case(5, zero=True)
    other = syn.make_draft_inputs(SHAPE, 2, 1, 1, 99)["feats"][:, 0]
    a = odf.dflash_block(w, SHAPE, kv["k_rows"], kv["v_rows"], ctx, anchors, 7, feats, 5, 1.0, u)
    b = odf.dflash_block(w, SHAPE, kv["k_rows"], kv["v_rows"], ctx, anchors, 7, other, 5, 1.0, u)
    np.testing.assert_array_equal(a["logits"], b["logits"])
    np.testing.assert_array_equal(a["tokens"], b["tokens"])
    w2 = syn.make_weights(SHAPE, 5)      # non-zero target-side columns: the feature matters
    c = odf.dflash_block(w2, SHAPE, kv["k_rows"], kv["v_rows"], ctx, anchors, 7, feats, 5, 1.0, u)
    d = odf.dflash_block(w2, SHAPE, kv["k_rows"], kv["v_rows"], ctx, anchors, 7, other, 5, 1.0, u)
    assert np.abs(c["logits"] - d["logits"]).max() > 1e-3


def _matrix_form_block(w, kv, ctx, anchor, mask, feat, block, b):
    """All block positions at once: x [n, d]; per layer QKV for every row from
    [c; RMSNorm(x)], rotary by position, K/V rounded to bf16, attention of the
    block queries over prefix + block keys with a causal mask (torch SDPA)."""
    W = od.widen_weights(w)
    sh = SHAPE
    Hq, Hkv, hd, d = sh.n_q_heads, sh.n_kv_heads, sh.head_dim, sh.d_model
    offs = np.concatenate([[0], np.cumsum(ctx)])
    n = block
    toks = [anchor] + [mask] * (n - 1)
    pos = np.arange(ctx[b], ctx[b] + n)
    c = torch.from_numpy(W["W_c"] @ widen(feat))
    x = torch.from_numpy(W["embed"][toks])
    # rotary as a complex multiply on (x_i, x_{i+hd/2}) pairs
    ang = torch.from_numpy(np.outer(pos, sh.rope_theta ** (-np.arange(hd // 2) * 2.0 / hd)))
    rot = torch.polar(torch.ones_like(ang), ang)

    def rope(t):   # [n, H, hd]
        zc = torch.complex(t[..., : hd // 2], t[..., hd // 2:]) * rot[:, None, :]
        return torch.cat([zc.real, zc.imag], dim=-1)

    for l in range(sh.n_layers):
        u = torch.cat([c.expand(n, d), F.rms_norm(x, (d,), torch.from_numpy(W["attn_norm"][l]), eps=sh.rms_eps)], 1)
        qkv = u @ torch.from_numpy(W["W_qkv"][l]).T
        q = rope(qkv[:, : Hq * hd].reshape(n, Hq, hd))
        k = torch.from_numpy(round_to_bf16(rope(qkv[:, Hq * hd:(Hq + Hkv) * hd].reshape(n, Hkv, hd)).numpy()))
        v = torch.from_numpy(round_to_bf16(qkv[:, (Hq + Hkv) * hd:].reshape(n, Hkv, hd).numpy()))
        kp = torch.from_numpy(widen(kv["k_rows"][l, offs[b]:offs[b + 1]]))
        vp = torch.from_numpy(widen(kv["v_rows"][l, offs[b]:offs[b + 1]]))
        K_ = torch.cat([kp, k]).permute(1, 0, 2)[None]
        V_ = torch.cat([vp, v]).permute(1, 0, 2)[None]
        m = int(ctx[b])
        allow = torch.arange(m + n)[None, :] <= (m + torch.arange(n))[:, None]
        a = F.scaled_dot_product_attention(q.permute(1, 0, 2)[None], K_, V_, attn_mask=allow, enable_gqa=True)
        x = x + a[0].permute(1, 0, 2).reshape(n, Hq * hd) @ torch.from_numpy(W["W_o"][l]).T
        h = F.rms_norm(x, (d,), torch.from_numpy(W["ffn_norm"][l]), eps=sh.rms_eps)
        x = x + (F.silu(h @ torch.from_numpy(W["W_gate"][l]).T) * (h @ torch.from_numpy(W["W_up"][l]).T)) \
            @ torch.from_numpy(W["W_down"][l]).T
    hf = F.rms_norm(x, (d,), torch.from_numpy(W["final_norm"]), eps=sh.rms_eps)
    return (hf @ torch.from_numpy(W["lm_head"]).T).numpy()


@pytest.mark.parametrize("block", [2, 4, 7])
def test_block_forward_equals_matrix_form_causal_forward(block):
    w, kv, ctx, anchors, feats, u = _case(11, block=block)
    o = odf.dflash_block(w, SHAPE, kv["k_rows"], kv["v_rows"], ctx, anchors, 3, feats, block, 1.0, u)
    for b in range(len(ctx)):
        ref = _matrix_form_block(w, kv, ctx, int(anchors[b]), 3, feats[b], block, b)
        # position k's logits predict token k + 1: rows 0..block-2
        np.testing.assert_allclose(o["logits"][b], ref[: block - 1], rtol=1e-9, atol=1e-11)


def test_block_of_two_is_the_chain_drafters_first_token():
    w, kv, ctx, anchors, feats, u = _case(17, block=2)
    for T in (0.0, 1.0):
        o = odf.dflash_block(w, SHAPE, kv["k_rows"], kv["v_rows"], ctx, anchors, 9, feats, 2, T, u)
        ch = od.draft_step(w, SHAPE, kv["k_rows"], kv["v_rows"], ctx, anchors[:, None], feats[:, None],
                           np.ones(len(ctx), np.int32), 1, T, u)
        np.testing.assert_array_equal(o["logits"], ch["logits"])
        np.testing.assert_array_equal(o["tokens"], ch["tokens"])
        np.testing.assert_array_equal(o["stats"], ch["stats"])


def test_causal_block_last_position_and_mask_token():
    w, kv, ctx, anchors, feats, u = _case(23, block=6)
    a = odf.dflash_block(w, SHAPE, kv["k_rows"], kv["v_rows"], ctx, anchors, 3, feats, 6, 1.0, u)
    full = odf.dflash_block(w, SHAPE, kv["k_rows"], kv["v_rows"], ctx, anchors, 3, feats, 6, 1.0, u,
                            full_block=True)
    np.testing.assert_array_equal(a["logits"], full["logits"])
    np.testing.assert_array_equal(a["new_k"][0], full["new_k"][0][:, :5])
    other = odf.dflash_block(w, SHAPE, kv["k_rows"], kv["v_rows"], ctx, anchors, 400, feats, 6, 1.0, u)
    np.testing.assert_array_equal(a["logits"][:, 0], other["logits"][:, 0])   # the anchor's row sees no mask
    assert np.abs(a["logits"][:, 1:] - other["logits"][:, 1:]).max() > 1e-4
