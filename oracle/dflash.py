"""Oracle EAGLE-style DFlash block drafter, float64.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

What it computes (Appendix, "EAGLE-Style Target Interface for DFlash", and
"Background on DFlash"):

* A block of size Bk is one drafter forward over Bk positions: position 0
  holds the verified anchor token, positions 1..Bk-1 the [MASK] placeholder
  token.  Position k sits at sequence position ctx + k (rotary angle included).
* Every attention layer keeps the drafter's own projections and adds
  target-side projections of the projected target feature c_t:
  Q = W_Q h + W_Q^tgt c_t (and the same for K and V).  That is the expanded
  projection of Eq. 2-3, W~_qkv [c_t; RMSNorm(h)] with the target-side columns
  first; zero target-side columns leave the pretrained drafter's forward.
* c_t = W_c [h_low; h_mid; h_high] (Eq. 1) is gathered once at the block's
  verified anchor position and the same vector is used at every position.
* Intra-block attention is causal: position k attends over the committed
  prefix and block positions 0..k (the drafter's own keys and values, cached
  in bf16 like every drafter row).
* Labels are shifted by one: the output at position k is the distribution of
  the token at position k + 1.  Positions 0..Bk-2 thus give the Bk - 1
  proposals of one forward pass; proposal k is drawn from its own
  q_k = softmax(logits_k / T) by the inverse CDF at u_draft[k] (argmax at
  T = 0), independently of the other proposals.
* The output at position Bk - 1 would predict a token past the block and,
  under causal attention, changes nothing before it; it is not computed
  (``dflash_block(..., full_block=True)`` computes it, for the pin that shows
  the proposals do not depend on it).

The backbone layers, RMSNorm, RoPE, GQA, SwiGLU, final norm and LM head are
the drafter's (``oracle.drafter.forward_row``).  The anchor's K/V row is the
one committed position of the call; the mask rows are speculative.
"""
from __future__ import annotations

import numpy as np

from .bf16 import widen
from .drafter import _SeqCache, feature_projection, forward_row, rmsnorm, sample, widen_weights


def dflash_block(weights: dict, shape, prefix_k: np.ndarray, prefix_v: np.ndarray, ctx_lens: np.ndarray,
                 anchors: np.ndarray, mask_token: int, feats: np.ndarray, block: int, temperature: float,
                 u_draft: np.ndarray, widened: dict | None = None, full_block: bool = False) -> dict:
    """One block-drafting call for a batch of sequences.

    prefix_k/prefix_v: [L, sum(ctx), Hkv, hd] bf16 bits, sequence b owning rows
    [sum(ctx[:b]), sum(ctx[:b+1])).  anchors [B] int: the verified anchor token
    of each sequence, at position ctx[b].  feats [B, 3H] bf16 bits: the target
    feature gathered at the anchor.  u_draft [B, block - 1].

    Returns logits [B, block-1, V], tokens/qx [B, block-1], stats [B, block-1, 2]
    ((M, log S) of logits/T), margins [B, block-1], new_k/new_v per sequence
    [L, n_rows, Hkv, hd] (n_rows = block - 1, or block with ``full_block``), with
    new_k_mag/new_v_mag the error scale of each element (oracle.drafter.forward_row).
    """
    W = widened if widened is not None else widen_weights(weights)
    B, V, L = len(ctx_lens), shape.vocab, shape.n_layers
    P = block - 1
    offs = np.concatenate([[0], np.cumsum(ctx_lens)]).astype(np.int64)
    out = {"logits": np.zeros((B, P, V)), "tokens": np.zeros((B, P), np.int64), "qx": np.zeros((B, P)),
           "stats": np.zeros((B, P, 2)), "margins": np.zeros((B, P)), "new_k": [], "new_v": [],
           "new_k_mag": [], "new_v_mag": []}
    for b in range(B):
        cache = _SeqCache([widen(prefix_k[l, offs[b]:offs[b + 1]]) for l in range(L)],
                          [widen(prefix_v[l, offs[b]:offs[b + 1]]) for l in range(L)])
        new_k = [[] for _ in range(L)]
        new_v = [[] for _ in range(L)]
        new_mag = [[] for _ in range(L)]
        c = feature_projection(W["W_c"], widen(feats[b]))          # gathered once, at the anchor
        for k in range(block if full_block else P):
            tok = int(anchors[b]) if k == 0 else int(mask_token)
            x = forward_row(W, shape, cache, tok, c, int(ctx_lens[b]) + k, new_k, new_v, new_mag=new_mag)
            if k < P:                                              # position k predicts token k + 1
                z = W["lm_head"] @ rmsnorm(x, W["final_norm"], shape.rms_eps)
                smp = sample(z, temperature, float(u_draft[b, k]))
                out["logits"][b, k] = z
                out["tokens"][b, k] = smp["token"]
                out["qx"][b, k] = smp["qx"]
                out["stats"][b, k] = (smp["M"], smp["logS"])
                out["margins"][b, k] = smp["margin"]
        out["new_k"].append(np.asarray(new_k))
        out["new_v"].append(np.asarray(new_v))
        out["new_k_mag"].append(np.asarray([[m[0] for m in ml] for ml in new_mag]))
        out["new_v_mag"].append(np.asarray([[m[1] for m in ml] for ml in new_mag]))
    return out
