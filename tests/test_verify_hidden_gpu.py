"""Logits-free sampled verification (the Sec. 3.1 rule with the draft rows
defined by the drafter's final norm and LM head over its kept states,
Sec. 3.3-3.4) through the C ABI, against the oracle."""
from dataclasses import replace

import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from oracle import verify as ov  # noqa: E402
from oracle.drafter import inverse_cdf  # noqa: E402
from paper_2609_09338_gb300 import synthetic as syn  # noqa: E402
from paper_2609_09338_gb300.workloads import TINY  # noqa: E402
from parity import check_verify  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__ as g
    g.build()


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def _inputs(shape, w, B, K, T, sigma, seed):
    """Kept states, the draft tokens drawn from their rows, the draft step's
    q(x) and (M, log S), target logits near the draft rows, uniforms."""
    rng = np.random.default_rng(seed)
    hidden = rng.standard_normal((B, K, shape.d_model)).astype(np.float32)
    zq = ov.draft_logits_from_hidden(hidden, w["lm_head"], w["final_norm"], shape.rms_eps)
    y = zq / T
    M = y.max(-1)
    e = np.exp(y - M[..., None])
    S = e.sum(-1)
    x = np.array([[inverse_cdf(e[b, i], rng.random())[0] for i in range(K)] for b in range(B)], np.int32)
    qx = (np.take_along_axis(e, x[..., None].astype(np.int64), -1)[..., 0] / S).astype(np.float32)
    stats = np.stack([M, np.log(S)], -1).astype(np.float32)
    zp = np.concatenate([zq + sigma * rng.standard_normal(zq.shape),
                         3 * rng.standard_normal((B, 1, shape.vocab))], axis=1).astype(np.float32)
    return dict(hidden=hidden, x=x, qx=qx, stats=stats, target=zp,
                u_accept=rng.random((B, K), dtype=np.float32), u_sample=rng.random((B, K + 1), dtype=np.float32))


def _run_hidden(ctx, inp, T, dtype):
    from paper_2609_09338_gb300.binding import to_device_bf16
    from paper_2609_09338_gb300.session import VerifyHiddenBuffers
    B, K = inp["x"].shape
    vb = VerifyHiddenBuffers(ctx, B, K)
    tgt = _dev(inp["target"]) if dtype == "f32" else to_device_bf16(syn.bf16_bits(inp["target"]))
    vb.run_hidden(tgt, _dev(inp["hidden"]), _dev(inp["qx"]), _dev(inp["stats"]), _dev(inp["x"]), T,
                  _dev(inp["u_accept"]), _dev(inp["u_sample"]))
    torch.cuda.synchronize()
    return {"status": int(vb.status.item()), **{k: getattr(vb, k).cpu().numpy()
                                                  for k in ("out_tokens", "n_accepted", "flags", "probs")}}


CASES = [
    # vocab, B, K, T, dtype   (chunks with a ragged tail; two groups of sequences at B 96)
    (4096, 1, 4, 1.0, "f32"),
    (20000, 7, 3, 0.7, "bf16"),
    (20003, 5, 2, 1.0, "f32"),      # vocab not a multiple of 8: scalar loads, partial last LM tile
    (8192, 96, 3, 1.0, "f32"),      # two groups (80 + 16 sequences)
    (4096, 3, 15, 1.3, "f32"),      # longest chain
]


@pytest.mark.parametrize("V,B,K,T,dtype", CASES)
def test_verify_hidden_matches_oracle(V, B, K, T, dtype):
    from paper_2609_09338_gb300 import binding as ob
    shape = replace(TINY, vocab=V)
    w = syn.make_weights(shape, seed=V + B)
    ctx = ob.osprey_create(shape, ob.upload_weights(w))
    inp = _inputs(shape, w, B, K, T, 0.7, seed=V + K)
    g = _run_hidden(ctx, inp, T, dtype)
    assert g["status"] == 0
    tgt = inp["target"] if dtype == "f32" else syn.bf16_bits(inp["target"])
    o = ov.verify_hidden(tgt, inp["hidden"], w["lm_head"], w["final_norm"], shape.rms_eps, inp["x"], T,
                         inp["u_accept"], inp["u_sample"])
    check_verify(g["out_tokens"], g["n_accepted"], o, K)
    np.testing.assert_allclose(g["probs"][..., 0], o["p_x"], atol=1e-5)
    np.testing.assert_array_equal(g["probs"][..., 1], inp["qx"])          # the draft step's own q(x)
    assert (g["flags"] & 8).sum() == 0
    rej = (o["n_accepted"] < K).sum()
    assert 0 < rej or B < 4                                                # residual draws are exercised


def test_invalid_draft_token_is_reported():
    from paper_2609_09338_gb300 import binding as ob
    shape = TINY
    w = syn.make_weights(shape, seed=3)
    ctx = ob.osprey_create(shape, ob.upload_weights(w))
    inp = _inputs(shape, w, 4, 3, 1.0, 0.7, seed=4)
    inp["x"][2, 1] = -1                                                    # a skipped sequence's tokens
    g = _run_hidden(ctx, inp, 1.0, "f32")
    assert ob.ERRORS[g["status"]] == "INVALID_ARG"
    assert g["n_accepted"][2] == 0 and (g["out_tokens"][2] == -1).all()
    o = ov.verify_hidden(inp["target"][[0, 1, 3]], inp["hidden"][[0, 1, 3]], w["lm_head"], w["final_norm"],
                         shape.rms_eps, inp["x"][[0, 1, 3]], 1.0, inp["u_accept"][[0, 1, 3]],
                         inp["u_sample"][[0, 1, 3]])
    check_verify(g["out_tokens"][[0, 1, 3]], g["n_accepted"][[0, 1, 3]], o, 3)


@pytest.mark.parametrize("B,max_new", [(1, 1), (4, 3), (33, 2)])
def test_draft_then_verify_without_logits(B, max_new):
    """draft_step_hidden matches draft_step (tokens, q(x), stats bit for bit);
    each kept state maps to its draft logits row through the final norm and the
    LM head (a float64 restatement here); the logits-free verify of the kept
    states decides as osprey_verify does on the draft logits.  From 3 to 80
    sequences both recompute the decision row with the same tensor-core GEMM
    (same planes, same split), so the two agree exactly; at batch 1 the draft
    logits come from the streamed GEMV and the acceptance decisions agree."""
    from paper_2609_09338_gb300.binding import to_device_bf16
    from paper_2609_09338_gb300.session import DraftSession, VerifyBuffers
    shape, K, T = TINY, 4, 1.0
    ctx_lens = np.random.default_rng(B).integers(40, 200, B).astype(np.int32)
    w = syn.make_weights(shape, seed=11)
    kv = syn.make_kv_prefix(shape, ctx_lens, max_new + K, seed=12)
    di = syn.make_draft_inputs(shape, B, max_new, K, seed=13)
    di["n_new"] = np.random.default_rng(B + 1).integers(1, max_new + 1, B).astype(np.int32)
    outs = []
    for keep in (False, True):
        sess = DraftSession(shape, w, kv["page_table"], kv["n_pages"], K, max_new)
        sess.append(ctx_lens, kv["k_rows"], kv["v_rows"])
        out = sess.draft_buffers(with_logits=not keep)
        args = (_dev(di["n_new"]), _dev(di["tokens"]), to_device_bf16(di["feats"]), T, _dev(di["u_draft"]), out)
        hidden = torch.full((B, K, shape.d_model), float("nan"), device="cuda")
        if keep:
            sess.draft_hidden(*args, hidden)
        else:
            sess.draft(*args)
        torch.cuda.synchronize()
        assert int(sess.status.item()) == 0
        outs.append({**{k: v.cpu().numpy() for k, v in out.items() if v is not None},
                     "hidden": hidden.cpu().numpy(), "sess": sess})
    a, h = outs
    for k in ("draft_tokens", "draft_qx", "draft_stats"):
        np.testing.assert_array_equal(a[k], h[k])
    g = h["hidden"].astype(np.float64)
    wide = lambda bits: (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    nrm = g / np.sqrt((g * g).mean(-1, keepdims=True) + shape.rms_eps) * wide(w["final_norm"])
    assert np.abs(nrm @ wide(w["lm_head"]).T - a["draft_logits"]).max() < 1e-3
    rng = np.random.default_rng(5)
    target = np.concatenate([a["draft_logits"] + 0.7 * rng.standard_normal(a["draft_logits"].shape),
                             rng.standard_normal((B, 1, shape.vocab))], axis=1).astype(np.float32)
    u_acc, u_smp = rng.random((B, K), dtype=np.float32), rng.random((B, K + 1), dtype=np.float32)
    inp = dict(hidden=h["hidden"], x=h["draft_tokens"], qx=h["draft_qx"], stats=h["draft_stats"], target=target,
               u_accept=u_acc, u_sample=u_smp)
    gh = _run_hidden(h["sess"].ctx, inp, T, "f32")
    vb = VerifyBuffers(B, K, shape.vocab)
    vb.run(_dev(target), _dev(a["draft_logits"]), _dev(a["draft_tokens"]), T, _dev(u_acc), _dev(u_smp))
    torch.cuda.synchronize()
    assert gh["status"] == 0 and int(vb.status.item()) == 0
    np.testing.assert_array_equal(gh["n_accepted"], vb.n_accepted.cpu().numpy())
    if B >= 3:
        np.testing.assert_array_equal(gh["out_tokens"], vb.out_tokens.cpu().numpy())
