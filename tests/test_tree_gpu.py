"""Tree drafting (topk > 1) on the GPU, through the C ABI, against the oracle.

* osprey_verify_tree against oracle.tree.verify_tree: token ids, accepted
  lengths and the accepted branch bit-exact at every unflagged decision (the
  comparison of a sequence stops at its first flagged one).  The ratio band
  is 1e-4 here: after a rejection the tested ratio is max(0, p - c q) / W / q,
  whose float32 value carries the cancellation in p - c q.
* topk = 1 gives osprey_verify's result.
* osprey_draft_step_topk: candidate 0 is the chain drafter's token (same
  logits, statistics and cached rows, bit for bit); the other candidates are
  the inverse CDF of the GPU's own logits at their uniforms (sampled) or the
  next-highest logits (greedy), and the oracle's where the decision is not
  within the measured logit error of a tie."""
from dataclasses import replace

import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from oracle import drafter as od  # noqa: E402
from oracle import tree as ot  # noqa: E402
from paper_2609_09338_gb300 import synthetic as syn  # noqa: E402
from paper_2609_09338_gb300.workloads import TINY, WORKLOADS  # noqa: E402

RATIO_BAND = 1e-4


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__ as g
    g.build()


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def _run_tree(ti, T, dtype):
    from paper_2609_09338_gb300.binding import to_device_bf16
    from paper_2609_09338_gb300.session import TreeVerifyBuffers
    B, K, k = ti["cand"].shape
    conv = (lambda a: _dev(a)) if dtype == "f32" else (lambda a: to_device_bf16(syn.bf16_bits(a)))
    tb = TreeVerifyBuffers(B, K)
    tb.run(conv(ti["target_logits"]), conv(ti["draft_logits"]) if T > 0 else None, _dev(ti["cand"]), T,
           _dev(ti["u_accept"]), _dev(ti["u_sample"]))
    torch.cuda.synchronize()
    return {"status": int(tb.status.item()), **{n: getattr(tb, n).cpu().numpy()
                                                  for n in ("out_tokens", "n_accepted", "branch", "flags")}}


def check_tree(g, o, K):
    """Bit-exact under the flagging rule; returns the number of flagged sequences."""
    B = g["out_tokens"].shape[0]
    flagged = 0
    for b in range(B):
        fl = o["flags"][b]
        stop = next((i for i in range(K + 1) if fl[i] & (ot.FLAG_RATIO | ot.FLAG_CDF)), None)
        if stop is not None:
            flagged += 1
            np.testing.assert_array_equal(g["out_tokens"][b, :stop], o["out_tokens"][b, :stop], err_msg=str(b))
            continue
        assert g["n_accepted"][b] == o["n_accepted"][b], (b, g["n_accepted"][b], o["n_accepted"][b])
        assert g["branch"][b] == o["branch"][b], (b, g["branch"][b], o["branch"][b])
        np.testing.assert_array_equal(g["out_tokens"][b], o["out_tokens"][b], err_msg=str(b))
    return flagged


@pytest.mark.parametrize("V,B,K,k,T,dtype", [
    (4096, 24, 4, 3, 1.0, "f32"),
    (20003, 9, 5, 2, 0.7, "f32"),     # vocabulary not a multiple of 8: scalar loads
    (20000, 12, 3, 4, 1.0, "bf16"),
    (4096, 16, 6, 3, 0.0, "f32"),
    (151936, 4, 7, 4, 1.0, "f32"),
    (151936, 4, 7, 4, 0.0, "bf16"),
])
def test_verify_tree_matches_oracle(V, B, K, k, T, dtype):
    ti = syn.make_tree_inputs(V, B, K, k, T, 0.7, seed=V + B + k)
    g = _run_tree(ti, T, dtype)
    assert g["status"] == 0
    tgt = ti["target_logits"] if dtype == "f32" else syn.bf16_bits(ti["target_logits"])
    drf = ti["draft_logits"] if dtype == "f32" else syn.bf16_bits(ti["draft_logits"])
    o = ot.verify_tree(tgt, drf if T > 0 else None, ti["cand"], T, ti["u_accept"], ti["u_sample"],
                       ratio_band=RATIO_BAND)
    flagged = check_tree(g, o, K)
    assert flagged <= max(1, B // 8)
    if T > 0:   # leaves and residual draws are exercised
        assert (o["branch"] > 0).any() or (o["n_accepted"] < K).any()


def test_topk1_tree_is_the_chain_verify():
    from paper_2609_09338_gb300.session import VerifyBuffers
    V, B, K, T = 8192, 16, 5, 1.0
    vi = syn.make_verify_inputs(V, B, K, T, 0.7, seed=77)
    ti = {"target_logits": vi["target_logits"], "draft_logits": vi["draft_logits"],
          "cand": vi["draft_tokens"][..., None], "u_accept": vi["u_accept"][..., None], "u_sample": vi["u_sample"]}
    g = _run_tree(ti, T, "f32")
    vb = VerifyBuffers(B, K, V)
    vb.run(_dev(vi["target_logits"]), _dev(vi["draft_logits"]), _dev(vi["draft_tokens"]), T, _dev(vi["u_accept"]),
           _dev(vi["u_sample"]))
    torch.cuda.synchronize()
    flagged_chain = vb.flags.cpu().numpy()
    for b in range(B):
        if flagged_chain[b].any() or g["flags"][b].any():
            continue
        assert g["n_accepted"][b] == int(vb.n_accepted[b])
        np.testing.assert_array_equal(g["out_tokens"][b], vb.out_tokens[b].cpu().numpy())


def test_candidate_out_of_range_is_reported():
    ti = syn.make_tree_inputs(4096, 4, 3, 2, 1.0, 0.7, seed=5)
    ti["cand"][2, 1, 1] = 4096
    g = _run_tree(ti, 1.0, "f32")
    assert g["status"] == -1
    assert g["n_accepted"][2] == 0 and (g["out_tokens"][2] == -1).all()


def _draft_topk(shape, ctx, K, k, T, seed, peaked=False):
    from paper_2609_09338_gb300.binding import to_device_bf16
    from paper_2609_09338_gb300.session import DraftSession
    ctx = np.asarray(ctx, np.int32)
    B = len(ctx)
    w = syn.make_weights(shape, seed, peaked_vocab=peaked)
    kv = syn.make_kv_prefix(shape, ctx, 1 + K, seed + 1)
    di = syn.make_draft_inputs(shape, B, 1, K, seed + 2)
    u = np.random.default_rng(seed + 3).random((B, K, k), dtype=np.float32)
    u[..., 0] = di["u_draft"]
    res = {}
    for mode in ("chain", "tree"):
        sess = DraftSession(shape, w, kv["page_table"], kv["n_pages"], K)
        sess.append(ctx, kv["k_rows"], kv["v_rows"])
        args = (_dev(di["n_new"]), _dev(di["tokens"]), to_device_bf16(di["feats"]), T)
        if mode == "chain":
            out = sess.draft_buffers(with_logits=True)
            sess.draft(*args, _dev(di["u_draft"]), out)
        else:
            out = sess.tree_buffers(k, with_logits=True)
            sess.draft_tree(*args, _dev(u), out)
        torch.cuda.synchronize()
        r = {n: v.cpu().numpy() for n, v in out.items() if v is not None}
        r["status"] = int(sess.status.item())
        r["k_pages"] = sess.kv.k_pages.float().cpu().numpy()
        res[mode] = r
        del sess
    return res, dict(w=w, kv=kv, di=di, ctx=ctx, u=u)


@pytest.mark.parametrize("name,B,T", [("tiny", 1, 1.0), ("tiny", 5, 1.0), ("tiny", 5, 0.0),
                                      ("qwen3", 1, 1.0), ("qwen3", 4, 0.0)])
def test_draft_topk_candidates(name, B, T):
    k, K = 3, 4
    shape = TINY if name == "tiny" else WORKLOADS["qwen3-8b-d1024-v151936-b1-k7"].shape
    ctx = [40 + 11 * b for b in range(B)]
    res, inp = _draft_topk(shape, ctx, K, k, T, 91, peaked=T > 0)
    ch, tr = res["chain"], res["tree"]
    assert ch["status"] == 0 and tr["status"] == 0
    z = tr["draft_logits"].astype(np.float64)
    if B >= 3:
        # the same tensor-core LM head and pick: candidate 0 is the chain, bit for bit
        np.testing.assert_array_equal(tr["cand"][..., 0], ch["draft_tokens"])
        np.testing.assert_array_equal(tr["draft_logits"], ch["draft_logits"])
        np.testing.assert_array_equal(tr["k_pages"], ch["k_pages"])
        np.testing.assert_array_equal(tr["draft_stats"], ch["draft_stats"])
    else:
        # one or two rows: the chain samples on the streamed LM head, topk on the
        # tensor-core one; candidate 0 agrees wherever its draw is clear of a bin edge.
        # The tensor-core head carries each final-norm activation in two bf16 planes
        # (error at most 2^-18 relative per element), so the two heads' logits part by
        # a few parts in 1e6 of their magnitude on top of the accumulation order.
        np.testing.assert_allclose(tr["draft_logits"], ch["draft_logits"], atol=1e-4, rtol=1e-5)
        for b in range(B):
            for i in range(K):
                own = od.sample(z[b, i], T, float(inp["u"][b, i, 0]))
                if own["margin"] > 1e-4:
                    assert tr["cand"][b, i, 0] == ch["draft_tokens"][b, i], (b, i)
                else:
                    return   # the chains may part here: nothing after it is comparable
    z = tr["draft_logits"].astype(np.float64)
    o = od.draft_step(inp["w"], shape, inp["kv"]["k_rows"], inp["kv"]["v_rows"], inp["ctx"], inp["di"]["tokens"],
                      inp["di"]["feats"], inp["di"]["n_new"], K, T, inp["di"]["u_draft"],
                      forced_tokens=ch["draft_tokens"])
    err = float(np.abs(z - o["logits"]).max())
    assert err < 2e-2
    for b in range(B):
        for i in range(K):
            if T == 0:
                zr = z[b, i]
                order = np.lexsort((np.arange(zr.size), -zr))
                # the GPU's own logits: strictly ordered where the gaps exceed their recomputation error
                gaps = -np.diff(zr[order[:k + 1]])
                for j in range(1, k):
                    if gaps[j - 1] > 1e-4 and gaps[j] > 1e-4:
                        assert tr["cand"][b, i, j] == order[j], (b, i, j)
                zo = o["logits"][b, i]
                oo = np.lexsort((np.arange(zo.size), -zo))
                go = -np.diff(zo[oo[:k + 1]])
                for j in range(1, k):
                    if go[j - 1] > 2 * err + 1e-6 and go[j] > 2 * err + 1e-6:
                        assert tr["cand"][b, i, j] == oo[j], (b, i, j)
            else:
                for j in range(1, k):
                    own = od.sample(z[b, i], T, float(inp["u"][b, i, j]))
                    if own["margin"] > 1e-5:
                        assert tr["cand"][b, i, j] == own["token"], (b, i, j)
                    ref = od.sample(o["logits"][b, i], T, float(inp["u"][b, i, j]))
                    if ref["margin"] > np.expm1(2 * err / T) + 1e-5:
                        assert tr["cand"][b, i, j] == ref["token"], (b, i, j)
                y = z[b, i] / T
                e = np.exp(y - y.max())
                np.testing.assert_allclose(tr["cand_qx"][b, i], e[tr["cand"][b, i]] / e.sum(), rtol=1e-3, atol=1e-7)


def test_tree_end_to_end_smoke():
    """Draft candidates, target rows around them, tree verification: a run
    through both entry points with consistent outputs."""
    shape = replace(TINY, vocab=4096)
    K, k, T = 4, 3, 1.0
    res, _ = _draft_topk(shape, [64, 20], K, k, T, 95, peaked=True)
    tr = res["tree"]
    B = 2
    rng = np.random.default_rng(3)
    zq = tr["draft_logits"]
    zp = np.empty((B, 1 + K * k, shape.vocab), np.float32)
    zp[:, 0] = zq[:, 0] + 0.5 * rng.standard_normal((B, shape.vocab))
    for i in range(K):
        for j in range(k):
            src = zq[:, i + 1] if (j == 0 and i < K - 1) else zq[:, i]
            zp[:, 1 + i * k + j] = src + 0.5 * rng.standard_normal((B, shape.vocab))
    ti = {"target_logits": zp, "draft_logits": zq, "cand": tr["cand"],
          "u_accept": rng.random((B, K, k), dtype=np.float32), "u_sample": rng.random((B, K + 1), dtype=np.float32)}
    g = _run_tree(ti, T, "f32")
    assert g["status"] == 0
    o = ot.verify_tree(zp, zq, tr["cand"], T, ti["u_accept"], ti["u_sample"], ratio_band=RATIO_BAND)
    check_tree(g, o, K)
