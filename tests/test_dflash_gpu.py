"""CUDA block drafting (EAGLE-style DFlash, Appendix "EAGLE-Style Target
Interface for DFlash") against the oracle, through the C ABI.

One call is one drafter forward over the anchor and block - 1 mask positions
of each sequence, with the target feature broadcast through the expanded QKV
and causal attention inside the block; position j proposes the token at j + 1.
Logits within 2e-2 of the oracle; tokens equal wherever the decision is not
within the error of a tie (as for the chain drafter); the anchor's K/V row is
committed and the mask rows are cached speculatively after it."""
from dataclasses import replace

import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from oracle import dflash as odf  # noqa: E402
from oracle import drafter as od  # noqa: E402
from paper_2609_09338_gb300 import synthetic as syn  # noqa: E402
from paper_2609_09338_gb300.workloads import TINY, WORKLOADS  # noqa: E402
from parity import check_kv_rows, gather_positions  # noqa: E402

LOGIT_TOL = 2e-2


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__ as g
    g.build()


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def run_block(shape, ctx, block, T, seed, mask=7, zero=False, peaked=False, feats_seed=None):
    from paper_2609_09338_gb300.binding import to_device_bf16
    from paper_2609_09338_gb300.session import DflashSession
    ctx = np.asarray(ctx, np.int32)
    B = len(ctx)
    w = syn.make_weights(shape, seed, zero_expansion=zero, peaked_vocab=peaked)
    kv = syn.make_kv_prefix(shape, ctx, block, seed + 1)
    rng = np.random.default_rng(seed + 2)
    anchors = rng.integers(0, shape.vocab, B).astype(np.int32)
    feats = syn.make_draft_inputs(shape, B, 1, 1, seed + 3 if feats_seed is None else feats_seed)["feats"][:, 0]
    u = rng.random((B, block - 1), dtype=np.float32)
    sess = DflashSession(shape, w, kv["page_table"], kv["n_pages"], block)
    sess.append(ctx, kv["k_rows"], kv["v_rows"])
    out = sess.block_buffers(with_logits=True)
    sess.propose(_dev(anchors), mask, to_device_bf16(feats), T, _dev(u), out)
    torch.cuda.synchronize()
    g = {k: v.cpu().numpy() for k, v in out.items()}
    g["status"] = int(sess.status.item())
    g["seq_len"] = sess.kv.seq_len.cpu().numpy()
    g["k_pages"] = sess.kv.k_pages.float().cpu().numpy()
    g["v_pages"] = sess.kv.v_pages.float().cpu().numpy()
    del sess
    return dict(w=w, kv=kv, ctx=ctx, anchors=anchors, feats=feats, u=u, g=g, shape=shape, block=block, T=T,
                mask=mask)


def check_block(case, seqs=None):
    g, T, sh, P = case["g"], case["T"], case["shape"], case["block"] - 1
    ctx, kv = case["ctx"], case["kv"]
    idx = list(range(len(ctx))) if seqs is None else seqs
    offs = np.concatenate([[0], np.cumsum(ctx)])
    rows = np.concatenate([np.arange(offs[b], offs[b + 1]) for b in idx]).astype(np.int64)
    o = odf.dflash_block(case["w"], sh, kv["k_rows"][:, rows], kv["v_rows"][:, rows], ctx[idx], case["anchors"][idx],
                         case["mask"], case["feats"][idx], case["block"], T, case["u"][idx])
    assert g["status"] == 0
    np.testing.assert_array_equal(g["seq_len"], ctx + 1)                     # only the anchor is committed
    gl = g["draft_logits"][idx]
    err = float(np.abs(gl - o["logits"]).max())
    assert err < LOGIT_TOL, f"logits max abs err {err}"
    toks = g["draft_tokens"][idx]
    checked = 0
    for i, b in enumerate(idx):
        for j in range(P):
            if T == 0:
                if o["margins"][i, j] > 2 * err + 1e-6:
                    assert toks[i, j] == o["tokens"][i, j], (b, j)
                    checked += 1
            else:
                own = od.sample(gl[i, j].astype(np.float64), T, float(case["u"][b, j]))
                if own["margin"] > 1e-5:
                    assert toks[i, j] == own["token"], (b, j)
                if o["margins"][i, j] > np.expm1(2 * err / T) + 1e-5:
                    assert toks[i, j] == o["tokens"][i, j], (b, j)
                    checked += 1
    if T > 0:
        np.testing.assert_allclose(g["draft_stats"][idx][..., 0], o["stats"][..., 0], atol=err / T + 1e-5)
        np.testing.assert_allclose(g["draft_stats"][idx][..., 1], o["stats"][..., 1], atol=2 * err / T + 1e-4)
    for i, b in enumerate(idx):
        pos = np.arange(ctx[b], ctx[b] + P)                                   # anchor + mask rows
        for name, pages in (("new_k", g["k_pages"]), ("new_v", g["v_pages"])):
            got = gather_positions(pages, kv["page_table"][b], pos)
            check_kv_rows(got, o[name][i], o[name + "_mag"][i])
    return checked, len(idx) * P


@pytest.mark.parametrize("T", [0.0, 1.0])
def test_block_matches_oracle(T):
    shape = replace(TINY, n_layers=2, n_q_heads=8, n_kv_heads=2)
    checked, total = check_block(run_block(shape, [40, 3, 77], 5, T, 81, peaked=T > 0))
    assert checked >= total // 2


def test_blocks_in_several_tensor_core_groups():
    """6 sequences x 16 proposals = 96 rows: one group of 5 sequences (80 rows),
    then one of 1, each a pass over the weights."""
    checked, total = check_block(run_block(TINY, [30, 1, 64, 17, 5, 90], 17, 0.0, 83), seqs=[0, 4, 5])
    assert checked >= total // 2


def test_zero_target_projection_bitwise_feature_independent():
    """The appendix's zero-initialised target-side projections: proposals,
    logits and cached rows do not depend on the target feature, bit for bit."""
    a = run_block(TINY, [50, 9], 6, 0.0, 85, zero=True)
    b = run_block(TINY, [50, 9], 6, 0.0, 85, zero=True, feats_seed=999)
    for k in ("draft_logits", "draft_tokens", "k_pages", "v_pages"):
        np.testing.assert_array_equal(a["g"][k], b["g"][k])
    c = run_block(TINY, [50, 9], 6, 0.0, 85, zero=False, feats_seed=999)
    d = run_block(TINY, [50, 9], 6, 0.0, 85, zero=False)
    assert np.abs(c["g"]["draft_logits"] - d["g"]["draft_logits"]).max() > 1e-3
    check_block(a)


def test_paper_block_size_four_layers():
    """Block size 16 (the appendix's B), a four-layer drafter of the workload's
    head layout at a reduced width and vocabulary, sampled."""
    shape = replace(WORKLOADS["dflash-d4096-l4-v151936-b1-blk16"].shape, d_model=1024, ffn_dim=3072,
                    feat_dim=3072, vocab=8192)
    checked, total = check_block(run_block(shape, [700], 16, 1.0, 87, peaked=True))
    assert checked >= total // 2
