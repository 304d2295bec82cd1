"""osprey_kv_append: rows land in the pages the table names; lengths advance;
capacity violations are reported on the device and leave lengths unchanged."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from dataclasses import replace  # noqa: E402

from paper_2609_09338_gb300 import synthetic as syn  # noqa: E402
from paper_2609_09338_gb300.workloads import TINY, QWEN3_8B_DRAFTER  # noqa: E402
from parity import gather_positions  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__ as g
    g.build()


def _session(shape, ctx, reserve, seed, spare=0):
    from paper_2609_09338_gb300.session import DraftSession
    kv = syn.make_kv_prefix(shape, ctx, reserve, seed, spare_pages=spare)
    w = syn.make_weights(replace(shape, vocab=256), 1)
    sess = DraftSession(replace(shape, vocab=256), w, kv["page_table"], kv["n_pages"], K=2)
    return sess, kv


@pytest.mark.parametrize("shape,ctx", [(TINY, [0, 1, 15, 16, 17, 100]),
                                       (replace(TINY, n_layers=2), [33, 7]),
                                       (QWEN3_8B_DRAFTER, [2048, 1, 300])])
def test_append_scatters_rows_exactly(shape, ctx):
    ctx = np.asarray(ctx, np.int32)
    sess, kv = _session(shape, ctx, 8, 11, spare=3)
    sess.append(ctx, kv["k_rows"], kv["v_rows"])
    torch.cuda.synchronize()
    assert int(sess.status.item()) == 0
    np.testing.assert_array_equal(sess.kv.seq_len.cpu().numpy(), ctx)
    kp = sess.kv.k_pages.view(torch.int16).cpu().numpy().view(np.uint16)
    vp = sess.kv.v_pages.view(torch.int16).cpu().numpy().view(np.uint16)
    off = 0
    for b, n in enumerate(ctx):
        got_k = gather_positions(kp, kv["page_table"][b], np.arange(n))
        got_v = gather_positions(vp, kv["page_table"][b], np.arange(n))
        np.testing.assert_array_equal(got_k, kv["k_rows"][:, off:off + n])
        np.testing.assert_array_equal(got_v, kv["v_rows"][:, off:off + n])
        off += n
    # a second append continues after the committed length
    more = np.array([3] * len(ctx), np.int32)
    rows = syn.make_kv_prefix(shape, more, 0, 12)
    sess.append(more, rows["k_rows"], rows["v_rows"])
    torch.cuda.synchronize()
    np.testing.assert_array_equal(sess.kv.seq_len.cpu().numpy(), ctx + 3)
    kp = sess.kv.k_pages.view(torch.int16).cpu().numpy().view(np.uint16)
    got = gather_positions(kp, kv["page_table"][0], np.arange(ctx[0], ctx[0] + 3))
    np.testing.assert_array_equal(got, rows["k_rows"][:, 0:3])


def test_append_past_capacity_is_reported_and_not_committed():
    ctx = np.array([10, 20], np.int32)
    sess, kv = _session(TINY, ctx, 0, 13)
    big = np.array([0, sess.kv.max_pages * 16 - 20 + 1], np.int32)   # one row too many for sequence 1
    rows = syn.make_kv_prefix(TINY, big, 0, 14)
    sess.append(ctx, kv["k_rows"], kv["v_rows"])
    sess.append(big, rows["k_rows"], rows["v_rows"])
    torch.cuda.synchronize()
    assert int(sess.status.item()) == -4
    np.testing.assert_array_equal(sess.kv.seq_len.cpu().numpy(), ctx)


def test_append_row_count_mismatch_is_rejected():
    ctx = np.array([4, 4], np.int32)
    sess, kv = _session(TINY, ctx, 4, 15)
    from paper_2609_09338_gb300 import binding as ob
    n_rows = torch.tensor([4, 5], dtype=torch.int32, device="cuda")       # sums to 9, rows hold 8
    ob.osprey_kv_append(sess.ctx, sess.kv, n_rows, ob.to_device_bf16(kv["k_rows"]),
                        ob.to_device_bf16(kv["v_rows"]), sess.status)
    torch.cuda.synchronize()
    assert int(sess.status.item()) == -1
    np.testing.assert_array_equal(sess.kv.seq_len.cpu().numpy(), [0, 0])
