"""Failure detection without a GPU fault: a bounded device wait that runs out
(a barrier nothing completes) reports OSPREY_ERR_TIMEOUT through the status
word, and the context stays usable for the next call."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from paper_2609_09338_gb300 import synthetic as syn  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__ as g
    g.build()


def test_bounded_wait_reports_timeout_and_context_survives():
    from paper_2609_09338_gb300 import binding as ob
    from paper_2609_09338_gb300.session import VerifyBuffers
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    ob.osprey_selftest_wait_timeout(1_000_000, status)     # about half a millisecond of SM clocks
    torch.cuda.synchronize()
    assert ob.ERRORS[int(status.item())] == "TIMEOUT"
    # the next call on the same context and stream runs normally
    vi = syn.make_verify_inputs(4096, 2, 3, 1.0, 0.7, seed=5)
    dev = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    vb = VerifyBuffers(2, 3, 4096)
    vb.run(dev(vi["target_logits"]), dev(vi["draft_logits"]), dev(vi["draft_tokens"]), 1.0,
           dev(vi["u_accept"]), dev(vi["u_sample"]))
    torch.cuda.synchronize()
    assert int(vb.status.item()) == 0
    assert (vb.n_accepted.cpu().numpy() >= 0).all()
