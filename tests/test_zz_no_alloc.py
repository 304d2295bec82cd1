"""osprey_verify_static: the verify entry point that allocates nothing.

Some callers cannot allocate device memory - an engine that has reserved nearly
all HBM for its weights and KV cache, or code on a latency-critical path where
cudaMalloc/cudaFree may block or synchronise the device.  For them the library
keeps verify's scratch in a fixed device array of its own.  This file checks,
through the C ABI, that two calls in a row give what the workspace entry point
gives, that a call changes neither the device's free memory nor torch's
allocations, and that requests too large for the array are refused with a
message.  Kept in a file that pytest collects last."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from paper_2609_09338_gb300 import synthetic as syn  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__ as g
    g.build()


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def _outputs(B, K):
    return {"out_tokens": torch.full((B, K + 1), -9, dtype=torch.int32, device="cuda"),
            "n_accepted": torch.full((B,), -9, dtype=torch.int32, device="cuda"),
            "flags": torch.full((B, K + 1), 255, dtype=torch.uint8, device="cuda"),
            "probs": torch.zeros((B, K, 2), dtype=torch.float32, device="cuda"),
            "status": torch.zeros(1, dtype=torch.int32, device="cuda")}


@pytest.mark.parametrize("V,B,K,T", [(20000, 7, 3, 1.0), (151936, 4, 7, 1.0), (4096, 16, 4, 0.0)])
def test_static_scratch_matches_workspace_entry_point(V, B, K, T):
    from paper_2609_09338_gb300 import binding as ob
    vi = syn.make_verify_inputs(V, B, K, T, 0.7, seed=V + 5 * B)
    args = (_dev(vi["target_logits"]), _dev(vi["draft_logits"]) if T > 0 else None, _dev(vi["draft_tokens"]), T,
            _dev(vi["u_accept"]), _dev(vi["u_sample"]))
    ref = _outputs(B, K)
    ws = torch.zeros(ob.osprey_verify_workspace_bytes(B, K, V), dtype=torch.uint8, device="cuda")
    ob.osprey_verify(*args, ref["out_tokens"], ref["n_accepted"], ref["flags"], ref["probs"], ws, ref["status"])
    outs = [_outputs(B, K) for _ in range(2)]   # allocated before the calls are measured
    torch.cuda.synchronize()
    for i, got in enumerate(outs):              # two calls in a row share the static array
        free0, alloc0 = torch.cuda.mem_get_info()[0], torch.cuda.memory_allocated()
        ob.osprey_verify_static(*args, got["out_tokens"], got["n_accepted"], got["flags"], got["probs"],
                                got["status"])
        torch.cuda.synchronize()
        if i == 1:   # the first call may load the library's device code; the second allocates nothing
            assert torch.cuda.mem_get_info()[0] == free0
            assert torch.cuda.memory_allocated() == alloc0
        assert int(got["status"].item()) == 0
        for k in ("out_tokens", "n_accepted", "flags"):
            np.testing.assert_array_equal(got[k].cpu().numpy(), ref[k].cpu().numpy())
        if T > 0:
            np.testing.assert_allclose(got["probs"].cpu().numpy(), ref["probs"].cpu().numpy(), atol=1e-5)


def test_static_scratch_refuses_oversized_requests():
    from paper_2609_09338_gb300 import binding as ob
    B, K, V = 4096, 8, 200064
    assert ob.osprey_verify_workspace_bytes(B, K, V) > ob.VERIFY_STATIC_SCRATCH_BYTES
    t = torch.zeros(1, dtype=torch.float32, device="cuda")
    i = torch.zeros(1, dtype=torch.int32, device="cuda")
    p = ob._ptr
    code = ob._c_verify_static(B, K, V, ob.OSPREY_F32, p(t), p(t), p(i), 1.0, p(t), p(t), p(i), p(i), p(i), None,
                               p(i), None)
    assert code == -4
    assert "static scratch" in ob.osprey_last_error()
