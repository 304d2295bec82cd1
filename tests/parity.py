"""Shared parity checks between the CUDA path and the oracle (test helpers)."""
import numpy as np

from oracle import verify as ov


def check_verify(gpu_tokens, gpu_nacc, o, K):
    """Bit-exact comparison under the flagging rule: token ids and accepted
    lengths must match at every unflagged decision; comparison of a sequence
    stops at its first flagged decision.  Returns the number of sequences that
    hit a flag."""
    B = gpu_tokens.shape[0]
    flagged = 0
    for b in range(B):
        fl = o["flags"][b]
        r = int(o["n_accepted"][b])
        stop = next((i for i in range(K + 1) if fl[i] & ov.FLAG_RATIO), None)
        if stop is not None:
            flagged += 1
            assert (gpu_tokens[b, :stop] == o["out_tokens"][b, :stop]).all(), b
            assert gpu_nacc[b] >= stop, b
            continue
        assert gpu_nacc[b] == r, (b, gpu_nacc[b], r)
        assert (gpu_tokens[b, :r] == o["out_tokens"][b, :r]).all(), b
        if fl[r] & ov.FLAG_CDF:
            flagged += 1
        else:
            assert gpu_tokens[b, r] == o["out_tokens"][b, r], (b, r, gpu_tokens[b, r], o["out_tokens"][b, r])
        assert (gpu_tokens[b, r + 1:] == -1).all(), b
    return flagged


def gather_positions(pages, page_table_row, positions):
    """pages [L, n_pages, Hkv, P, hd] (numpy float32) -> [L, len(positions), Hkv, hd]."""
    P = pages.shape[3]
    pos = np.asarray(positions)
    # advanced indices split by a slice put the position axis first: move it back
    return np.moveaxis(pages[:, page_table_row[pos // P], :, pos % P, :], 0, 1)


def bf16_to_f32(t):
    """torch bf16 tensor -> numpy float32 (exact)."""
    import torch
    return t.to(torch.float32).cpu().numpy()
