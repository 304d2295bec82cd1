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


def check_kv_rows(got, want, mag):
    """Cached bf16 K/V rows of the GPU against the oracle's.

    Each side rounds its own unrounded value a (GPU, float32) or a* (oracle,
    float64) to bf16, which moves it by at most half a bf16 step, 2^-8 |value|:
        |got - want| <= 2^-8 (|got| + |want|) + |a - a*|.
    a - a* is the float32 error of the projection that made the element, a dot
    product of the row's inputs u with a row of W~_qkv, so it scales with
    mag = sum_j |W_ij| |u_j| (the oracle's ``*_mag``; for a rotated key, summed
    over its rotation pair): |a - a*| <= c * mag.  The inputs u of a chain row
    carry the float32 error of every step before it (the fed-back state runs
    through attention over up to 8k cached keys).  Over the workloads the
    largest element needs c = 2^-13.8: a row of the sixth chain step of the
    two-layer Llama-shaped drafter drafting greedily (2^-15.0 when it samples);
    the one-layer drafters fit 2^-16.  c = 2^-13 keeps a factor 1.7 above it."""
    import numpy as np
    np.testing.assert_array_less(np.abs(got - want), 2.0 ** -8 * (np.abs(got) + np.abs(want)) + 2.0 ** -13 * mag + 1e-30)
