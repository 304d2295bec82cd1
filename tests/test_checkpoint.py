"""Drafter weight files: a round trip keeps every bf16 byte; a wrong shape or a
foreign file is refused."""
from dataclasses import replace

import numpy as np
import pytest

from paper_2609_09338_gb300 import checkpoint as ck
from paper_2609_09338_gb300 import synthetic as syn
from paper_2609_09338_gb300.workloads import TINY


def test_round_trip_keeps_every_byte(tmp_path):
    shape = replace(TINY, n_layers=2)
    w = syn.make_weights(shape, 5)
    p = str(tmp_path / "w.npz")
    ck.save_weights(p, shape, w)
    got_shape, got = ck.load_weights(p, shape)
    assert got_shape == shape
    for name, a in w.items():
        if isinstance(a, list):
            assert len(got[name]) == len(a)
            for x, y in zip(a, got[name]):
                np.testing.assert_array_equal(x, y)
                assert y.dtype == np.uint16
        else:
            np.testing.assert_array_equal(a, got[name])


def test_wrong_shape_and_foreign_files_are_refused(tmp_path):
    w = syn.make_weights(TINY, 6)
    p = str(tmp_path / "w.npz")
    ck.save_weights(p, TINY, w)
    with pytest.raises(ValueError, match="expected"):
        ck.load_weights(p, replace(TINY, vocab=TINY.vocab + 8))
    bad = dict(w)
    bad["lm_head"] = bad["lm_head"][:-1]
    with pytest.raises(ValueError, match="lm_head"):
        ck.save_weights(str(tmp_path / "bad.npz"), TINY, bad)
    q = str(tmp_path / "other.npz")
    np.savez(q, __meta__=np.frombuffer(b'{"format": "something else"}', dtype=np.uint8))
    with pytest.raises(ValueError, match="not a drafter weight file"):
        ck.load_weights(q)
