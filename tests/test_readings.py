"""The reading of Eq. 1-2 (W_c maps the 3H target tap to d; the expanded QKV
reads 2d inputs) reproduces the body sizes the paper prints in its draft-size
table (Appendix, "Draft Model Sizes")."""
import json
import os

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "draft_sizes.json")))


def _body_params(r):
    d, hd = r["d_h"], r["head_dim"]
    qkv_rows = (r["n_q_heads"] + 2 * r["n_kv_heads"]) * hd
    per_layer = qkv_rows * 2 * d + d * r["n_q_heads"] * hd + 3 * r["ffn"] * d
    return r["L"] * per_layer + r["f_c_in"] * d


def test_body_sizes_match_paper_table():
    for r in GOLD["rows"]:
        got = _body_params(r) / 1e6
        assert abs(got - r["body_m"]) <= GOLD["tolerance_m"], (r["draft"], got)


def test_unexpanded_reading_does_not_match():
    r = next(r for r in GOLD["rows"] if r["draft"] == "Osprey")
    d, hd = r["d_h"], r["head_dim"]
    qkv_rows = (r["n_q_heads"] + 2 * r["n_kv_heads"]) * hd
    unexpanded = r["L"] * (qkv_rows * d + d * r["n_q_heads"] * hd + 3 * r["ffn"] * d) + r["f_c_in"] * d
    assert abs(unexpanded / 1e6 - r["body_m"]) > 20
