"""Drafter weight files: the bf16 weights of one drafter shape in one .npz.

A file holds the shape (as JSON) and every weight as its bf16 bit pattern
(uint16), so a reload gives the same bytes to the CUDA path (through
``binding.upload_weights``) and to the oracle (which widens them exactly).  The
seeded generator in ``synthetic`` writes such a file once; later runs, or runs
on another machine, read it back instead of drawing the weights again.
"""
from __future__ import annotations

import json
import os
from dataclasses import asdict

import numpy as np

from .workloads import DrafterShape

_LAYERED = ("attn_norm", "W_qkv", "W_o", "ffn_norm", "W_gate", "W_up", "W_down")
_GLOBAL = ("W_c", "embed", "final_norm", "lm_head")
FORMAT = "osprey-drafter-weights-v1"


def expected_shapes(shape: DrafterShape) -> dict:
    """Array shape of every weight (the layout of include/osprey.h)."""
    d, a = shape.d_model, shape.n_q_heads * shape.head_dim
    return {"W_c": (d, shape.feat_dim), "embed": (shape.vocab, d), "final_norm": (d,),
            "lm_head": (shape.vocab, d), "attn_norm": (d,), "W_qkv": (shape.qkv_rows, 2 * d), "W_o": (d, a),
            "ffn_norm": (d,), "W_gate": (shape.ffn_dim, d), "W_up": (shape.ffn_dim, d),
            "W_down": (d, shape.ffn_dim)}


def _check(shape: DrafterShape, weights: dict):
    want = expected_shapes(shape)
    for name in _GLOBAL:
        a = weights[name]
        if a.dtype != np.uint16 or a.shape != want[name]:
            raise ValueError(f"{name}: {a.dtype} {a.shape}, expected uint16 {want[name]}")
    for name in _LAYERED:
        if len(weights[name]) != shape.n_layers:
            raise ValueError(f"{name}: {len(weights[name])} layers, expected {shape.n_layers}")
        for l, a in enumerate(weights[name]):
            if a.dtype != np.uint16 or a.shape != want[name]:
                raise ValueError(f"{name}[{l}]: {a.dtype} {a.shape}, expected uint16 {want[name]}")


def save_weights(path: str, shape: DrafterShape, weights: dict) -> None:
    """Write the weights (bf16 bit patterns, as ``synthetic.make_weights`` returns them)."""
    _check(shape, weights)
    arrays = {name: weights[name] for name in _GLOBAL}
    for name in _LAYERED:
        for l, a in enumerate(weights[name]):
            arrays[f"{name}.{l}"] = a
    meta = json.dumps({"format": FORMAT, "shape": asdict(shape)})
    tmp = f"{path}.tmp{os.getpid()}"
    with open(tmp, "wb") as f:
        np.savez(f, __meta__=np.frombuffer(meta.encode(), dtype=np.uint8), **arrays)
    os.replace(tmp, path)   # readers never see a partial file


def load_weights(path: str, shape: DrafterShape | None = None) -> tuple[DrafterShape, dict]:
    """Read a weight file; with ``shape`` given, the file must hold that shape."""
    with np.load(path, allow_pickle=False) as z:
        meta = json.loads(bytes(z["__meta__"]).decode())
        if meta.get("format") != FORMAT:
            raise ValueError(f"{path}: not a drafter weight file ({meta.get('format')!r})")
        got = DrafterShape(**meta["shape"])
        if shape is not None and got != shape:
            raise ValueError(f"{path}: holds {got}, expected {shape}")
        weights = {name: z[name] for name in _GLOBAL}
        for name in _LAYERED:
            weights[name] = [z[f"{name}.{l}"] for l in range(got.n_layers)]
    _check(got, weights)
    return got, weights
