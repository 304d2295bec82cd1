"""ctypes binding of libosprey.so (include/osprey.h), same names as the C ABI.

Argument marshalling only: tensors are checked for device, dtype, shape and
contiguity and passed as raw pointers; every step of the path runs in the
library's CUDA kernels.  Importing this module fails loudly when the library
has not been built - there is no other implementation to fall back to.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import numpy as np
import torch

from .workloads import DrafterShape

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libosprey.so")
MAX_LAYERS = 8
OSPREY_F32, OSPREY_BF16 = 0, 1
ERRORS = {0: "OK", -1: "INVALID_ARG", -2: "SHAPE", -3: "DTYPE", -4: "CAPACITY", -5: "CUDA", -6: "TIMEOUT"}


def status_name(code: int) -> str:
    """Name of a status code; a bounds-checked build (-DOSP_BOUNDS=1) reports a
    failed check as -(1000 + source line)."""
    if code <= -1000:
        return f"BOUNDS(line {-code - 1000})"
    return ERRORS.get(code, f"UNKNOWN({code})")


class OspreyError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"osprey error {code} ({ERRORS.get(code, '?')}): {msg}")
        self.code = code


def _load():
    if not os.path.exists(_LIB_PATH):
        raise ImportError(f"{_LIB_PATH} is missing: run `python -c 'import __graft_entry__ as g; g.build()'`")
    return ctypes.CDLL(_LIB_PATH)


_lib = _load()
_vp, _i32, _i64, _f32, _sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_float, ctypes.c_size_t


class osprey_config(ctypes.Structure):
    _fields_ = [(n, _i32) for n in ("d_model", "n_layers", "n_q_heads", "n_kv_heads", "head_dim",
                                     "ffn_dim", "vocab", "feat_dim", "page_size")] + \
               [("rms_eps", _f32), ("rope_theta", _f32)]


class osprey_weights(ctypes.Structure):
    _fields_ = [(n, _vp) for n in ("W_c", "embed", "final_norm", "lm_head")] + \
               [(n, _vp * MAX_LAYERS) for n in ("attn_norm", "W_qkv", "W_o", "ffn_norm", "W_gate", "W_up", "W_down")]


class osprey_kv(ctypes.Structure):
    _fields_ = [("k_pages", _vp), ("v_pages", _vp), ("page_table", _vp), ("seq_len", _vp),
                ("max_pages_per_seq", _i32), ("n_pages", _i32)]


def _sig(name, res, args):
    f = getattr(_lib, name)
    f.restype, f.argtypes = res, args
    return f


_c_last_error = _sig("osprey_last_error", ctypes.c_char_p, [])
_c_create = _sig("osprey_create", ctypes.c_int, [ctypes.POINTER(osprey_config), ctypes.POINTER(osprey_weights),
                                                  ctypes.POINTER(_vp)])
_c_destroy = _sig("osprey_destroy", None, [_vp])
_c_draft_ws = _sig("osprey_draft_workspace_bytes", _sz, [_vp, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int])
_c_kv_append = _sig("osprey_kv_append", ctypes.c_int, [_vp, ctypes.POINTER(osprey_kv), ctypes.c_int, _vp, _i64,
                                                        _vp, _vp, _vp, _vp])
_c_draft = _sig("osprey_draft_step", ctypes.c_int,
                [_vp, ctypes.POINTER(osprey_kv), ctypes.c_int, ctypes.c_int, ctypes.c_int, _vp, _vp, _vp, _f32, _vp,
                 _vp, _vp, _vp, _vp, _vp, _sz, _vp, _vp])
_c_draft_hidden = _sig("osprey_draft_step_hidden", ctypes.c_int,
                       [_vp, ctypes.POINTER(osprey_kv), ctypes.c_int, ctypes.c_int, ctypes.c_int, _vp, _vp, _vp, _f32,
                        _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp, _vp])
_c_draft_topk = _sig("osprey_draft_step_topk", ctypes.c_int,
                     [_vp, ctypes.POINTER(osprey_kv), ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int, _vp, _vp,
                      _vp, ctypes.c_float, _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp, _vp])
_c_verify_tree = _sig("osprey_verify_tree", ctypes.c_int,
                      [ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int, _vp, _vp, _vp,
                       ctypes.c_float, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp])
_c_dflash_ws = _sig("osprey_dflash_workspace_bytes", _sz, [_vp, ctypes.c_int, ctypes.c_int, ctypes.c_int])
_c_dflash = _sig("osprey_dflash_step", ctypes.c_int,
                 [_vp, ctypes.POINTER(osprey_kv), ctypes.c_int, ctypes.c_int, _vp, ctypes.c_int32, _vp,
                  ctypes.c_float, _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp, _vp])
_c_verify_hidden_ws = _sig("osprey_verify_hidden_workspace_bytes", _sz, [_vp, ctypes.c_int, ctypes.c_int])
_c_verify_hidden = _sig("osprey_verify_hidden", ctypes.c_int,
                        [_vp, ctypes.c_int, ctypes.c_int, ctypes.c_int, _vp, _vp, _vp, _vp, _vp, _f32, _vp, _vp, _vp,
                         _vp, _vp, _vp, _vp, _sz, _vp, _vp])
_c_verify_ws = _sig("osprey_verify_workspace_bytes", _sz, [ctypes.c_int, ctypes.c_int, ctypes.c_int])
_c_verify = _sig("osprey_verify", ctypes.c_int,
                 [ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int, _vp, _vp, _vp, _f32, _vp, _vp, _vp, _vp,
                  _vp, _vp, _vp, _sz, _vp, _vp])
_c_verify_static = _sig("osprey_verify_static", ctypes.c_int,
                        [ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int, _vp, _vp, _vp, _f32, _vp, _vp, _vp,
                         _vp, _vp, _vp, _vp, _vp])
_c_probe_enable = _sig("osprey_probe_enable", ctypes.c_int, [_vp, ctypes.c_int])
_c_probe_select = _sig("osprey_probe_select", ctypes.c_int, [_vp, ctypes.c_int])
_c_probe_read = _sig("osprey_probe_read", ctypes.c_int, [_vp, ctypes.POINTER(_f32), ctypes.c_int])
_c_launch_count = _sig("osprey_launch_count", _i64, [])
_c_selftest_wait = _sig("osprey_selftest_wait_timeout", ctypes.c_int, [_i64, _vp, _vp])

EXPORTED = ["osprey_last_error", "osprey_create", "osprey_destroy", "osprey_draft_workspace_bytes",
            "osprey_kv_append", "osprey_draft_step", "osprey_draft_step_hidden", "osprey_draft_step_topk",
            "osprey_verify_tree", "osprey_dflash_workspace_bytes",
            "osprey_dflash_step", "osprey_verify_workspace_bytes",
            "osprey_verify", "osprey_verify_static", "osprey_verify_hidden_workspace_bytes", "osprey_verify_hidden",
            "osprey_probe_enable", "osprey_probe_select", "osprey_probe_read", "osprey_launch_count", "osprey_selftest_wait_timeout"]


def osprey_last_error() -> str:
    return _c_last_error().decode()


def _check(code: int):
    if code != 0:
        raise OspreyError(code, osprey_last_error())


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _need(t, dtype, shape=None, name="tensor", device=True):
    if t is None:
        raise ValueError(f"{name} is required")
    if t.dtype != dtype:
        raise TypeError(f"{name}: dtype {t.dtype}, expected {dtype}")
    if device and not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name}: shape {tuple(t.shape)}, expected {tuple(shape)}")
    return t


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


# ---------------------------------------------------------------------------- context

class Ctx:
    """An osprey_ctx plus references to the weight tensors it borrows."""

    def __init__(self, shape: DrafterShape, weights: dict):
        self.shape = shape
        self._weights = weights        # keep the device tensors alive
        cfg = osprey_config(shape.d_model, shape.n_layers, shape.n_q_heads, shape.n_kv_heads, shape.head_dim,
                            shape.ffn_dim, shape.vocab, shape.feat_dim, shape.page_size, shape.rms_eps,
                            shape.rope_theta)
        w = osprey_weights()
        bf = torch.bfloat16
        d, V = shape.d_model, shape.vocab
        w.W_c = _ptr(_need(weights["W_c"], bf, (d, shape.feat_dim), "W_c"))
        w.embed = _ptr(_need(weights["embed"], bf, (V, d), "embed"))
        w.final_norm = _ptr(_need(weights["final_norm"], bf, (d,), "final_norm"))
        w.lm_head = _ptr(_need(weights["lm_head"], bf, (V, d), "lm_head"))
        a = shape.n_q_heads * shape.head_dim
        shapes = {"attn_norm": (d,), "W_qkv": (shape.qkv_rows, 2 * d), "W_o": (d, a), "ffn_norm": (d,),
                  "W_gate": (shape.ffn_dim, d), "W_up": (shape.ffn_dim, d), "W_down": (d, shape.ffn_dim)}
        for name, shp in shapes.items():
            arr = getattr(w, name)
            for l in range(shape.n_layers):
                arr[l] = _ptr(_need(weights[name][l], bf, shp, f"{name}[{l}]")).value
        self._cfg, self._w = cfg, w
        h = _vp()
        _check(_c_create(ctypes.byref(cfg), ctypes.byref(w), ctypes.byref(h)))
        self.handle = h

    def close(self):
        if self.handle:
            _c_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def osprey_create(shape: DrafterShape, weights: dict) -> Ctx:
    return Ctx(shape, weights)


def osprey_destroy(ctx: Ctx):
    ctx.close()


# ---------------------------------------------------------------------------- KV cache

@dataclass
class KvCache:
    k_pages: torch.Tensor      # [L, n_pages, Hkv, P, hd] bf16
    v_pages: torch.Tensor
    page_table: torch.Tensor   # [B, max_pages] int32
    seq_len: torch.Tensor      # [B] int32

    @property
    def max_pages(self) -> int:
        return self.page_table.shape[1]

    @property
    def n_pages(self) -> int:
        return self.k_pages.shape[1]

    def c_struct(self) -> osprey_kv:
        return osprey_kv(self.k_pages.data_ptr(), self.v_pages.data_ptr(), self.page_table.data_ptr(),
                         self.seq_len.data_ptr(), self.max_pages, self.n_pages)


def alloc_kv(shape: DrafterShape, page_table: np.ndarray, n_pages: int, device="cuda") -> KvCache:
    B = page_table.shape[0]
    pages = (shape.n_layers, n_pages, shape.n_kv_heads, shape.page_size, shape.head_dim)
    return KvCache(torch.zeros(pages, dtype=torch.bfloat16, device=device),
                   torch.zeros(pages, dtype=torch.bfloat16, device=device),
                   torch.from_numpy(np.ascontiguousarray(page_table, np.int32)).to(device),
                   torch.zeros(B, dtype=torch.int32, device=device))


def to_device_bf16(bits: np.ndarray, device="cuda") -> torch.Tensor:
    """bf16 bit patterns (uint16 numpy) -> a bf16 device tensor with the same bytes."""
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).to(device)


def upload_weights(w: dict, device="cuda") -> dict:
    out = {}
    for k, v in w.items():
        out[k] = [to_device_bf16(a, device) for a in v] if isinstance(v, list) else to_device_bf16(v, device)
    return out


# ---------------------------------------------------------------------------- calls

def osprey_draft_workspace_bytes(ctx: Ctx, B: int, K: int, max_new: int, max_pages: int) -> int:
    return int(_c_draft_ws(ctx.handle, B, K, max_new, max_pages))


def osprey_kv_append(ctx: Ctx, kv: KvCache, n_rows: torch.Tensor, k_rows: torch.Tensor, v_rows: torch.Tensor,
                     status: torch.Tensor, stream=None):
    B = kv.page_table.shape[0]
    _need(n_rows, torch.int32, (B,), "n_rows")
    s = ctx.shape
    total = k_rows.shape[1] if k_rows.dim() == 4 else 0
    _need(k_rows, torch.bfloat16, (s.n_layers, total, s.n_kv_heads, s.head_dim), "k_rows")
    _need(v_rows, torch.bfloat16, (s.n_layers, total, s.n_kv_heads, s.head_dim), "v_rows")
    _need(status, torch.int32, (1,), "status")
    kvs = kv.c_struct()
    _check(_c_kv_append(ctx.handle, ctypes.byref(kvs), B, _ptr(n_rows), total, _ptr(k_rows), _ptr(v_rows),
                        _ptr(status), _stream(stream)))


def osprey_draft_step(ctx: Ctx, kv: KvCache, n_new: torch.Tensor, tokens: torch.Tensor, feats: torch.Tensor,
                      temperature: float, u_draft, draft_tokens: torch.Tensor, draft_qx=None, draft_stats=None,
                      draft_logits=None, workspace: torch.Tensor = None, status: torch.Tensor = None, stream=None):
    s = ctx.shape
    B, max_new = tokens.shape
    K = draft_tokens.shape[1]
    _need(n_new, torch.int32, (B,), "n_new")
    _need(tokens, torch.int32, (B, max_new), "tokens")
    _need(feats, torch.bfloat16, (B, max_new, s.feat_dim), "feats")
    _need(draft_tokens, torch.int32, (B, K), "draft_tokens")
    if u_draft is not None:
        _need(u_draft, torch.float32, (B, K), "u_draft")
    if draft_qx is not None:
        _need(draft_qx, torch.float32, (B, K), "draft_qx")
    if draft_stats is not None:
        _need(draft_stats, torch.float32, (B, K, 2), "draft_stats")
    if draft_logits is not None:
        _need(draft_logits, torch.float32, (B, K, s.vocab), "draft_logits")
    _need(workspace, torch.uint8, None, "workspace")
    _need(status, torch.int32, (1,), "status")
    if kv.page_table.shape[0] != B:
        raise ValueError("page table rows must equal the batch")
    kvs = kv.c_struct()
    _check(_c_draft(ctx.handle, ctypes.byref(kvs), B, K, max_new, _ptr(n_new), _ptr(tokens), _ptr(feats),
                    float(temperature), _ptr(u_draft), _ptr(draft_tokens), _ptr(draft_qx), _ptr(draft_stats),
                    _ptr(draft_logits), _ptr(workspace), workspace.numel(), _ptr(status), _stream(stream)))


def osprey_draft_step_hidden(ctx: Ctx, kv: KvCache, n_new: torch.Tensor, tokens: torch.Tensor, feats: torch.Tensor,
                             temperature: float, u_draft, draft_tokens: torch.Tensor, draft_qx: torch.Tensor,
                             draft_stats: torch.Tensor, draft_hidden: torch.Tensor, workspace: torch.Tensor = None,
                             status: torch.Tensor = None, stream=None):
    """osprey_draft_step without draft logits, keeping the state behind every
    draft token in draft_hidden [B, K, d] float32 (for osprey_verify_hidden)."""
    s = ctx.shape
    B, max_new = tokens.shape
    K = draft_tokens.shape[1]
    _need(n_new, torch.int32, (B,), "n_new")
    _need(tokens, torch.int32, (B, max_new), "tokens")
    _need(feats, torch.bfloat16, (B, max_new, s.feat_dim), "feats")
    _need(draft_tokens, torch.int32, (B, K), "draft_tokens")
    if u_draft is not None:
        _need(u_draft, torch.float32, (B, K), "u_draft")
    if draft_qx is not None:
        _need(draft_qx, torch.float32, (B, K), "draft_qx")
    if draft_stats is not None:
        _need(draft_stats, torch.float32, (B, K, 2), "draft_stats")
    _need(draft_hidden, torch.float32, (B, K, s.d_model), "draft_hidden")
    _need(workspace, torch.uint8, None, "workspace")
    _need(status, torch.int32, (1,), "status")
    if kv.page_table.shape[0] != B:
        raise ValueError("page table rows must equal the batch")
    kvs = kv.c_struct()
    _check(_c_draft_hidden(ctx.handle, ctypes.byref(kvs), B, K, max_new, _ptr(n_new), _ptr(tokens), _ptr(feats),
                           float(temperature), _ptr(u_draft), _ptr(draft_tokens), _ptr(draft_qx), _ptr(draft_stats),
                           _ptr(draft_hidden), _ptr(workspace), workspace.numel(), _ptr(status), _stream(stream)))


def osprey_draft_step_topk(ctx: Ctx, kv: KvCache, n_new: torch.Tensor, tokens: torch.Tensor, feats: torch.Tensor,
                           temperature: float, u_draft, cand: torch.Tensor, cand_qx=None, draft_stats=None,
                           draft_logits=None, workspace: torch.Tensor = None, status: torch.Tensor = None, stream=None):
    """A draft call drawing topk candidates per chain step (cand [B, K, topk]);
    candidate 0 continues the chain."""
    s = ctx.shape
    B, max_new = tokens.shape
    K, k = cand.shape[1], cand.shape[2]
    _need(n_new, torch.int32, (B,), "n_new")
    _need(tokens, torch.int32, (B, max_new), "tokens")
    _need(feats, torch.bfloat16, (B, max_new, s.feat_dim), "feats")
    _need(cand, torch.int32, (B, K, k), "cand")
    if u_draft is not None:
        _need(u_draft, torch.float32, (B, K, k), "u_draft")
    if cand_qx is not None:
        _need(cand_qx, torch.float32, (B, K, k), "cand_qx")
    if draft_stats is not None:
        _need(draft_stats, torch.float32, (B, K, 2), "draft_stats")
    if draft_logits is not None:
        _need(draft_logits, torch.float32, (B, K, s.vocab), "draft_logits")
    _need(workspace, torch.uint8, None, "workspace")
    _need(status, torch.int32, (1,), "status")
    if kv.page_table.shape[0] != B:
        raise ValueError("page table rows must equal the batch")
    kvs = kv.c_struct()
    _check(_c_draft_topk(ctx.handle, ctypes.byref(kvs), B, K, k, max_new, _ptr(n_new), _ptr(tokens), _ptr(feats),
                         float(temperature), _ptr(u_draft), _ptr(cand), _ptr(cand_qx), _ptr(draft_stats),
                         _ptr(draft_logits), _ptr(workspace), workspace.numel(), _ptr(status), _stream(stream)))


def osprey_verify_tree(target_logits: torch.Tensor, draft_logits, cand: torch.Tensor, temperature: float, u_accept,
                       u_sample, out_tokens: torch.Tensor, n_accepted: torch.Tensor, branch: torch.Tensor,
                       flags: torch.Tensor, status: torch.Tensor, stream=None):
    """Verify a branching-chain draft tree: target [B, 1 + K*topk, V], draft
    [B, K, V] (None when greedy), cand [B, K, topk]."""
    B, K, k = cand.shape
    V = target_logits.shape[-1]
    dt = {torch.float32: OSPREY_F32, torch.bfloat16: OSPREY_BF16}.get(target_logits.dtype)
    if dt is None:
        raise ValueError("logits must be float32 or bfloat16")
    _need(target_logits, target_logits.dtype, (B, 1 + K * k, V), "target_logits")
    if draft_logits is not None:
        _need(draft_logits, target_logits.dtype, (B, K, V), "draft_logits")
    _need(cand, torch.int32, (B, K, k), "cand")
    if temperature > 0:
        _need(u_accept, torch.float32, (B, K, k), "u_accept")
        _need(u_sample, torch.float32, (B, K + 1), "u_sample")
    _need(out_tokens, torch.int32, (B, K + 1), "out_tokens")
    _need(n_accepted, torch.int32, (B,), "n_accepted")
    _need(branch, torch.int32, (B,), "branch")
    _need(flags, torch.uint8, (B, K + 1), "flags")
    _need(status, torch.int32, (1,), "status")
    _check(_c_verify_tree(B, K, k, V, dt, _ptr(target_logits), _ptr(draft_logits), _ptr(cand), float(temperature),
                          _ptr(u_accept), _ptr(u_sample), _ptr(out_tokens), _ptr(n_accepted), _ptr(branch),
                          _ptr(flags), _ptr(status), _stream(stream)))


def osprey_dflash_workspace_bytes(ctx: Ctx, B: int, block: int, max_pages: int) -> int:
    return int(_c_dflash_ws(ctx.handle, B, block, max_pages))


def osprey_dflash_step(ctx: Ctx, kv: KvCache, anchors: torch.Tensor, mask_token: int, feats: torch.Tensor,
                       temperature: float, u_draft, draft_tokens: torch.Tensor, draft_qx=None, draft_stats=None,
                       draft_logits=None, workspace: torch.Tensor = None, status: torch.Tensor = None, stream=None):
    """Block drafting (EAGLE-style DFlash): one forward over anchor + block-1
    mask positions per sequence; draft_tokens [B, block-1] are its proposals."""
    s = ctx.shape
    B = anchors.shape[0]
    P = draft_tokens.shape[1]
    _need(anchors, torch.int32, (B,), "anchors")
    _need(feats, torch.bfloat16, (B, s.feat_dim), "feats")
    _need(draft_tokens, torch.int32, (B, P), "draft_tokens")
    if u_draft is not None:
        _need(u_draft, torch.float32, (B, P), "u_draft")
    if draft_qx is not None:
        _need(draft_qx, torch.float32, (B, P), "draft_qx")
    if draft_stats is not None:
        _need(draft_stats, torch.float32, (B, P, 2), "draft_stats")
    if draft_logits is not None:
        _need(draft_logits, torch.float32, (B, P, s.vocab), "draft_logits")
    _need(workspace, torch.uint8, None, "workspace")
    _need(status, torch.int32, (1,), "status")
    if kv.page_table.shape[0] != B:
        raise ValueError("page table rows must equal the batch")
    kvs = kv.c_struct()
    _check(_c_dflash(ctx.handle, ctypes.byref(kvs), B, P + 1, _ptr(anchors), int(mask_token), _ptr(feats),
                     float(temperature), _ptr(u_draft), _ptr(draft_tokens), _ptr(draft_qx), _ptr(draft_stats),
                     _ptr(draft_logits), _ptr(workspace), workspace.numel(), _ptr(status), _stream(stream)))


def osprey_verify_hidden_workspace_bytes(ctx: Ctx, B: int, K: int) -> int:
    return int(_c_verify_hidden_ws(ctx.handle, B, K))


def osprey_verify_hidden(ctx: Ctx, target_logits: torch.Tensor, draft_hidden: torch.Tensor, draft_qx: torch.Tensor,
                         draft_stats: torch.Tensor, draft_tokens: torch.Tensor, temperature: float,
                         u_accept: torch.Tensor, u_sample: torch.Tensor, out_tokens: torch.Tensor,
                         n_accepted: torch.Tensor, flags: torch.Tensor, probs=None, workspace: torch.Tensor = None,
                         status: torch.Tensor = None, stream=None):
    """Sampled verification without draft logits: the decision row's draft
    logits are recomputed from draft_hidden by ctx's LM head."""
    B, K1, V = target_logits.shape
    K = K1 - 1
    dt = {torch.float32: OSPREY_F32, torch.bfloat16: OSPREY_BF16}.get(target_logits.dtype)
    if dt is None:
        raise TypeError("logits must be float32 or bfloat16")
    if V != ctx.shape.vocab:
        raise ValueError(f"target vocab {V} differs from the drafter's {ctx.shape.vocab}")
    _need(target_logits, target_logits.dtype, (B, K + 1, V), "target_logits")
    _need(draft_hidden, torch.float32, (B, K, ctx.shape.d_model), "draft_hidden")
    _need(draft_qx, torch.float32, (B, K), "draft_qx")
    _need(draft_stats, torch.float32, (B, K, 2), "draft_stats")
    _need(draft_tokens, torch.int32, (B, K), "draft_tokens")
    _need(u_accept, torch.float32, (B, K), "u_accept")
    _need(u_sample, torch.float32, (B, K + 1), "u_sample")
    _need(out_tokens, torch.int32, (B, K + 1), "out_tokens")
    _need(n_accepted, torch.int32, (B,), "n_accepted")
    _need(flags, torch.uint8, (B, K + 1), "flags")
    if probs is not None:
        _need(probs, torch.float32, (B, K, 2), "probs")
    _need(workspace, torch.uint8, None, "workspace")
    _need(status, torch.int32, (1,), "status")
    _check(_c_verify_hidden(ctx.handle, B, K, dt, _ptr(target_logits), _ptr(draft_hidden), _ptr(draft_qx),
                            _ptr(draft_stats), _ptr(draft_tokens), float(temperature), _ptr(u_accept),
                            _ptr(u_sample), _ptr(out_tokens), _ptr(n_accepted), _ptr(flags), _ptr(probs),
                            _ptr(workspace), workspace.numel(), _ptr(status), _stream(stream)))


def osprey_verify_workspace_bytes(B: int, K: int, V: int) -> int:
    return int(_c_verify_ws(B, K, V))


def osprey_verify(target_logits: torch.Tensor, draft_logits, draft_tokens: torch.Tensor, temperature: float,
                  u_accept, u_sample, out_tokens: torch.Tensor, n_accepted: torch.Tensor, flags: torch.Tensor,
                  probs=None, workspace: torch.Tensor = None, status: torch.Tensor = None, stream=None):
    B, K1, V = target_logits.shape
    K = K1 - 1
    dt = {torch.float32: OSPREY_F32, torch.bfloat16: OSPREY_BF16}.get(target_logits.dtype)
    if dt is None:
        raise TypeError("logits must be float32 or bfloat16")
    _need(target_logits, target_logits.dtype, (B, K + 1, V), "target_logits")
    if draft_logits is not None:
        _need(draft_logits, target_logits.dtype, (B, K, V), "draft_logits")
    _need(draft_tokens, torch.int32, (B, K), "draft_tokens")
    if u_accept is not None:
        _need(u_accept, torch.float32, (B, K), "u_accept")
    if u_sample is not None:
        _need(u_sample, torch.float32, (B, K + 1), "u_sample")
    _need(out_tokens, torch.int32, (B, K + 1), "out_tokens")
    _need(n_accepted, torch.int32, (B,), "n_accepted")
    _need(flags, torch.uint8, (B, K + 1), "flags")
    if probs is not None:
        _need(probs, torch.float32, (B, K, 2), "probs")
    _need(workspace, torch.uint8, None, "workspace")
    _need(status, torch.int32, (1,), "status")
    _check(_c_verify(B, K, V, dt, _ptr(target_logits), _ptr(draft_logits), _ptr(draft_tokens), float(temperature),
                     _ptr(u_accept), _ptr(u_sample), _ptr(out_tokens), _ptr(n_accepted), _ptr(flags), _ptr(probs),
                     _ptr(workspace), workspace.numel(), _ptr(status), _stream(stream)))


VERIFY_STATIC_SCRATCH_BYTES = 4 << 20


def osprey_verify_static(target_logits: torch.Tensor, draft_logits, draft_tokens: torch.Tensor, temperature: float,
                         u_accept, u_sample, out_tokens: torch.Tensor, n_accepted: torch.Tensor, flags: torch.Tensor,
                         probs=None, status: torch.Tensor = None, stream=None):
    """osprey_verify without a workspace argument, for callers that cannot
    allocate device memory: the library's own static scratch array is used
    (calls that can overlap on the GPU must be serialised by the caller)."""
    B, K1, V = target_logits.shape
    K = K1 - 1
    dt = {torch.float32: OSPREY_F32, torch.bfloat16: OSPREY_BF16}.get(target_logits.dtype)
    if dt is None:
        raise TypeError("logits must be float32 or bfloat16")
    _need(target_logits, target_logits.dtype, (B, K + 1, V), "target_logits")
    if draft_logits is not None:
        _need(draft_logits, target_logits.dtype, (B, K, V), "draft_logits")
    _need(draft_tokens, torch.int32, (B, K), "draft_tokens")
    _need(out_tokens, torch.int32, (B, K + 1), "out_tokens")
    _need(n_accepted, torch.int32, (B,), "n_accepted")
    _need(flags, torch.uint8, (B, K + 1), "flags")
    if probs is not None:
        _need(probs, torch.float32, (B, K, 2), "probs")
    _need(status, torch.int32, (1,), "status")
    _check(_c_verify_static(B, K, V, dt, _ptr(target_logits), _ptr(draft_logits), _ptr(draft_tokens),
                            float(temperature), _ptr(u_accept), _ptr(u_sample), _ptr(out_tokens), _ptr(n_accepted),
                            _ptr(flags), _ptr(probs), _ptr(status), _stream(stream)))


def osprey_probe_enable(ctx: Ctx, n_slots: int):
    _check(_c_probe_enable(ctx.handle, n_slots))


PROBE_LM_HEAD, PROBE_ATTENTION = 0, 1


def osprey_probe_select(ctx: Ctx, kind: int):
    _check(_c_probe_select(ctx.handle, kind))


def osprey_probe_read(ctx: Ctx, n: int) -> list:
    buf = (_f32 * n)()
    _check(_c_probe_read(ctx.handle, buf, n))
    return list(buf)


def osprey_launch_count() -> int:
    return int(_c_launch_count())


def osprey_selftest_wait_timeout(limit_cycles: int, status: torch.Tensor, stream=None):
    """Run the bounded-wait failure path once: status reads OSPREY_ERR_TIMEOUT afterwards."""
    _need(status, torch.int32, (1,), "status")
    _check(_c_selftest_wait(int(limit_cycles), _ptr(status), _stream(stream)))
