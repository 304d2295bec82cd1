"""Device-side state for one drafter: weights, paged KV cache, workspaces.

Plumbing only (allocation and uploads with torch); every computation is a
call into libosprey.so through ``binding``.
"""
from __future__ import annotations

import numpy as np
import torch

from . import binding as ob
from .workloads import DrafterShape


class DraftSession:
    def __init__(self, shape: DrafterShape, weights_np: dict, page_table: np.ndarray, n_pages: int,
                 K: int, max_new: int = 1, device: str = "cuda"):
        self.shape, self.K, self.max_new, self.device = shape, K, max_new, device
        self.weights = ob.upload_weights(weights_np, device)
        self.ctx = ob.osprey_create(shape, self.weights)
        self.kv = ob.alloc_kv(shape, page_table, n_pages, device)
        self.B = page_table.shape[0]
        nbytes = ob.osprey_draft_workspace_bytes(self.ctx, self.B, K, max_new, self.kv.max_pages)
        self.workspace = torch.zeros(nbytes, dtype=torch.uint8, device=device)
        self.status = torch.zeros(1, dtype=torch.int32, device=device)

    def append(self, n_rows: np.ndarray, k_rows: np.ndarray, v_rows: np.ndarray):
        """Fill the cache: rows [L, sum(n_rows), Hkv, hd] as bf16 bit patterns."""
        ob.osprey_kv_append(self.ctx, self.kv, torch.from_numpy(np.asarray(n_rows, np.int32)).to(self.device),
                            ob.to_device_bf16(k_rows, self.device), ob.to_device_bf16(v_rows, self.device),
                            self.status)

    def draft_buffers(self, with_logits: bool = False) -> dict:
        B, K, dev = self.B, self.K, self.device
        return {
            "draft_tokens": torch.full((B, K), -7, dtype=torch.int32, device=dev),
            "draft_qx": torch.zeros((B, K), dtype=torch.float32, device=dev),
            "draft_stats": torch.zeros((B, K, 2), dtype=torch.float32, device=dev),
            "draft_logits": torch.zeros((B, K, self.shape.vocab), dtype=torch.float32, device=dev)
            if with_logits else None,
        }

    def draft(self, n_new, tokens, feats, temperature: float, u_draft, out: dict, stream=None):
        ob.osprey_draft_step(self.ctx, self.kv, n_new, tokens, feats, temperature, u_draft, out["draft_tokens"],
                             out["draft_qx"], out["draft_stats"], out["draft_logits"], self.workspace,
                             self.status, stream)

    def tree_buffers(self, topk: int, with_logits: bool = False) -> dict:
        B, K, dev = self.B, self.K, self.device
        return {
            "cand": torch.full((B, K, topk), -7, dtype=torch.int32, device=dev),
            "cand_qx": torch.zeros((B, K, topk), dtype=torch.float32, device=dev),
            "draft_stats": torch.zeros((B, K, 2), dtype=torch.float32, device=dev),
            "draft_logits": torch.zeros((B, K, self.shape.vocab), dtype=torch.float32, device=dev)
            if with_logits else None,
        }

    def draft_tree(self, n_new, tokens, feats, temperature: float, u_draft, out: dict, stream=None):
        """The draft call with topk candidates per chain step (out from tree_buffers)."""
        ob.osprey_draft_step_topk(self.ctx, self.kv, n_new, tokens, feats, temperature, u_draft, out["cand"],
                                  out["cand_qx"], out["draft_stats"], out["draft_logits"], self.workspace,
                                  self.status, stream)

    def draft_hidden(self, n_new, tokens, feats, temperature: float, u_draft, out: dict, hidden, stream=None):
        """The draft call without logits, keeping each draft token's state in hidden [B, K, d]."""
        ob.osprey_draft_step_hidden(self.ctx, self.kv, n_new, tokens, feats, temperature, u_draft,
                                    out["draft_tokens"], out["draft_qx"], out["draft_stats"], hidden, self.workspace,
                                    self.status, stream)


class DflashSession(DraftSession):
    """A drafter that proposes blocks (EAGLE-style DFlash): each call is one
    forward over the anchor and block - 1 mask positions of every sequence."""

    def __init__(self, shape: DrafterShape, weights_np: dict, page_table: np.ndarray, n_pages: int, block: int,
                 device: str = "cuda"):
        super().__init__(shape, weights_np, page_table, n_pages, block - 1, block - 1, device)
        self.block = block
        nbytes = ob.osprey_dflash_workspace_bytes(self.ctx, self.B, block, self.kv.max_pages)
        self.workspace = torch.zeros(nbytes, dtype=torch.uint8, device=device)

    def block_buffers(self, with_logits: bool = False) -> dict:
        return self.draft_buffers(with_logits)

    def propose(self, anchors, mask_token: int, feats, temperature: float, u_draft, out: dict, stream=None):
        ob.osprey_dflash_step(self.ctx, self.kv, anchors, mask_token, feats, temperature, u_draft,
                              out["draft_tokens"], out["draft_qx"], out["draft_stats"], out["draft_logits"],
                              self.workspace, self.status, stream)


class VerifyBuffers:
    def __init__(self, B: int, K: int, V: int, device: str = "cuda", workspace_bytes: int | None = None):
        self.out_tokens = torch.zeros((B, K + 1), dtype=torch.int32, device=device)
        self.n_accepted = torch.zeros(B, dtype=torch.int32, device=device)
        self.flags = torch.zeros((B, K + 1), dtype=torch.uint8, device=device)
        self.probs = torch.zeros((B, K, 2), dtype=torch.float32, device=device)
        if workspace_bytes is None:
            workspace_bytes = ob.osprey_verify_workspace_bytes(B, K, V)
        self.workspace = torch.zeros(workspace_bytes, dtype=torch.uint8, device=device)
        self.status = torch.zeros(1, dtype=torch.int32, device=device)

    def run(self, target, draft, tokens, temperature, u_accept, u_sample, stream=None):
        ob.osprey_verify(target, draft, tokens, temperature, u_accept, u_sample, self.out_tokens,
                         self.n_accepted, self.flags, self.probs, self.workspace, self.status, stream)


class TreeVerifyBuffers:
    """Outputs of osprey_verify_tree for B sequences of depth K (no workspace)."""

    def __init__(self, B: int, K: int, device: str = "cuda"):
        self.out_tokens = torch.zeros((B, K + 1), dtype=torch.int32, device=device)
        self.n_accepted = torch.zeros(B, dtype=torch.int32, device=device)
        self.branch = torch.zeros(B, dtype=torch.int32, device=device)
        self.flags = torch.zeros((B, K + 1), dtype=torch.uint8, device=device)
        self.status = torch.zeros(1, dtype=torch.int32, device=device)

    def run(self, target, draft, cand, temperature, u_accept, u_sample, stream=None):
        ob.osprey_verify_tree(target, draft, cand, temperature, u_accept, u_sample, self.out_tokens,
                              self.n_accepted, self.branch, self.flags, self.status, stream)


class VerifyHiddenBuffers(VerifyBuffers):
    """Outputs and workspace of the logits-free verify for one drafter context."""

    def __init__(self, ctx: "ob.Ctx", B: int, K: int, device: str = "cuda"):
        super().__init__(B, K, ctx.shape.vocab, device, ob.osprey_verify_hidden_workspace_bytes(ctx, B, K))
        self.ctx = ctx

    def run_hidden(self, target, hidden, qx, stats, tokens, temperature, u_accept, u_sample, stream=None):
        ob.osprey_verify_hidden(self.ctx, target, hidden, qx, stats, tokens, temperature, u_accept, u_sample,
                                self.out_tokens, self.n_accepted, self.flags, self.probs, self.workspace,
                                self.status, stream)
