"""Drafter shapes and speculative-decoding workloads.

Each workload names a drafter shape (an Osprey-style drafter: a shallow
transformer whose QKV projection is widened to take the projected target
feature, Sec. 3.3 Eq. 1-3) and the serving axes of one measurement: batch,
chain length K (topk=1 chain drafting, Sec. 4 "Inference settings"), context
lengths and temperature (Appendix, serving-sensitivity table).

The shapes follow the targets the paper evaluates: a Qwen3-8B-shaped target
(hidden 4096), a Llama-3.3-70B-shaped target (hidden 8192) and a large-vocabulary
verify-heavy case; the drafter widths follow the draft-size table (Appendix,
"Draft Model Sizes").
"""
from __future__ import annotations

from dataclasses import dataclass, field, replace


@dataclass(frozen=True)
class DrafterShape:
    d_model: int          # drafter hidden width d
    n_layers: int         # transformer blocks kept after pruning (Sec. 3.2, N in 1..4)
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    ffn_dim: int          # SwiGLU inner width
    vocab: int            # target vocabulary after alignment (Sec. 3.3)
    feat_dim: int         # 3 x target hidden (low/mid/high tap, Eq. 1)
    rope_theta: float
    rms_eps: float = 1e-6
    page_size: int = 16

    @property
    def qkv_rows(self) -> int:
        return (self.n_q_heads + 2 * self.n_kv_heads) * self.head_dim

    @property
    def group(self) -> int:
        return self.n_q_heads // self.n_kv_heads

    def layer_params(self) -> int:
        d, a = self.d_model, self.n_q_heads * self.head_dim
        return self.qkv_rows * 2 * d + d * a + 3 * self.ffn_dim * d + 2 * d

    def weight_bytes_per_step(self) -> int:
        """bf16 bytes of every weight a chain step touches (all layers + LM head)."""
        return 2 * (self.n_layers * self.layer_params() + self.vocab * self.d_model + self.d_model)


@dataclass(frozen=True)
class Workload:
    name: str
    shape: DrafterShape
    batch: int
    K: int                      # draft chain length
    ctx_lo: int                 # committed context, uniform in [ctx_lo, ctx_hi]
    ctx_hi: int
    temperature: float          # 0 means greedy
    sigma_p: float              # target logits = draft logits + N(0, sigma_p^2)
    logits_dtype: str = "f32"   # "f32" or "bf16" target/draft logits for verify
    seed: int = 1000
    n_new: int = 1              # extend rows per sequence in one draft call
    extra: dict = field(default_factory=dict, compare=False)

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)


TINY = DrafterShape(d_model=256, n_layers=1, n_q_heads=4, n_kv_heads=2, head_dim=64,
                    ffn_dim=768, vocab=4096, feat_dim=3 * 512, rope_theta=1e6)
QWEN3_8B_DRAFTER = DrafterShape(d_model=1024, n_layers=1, n_q_heads=16, n_kv_heads=8,
                                head_dim=128, ffn_dim=3072, vocab=151936,
                                feat_dim=3 * 4096, rope_theta=1e6)
LLAMA70B_DRAFTER = DrafterShape(d_model=2048, n_layers=2, n_q_heads=16, n_kv_heads=4,
                                head_dim=128, ffn_dim=6144, vocab=128256,
                                feat_dim=3 * 8192, rope_theta=5e5)
LARGE_VOCAB_DRAFTER = DrafterShape(d_model=1024, n_layers=1, n_q_heads=16, n_kv_heads=8,
                                   head_dim=128, ffn_dim=3072, vocab=200064,
                                   feat_dim=3 * 3072, rope_theta=1e6)

# The paper's own drafter body (Sec. 3.2; Appendix "Draft Model Sizes"): two
# Qwen3-4B-shaped blocks, d 2560, 32/8 heads of 128, FFN 9728, on a
# Qwen3-8B-shaped target (3 x 4096 feature columns, vocabulary 151936).
OSPREY_PAPER_DRAFTER = DrafterShape(d_model=2560, n_layers=2, n_q_heads=32, n_kv_heads=8,
                                    head_dim=128, ffn_dim=9728, vocab=151936,
                                    feat_dim=3 * 4096, rope_theta=1e6)

# The appendix's DFlash drafter (Appendix, "Cross-Domain Warm-Start Ablation
# under DFlash"): a four-layer LayerSkip-Llama-8B-shaped body (d 4096, 32/8
# heads of 128, FFN 14336, rotary base 5e5) with its LM head row-mapped to the
# Qwen3-8B target vocabulary and the EAGLE-style target interface (the target
# feature 3 x 4096 projected to d and fed through the expanded QKV).
DFLASH_DRAFTER = DrafterShape(d_model=4096, n_layers=4, n_q_heads=32, n_kv_heads=8, head_dim=128,
                              ffn_dim=14336, vocab=151936, feat_dim=3 * 4096, rope_theta=5e5)

WORKLOADS = {
    # tiny correctness case: fits the oracle in well under a second
    "tiny-d256-v4096-b1-k4": Workload("tiny-d256-v4096-b1-k4", TINY, batch=1, K=4,
                                      ctx_lo=128, ctx_hi=128, temperature=1.0,
                                      sigma_p=0.7, seed=1000),
    # Qwen3-8B-shaped target, one stream: HBM-bound GEMV regime (LM head dominates)
    "qwen3-8b-d1024-v151936-b1-k7": Workload("qwen3-8b-d1024-v151936-b1-k7", QWEN3_8B_DRAFTER,
                                             batch=1, K=7, ctx_lo=2048, ctx_hi=2048,
                                             temperature=1.0, sigma_p=0.7, seed=1001),
    # same drafter, batch 32, ragged paged contexts
    "qwen3-8b-d1024-v151936-b32-k7": Workload("qwen3-8b-d1024-v151936-b32-k7", QWEN3_8B_DRAFTER,
                                              batch=32, K=7, ctx_lo=1024, ctx_hi=4096,
                                              temperature=1.0, sigma_p=0.7, seed=1002),
    # Llama-3.3-70B-shaped target, 2-layer drafter
    "llama70b-d2048-v128256-b16-k7": Workload("llama70b-d2048-v128256-b16-k7", LLAMA70B_DRAFTER,
                                              batch=16, K=7, ctx_lo=2048, ctx_hi=8192,
                                              temperature=0.7, sigma_p=0.5, seed=1003),
    # the paper-shaped drafter, one stream; each call extends by 3 accepted rows
    # (an acceptance length of about 3) before its 7-token chain
    "osprey-d2560-v151936-b1-k7-ext3": Workload("osprey-d2560-v151936-b1-k7-ext3", OSPREY_PAPER_DRAFTER,
                                                batch=1, K=7, ctx_lo=2048, ctx_hi=2048, temperature=1.0,
                                                sigma_p=0.7, seed=1005, n_new=3),
    # block drafting, one stream: one forward over anchor + 15 mask positions
    # (block size 16, the appendix's setting) proposes K = 15 tokens
    "dflash-d4096-l4-v151936-b1-blk16": Workload("dflash-d4096-l4-v151936-b1-blk16", DFLASH_DRAFTER,
                                                 batch=1, K=15, ctx_lo=2048, ctx_hi=2048, temperature=1.0,
                                                 sigma_p=0.7, seed=1006, extra={"block": 16}),
    # tree drafting: K = 5 chain steps (the paper's serving steps) with topk = 4
    # candidates each, batch 8, verified as a branching chain
    "qwen3-8b-d1024-v151936-b8-k5-topk4": Workload("qwen3-8b-d1024-v151936-b8-k5-topk4", QWEN3_8B_DRAFTER,
                                                   batch=8, K=5, ctx_lo=1024, ctx_hi=4096, temperature=1.0,
                                                   sigma_p=0.7, seed=1007, extra={"topk": 4}),
    # large vocabulary, verify-heavy
    "large-vocab-d1024-v200064-b64-k8": Workload("large-vocab-d1024-v200064-b64-k8",
                                                 LARGE_VOCAB_DRAFTER, batch=64, K=8,
                                                 ctx_lo=1024, ctx_hi=16384, temperature=1.0,
                                                 sigma_p=0.7, seed=1004),
}

BENCH_WORKLOAD = "large-vocab-d1024-v200064-b64-k8"
