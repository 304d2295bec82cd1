"""Benchmark: draft+verify steps/s of the speculative-decoding hot path on GB300.

One step = one osprey_draft_step (extend row + a K-token chain through the
drafter, LM head sampled on chip) + one osprey_verify over the workload's
synthetic target/draft logits, captured in one CUDA graph.  Inputs are seeded
synthetic data shaped like the workload (weights bf16 ~ N(0, 0.02^2)).

Default workload: the large-vocabulary drafter (d=1024, 1 layer, 16/8 heads of
128, FFN 3072, vocab 200064, 3 x 3072 feature columns), batch 64, K=8, ragged
paged contexts U[1024, 16384], temperature 1, float32 logits: the largest
single-GPU workload.  The other workloads are measured after it under
"other_workloads" (--no-extra skips them).

Prints ONE JSON line (rank 0).  ``--impl reference`` times the CPU oracle on
the same workload instead (a deliberately slow float64 program), on a bounded
sample of sequences per step.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2609_09338_gb300 import synthetic as syn  # noqa: E402
from paper_2609_09338_gb300.workloads import BENCH_WORKLOAD, WORKLOADS  # noqa: E402

# dram__bytes_read.sum + dram__bytes_write.sum of one streamed LM-head launch
# at batch 1 (qwen3-8b-d1024-v151936-b1-k7: the first LM head of a bench run,
# ncu --set full); valid only for the stream.cu it was taken on.
LM_TRAFFIC = {"source": "paper_2609_09338_gb300/csrc/stream.cu",
              "sha256": "52f460bbc3c87bb8a826df02e23cb78a1374cbd91b4bcbe4cc2ebfcecdf7d6bd",
              "bytes_per_launch": 311_286_528 + 2_934_016}
# DRAM bytes (read + write) of one attention launch at the large-vocabulary
# workload, from one ncu capture of this source (profiles/attn_large-vocab-*.md)
ATTN_TRAFFIC = {"source": "paper_2609_09338_gb300/csrc/draft.cu",
                "sha256": "945657d709f2eaf25536b42ea209467dc8ded111749c3da39e67f610b277bde6",
                "workload": "large-vocab-d1024-v200064-b64-k8",
                "bytes_per_launch": 2_162_905_856 + 16_101_376}


def _sha(path):
    with open(path, "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=200)
    p.add_argument("--warmup", type=int, default=10)
    p.add_argument("--impl", default="osprey", choices=["osprey", "reference"])
    p.add_argument("--workload", default=BENCH_WORKLOAD, choices=sorted(WORKLOADS))
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--temperature", type=float, default=None, help="override the workload's temperature")
    p.add_argument("--verify-sweep", action="store_true",
                   help="time verify alone over batch x K at V=200064 (fp32 and bf16 logits)")
    p.add_argument("--weights", default=None,
                   help="drafter weight file: read it if it exists (it must hold the workload's shape), "
                        "else write the seeded weights there")
    p.add_argument("--verify-hidden", action="store_true",
                   help="compare draft (logits written) + verify against draft (states kept) + logits-free verify")
    p.add_argument("--no-extra", action="store_true", help="measure the headline workload only")
    p.add_argument("--sweep", default=None,
                   help="verify sweep points as dtype:B:K[,dtype:B:K...] (default: all of f32/bf16 x B x K)")
    return p.parse_args()


# measured after the headline workload, each with its own dominant kernel
EXTRA_WORKLOADS = ["qwen3-8b-d1024-v151936-b1-k7", "qwen3-8b-d1024-v151936-b32-k7",
                   "llama70b-d2048-v128256-b16-k7", "osprey-d2560-v151936-b1-k7-ext3",
                   "dflash-d4096-l4-v151936-b1-blk16", "qwen3-8b-d1024-v151936-b8-k5-topk4"]


def make_inputs(wl, rank=0, weights_path=None):
    sh = wl.shape
    seed = wl.seed + 1000 * rank
    ctx = syn.make_contexts(wl, seed + 17)
    if weights_path and os.path.exists(weights_path):
        from paper_2609_09338_gb300 import checkpoint
        _, w = checkpoint.load_weights(weights_path, sh)
    else:
        w = syn.make_weights(sh, seed)
        if weights_path and rank == 0:
            from paper_2609_09338_gb300 import checkpoint
            checkpoint.save_weights(weights_path, sh, w)
    kv = syn.make_kv_prefix(sh, ctx, wl.extra.get("block", wl.n_new + wl.K), seed + 1)
    di = syn.make_draft_inputs(sh, wl.batch, wl.n_new, wl.K, seed + 2)
    topk = wl.extra.get("topk", 1)
    if topk > 1:
        vi = syn.make_tree_inputs(sh.vocab, wl.batch, wl.K, topk, wl.temperature, wl.sigma_p, seed + 3)
        di["u_draft"] = np.random.default_rng(seed + 4).random((wl.batch, wl.K, topk), dtype=np.float32)
    else:
        vi = syn.make_verify_inputs(sh.vocab, wl.batch, wl.K, wl.temperature, wl.sigma_p, seed + 3)
    return ctx, w, kv, di, vi


def algorithmic_bytes(wl, ctx):
    """Bytes the method must touch per step (no L2 reuse credited).

    attn_call: the K/V bytes of every attention launch of one draft call (chain
    step k of sequence b reads its ctx_b + n_new + k cached positions, K and V,
    bf16, for each of the L layers), over the K * L launches of the call."""
    sh = wl.shape
    B, K = wl.batch, wl.K
    w_step = sh.weight_bytes_per_step()
    kv_row = 2 * sh.n_layers * sh.n_kv_heads * sh.head_dim * 2           # K and V, bf16, all layers
    if wl.extra.get("block"):
        # block drafting: one forward over the block (weights once), every
        # sequence's cached positions read once, its block rows written
        blk = wl.extra["block"]
        kv = sum(kv_row * (int(c) + blk - 1) for c in ctx)
        draft = w_step + 2 * sh.d_model * sh.feat_dim + kv + B * sh.feat_dim * 2
        s = 4 if wl.logits_dtype == "f32" else 2
        return {"draft": draft, "verify": B * (2 * K + 1) * sh.vocab * s,
                "lm_head_launch": sh.vocab * sh.d_model * 2 + 2 * sh.d_model, "attn_call": kv,
                "attn_launches": sh.n_layers, "lm_launches": 1,
                "verify_f32": B * (2 * K + 1) * sh.vocab * 4, "verify_bf16": B * (2 * K + 1) * sh.vocab * 2}
    # chain step k attends over ctx + n_new + k positions (extend row: ctx + 1 with n_new = 1)
    kv = sum(kv_row * (int(c) + wl.n_new + k) for c in ctx for k in range(K))
    draft = K * w_step + 2 * sh.d_model * sh.feat_dim + kv + B * wl.n_new * sh.feat_dim * 2
    s = 4 if wl.logits_dtype == "f32" else 2
    # chain: every target and draft row once; tree: the rows of one root-to-leaf path
    # (K + 1 target rows and K draft rows), what a walk that accepts the chain reads
    verify = B * (K + 1) * sh.vocab * s + B * K * sh.vocab * s
    lm_launch = sh.vocab * sh.d_model * 2 * 1 + 2 * sh.d_model
    return {"draft": draft, "verify": verify, "lm_head_launch": lm_launch, "attn_call": kv,
            "attn_launches": K * sh.n_layers, "lm_launches": K,
            "verify_f32": B * (2 * K + 1) * sh.vocab * 4, "verify_bf16": B * (2 * K + 1) * sh.vocab * 2}


def dominant_kernel(nb):
    """The kernel class with the most algorithmic bytes per draft call."""
    return "attention" if nb["attn_call"] > nb["lm_head_launch"] * nb["lm_launches"] else "lm_head"


class ClockSampler:
    """nvidia-smi clocks and throttle reasons while the timed region runs."""
    Q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, index, path):
        self.index, self.path, self.proc = index, path, None

    def __enter__(self):
        try:
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "20"],
                                         stdout=self.fh, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc:
            time.sleep(0.1)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.fh.close()

    def summary(self):
        rows = []
        try:
            with open(self.path) as f:
                for line in f:
                    parts = [x.strip() for x in line.split(",")]
                    if len(parts) == 7:
                        rows.append(parts)
        except OSError:
            pass
        num = lambda x: float(x) if x.replace(".", "", 1).isdigit() else None
        sm = [num(r[0]) for r in rows if num(r[0]) is not None]
        mx = [num(r[1]) for r in rows if num(r[1]) is not None]
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": len(rows)}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[3 + i].lower() == "active"})
        busy = sorted(sm)[len(sm) // 4:]          # drop the idle samples around the region
        return {"sm_mhz": statistics.median(busy), "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return 6800.0, "fallback"


def _blas():
    """numpy's OpenBLAS (get, set) thread-count functions, or None."""
    import ctypes
    np.ones((64, 64)) @ np.ones((64, 64))   # make sure the library is loaded
    try:
        with open("/proc/self/maps") as f:
            libs = sorted({ln.split()[-1] for ln in f if "openblas" in ln.lower() and ".so" in ln.split()[-1]})
    except OSError:
        return None
    for path in libs:
        try:
            lib = ctypes.CDLL(path)
        except OSError:
            continue
        for suffix in ("64_", "", "_64"):
            for pre in ("scipy_openblas", "openblas"):
                try:
                    get = getattr(lib, f"{pre}_get_num_threads{suffix}")
                    put = getattr(lib, f"{pre}_set_num_threads{suffix}")
                except AttributeError:
                    continue
                get.restype = ctypes.c_int
                put.argtypes = [ctypes.c_int]
                return get, put
    return None


def oracle_sequence_step(wl, ctx, w, W, kv, di, vi, b):
    """One sequence's share of a step, run by the oracle: its draft call (extend
    rows + K-token chain) and its verification.  Returns the seconds each took."""
    from oracle import drafter as od
    from oracle import verify as ov
    offs = np.concatenate([[0], np.cumsum(ctx)]).astype(np.int64)
    sl = slice(int(offs[b]), int(offs[b + 1]))
    t0 = time.perf_counter()
    od.draft_step(w, wl.shape, kv["k_rows"][:, sl], kv["v_rows"][:, sl], ctx[b:b + 1], di["tokens"][b:b + 1],
                  di["feats"][b:b + 1], di["n_new"][b:b + 1], wl.K, wl.temperature, di["u_draft"][b:b + 1],
                  widened=W)
    t1 = time.perf_counter()
    ov.verify(vi["target_logits"][b:b + 1], vi["draft_logits"][b:b + 1], vi["draft_tokens"][b:b + 1],
              wl.temperature, vi["u_accept"][b:b + 1], vi["u_sample"][b:b + 1])
    return t1 - t0, time.perf_counter() - t1


def cpu_baseline(wl, ctx, w, kv, di, vi, budget_s=8.0):
    """The oracle as it stands on the host cores, on a bounded sample: whole
    sequences of the workload (draft call + verify of one sequence), scaled to
    steps/s as 1 / (B x mean seconds per sequence).  Timed with numpy's BLAS at
    its own thread count and again at one thread."""
    from oracle import drafter as od
    t0 = time.perf_counter()
    W = od.widen_weights(w)
    setup = time.perf_counter() - t0
    blas = _blas()
    threads = blas[0]() if blas else None

    def sample(budget):
        n, t_run, phases = 0, 0.0, []
        while True:
            b = n % wl.batch
            t1 = time.perf_counter()
            phases.append(oracle_sequence_step(wl, ctx, w, W, kv, di, vi, b))
            t_run += time.perf_counter() - t1
            n += 1
            if t_run > budget or n >= 4 * wl.batch:
                return n, t_run, phases
    n, t_run, phases = sample(budget_s)
    res = {"value": n / t_run / wl.batch, "unit": "steps/s", "cores": threads, "kind": "oracle",
           "sample": f"{n} sequence(s) of {wl.name} (draft call K={wl.K} + verify each, float64 numpy), "
                     f"scaled to steps of {wl.batch} sequences; weights widened once ({setup:.1f}s, untimed); "
                     f"cores = numpy BLAS threads; {os.cpu_count()} host cores visible",
           # per sequence, over the sample: the draft call and the verification apart
           "draft_call_s_median": float(np.median([p[0] for p in phases])),
           "verify_s_median": float(np.median([p[1] for p in phases]))}
    if blas and threads and threads > 1:
        blas[1](1)
        try:
            n1, t1, phases1 = sample(budget_s / 2)
        finally:
            blas[1](threads)
        res["one_core"] = {"value": n1 / t1 / wl.batch, "cores": 1, "sample": f"{n1} sequence(s)",
                           "draft_call_s_median": float(np.median([p[0] for p in phases1])),
                           "verify_s_median": float(np.median([p[1] for p in phases1]))}
    return res


def max_over_ranks(x: float, world: int, device="cpu") -> float:
    """The job's time is its slowest replica's: MAX over the ranks (identity for one rank)."""
    if world <= 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    wl = WORKLOADS[args.workload]
    ctx, w, kv, di, vi = make_inputs(wl, 0, args.weights)
    from oracle import drafter as od
    W = od.widen_weights(w)
    blas = _blas()
    cores = blas[0]() if blas else None
    # one step of the reference arm is a bounded sample of the workload: up to
    # ``per`` of its sequences (draft call + verify each), scaled to whole steps
    per = max(1, min(wl.batch, 2))

    def step(i):
        for j in range(per):
            oracle_sequence_step(wl, ctx, w, W, kv, di, vi, (i * per + j) % wl.batch)
    for i in range(args.warmup):
        step(i)
    t0 = time.perf_counter()
    for i in range(args.steps):
        step(args.warmup + i)
    dt = time.perf_counter() - t0
    v = args.steps * per / wl.batch / dt
    sample = (f"each step: {per} of the {wl.batch} sequences of {wl.name} (draft call K={wl.K} + verify), "
              f"scaled to steps/s as sequences / {wl.batch}; float64 numpy; cores = numpy BLAS threads")
    print(json.dumps({
        "impl": "reference", "metric": "draft+verify steps/s", "value": v, "unit": "steps/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 / v, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": config_of(wl, ctx),
        "cpu_baseline": {"value": v, "unit": "steps/s", "cores": cores, "kind": "oracle", "sample": sample},
        "e2e": {"value": v, "unit": "steps/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }))


def nvtx_push(name):
    """An NVTX range for a profiler's timeline; nothing when this torch build has no NVTX."""
    try:
        import torch
        torch.cuda.nvtx.range_push(name)
    except (RuntimeError, AttributeError):
        pass


def nvtx_pop():
    try:
        import torch
        torch.cuda.nvtx.range_pop()
    except (RuntimeError, AttributeError):
        pass


def lm_head_label(B, block=False):
    """The LM-head launches the probes bracket, by the number of rows (the draft
    step's kernel selection)."""
    if block:
        return ("tc_kernel<LM> + lm_pick_kernel over every block row (tcgen05 LM head with per-32-id sampling "
                "partials in its epilogue, then the pick; the operand planes come from the last down projection)")
    if B <= 2:
        return "stream_kernel<LM> (final RMSNorm + TMA-streamed LM-head GEMV + on-chip sampling)"
    if B <= 80:
        return ("tc_kernel<LM> + lm_pick_kernel (tcgen05 LM head, two weight tiles per stage, per-32-id sampling "
                "partials in its epilogue, then the pick)")
    return "lm_head_kernel (CUDA-core LM head + on-chip sampling)"


def config_of(wl, ctx):
    sh = wl.shape
    return {"workload": wl.name, "batch": wl.batch, "K": wl.K, "ctx": [int(ctx.min()), int(ctx.max())],
            "vocab": sh.vocab, "d_model": sh.d_model, "layers": sh.n_layers,
            "heads": f"{sh.n_q_heads}/{sh.n_kv_heads}x{sh.head_dim}", "ffn": sh.ffn_dim,
            "temperature": wl.temperature, "logits": wl.logits_dtype, "weights": "bf16",
            "l2": "flushed before every timed step (256 MB write, then 256 MB read)", "parallelism": "replicas"}


def verify_sweep(args):
    """Verify alone: GB/s against the HBM roofline over batch x K (V = 200064)."""
    import torch
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_09338_gb300.session import VerifyBuffers
    torch.cuda.set_device(0)
    V, T = 200064, 1.0
    peak, peak_kind = peaks()
    flush_w = torch.empty(256 * 1024 * 1024 // 4, dtype=torch.float32, device="cuda")
    flush_r = torch.ones(256 * 1024 * 1024 // 4, dtype=torch.float32, device="cuda")
    gen = torch.Generator(device="cuda").manual_seed(1234)
    points = []
    grid = [(dt, B, K) for dt in ("f32", "bf16") for B in (1, 8, 64, 256) for K in (1, 4, 8)]
    if args.sweep:
        grid = [(p.split(":")[0], int(p.split(":")[1]), int(p.split(":")[2])) for p in args.sweep.split(",")]
    for dname, B, K in grid:
        dtype = torch.float32 if dname == "f32" else torch.bfloat16
        zp = torch.randn((B, K + 1, V), generator=gen, device="cuda").to(dtype)
        zq = torch.randn((B, K, V), generator=gen, device="cuda").to(dtype)
        x = torch.randint(0, V, (B, K), generator=gen, device="cuda", dtype=torch.int32)
        ua = torch.rand((B, K), generator=gen, device="cuda")
        us = torch.rand((B, K + 1), generator=gen, device="cuda")
        vb = VerifyBuffers(B, K, V)
        st = torch.cuda.Stream()
        st.wait_stream(torch.cuda.current_stream())   # inputs and zeroed workspace first
        with torch.cuda.stream(st):
            vb.run(zp, zq, x, T, ua, us)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()   # replayed, so host marshalling stays out of the timing
        with torch.cuda.graph(g, stream=st):
            vb.run(zp, zq, x, T, ua, us)
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(args.steps + 3)]
        with torch.cuda.stream(st):
            for s_, e_ in ev:
                flush_w.zero_()
                flush_r.sum()
                s_.record(st)
                g.replay()
                e_.record(st)
        torch.cuda.synchronize()
        assert int(vb.status.item()) == 0
        ev = ev[3:]
        us_ = 1e3 * sum(s_.elapsed_time(e_) for s_, e_ in ev) / len(ev)
        nbytes = (B * (K + 1) * V + B * K * V) * zp.element_size()
        gbs = nbytes / (us_ * 1e-6) / 1e9
        points.append({"dtype": "f32" if dtype == torch.float32 else "bf16", "B": B, "K": K,
                       "bytes": nbytes, "us": round(us_, 2), "GBps": round(gbs, 1),
                       "frac": round(gbs / peak, 3), "roofline_us": round(nbytes / peak / 1e3, 2)})
        del zp, zq
    print(json.dumps({"metric": "verify GB/s sweep", "peak": peak, "peak_kind": peak_kind, "V": V,
                      "temperature": T, "steps": args.steps, "l2": "flushed before every call",
                      "verify_sweep": points}))


def verify_hidden_compare(args):
    """One sampled draft+verify step two ways on the workload's drafter: the draft
    step writes its logits [B, K, V] and osprey_verify reads them, or the draft
    step keeps each token's state [B, K, d] and osprey_verify_hidden recomputes
    only the decision rows.  Target logits are the workload's synthetic rows."""
    import torch
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_09338_gb300 import binding as ob
    from paper_2609_09338_gb300.session import DraftSession, VerifyBuffers, VerifyHiddenBuffers
    torch.cuda.set_device(0)
    wl = WORKLOADS[args.workload]
    if args.temperature is not None:
        wl = wl.with_(temperature=args.temperature)
    if wl.temperature <= 0:
        raise SystemExit("--verify-hidden needs a sampled workload (temperature > 0)")
    sh, B, K, T = wl.shape, wl.batch, wl.K, wl.temperature
    ctx, w, kv, di, vi = make_inputs(wl, 0, args.weights)
    dev = "cuda"
    T_ = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
    target = T_(vi["target_logits"]) if wl.logits_dtype == "f32" else \
        ob.to_device_bf16(syn.bf16_bits(vi["target_logits"]))
    d_in = (T_(di["n_new"]), T_(di["tokens"]), ob.to_device_bf16(di["feats"]), T, T_(di["u_draft"]))
    u_acc, u_smp = T_(vi["u_accept"]), T_(vi["u_sample"])
    flush_w = torch.empty(256 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)
    flush_r = torch.ones(256 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)
    res = {}
    for mode in ("logits", "hidden"):
        sess = DraftSession(sh, w, kv["page_table"], kv["n_pages"], K, wl.n_new)
        sess.append(ctx, kv["k_rows"], kv["v_rows"])
        torch.cuda.synchronize()
        seq0 = sess.kv.seq_len.clone()
        out = sess.draft_buffers(with_logits=mode == "logits")
        hidden = torch.zeros((B, K, sh.d_model), dtype=torch.float32, device=dev)
        vb = VerifyBuffers(B, K, sh.vocab) if mode == "logits" else VerifyHiddenBuffers(sess.ctx, B, K)
        # osprey_verify reads both rows in one dtype and the draft step writes float32
        tgt = target if mode == "hidden" or wl.logits_dtype == "f32" else target.float()

        def step():
            sess.kv.seq_len.copy_(seq0)
            if mode == "logits":
                sess.draft(*d_in, out)
                vb.run(tgt, out["draft_logits"], out["draft_tokens"], T, u_acc, u_smp)
            else:
                sess.draft_hidden(*d_in, out, hidden)
                vb.run_hidden(tgt, hidden, out["draft_qx"], out["draft_stats"], out["draft_tokens"], T, u_acc,
                              u_smp)
        st = torch.cuda.Stream()
        st.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(st):
            step()
        torch.cuda.synchronize()
        assert int(sess.status.item()) == 0 and int(vb.status.item()) == 0
        g = torch.cuda.CUDAGraph()
        n0 = ob.osprey_launch_count()
        with torch.cuda.graph(g, stream=st):
            step()
        launches = ob.osprey_launch_count() - n0
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(args.steps + max(args.warmup, 3))]
        with torch.cuda.stream(st):
            for s_, e_ in ev:
                flush_w.zero_()
                flush_r.sum()
                s_.record(st)
                g.replay()
                e_.record(st)
        torch.cuda.synchronize()
        assert int(sess.status.item()) == 0 and int(vb.status.item()) == 0
        ev = ev[max(args.warmup, 3):]
        res[mode] = {"ms_per_step": sum(s_.elapsed_time(e_) for s_, e_ in ev) / len(ev),
                     "launches_per_step": launches,
                     "mean_accepted": float(vb.n_accepted.float().mean().item())}
        del sess, vb, g
        torch.cuda.empty_cache()
    s_ = 4 if wl.logits_dtype == "f32" else 2
    print(json.dumps({"metric": "draft+verify ms per step, draft logits vs kept states",
                      "workload": wl.name, "temperature": T, "logits": wl.logits_dtype, "steps": args.steps,
                      "l2": "flushed before every step", **res,
                      "draft_logits_bytes": B * K * sh.vocab * 4,
                      "decision_row_lm_bytes": -(-B // 80) * sh.vocab * sh.d_model * 2 + B * sh.vocab * s_}))


def measure(wl, args, rank, world, local, full):
    """Time `args.steps` draft+verify steps of one workload (graph replays, L2
    flushed before each).  With ``full``: also verify alone (float32 and bf16
    logits), the end-to-end form from pinned host memory, clocks and the CPU
    baseline."""
    import torch
    from paper_2609_09338_gb300 import binding as ob
    from paper_2609_09338_gb300.session import DraftSession, VerifyBuffers

    sh, B, K, T = wl.shape, wl.batch, wl.K, wl.temperature
    ctx, w, kv, di, vi = make_inputs(wl, rank, args.weights if full else None)
    nb = algorithmic_bytes(wl, ctx)
    dom = dominant_kernel(nb)
    dev = "cuda"
    blk = wl.extra.get("block")
    if blk:
        from paper_2609_09338_gb300.session import DflashSession
        sess = DflashSession(sh, w, kv["page_table"], kv["n_pages"], blk)
    else:
        sess = DraftSession(sh, w, kv["page_table"], kv["n_pages"], K, wl.n_new)
    sess.append(ctx, kv["k_rows"], kv["v_rows"])
    torch.cuda.synchronize()
    assert int(sess.status.item()) == 0
    seq0 = sess.kv.seq_len.clone()
    T_ = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
    d_in = {"n_new": T_(di["n_new"]), "tokens": T_(di["tokens"]), "feats": ob.to_device_bf16(di["feats"]),
            "u_draft": T_(di["u_draft"])}
    if wl.logits_dtype == "f32":
        v_in = {"target": T_(vi["target_logits"]), "draft": T_(vi["draft_logits"])}
    else:
        v_in = {"target": ob.to_device_bf16(syn.bf16_bits(vi["target_logits"])),
                "draft": ob.to_device_bf16(syn.bf16_bits(vi["draft_logits"]))}
    v_in.update({"tokens": T_(vi["cand"] if "cand" in vi else vi["draft_tokens"]), "u_accept": T_(vi["u_accept"]),
                 "u_sample": T_(vi["u_sample"])})
    topk = wl.extra.get("topk", 1)
    if topk > 1:
        from paper_2609_09338_gb300.session import TreeVerifyBuffers
        out = sess.tree_buffers(topk)
        vb = TreeVerifyBuffers(B, K)
    else:
        out = sess.draft_buffers()
        vb = VerifyBuffers(B, K, sh.vocab)
    n_probe = nb["attn_launches"] if dom == "attention" else nb["lm_launches"]
    ob.osprey_probe_select(sess.ctx, ob.PROBE_ATTENTION if dom == "attention" else ob.PROBE_LM_HEAD)
    ob.osprey_probe_enable(sess.ctx, n_probe)
    stream = torch.cuda.Stream()
    stream.wait_stream(torch.cuda.current_stream())   # inputs and buffers first

    if blk:   # the block's anchor and feature: the first extend row's token and feature
        d_in["anchors"] = d_in["tokens"][:, 0].contiguous()
        d_in["feats1"] = d_in["feats"][:, 0].contiguous()

    def step():
        sess.kv.seq_len.copy_(seq0)
        if blk:
            sess.propose(d_in["anchors"], 0, d_in["feats1"], T, d_in["u_draft"], out)
        elif topk > 1:
            sess.draft_tree(d_in["n_new"], d_in["tokens"], d_in["feats"], T, d_in["u_draft"], out)
        else:
            sess.draft(d_in["n_new"], d_in["tokens"], d_in["feats"], T, d_in["u_draft"], out)
        vb.run(v_in["target"], v_in["draft"] if T > 0 else None, v_in["tokens"], T, v_in["u_accept"],
               v_in["u_sample"])

    # eager warm-up, then capture one step in a graph
    with torch.cuda.stream(stream):
        step()
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    n0 = ob.osprey_launch_count()
    with torch.cuda.graph(graph, stream=stream):
        step()
    launches_per_step = ob.osprey_launch_count() - n0
    torch.cuda.synchronize()
    flush_w = torch.empty(256 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)
    flush_r = torch.ones(256 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)

    def flush():
        """Evict L2: write a 256 MB buffer, then read another so no dirty line is left."""
        flush_w.zero_()
        flush_r.sum()

    for _ in range(max(args.warmup, 3)):
        flush()
        graph.replay()
    torch.cuda.synchronize()
    assert int(sess.status.item()) == 0 and int(vb.status.item()) == 0

    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    probe_ms = []
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    torch.cuda.synchronize()
    clk_file = tempfile.NamedTemporaryFile(prefix=f"osprey_clocks_{rank}_", suffix=".csv", delete=False)
    clk_file.close()
    with ClockSampler(local, clk_file.name) as clk:
        with torch.cuda.stream(stream):
            for i in range(args.steps):
                flush()
                nvtx_push(f"step {i}")
                starts[i].record(stream)
                graph.replay()
                ends[i].record(stream)
                nvtx_pop()
                ends[i].synchronize()
                probe_ms.append(ob.osprey_probe_read(sess.ctx, n_probe))
        torch.cuda.synchronize()
    clocks = clk.summary()
    try:
        os.unlink(clk_file.name)
    except OSError:
        pass
    if world > 1:
        dist.barrier()
    assert int(sess.status.item()) == 0 and int(vb.status.item()) == 0
    step_ms = [s_.elapsed_time(e_) for s_, e_ in zip(starts, ends)]
    ms = max_over_ranks(sum(step_ms) / len(step_ms), world, dev)
    peak, peak_kind = peaks()
    acc = vb.n_accepted.float()
    if dom == "attention":
        # bytes of all the call's attention launches / their summed duration
        call_ms = sum(sum(p) for p in probe_ms) / len(probe_ms)
        achieved = nb["attn_call"] / (call_ms * 1e-3) / 1e9
        attn_sha = _sha(os.path.join(ROOT, ATTN_TRAFFIC["source"]))
        traffic = (ATTN_TRAFFIC["bytes_per_launch"]
                   if attn_sha == ATTN_TRAFFIC["sha256"] and wl.name == ATTN_TRAFFIC["workload"] else None)
        roof = {"kernel": "split-KV GQA decode attention (attn_kernel / attn_cluster_kernel), all launches of a call",
                "bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                "traffic": traffic, "peak_kind": peak_kind,
                "bytes_per_launch": nb["attn_call"] / nb["attn_launches"],
                "mean_launch_us": 1e3 * call_ms / nb["attn_launches"], "launches_timed": len(probe_ms) * n_probe}
    else:
        lm = [x for p in probe_ms for x in p]
        lm_mean_ms = sum(lm) / len(lm)
        achieved = nb["lm_head_launch"] / (lm_mean_ms * 1e-3) / 1e9
        sha = _sha(os.path.join(ROOT, LM_TRAFFIC["source"]))
        roof = {"kernel": lm_head_label(B, bool(blk)), "bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                "frac": achieved / peak,
                "traffic": LM_TRAFFIC["bytes_per_launch"] if LM_TRAFFIC["sha256"] == sha and B <= 2 else None,
                "peak_kind": peak_kind, "bytes_per_launch": nb["lm_head_launch"], "mean_launch_us": lm_mean_ms * 1e3,
                "launches_timed": len(lm)}
    res = {"ms_per_step": ms, "steps_per_s": world * 1e3 / ms, "drafted_tokens_per_s": world * B * K * 1e3 / ms,
           "draft_step_bytes": nb["draft"], "verify_bytes": nb["verify"],
           "step_hbm_frac": (nb["draft"] + nb["verify"]) / (ms * 1e-3) / 1e9 / peak,
           "synthetic_al": float(acc.mean().item()) + 1.0, "synthetic_al_sequences": B,
           "roofline": roof, "launches_per_step": launches_per_step, "clocks": clocks, "config": config_of(wl, ctx)}
    if not full:
        del sess, vb, graph
        return res

    # verify alone (same inputs, L2 flushed): verify GB/s in the workload's dtype and in bf16
    def time_verify(tgt, drf):
        vgraph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(vgraph, stream=stream):
            vb.run(tgt, drf if T > 0 else None, v_in["tokens"], T, v_in["u_accept"], v_in["u_sample"])
        vs = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 3)]
        ve = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 3)]
        with torch.cuda.stream(stream):
            for i in range(args.steps + 3):
                flush()
                vs[i].record(stream)
                vgraph.replay()
                ve[i].record(stream)
        torch.cuda.synchronize()
        assert int(vb.status.item()) == 0
        return sum(s_.elapsed_time(e_) for s_, e_ in zip(vs[3:], ve[3:])) / args.steps
    v_ms = time_verify(v_in["target"], v_in["draft"])
    tb, db = v_in["target"].to(torch.bfloat16), v_in["draft"].to(torch.bfloat16)
    vbf_ms = time_verify(tb, db)
    del tb, db
    res["verify_us"] = v_ms * 1e3
    res["verify_gbs"] = nb["verify"] / (v_ms * 1e-3) / 1e9
    res["verify_frac"] = res["verify_gbs"] / peak
    res["verify_bf16_us"] = vbf_ms * 1e3
    res["verify_bf16_gbs"] = nb["verify_bf16"] / (vbf_ms * 1e-3) / 1e9
    res["verify_bf16_frac"] = res["verify_bf16_gbs"] / peak

    # end to end: every step's inputs copied from pinned host memory and its
    # results read back, inside the timed region.  Two device input sets, each
    # with its own captured step, so that a copy stream fills one set while the
    # step on the other computes (the inputs, 0.9 GB at the large-vocabulary
    # workload, exceed L2, so no flush runs between these steps).
    # (the draft call's and verify's inputs both have "tokens": keys carry their side)
    both = {**{"d." + k: v for k, v in d_in.items()}, **{"v." + k: v for k, v in v_in.items()}}
    h_in = {k: v.cpu().pin_memory() for k, v in both.items()}
    h_out = [{"draft_tokens": torch.empty_like(out["draft_tokens"], device="cpu").pin_memory(),
              "out_tokens": torch.empty_like(vb.out_tokens, device="cpu").pin_memory(),
              "n_accepted": torch.empty_like(vb.n_accepted, device="cpu").pin_memory()} for _ in range(2)]
    sets = [both, {k: v.clone() for k, v in both.items()}]
    graphs = [graph]
    d_save, v_save = dict(d_in), dict(v_in)
    for k in d_in:
        d_in[k] = sets[1]["d." + k]
    for k in v_in:
        v_in[k] = sets[1]["v." + k]
    g2 = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g2, stream=stream):
        step()
    graphs.append(g2)
    d_in.update(d_save)
    v_in.update(v_save)
    copy_stream = torch.cuda.Stream()
    filled = [torch.cuda.Event() for _ in range(2)]
    consumed = [torch.cuda.Event() for _ in range(2)]
    torch.cuda.synchronize()
    e_start, e_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e_start.record(stream)
    copy_stream.wait_stream(stream)
    for i in range(args.steps):
        k = i % 2
        with torch.cuda.stream(copy_stream):
            if i >= 2:
                copy_stream.wait_event(consumed[k])   # the step that last read set k is done
            for name, v in h_in.items():
                sets[k][name].copy_(v, non_blocking=True)
            filled[k].record(copy_stream)
        with torch.cuda.stream(stream):
            stream.wait_event(filled[k])
            graphs[k].replay()
            consumed[k].record(stream)
            h_out[k]["draft_tokens"].copy_(out["draft_tokens"], non_blocking=True)
            h_out[k]["out_tokens"].copy_(vb.out_tokens, non_blocking=True)
            h_out[k]["n_accepted"].copy_(vb.n_accepted, non_blocking=True)
    e_end.record(stream)
    torch.cuda.synchronize()
    assert int(sess.status.item()) == 0 and int(vb.status.item()) == 0
    e2e_ms = max_over_ranks(e_start.elapsed_time(e_end) / args.steps, world, dev)
    res["e2e"] = {"value": world * 1e3 / e2e_ms, "unit": "steps/s",
                  "h2d_bytes_per_step": sum(v.numel() * v.element_size() for v in h_in.values()),
                  "d2h_bytes_per_step": sum(v.numel() * v.element_size() for v in h_out[0].values()),
                  "timing": "one span over all steps; the next step's inputs are copied (second stream, second "
                            "input set) while this step computes; inputs larger than L2, no flush between steps"}
    res["gpu_launches"] = launches_per_step * args.steps
    if rank == 0 and not args.no_cpu_baseline:
        res["cpu_baseline"] = cpu_baseline(wl, ctx, w, kv, di, vi)
    del sess, vb, graph, graphs, g2, sets, h_in
    return res


def main():
    args = parse()
    if args.impl == "reference":
        return run_reference(args)
    if args.verify_sweep:
        return verify_sweep(args)
    if args.verify_hidden:
        return verify_hidden_compare(args)
    import torch
    import torch.distributed as dist
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    import __graft_entry__
    __graft_entry__.build()

    wl = WORKLOADS[args.workload]
    if args.temperature is not None:
        wl = wl.with_(temperature=args.temperature)
    r = measure(wl, args, rank, world, local, full=True)
    torch.cuda.empty_cache()
    others = {}
    if not args.no_extra and world == 1:
        for name in EXTRA_WORKLOADS:
            if name == wl.name:
                continue
            o = measure(WORKLOADS[name], args, rank, world, local, full=False)
            torch.cuda.empty_cache()
            others[name] = {k: o[k] for k in ("ms_per_step", "steps_per_s", "step_hbm_frac", "synthetic_al",
                                              "launches_per_step")}
            others[name]["roofline"] = {k: o["roofline"][k] for k in ("kernel", "achieved", "frac",
                                                                      "mean_launch_us")}
            others[name]["clocks"] = o["clocks"]
    if rank == 0:
        res = {
            "metric": "draft+verify steps/s", "value": r["steps_per_s"], "unit": "steps/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": r["ms_per_step"], "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": r["config"],
            **{k: r[k] for k in ("drafted_tokens_per_s", "verify_gbs", "verify_us", "verify_frac", "verify_bf16_gbs",
                                 "verify_bf16_us", "verify_bf16_frac", "draft_step_bytes", "step_hbm_frac",
                                 "synthetic_al", "synthetic_al_sequences", "roofline", "e2e", "gpu_launches",
                                 "clocks")},
        }
        if "cpu_baseline" in r:
            res["cpu_baseline"] = r["cpu_baseline"]
        if others:
            res["other_workloads"] = others
        print(json.dumps(res))
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
