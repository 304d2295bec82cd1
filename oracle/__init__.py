"""CPU oracle for the Osprey speculative-decoding hot path.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path imports this package:
only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` use it.  It shares no code with the CUDA path (no kernels,
headers, helpers or tables); the two meet only in the seeded inputs of
``paper_2609_09338_gb300.synthetic``.

Everything is plain numpy in float64, written from the paper:

* ``oracle.drafter`` - the drafter forward and chain (Sec. 3.3 Eq. 1-3, Sec. 3.4),
  with the inputs widened exactly from the same bf16 bytes the GPU reads;
* ``oracle.verify`` - speculative-sampling verification (Sec. 3.1, the
  unmodified acceptance rule of Leviathan et al.), its greedy form, and the
  exact emission distribution obtained by integrating the rule over its
  uniforms;
* ``oracle.dflash`` - the EAGLE-style DFlash block drafter (Appendix, "EAGLE-
  Style Target Interface for DFlash"): one causal forward over an anchor and
  mask placeholders, the target feature broadcast through the expanded QKV;
* ``oracle.tree`` - verification of a draft tree (topk > 1): the multi-
  candidate form of the Sec. 3.1 rule over a branching chain, which is the
  chain rule at topk = 1.

Every function below is pinned by a ``-m "not gpu"`` test against something
other than itself (closed forms, library routines, invariants, brute force).
"""
from . import bf16, dflash, drafter, tree, verify  # noqa: F401
