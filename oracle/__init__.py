"""CPU oracle for MeBP's training step — TEST INFRASTRUCTURE ONLY.

A plain, slow, obviously correct numpy (fp64) restatement of what the hot path
computes, written from the paper's text:

* ``quant``  — the 4-bit symmetric weight compression and its decode (Section 3,
  "Base model weights compression").
* ``model``  — the LoRA-adapted pre-norm decoder block, its backward (the block
  VJP of Section 3, "Gradient checkpointing compilation"), the LM-head
  cross-entropy, and Algorithm 1 (checkpointed forward loop, then reverse
  backward loop that recomputes each block from its stored input).
* ``optim``  — the AdamW update of the LoRA weights (Section 4 trains with AdamW).

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline leg may
import this package.  It shares no code with the CUDA path and the product
never calls it.
"""
from . import quant, model, optim  # noqa: F401
