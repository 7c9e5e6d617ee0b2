"""Plain, slow CPU oracle of DVI (Draft, Verify & Improve, arxiv 2510.05421).

TEST INFRASTRUCTURE ONLY.  Nothing in the product path imports this package:
only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg (and its
`--impl reference` arm) may call it.  It shares no code with the CUDA path;
both sides take their inputs from the seeded generators in `workloads`.

Arithmetic is numpy in float64 by default (float32 on request for the large
shapes), written to follow the paper's definitions step by step:

  model.py   layer-split decoder f_{0->k}, f_{k->L}, both heads (Sec. 3.1)
  decode.py  greedy AR, and the DVI draft / verify / commit / log loop
             (Sec. 3.3)
  update.py  the objective of Sec. 3.4 (KL, reward-masked CE, entropy, CE,
             REINFORCE with an EMA baseline), its analytic gradient, the
             KL->RL schedule and the optimizer step

Pins (tests/test_oracle_*.py) tie each part to something other than itself:
closed forms, invariants of the method (losslessness, full acceptance when the
drafter is the whole model), finite differences and brute force.
Parity unpinned: the acceptance values (MAT) on synthetic weights -- the
paper's MAT needs Vicuna-7B and Spec-Bench.
"""
from .model import OracleModel, KVCache, rmsnorm, rope, softmax, log_softmax, silu
from .decode import greedy_ar, dvi_generate, DVIResult, StepRecord
from .update import (ObjectiveWeights, objective_weights, head_logits,
                     loss_terms, total_loss, grad_logits, param_grads,
                     AdamState, adam_step, DrafterUpdater)

__all__ = [
    "OracleModel", "KVCache", "rmsnorm", "rope", "softmax", "log_softmax",
    "silu", "greedy_ar", "dvi_generate", "DVIResult", "StepRecord",
    "ObjectiveWeights", "objective_weights", "head_logits", "loss_terms",
    "total_loss", "grad_logits", "param_grads", "AdamState", "adam_step",
    "DrafterUpdater",
]
