"""Write tests/golden/tiny_dvi.json from the CPU oracle alone.

Workload: the tiny fp32 decoder (L4 d256 V1024, layers 3-4 output projections
x0.1), split k=2, k_spec=4, 32 uniform prompt ids, 64 greedy tokens, KL-only
drafter update every 8 steps, lr 1e-3 (Sec. 3.3 rollout, Sec. 3.4 update).
The oracle runs in float64.  Stored: the greedy AR stream, the DVI stream,
per-step accept lengths m and the per-update losses.

    python tests/golden/make_golden.py
"""
import json
import os
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

from oracle import OracleModel, greedy_ar, dvi_generate, DrafterUpdater  # noqa: E402
from workloads import workload, make_weights, make_prompts  # noqa: E402


def main():
    w = workload("tiny")
    W = make_weights(w)
    P = make_prompts(w)
    m = OracleModel(W, w.shape, w.lora_gamma)
    ar = greedy_ar(OracleModel(W, w.shape, w.lora_gamma), P[0], w.gen_tokens)
    res = dvi_generate(m, P, w.gen_tokens, w.split_k, w.k_spec, w.update_every,
                       DrafterUpdater(m, w.update))
    out = dict(
        source="oracle float64 via tests/golden/make_golden.py",
        workload=w.name, prompt=[int(x) for x in P[0]],
        ar_tokens=[int(x) for x in ar],
        dvi_tokens=[int(x) for x in res.tokens[0]],
        accept_lengths=[s.m for s in res.steps],
        update_losses=[u["loss"] for u in res.updates],
        update_rows=[u["n"] for u in res.updates],
    )
    with open(os.path.join(HERE, "tiny_dvi.json"), "w") as f:
        json.dump(out, f, indent=1)


if __name__ == "__main__":
    main()
