"""Objective ablations of the online drafter update (Sec. 4.3): the full
KL->RL schedule against KL-only, PG-only (REINFORCE) and CE-only
(reward-masked cross-entropy), as acceptance per update window on a
drifting stream.

    python -m paper_2510_05421_gb300.ablation --workload tiny --objectives dvi,kl,pg,ce

Every objective starts from the same weights and decodes the same prompts:
two waves of prompts (the workload's shifted id ranges when it has them,
else a second prompt seed), one context for both, so the drafter keeps
adapting while the stream moves.  Prints one JSON line per objective with
the mean accepted length per window of `update_every` decode steps.  The
inputs are synthetic random-weight models, so the numbers show how each
objective moves acceptance on this stream, not the paper's values.
"""
from __future__ import annotations

import argparse
import json
from dataclasses import replace

import numpy as np


def run(workload_name: str, objectives, tokens: int, t_warmup: int, t_ramp: int, lr: float, device: int = 0):
    from workloads import workload, make_weights, make_prompts
    from .dvi import DVIEngine, DeviceWeights

    w = workload(workload_name)
    W = make_weights(w)
    waves = [make_prompts(w, 0), make_prompts(w, 1)]
    U = w.update_every
    cap = max(len(p) for P in waves for p in P) + 2 * tokens * (w.k_spec + 1) + 64
    out = []
    for obj in objectives:
        hyper = replace(w.update, objective=obj, t_warmup=t_warmup, t_ramp=t_ramp, lr=lr)
        dw = DeviceWeights.from_host(W, w.dtype, device=f"cuda:{device}")
        eng = DVIEngine(w.shape, w.dtype, dw, batch=w.batch, k_spec=w.k_spec, split_k=w.split_k,
                        lora_rank=w.lora_rank, lora_gamma=w.lora_gamma, max_seq_len=cap, log_steps=U,
                        device=device)
        windows = []
        for P in waves:
            _, mats, _, _ = eng.generate(P, tokens, update_every=U, hyper=hyper)
            m = mats.mean(axis=1)
            windows += [float(np.mean(m[i:i + U])) for i in range(0, len(m), U)]
        st = eng.stats()
        eng.close()
        out.append({"workload": w.name, "objective": obj, "update_every": U, "updates": st["updates"],
                    "mat_per_window": [round(x, 4) for x in windows],
                    "mat_wave1": round(float(np.mean(windows[:len(windows) // 2])), 4),
                    "mat_wave2": round(float(np.mean(windows[len(windows) // 2:])), 4),
                    "device_flags": st["device_flags"]})
    return out


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--workload", default="tiny")
    ap.add_argument("--objectives", default="dvi,kl,pg,ce")
    ap.add_argument("--tokens", type=int, default=128, help="tokens per sequence and wave")
    ap.add_argument("--t-warmup", type=int, default=4, help="updates of KL-only warm-up in the dvi schedule")
    ap.add_argument("--t-ramp", type=int, default=4)
    ap.add_argument("--lr", type=float, default=1e-3)
    args = ap.parse_args(argv)
    for line in run(args.workload, args.objectives.split(","), args.tokens, args.t_warmup, args.t_ramp, args.lr):
        print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
