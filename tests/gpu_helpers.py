"""Shared set-up for the GPU tests: engines built from seeded workloads."""
from __future__ import annotations

import numpy as np
import torch

from workloads import make_weights, make_prompts
from workloads.gen import bf16_round


def engine_for(w, W=None, dtype=None, use_graphs=True, max_seq_len=None, batch=None, **kw):
    from paper_2510_05421_gb300 import DVIEngine, DeviceWeights
    W = W if W is not None else make_weights(w)
    dtype = dtype or w.dtype
    dw = DeviceWeights.from_host(W, dtype)
    B = batch or w.batch
    msl = max_seq_len or (w.prompt_len[1] + w.gen_tokens + 4 * w.k_spec + 16)
    eng = DVIEngine(w.shape, dtype, dw, batch=B, k_spec=w.k_spec, split_k=kw.pop("split_k", w.split_k),
                    lora_rank=w.lora_rank, lora_gamma=w.lora_gamma, max_seq_len=msl,
                    log_steps=kw.pop("log_steps", w.update_every), use_graphs=use_graphs, **kw)
    return eng, W, dw


def logged_u(eng, w):
    """The replay buffer's head inputs u as float64 [cap][d] (bf16: hi + lo planes)."""
    d = w.shape.d_model
    if eng.dtype == "bf16":
        lu = eng.buffer("LOG_U", torch.bfloat16).view(2, -1, d).double()
        return (lu[0] + lu[1]).cpu().numpy()
    return eng.buffer("LOG_U", torch.float32).view(-1, d).double().cpu().numpy()


def rounded_weights(W):
    """The bf16-rounded weights promoted back to float32 (the oracle's view of a bf16 run)."""
    return W.map(bf16_round)


def teacher_forced_logits(model, seq_tokens):
    """Verifier logits of every position of one full sequence, in one causal pass."""
    L = model.s.n_layers
    cache = model.new_cache(len(seq_tokens) + 1)
    x = model.layers_range(0, L, model.embed(seq_tokens), 0, cache)
    return model.verifier_logits(x)
