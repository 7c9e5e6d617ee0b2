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


def teacher_forced_tail(model, seq_tokens, start):
    """Verifier logits at input positions start.. of one full sequence (one
    causal pass through every layer; the head only on the rows asked for)."""
    L = model.s.n_layers
    cache = model.new_cache(len(seq_tokens) + 1)
    x = model.layers_range(0, L, model.embed(seq_tokens), 0, cache)
    return model.verifier_logits(x[start:])


def run_logged_steps(eng, prompts, n_steps, update_every=0, hyper=None):
    """Prefill every prompt, then run `n_steps` decode steps one at a time and
    read the replay buffer after each: the verify rows every step logged.

    Returns (committed tokens per sequence including the prefill's first
    token, rows) with rows = [(b, input position, logits float64 [V], y*)];
    row i of a step for a sequence at committed length n has its input token
    at position n + i, so the oracle's teacher-forced logits at that position
    are its reference.  The drafter is updated every `update_every` steps."""
    B, K, V = eng.B, eng.K, eng.shape.vocab
    for b, p in enumerate(prompts):
        eng.prefill(b, torch.from_numpy(np.ascontiguousarray(p, dtype=np.int32)).to(eng.device))
    eng.log(True)
    eng.sync()
    first = eng.first.cpu().numpy()
    toks = [[int(first[b])] for b in range(B)]
    n = [len(p) for p in prompts]
    rows = []
    j = 0
    meta_all = eng.buffer("LOG_META", torch.int32).view(-1, 6)
    lg_all = eng.buffer("LOG_LOGITS", torch.float32).view(-1, V)
    for _ in range(n_steps):
        ids, cnt, _ = eng.step()
        eng.sync()
        ids, cnt = ids.cpu().numpy(), cnt.cpu().numpy()
        base = j * B * K
        meta = meta_all[base:base + B * K].cpu().numpy()
        lg = lg_all[base:base + B * K].double().cpu().numpy()
        for b in range(B):
            c = int(cnt[b])
            assert 1 <= c <= K
            for i in range(K):
                slot = b * K + i
                assert meta[slot, 0] == (1 if i < c else 0), (b, i, meta[slot])
                if i < c:
                    rows.append((b, n[b] + i, lg[slot], int(meta[slot, 5])))
            toks[b].extend(int(t) for t in ids[b, :c])
            n[b] += c
        j += 1
        if update_every and hyper is not None and j == update_every:
            eng.update(hyper)
            j = 0
    return toks, rows


def check_rows_against_oracle(model, prompts, toks, rows, tol):
    """Every logged verify row within `tol` (max abs) of the oracle's
    teacher-forced logits on the committed sequence, y* the argmax of the
    GPU row, and y* equal to the oracle's argmax wherever the oracle's top-2
    gap exceeds 2 tol.  Returns the largest error seen."""
    worst = 0.0
    by_seq = {}
    for b, pos, lg, ys in rows:
        by_seq.setdefault(b, []).append((pos, lg, ys))
    for b, rs in by_seq.items():
        seq = np.concatenate([prompts[b], np.asarray(toks[b], dtype=np.int32)])
        start = len(prompts[b])
        ref = teacher_forced_tail(model, seq, start)
        for pos, lg, ys in rs:
            r = ref[pos - start]
            err = float(np.abs(lg - r).max())
            worst = max(worst, err)
            assert err < tol, (b, pos, err)
            assert int(np.argmax(lg)) == ys, (b, pos)
            top2 = np.partition(r, -2)[-2:]
            if top2[1] - top2[0] > 2 * tol:
                assert int(np.argmax(r)) == ys, (b, pos)
    return worst
