"""Oracle decode loops: greedy AR and DVI (test infrastructure only).

Greedy AR (the speedup denominator and the losslessness reference of Sec. 3.1
and Sec. 4.1): prefill the prompt, then emit argmax_y p_phi(y | h_L) one token
at a time.

DVI step (Sec. 3.3), per sequence with committed cache length n and pending
token x_n (the last committed token, not yet in any cache):
  draft    for j = 0..K-1: h_{k,n+j} = f_{0->k}(tok_j) with tok_0 = x_n and
           tok_j = t~_j; t~_{j+1} = argmax p_theta(. | h_{k,n+j})   (greedy)
  verify   one pass of f_{k->L} over the K rows h_{k,n..n+K-1} with
           block-causal attention; y*_{n+i} = argmax p_phi(. | h_{L,n+i-1})
  accept   m = max{i in 0..K : t~_j = y*_{n+j} for all j <= i}
  commit   t~_1..t~_m, then the correction y*_{n+m+1} when m < K; with m = K
           no token beyond the block was verified, so the step commits K
           tokens and t~_K becomes the pending token (no bonus token).  With
           bonus=True the draft path also runs t~_K and the verifier checks
           K+1 rows, so every step commits m+1 tokens.
  log      tuples for i = 1..(number committed): (u = RMSNorm_final(h_{k,n+i-1}),
           a = t~_i, logits^phi_{n+i}, r = 1 if i <= m else 0, i, prev_id)
Cache rows past the new length are dead and get overwritten by later steps.
Every `update_every` steps the logged tuples of all sequences drive one
drafter update (update.py) and the buffer is cleared.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import List, Optional, Sequence

import numpy as np

from .model import OracleModel, KVCache


def _argmax(z: np.ndarray) -> int:
    if not np.all(np.isfinite(z)):
        raise FloatingPointError("non-finite logits")
    return int(np.argmax(z))          # lowest index wins a tie


def _top2_gap(z: np.ndarray) -> float:
    t = np.partition(z, -2)[-2:]
    return float(t[1] - t[0])


def prefill(model: OracleModel, cache: KVCache, prompt: Sequence[int]):
    """Run the whole prompt through all L layers; return (first token, logits row)."""
    x = model.embed(prompt)
    x = model.layers_range(0, model.s.n_layers, x, 0, cache)
    logits = model.verifier_logits(x[-1:])[0]
    return _argmax(logits), logits


def ar_step(model: OracleModel, cache: KVCache, n: int, tok: int):
    """One greedy AR step: the pending token x_n (at position n) through all
    L layers, then argmax of the verifier head; returns (next token, logits)."""
    x = model.embed([tok])
    x = model.layers_range(0, model.s.n_layers, x, n, cache)
    logits = model.verifier_logits(x)[0]
    return _argmax(logits), logits


def greedy_ar(model: OracleModel, prompt: Sequence[int], n_gen: int,
              return_logits: bool = False):
    """Greedy autoregressive decoding of n_gen tokens after the prompt."""
    P = len(prompt)
    cache = model.new_cache(P + n_gen + 1)
    tok, logits = prefill(model, cache, prompt)
    out, rows, gaps = [tok], [logits], [_top2_gap(logits)]
    n = P
    while len(out) < n_gen:
        tok, logits = ar_step(model, cache, n, tok)
        out.append(tok)
        rows.append(logits)
        gaps.append(_top2_gap(logits))
        n += 1
    out = np.array(out[:n_gen], dtype=np.int32)
    if return_logits:
        return out, np.stack(rows[:n_gen]), np.array(gaps[:n_gen])
    return out


@dataclass
class StepRecord:
    step: int
    seq: int
    n: int                       # committed cache length before the step
    drafts: List[int]            # t~_1..t~_K
    ystar: List[int]             # y*_{n+1}..y*_{n+K} (K+1 entries with bonus)
    m: int                       # accepted drafted tokens
    committed: List[int]
    verify_logits: Optional[np.ndarray] = None   # [K, V]
    draft_gap: float = np.inf    # smallest top-2 gap among the drafter argmaxes
    verify_gap: float = np.inf   # smallest top-2 gap among the verifier argmaxes


@dataclass
class LoggedTuple:
    seq: int
    u: np.ndarray                # RMSNorm_final(h_{k,n+i-1})
    a: int                       # drafted token t~_i
    logits: np.ndarray           # logits^phi_{n+i}
    r: int                       # 1 accepted, 0 first reject
    i: int                       # 1-based position in the block
    prev_id: int
    ystar: int


@dataclass
class DVIResult:
    tokens: List[np.ndarray]                   # per sequence, n_gen tokens
    steps: List[StepRecord] = field(default_factory=list)
    updates: List[dict] = field(default_factory=list)
    prefill_logits: List[np.ndarray] = field(default_factory=list)

    def mean_accepted(self) -> float:
        return float(np.mean([s.m for s in self.steps])) if self.steps else 0.0


def dvi_step(model: OracleModel, cache: KVCache, n: int, pending: int, k: int,
             K: int, bonus: bool = False):
    """One draft -> verify -> accept -> commit pass for one sequence.

    Returns (record fields, logged tuples, new n, new pending).
    """
    L = model.s.n_layers
    toks = [pending]
    hk = []
    dgap = np.inf
    for j in range(K):
        x = model.embed([toks[j]])
        x = model.layers_range(0, k, x, n + j, cache)
        hk.append(x[0])
        z = model.drafter_logits(x)[0]
        dgap = min(dgap, _top2_gap(z))
        toks.append(_argmax(z))
    rows = K
    if bonus:
        x = model.embed([toks[K]])
        x = model.layers_range(0, k, x, n + K, cache)
        hk.append(x[0])
        rows = K + 1
    X = np.stack(hk)                                   # [rows, d] = h_{k,n..}
    X = model.layers_range(k, L, X, n, cache)          # one verify pass
    logits = model.verifier_logits(X)                  # [rows, V]
    ystar = [_argmax(logits[i]) for i in range(rows)]
    vgap = min(_top2_gap(logits[i]) for i in range(rows))
    m = 0
    while m < K and toks[m + 1] == ystar[m]:
        m += 1
    if m < rows:
        committed = toks[1:m + 1] + [ystar[m]]
    else:
        committed = toks[1:K + 1]
    c = len(committed)
    U = model.final_norm(np.stack(hk[:K]))
    tuples = []
    for i in range(1, min(c, K) + 1):
        tuples.append(LoggedTuple(seq=-1, u=U[i - 1], a=toks[i],
                                  logits=logits[i - 1], r=1 if i <= m else 0,
                                  i=i, prev_id=toks[i - 1], ystar=ystar[i - 1]))
    return (toks[1:K + 1], ystar, m, committed, logits[:K], dgap, vgap), tuples, n + c, committed[-1]


def dvi_generate(model: OracleModel, prompts: Sequence[Sequence[int]], n_gen: int,
                 k: int, K: int, update_every: Optional[int] = None,
                 updater=None, bonus: bool = False, log: bool = True,
                 keep_logits: bool = False, max_steps: Optional[int] = None,
                 caches: Optional[List[KVCache]] = None) -> DVIResult:
    """Self-speculative generation of n_gen tokens for every prompt.

    All sequences run every step until each has n_gen tokens (a finished
    sequence keeps stepping and its extra tokens are dropped), mirroring one
    batched decode.  Tuples from all sequences share one buffer; every
    `update_every` steps `updater.update(tuples)` runs and the buffer clears.
    """
    B = len(prompts)
    if caches is None:
        caches = [model.new_cache(len(p) + n_gen + 2 * K + 2) for p in prompts]
    res = DVIResult(tokens=[])
    out, ns, pend = [], [], []
    for b, p in enumerate(prompts):
        tok, lg = prefill(model, caches[b], p)
        res.prefill_logits.append(lg)
        out.append([tok])
        ns.append(len(p))
        pend.append(tok)
    buf: List[LoggedTuple] = []
    step = 0
    while any(len(o) < n_gen for o in out):
        if max_steps is not None and step >= max_steps:
            break
        for b in range(B):
            (drafts, ystar, m, committed, vlog, dg, vg), tuples, ns[b], pend[b] = dvi_step(
                model, caches[b], ns[b], pend[b], k, K, bonus)
            out[b].extend(committed)
            res.steps.append(StepRecord(step=step, seq=b, n=ns[b] - len(committed),
                                        drafts=drafts, ystar=ystar, m=m,
                                        committed=committed,
                                        verify_logits=vlog if keep_logits else None,
                                        draft_gap=dg, verify_gap=vg))
            if log:
                for t in tuples:
                    t.seq = b
                buf.extend(tuples)
        step += 1
        if updater is not None and update_every and step % update_every == 0:
            res.updates.append(updater.update(buf))
            buf = []
    res.tokens = [np.array(o[:n_gen], dtype=np.int32) for o in out]
    return res
