"""Seeded weights and prompts.

Weights are N(0, 0.02) draws from numpy's PCG64 in float32, one SeedSequence
child per tensor, each tensor cut into fixed 4 Mi-element blocks with a
grandchild seed each so blocks can be drawn in parallel threads without
changing the values.  Norm gains are 1.  The drafter head W^(S) starts as a
copy of the LM head W^(V); the LoRA factor A starts at 0 and B is N(0, 0.02),
so the initial drafter head equals W^(S).

Prompt ids are uniform or a finite Zipf(s) law p(rank r) ~ (r+1)^-s over an
id range, drawn by inverse CDF.

No arithmetic of the method lives here.
"""
from __future__ import annotations

import os
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass
from typing import List, Optional, Sequence

import numpy as np

from .configs import Workload

_BLOCK = 1 << 22
_STD = np.float32(0.02)


@dataclass
class LayerWeights:
    attn_norm: np.ndarray
    wq: np.ndarray
    wk: np.ndarray
    wv: np.ndarray
    wo: np.ndarray
    ffn_norm: np.ndarray
    w_gate: np.ndarray
    w_up: np.ndarray
    w_down: np.ndarray


@dataclass
class Weights:
    embed: np.ndarray            # [V, d]
    layers: List[LayerWeights]
    final_norm: np.ndarray       # [d]
    lm_head: np.ndarray          # W^(V) [V, d]
    draft_head: np.ndarray       # W^(S) [V, d]
    lora_a: np.ndarray           # A [V, r]
    lora_b: np.ndarray           # B [r, d]

    def map(self, fn) -> "Weights":
        """Apply fn to every matrix (not to the norm gains or LoRA factors)."""
        return Weights(
            embed=fn(self.embed),
            layers=[LayerWeights(attn_norm=l.attn_norm, wq=fn(l.wq), wk=fn(l.wk),
                                 wv=fn(l.wv), wo=fn(l.wo), ffn_norm=l.ffn_norm,
                                 w_gate=fn(l.w_gate), w_up=fn(l.w_up),
                                 w_down=fn(l.w_down)) for l in self.layers],
            final_norm=self.final_norm, lm_head=fn(self.lm_head),
            draft_head=fn(self.draft_head), lora_a=self.lora_a,
            lora_b=self.lora_b)


def _normal(seed: np.random.SeedSequence, shape, pool) -> np.ndarray:
    n = int(np.prod(shape))
    out = np.empty(n, dtype=np.float32)
    nblk = (n + _BLOCK - 1) // _BLOCK
    kids = seed.spawn(nblk)

    def fill(i):
        lo, hi = i * _BLOCK, min(n, (i + 1) * _BLOCK)
        g = np.random.Generator(np.random.PCG64(kids[i]))
        out[lo:hi] = g.standard_normal(hi - lo, dtype=np.float32)
        out[lo:hi] *= _STD

    list(pool.map(fill, range(nblk)))
    return out.reshape(shape)


def make_weights(w: Workload, threads: Optional[int] = None) -> Weights:
    """float32 weights of the workload's shape, reproducible from w.weight_seed."""
    s = w.shape
    L, d, V, F, r = s.n_layers, s.d_model, s.vocab, s.d_ffn, w.lora_rank
    dq, dkv = s.n_heads * s.head_dim, s.n_kv_heads * s.head_dim
    kids = np.random.SeedSequence(w.weight_seed).spawn(2 + 7 * L + 1)
    threads = threads or min(32, os.cpu_count() or 1)
    with ThreadPoolExecutor(threads) as pool:
        embed = _normal(kids[0], (V, d), pool)
        layers = []
        for l in range(L):
            k = kids[1 + 7 * l: 1 + 7 * (l + 1)]
            wq = _normal(k[0], (dq, d), pool)
            wk = _normal(k[1], (dkv, d), pool)
            wv = _normal(k[2], (dkv, d), pool)
            wo = _normal(k[3], (d, dq), pool)
            wg = _normal(k[4], (F, d), pool)
            wu = _normal(k[5], (F, d), pool)
            wd = _normal(k[6], (d, F), pool)
            if (l + 1) in w.scaled_layers:
                f = np.float32(w.scale)
                wo *= f
                wd *= f
            layers.append(LayerWeights(
                attn_norm=np.ones(d, np.float32), wq=wq, wk=wk, wv=wv, wo=wo,
                ffn_norm=np.ones(d, np.float32), w_gate=wg, w_up=wu, w_down=wd))
        lm_head = _normal(kids[1 + 7 * L], (V, d), pool)
        lora_b = _normal(kids[2 + 7 * L], (max(r, 1), d), pool)[:r]
    return Weights(embed=embed, layers=layers, final_norm=np.ones(d, np.float32),
                   lm_head=lm_head, draft_head=lm_head.copy(),
                   lora_a=np.zeros((V, r), np.float32), lora_b=np.ascontiguousarray(lora_b))


def bf16_round(x: np.ndarray) -> np.ndarray:
    """Round float32 to the nearest bfloat16 (ties to even), returned as float32."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    rnd = ((b >> 16) & 1) + np.uint32(0x7FFF)
    return ((b + rnd) & np.uint32(0xFFFF0000)).view(np.float32)


def zipf_ids(rng: np.random.Generator, n: int, lo: int, hi: int, s: float) -> np.ndarray:
    """n ids in [lo, hi) with p(lo + r) proportional to (r+1)^-s, by inverse CDF."""
    ranks = np.arange(hi - lo, dtype=np.float64)
    p = (ranks + 1.0) ** (-s)
    cdf = np.cumsum(p)
    cdf /= cdf[-1]
    u = rng.random(n)
    idx = np.minimum(np.searchsorted(cdf, u, side="right"), hi - lo - 1)
    return (lo + idx).astype(np.int32)


def make_prompts(w: Workload, wave: int = 0) -> List[np.ndarray]:
    """One int32 prompt per sequence of the batch, reproducible from w.prompt_seed."""
    kids = np.random.SeedSequence(w.prompt_seed + wave).spawn(w.batch + 1)
    lo_len, hi_len = w.prompt_len
    lens = np.random.Generator(np.random.PCG64(kids[0])).integers(
        lo_len, hi_len + 1, size=w.batch)
    lo, hi = (w.waves[wave] if w.waves else (0, w.shape.vocab))
    out = []
    for b in range(w.batch):
        g = np.random.Generator(np.random.PCG64(kids[b + 1]))
        n = int(lens[b])
        if w.prompt_dist == "uniform":
            out.append(g.integers(lo, hi, size=n).astype(np.int32))
        else:
            out.append(zipf_ids(g, n, lo, hi, w.zipf_s))
    return out
