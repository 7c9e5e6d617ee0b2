"""Oracle forward pass of the layer-split decoder (test infrastructure only).

Sec. 3.1 writes the backbone as layers 0:L split at k (0 < k < L):
h_k = f_{0->k}(x), h_L = f_{k->L}(h_k), a frozen verifier head
p_phi = softmax(W^(V) h_L) and a drafter head
p_theta = softmax((W^(S) + gamma_s A_s B_s) h_k).  The paper does not restate
the backbone; it is Vicuna/Llama, so each layer here is the Llama pre-norm
block:

    x += W_o . Attn(RoPE(W_q n1), RoPE(W_k n1), W_v n1),   n1 = RMSNorm(x) * g1
    x += W_down . (SiLU(W_gate n2) * (W_up n2)),           n2 = RMSNorm(x) * g2

with causal attention scaled by 1/sqrt(head_dim), GQA mapping query head h to
KV head floor(h * H_kv / H), RoPE "rotate-half" with theta = 10000 and
RMSNorm eps = 1e-5.  Both heads read RMSNorm_final(h) (the model's frozen
final norm).  Layer indices in the API are 0-based: the draft path is layers
[0, k), the verify path [k, L).

Storage precision: the bf16 workloads keep their KV cache in bf16 (two bytes
per element: 16384 positions x 32 layers x 4096 x 2 tensors is the ~8 GB
cache of the long-context workload), so with kv_dtype="bf16" every K/V row is
rounded to the nearest bfloat16 when it is written to the cache; all other
arithmetic stays in the model's dtype (fp64 by default).
"""
from __future__ import annotations

import numpy as np

from workloads.configs import ModelShape
from workloads.gen import Weights


def rmsnorm(x: np.ndarray, g: np.ndarray, eps: float) -> np.ndarray:
    """x / sqrt(mean(x^2) + eps) * g over the last axis."""
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return x / np.sqrt(ms + eps) * g


def rope(x: np.ndarray, pos: np.ndarray, theta: float) -> np.ndarray:
    """Rotary embedding, rotate-half pairing (i, i + hd/2).

    x: [R, H, hd]; pos: [R] absolute positions.  Pair i turns by the angle
    pos * theta^(-2i/hd).
    """
    hd = x.shape[-1]
    half = hd // 2
    inv = theta ** (-np.arange(half, dtype=np.float64) * 2.0 / hd)
    ang = pos.astype(np.float64)[:, None] * inv[None, :]           # [R, half]
    cos = np.cos(ang).astype(x.dtype)[:, None, :]
    sin = np.sin(ang).astype(x.dtype)[:, None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * cos - x2 * sin, x2 * cos + x1 * sin], axis=-1)


def to_bf16(a: np.ndarray) -> np.ndarray:
    """Nearest bfloat16 value (ties to even) of every element, as float32.

    bfloat16 is the top 16 bits of an IEEE float32; rounding adds half an
    ulp of the kept part (minus one when the kept part is even) before the
    low 16 bits are cleared.
    """
    b = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32)
    bias = ((b >> np.uint32(16)) & np.uint32(1)) + np.uint32(0x7FFF)
    return ((b + bias) & np.uint32(0xFFFF0000)).view(np.float32)


def softmax(z: np.ndarray) -> np.ndarray:
    e = np.exp(z - z.max(axis=-1, keepdims=True))
    return e / e.sum(axis=-1, keepdims=True)


def log_softmax(z: np.ndarray) -> np.ndarray:
    zm = z - z.max(axis=-1, keepdims=True)
    return zm - np.log(np.exp(zm).sum(axis=-1, keepdims=True))


def silu(x: np.ndarray) -> np.ndarray:
    return x / (1.0 + np.exp(-x))


class KVCache:
    """Per-sequence K/V rows for every layer; rows past `n` are dead."""

    def __init__(self, shape: ModelShape, max_len: int, dtype):
        self.k = np.zeros((shape.n_layers, max_len, shape.n_kv_heads, shape.head_dim), dtype)
        self.v = np.zeros_like(self.k)
        self.max_len = max_len


class OracleModel:
    def __init__(self, weights: Weights, shape: ModelShape, lora_gamma: float = 1.0,
                 dtype=np.float64, kv_dtype: str | None = None):
        self.s = shape
        self.dtype = dtype
        assert kv_dtype in (None, "bf16")
        self.kv_bf16 = kv_dtype == "bf16"
        self.gamma = lora_gamma
        c = lambda a: np.asarray(a, dtype=dtype)
        self.embed_w = c(weights.embed)
        self.layers = [{f: c(getattr(l, f)) for f in
                        ("attn_norm", "wq", "wk", "wv", "wo", "ffn_norm",
                         "w_gate", "w_up", "w_down")} for l in weights.layers]
        self.final_g = c(weights.final_norm)
        self.w_v = c(weights.lm_head)          # W^(V), frozen
        self.w_s = c(weights.draft_head)       # W^(S)
        self.lora_a = c(weights.lora_a)        # A_s [V, r]
        self.lora_b = c(weights.lora_b)        # B_s [r, d]

    # ---- backbone -------------------------------------------------------
    def new_cache(self, max_len: int) -> KVCache:
        return KVCache(self.s, max_len, self.dtype)

    def embed(self, toks) -> np.ndarray:
        return self.embed_w[np.asarray(toks, dtype=np.int64)].copy()

    def attention(self, q, ck, cv, pos0: int) -> np.ndarray:
        """softmax(q K^T / sqrt(hd) + causal mask) V for R query rows.

        q: [R, H, hd] for positions pos0..pos0+R-1; ck, cv: [>=pos0+R, H_kv, hd].
        Row i sees cache positions 0..pos0+i.
        """
        s = self.s
        R = q.shape[0]
        T = pos0 + R
        out = np.empty_like(q)
        mask = np.arange(T)[None, :] <= (pos0 + np.arange(R))[:, None]   # [R, T]
        for h in range(s.n_heads):
            g = h * s.n_kv_heads // s.n_heads
            sc = q[:, h, :] @ ck[:T, g, :].T / np.sqrt(s.head_dim)
            sc = np.where(mask, sc, -np.inf)
            out[:, h, :] = softmax(sc) @ cv[:T, g, :]
        return out

    def layer(self, l: int, x: np.ndarray, pos0: int, cache: KVCache) -> np.ndarray:
        """One pre-norm block on rows x [R, d] at positions pos0.. ; writes K/V rows."""
        s, w = self.s, self.layers[l]
        R = x.shape[0]
        n1 = rmsnorm(x, w["attn_norm"], s.rms_eps)
        pos = pos0 + np.arange(R)
        q = (n1 @ w["wq"].T).reshape(R, s.n_heads, s.head_dim)
        k = (n1 @ w["wk"].T).reshape(R, s.n_kv_heads, s.head_dim)
        v = (n1 @ w["wv"].T).reshape(R, s.n_kv_heads, s.head_dim)
        q = rope(q, pos, s.rope_theta)
        k = rope(k, pos, s.rope_theta)
        if pos0 + R > cache.max_len:
            raise ValueError("KV cache capacity exceeded")
        if self.kv_bf16:
            k, v = to_bf16(k).astype(self.dtype), to_bf16(v).astype(self.dtype)
        cache.k[l, pos0:pos0 + R] = k
        cache.v[l, pos0:pos0 + R] = v
        o = self.attention(q, cache.k[l], cache.v[l], pos0)
        x = x + o.reshape(R, -1) @ w["wo"].T
        n2 = rmsnorm(x, w["ffn_norm"], s.rms_eps)
        hmid = silu(n2 @ w["w_gate"].T) * (n2 @ w["w_up"].T)
        return x + hmid @ w["w_down"].T

    def layers_range(self, lo: int, hi: int, x, pos0: int, cache: KVCache):
        for l in range(lo, hi):
            x = self.layer(l, x, pos0, cache)
        return x

    # ---- heads (Sec. 3.1) ----------------------------------------------
    def final_norm(self, h: np.ndarray) -> np.ndarray:
        return rmsnorm(h, self.final_g, self.s.rms_eps)

    def verifier_logits(self, h_L: np.ndarray) -> np.ndarray:
        """logits^phi = W^(V) RMSNorm_final(h_L)."""
        return self.final_norm(h_L) @ self.w_v.T

    def drafter_logits(self, h_k: np.ndarray) -> np.ndarray:
        """(W^(S) + gamma A B) RMSNorm_final(h_k), evaluated as W^S u + gamma A (B u)."""
        u = self.final_norm(h_k)
        z = u @ self.w_s.T
        if self.lora_a.shape[1] > 0:
            z = z + self.gamma * (u @ self.lora_b.T) @ self.lora_a.T
        return z
