"""Model shapes, decoding settings and drafter-update hyper-parameters.

The five workloads stand in for Vicuna-7B on Spec-Bench (the paper's setup,
Sec. 4.1 and App. A), which is not available here.  Where the paper gives no
constant (schedule breakpoints, optimizer, LoRA rank, beta decay) the values
below are this project's readings; each is listed with its reason in the
design notes.
"""
from __future__ import annotations

from dataclasses import dataclass, field, replace
from typing import Optional, Tuple


@dataclass(frozen=True)
class ModelShape:
    """Llama-style pre-norm decoder (Sec. 3.1 names only layers 0:L)."""
    n_layers: int
    d_model: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    d_ffn: int
    vocab: int
    rms_eps: float = 1e-5
    rope_theta: float = 10000.0

    def __post_init__(self):
        assert self.n_heads * self.head_dim > 0
        assert self.n_heads % self.n_kv_heads == 0
        assert self.head_dim % 2 == 0


@dataclass(frozen=True)
class UpdateHyper:
    """Drafter-head update (Sec. 3.4): objective weights, schedule, optimizer.

    objective: "dvi" (the KL->RL schedule of Sec. 3.4), or one of the
    single-term ablations of Sec. 4.3: "kl", "pg" (REINFORCE), "ce"
    (reward-masked cross-entropy).
    """
    objective: str = "dvi"
    lr: float = 1e-3
    beta1: float = 0.9
    beta2: float = 0.999
    adam_eps: float = 1e-8
    optimizer: str = "adam"          # "adam" | "sgd"
    tau: float = 1.0                 # KD temperature of p_phi^(tau)
    lambda0: float = 1.0             # lambda_kl during warmup
    lambda_kl_min: float = 0.1
    lambda_pg_max: float = 1.0
    t_warmup: int = 32
    t_ramp: int = 32
    w_ce: float = 0.0
    w_ent: float = 0.0
    w_rl_max: float = 0.1
    beta0: float = 0.1               # weight of KL(p_theta || p_phi) in L_policy
    beta_min: float = 0.01
    t_beta: float = 100.0
    baseline_rho: float = 0.9        # EMA of rewards (the baseline b)

    def __post_init__(self):
        assert self.objective in ("dvi", "kl", "pg", "ce")
        assert self.optimizer in ("adam", "sgd")


@dataclass(frozen=True)
class Workload:
    name: str
    shape: ModelShape
    dtype: str                       # "f32" | "bf16": weights, KV cache, activations
    batch: int
    split_k: int                     # draft = layers 1..k, verify = k+1..L
    k_spec: int
    lora_rank: int
    lora_gamma: float
    update_every: int                # U: decode steps between drafter updates
    update: UpdateHyper
    prompt_len: Tuple[int, int]      # inclusive range; (P, P) for a fixed length
    prompt_dist: str                 # "uniform" | "zipf"
    gen_tokens: int
    # output projections (W_o, W_down) of these 1-based layers are scaled
    scaled_layers: Tuple[int, ...] = ()
    scale: float = 1.0
    # batch workloads whose prompt distribution shifts midway: id ranges per wave
    waves: Tuple[Tuple[int, int], ...] = ()
    weight_seed: int = 0
    prompt_seed: int = 1
    zipf_s: float = 1.1

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)


def tiny_shape(**kw) -> ModelShape:
    base = dict(n_layers=4, d_model=256, n_heads=4, n_kv_heads=4, head_dim=64,
                d_ffn=688, vocab=1024)
    base.update(kw)
    return ModelShape(**base)


SHAPE_1B = ModelShape(n_layers=16, d_model=2048, n_heads=16, n_kv_heads=8,
                      head_dim=128, d_ffn=5632, vocab=32000)
SHAPE_7B = ModelShape(n_layers=32, d_model=4096, n_heads=32, n_kv_heads=32,
                      head_dim=128, d_ffn=11008, vocab=32000)

WORKLOADS = {
    # 1: tiny oracle model, fp32, KL-only update every 8 steps.
    "tiny": Workload(
        name="tiny-L4-d256-V1024-f32-b1", shape=tiny_shape(), dtype="f32",
        batch=1, split_k=2, k_spec=4, lora_rank=8, lora_gamma=1.0,
        update_every=8, update=UpdateHyper(objective="kl", lr=1e-3),
        prompt_len=(32, 32), prompt_dist="uniform", gen_tokens=64,
        scaled_layers=(3, 4), scale=0.1),
    # 2: ~1B GQA decoder, bf16; KL->RL switch after 32 updates.
    "1b": Workload(
        name="llama1b-shape-bf16-b1-k8-kspec5", shape=SHAPE_1B, dtype="bf16",
        batch=1, split_k=8, k_spec=5, lora_rank=16, lora_gamma=1.0,
        update_every=4, update=UpdateHyper(objective="dvi", t_warmup=32),
        prompt_len=(512, 512), prompt_dist="zipf", gen_tokens=256,
        scaled_layers=tuple(range(9, 17)), scale=0.3),
    # 3: Llama-2-7B shape, bf16, split at layer 2 as in the paper (Sec. 4.1).
    "7b": Workload(
        name="llama7b-shape-bf16-b1-k2-kspec5-prompt1024", shape=SHAPE_7B,
        dtype="bf16", batch=1, split_k=2, k_spec=5, lora_rank=16,
        lora_gamma=1.0, update_every=4, update=UpdateHyper(objective="dvi"),
        prompt_len=(1024, 1024), prompt_dist="zipf", gen_tokens=512),
    # 4: 7B shape, batch 8 ragged, two prompt waves over shifted id ranges.
    "7b-b8": Workload(
        name="llama7b-shape-bf16-b8-ragged-shift", shape=SHAPE_7B,
        dtype="bf16", batch=8, split_k=2, k_spec=5, lora_rank=16,
        lora_gamma=1.0, update_every=4, update=UpdateHyper(objective="dvi"),
        prompt_len=(128, 2048), prompt_dist="zipf", gen_tokens=512,
        waves=((0, 16000), (16000, 32000))),
    # 5: 7B shape, batch 1, 16K-token prompt, k_spec 8.
    "7b-16k": Workload(
        name="llama7b-shape-bf16-b1-k2-kspec8-prompt16384", shape=SHAPE_7B,
        dtype="bf16", batch=1, split_k=2, k_spec=8, lora_rank=16,
        lora_gamma=1.0, update_every=4, update=UpdateHyper(objective="dvi"),
        prompt_len=(16384, 16384), prompt_dist="zipf", gen_tokens=1024),
}


def workload(name: str, **overrides) -> Workload:
    w = WORKLOADS[name]
    return w.with_(**overrides) if overrides else w
