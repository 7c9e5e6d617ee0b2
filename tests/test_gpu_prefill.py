"""bf16 prompt passes on the prefill kernel (128 token rows x 256 features
per tile, activations as bf16 hi + lo pairs on the MMA's M side).

* The K/V cache a prefill writes, layer by layer, against the oracle's
  (float64 on the bf16-rounded weights, K/V rounded to bf16 as cached):
  every row of every layer within two bf16 steps of the largest entry, and
  the first generated token equal to the oracle's wherever its top-2 gap is
  clear.  Prompts are ragged (several 128-row tiles and a partial one); the
  shapes cover head_dim 64 and 128, GQA, a gate/up tail tile (d_ffn 688 is
  not a multiple of 128) and a K tail (688 is not a multiple of 64).
* A row's result does not depend on the pass it sits in: chunk sizes 16,
  128, 992 and the default (1024) write bit-identical caches.
"""
from dataclasses import replace

import numpy as np
import pytest
import torch

from oracle import OracleModel
from oracle.decode import prefill as oracle_prefill
from workloads import workload, make_weights, make_prompts
from gpu_helpers import rounded_weights

pytestmark = pytest.mark.gpu


def _case(name):
    if name == "tiny":
        return workload("tiny").with_(dtype="bf16", prompt_len=(300, 300))
    w = workload("1b")      # GQA 16/8, head_dim 128, d 2048, F 5632, two layers
    return w.with_(shape=replace(w.shape, n_layers=2), split_k=1, prompt_len=(700, 700))


def _prefill(w, dw, P, chunk):
    from paper_2510_05421_gb300 import DVIEngine
    eng = DVIEngine(w.shape, "bf16", dw, batch=1, k_spec=w.k_spec, split_k=w.split_k, lora_rank=w.lora_rank,
                    lora_gamma=w.lora_gamma, max_seq_len=len(P[0]) + 64, log_steps=w.update_every,
                    prefill_chunk=chunk)
    eng.prefill(0, torch.from_numpy(P[0]).cuda())
    st = eng.stats()
    s = w.shape
    shape = (s.n_layers, 1, s.n_kv_heads, len(P[0]) + 64, s.head_dim)
    k = eng.buffer("K_CACHE", torch.bfloat16).view(shape)[:, 0, :, :len(P[0])].float().cpu().numpy()
    v = eng.buffer("V_CACHE", torch.bfloat16).view(shape)[:, 0, :, :len(P[0])].float().cpu().numpy()
    first = int(eng.first[0].item())
    eng.close()
    assert st["device_status"] == 0, st["device_flags"]
    return k, v, first


@pytest.mark.parametrize("name", ["tiny", "1b-L2"])
def test_prefill_cache_matches_oracle(name):
    from paper_2510_05421_gb300 import DeviceWeights
    w = _case(name.split("-")[0])
    W = make_weights(w)
    P = make_prompts(w)
    n = len(P[0])
    k, v, first = _prefill(w, DeviceWeights.from_host(W, "bf16"), P, 0)
    m = OracleModel(rounded_weights(W), w.shape, w.lora_gamma, dtype=np.float64, kv_dtype="bf16")
    cache = m.new_cache(n + 1)
    tok, logits = oracle_prefill(m, cache, P[0])
    for l in range(w.shape.n_layers):
        for got, ref in ((k[l], cache.k[l, :n]), (v[l], cache.v[l, :n])):
            ref = ref.transpose(1, 0, 2)                 # [H_kv, n, hd] as the GPU stores it
            err = np.abs(got - ref).max() / np.abs(ref).max()
            assert err < 2 ** -7, (l, err)
    top2 = np.partition(logits, -2)[-2:]
    if top2[1] - top2[0] > 0.06:
        assert first == tok


def test_prefill_chunk_size_does_not_change_the_cache():
    from paper_2510_05421_gb300 import DeviceWeights
    w = _case("tiny")
    W = make_weights(w)
    P = make_prompts(w)
    dw = DeviceWeights.from_host(W, "bf16")
    outs = [_prefill(w, dw, P, c) for c in (16, 128, 992, 0)]
    for k, v, first in outs[1:]:
        assert np.array_equal(k, outs[0][0])
        assert np.array_equal(v, outs[0][1])
        assert first == outs[0][2]
