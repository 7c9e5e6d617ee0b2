"""Verifier logits of every decode step against the oracle, in the shapes
where only the GPU's own greedy stream checked them before.

The batched and long-context workloads keep their width (Llama-2-7B:
d 4096, 32 heads of 128, SwiGLU 11008, vocabulary 32000), their split,
k_spec, prompt lengths, update schedule and launch configuration (CUDA
graphs), with the layer count cut to four (split k = 2: two draft layers,
two verify layers) so the float64 oracle finishes in about a minute:

* the 8-sequence ragged batch (prompt lengths uniform in 128..2048): the
  decode attention's rows of eight sequences of different lengths in one
  launch, each row's position split evenly over the cluster's splits;
* a 4096-token prompt with k_spec = 8: the split plan at its largest (8
  splits per KV head) over 65+ 64-position chunks per row, and the prefill
  attention over 32 chunks of 128 rows.

Every logged verify row of every step (Sec. 3.3: row i verifies the prefix
up to t~_i) is compared with the oracle's teacher-forced logits on the
committed sequence (float64 arithmetic on the bf16-rounded weights, the KV
cache rounded to bf16 as the GPU stores it), within 3e-2, with y* the row's
argmax and equal to the oracle's wherever its top-2 gap is clear.
"""
from dataclasses import replace

import numpy as np
import pytest

from oracle import OracleModel
from workloads import workload, make_weights, make_prompts
from gpu_helpers import rounded_weights, run_logged_steps, check_rows_against_oracle

pytestmark = pytest.mark.gpu
TOL = 3e-2


def _reduced(name, layers=4, **kw):
    w = workload(name)
    return w.with_(shape=replace(w.shape, n_layers=layers), name=f"{w.name}-L{layers}", **kw)


def _engine(w, dw, P, n_steps):
    from paper_2510_05421_gb300 import DVIEngine
    # KV capacity as the benchmark sizes it: prompt + K per step + slack
    cap = max(len(p) for p in P) + (n_steps + 2) * w.k_spec + 64
    return DVIEngine(w.shape, w.dtype, dw, batch=w.batch, k_spec=w.k_spec, split_k=w.split_k,
                     lora_rank=w.lora_rank, lora_gamma=w.lora_gamma, max_seq_len=cap,
                     log_steps=w.update_every)


def _run(w, P, n_steps):
    from paper_2510_05421_gb300 import DeviceWeights
    W = make_weights(w)
    dw = DeviceWeights.from_host(W, w.dtype)
    eng = _engine(w, dw, P, n_steps)
    toks, rows = run_logged_steps(eng, P, n_steps, update_every=w.update_every, hyper=w.update)
    st = eng.stats()
    eng.close()
    assert st["device_status"] == 0, st["device_flags"]
    assert st["updates"] == n_steps // w.update_every
    model = OracleModel(rounded_weights(W), w.shape, w.lora_gamma, dtype=np.float64, kv_dtype="bf16")
    return check_rows_against_oracle(model, P, toks, rows, TOL), rows


def test_batch8_ragged_every_step_against_oracle():
    w = _reduced("7b-b8")
    P = make_prompts(w)
    lens = sorted(len(p) for p in P)
    # lengths that straddle many 64-position chunks and differ per sequence
    assert len(set(lens)) == len(lens) and lens[-1] - lens[0] > 64 * 8
    n_steps = 2 * w.update_every
    worst, rows = _run(w, P, n_steps)
    # every sequence logged at least one row per step
    assert len(rows) >= w.batch * n_steps
    assert {b for b, _, _, _ in rows} == set(range(w.batch))
    print("batch-8 ragged: rows", len(rows), "max |dlogit|", worst)


def test_long_prompt_every_step_against_oracle():
    w = _reduced("7b-16k", prompt_len=(4096, 4096))
    P = make_prompts(w)
    assert len(P[0]) == 4096 and w.k_spec == 8
    n_steps = 2 * w.update_every
    worst, rows = _run(w, P, n_steps)
    assert len(rows) >= n_steps
    print("4096-token prompt: rows", len(rows), "max |dlogit|", worst)
