"""The decode path at the full sizes of the measured workloads.

Shapes, split points, K, prompt lengths and launch configuration (CUDA
graphs, KV capacity as the benchmark sizes it) are the workloads' own; only
the number of generated tokens is cut.  At these sizes the oracle is used on
sampled outputs, and the rest is checked through properties that hold at any
size:

* losslessness (Sec. 3.3): the committed DVI stream equals the GPU's own
  greedy autoregressive stream bit for bit, with the drafter training online;
* teacher-forced verifier logits of every logged verify row of an 8-step
  run with the drafter training, against the oracle (float32 arithmetic on
  the bf16-rounded weights, bf16 KV cache; float32 keeps the 7B oracle
  within minutes, and its rounding is far below the bound), within 3e-2,
  with y* the row's argmax (1B and 7B);
* the 8-sequence ragged batch over two prompt waves whose drafter state
  carries over, and the 16K-token prompt with K = 8;
* one LoRA update at the 7B shape: dA, dB against the oracle's closed-form
  gradients on the GPU's own logged tuples, within 1e-3.
"""
import functools

import numpy as np
import pytest
import torch

from oracle import OracleModel
from workloads import workload, make_weights, make_prompts
from gpu_helpers import rounded_weights, run_logged_steps, check_rows_against_oracle

pytestmark = pytest.mark.gpu
GEN = 24


@functools.lru_cache(maxsize=1)
def _weights(name):
    from paper_2510_05421_gb300 import DeviceWeights
    w = workload(name)
    W = make_weights(w)
    return W, DeviceWeights.from_host(W, w.dtype)


def _engine(w, dw, max_seq_len):
    from paper_2510_05421_gb300 import DVIEngine
    return DVIEngine(w.shape, w.dtype, dw, batch=w.batch, k_spec=w.k_spec, split_k=w.split_k,
                     lora_rank=w.lora_rank, lora_gamma=w.lora_gamma, max_seq_len=max_seq_len,
                     log_steps=w.update_every)


def _capacity(w, P):
    # as the benchmark sizes the KV cache: prompt + K per generated token + slack
    return max(len(p) for p in P) + w.gen_tokens * w.k_spec + 64


def _lossless(w, dw, P, n_gen=GEN):
    eng = _engine(w, dw, _capacity(w, P))
    ar = eng.generate_ar(P, n_gen)
    eng.close()
    eng = _engine(w, dw, _capacity(w, P))
    toks, mats, _, _ = eng.generate(P, n_gen, update_every=w.update_every, hyper=w.update)
    st = eng.stats()
    eng.close()
    assert st["device_status"] == 0, st["device_flags"]
    for b in range(len(P)):
        assert toks[b] == list(ar[b]), b
    assert ((mats >= 0) & (mats <= w.k_spec)).all()
    return toks, mats


def _every_step_logits(w, dw, W, P, n_steps=8):
    """Verify-row logits of every step of an 8-step run: GPU log against the oracle."""
    eng = _engine(w, dw, _capacity(w, P))
    toks, rows = run_logged_steps(eng, P, n_steps, update_every=w.update_every, hyper=w.update)
    st = eng.stats()
    eng.close()
    assert st["device_status"] == 0, st["device_flags"]
    assert len(rows) >= n_steps
    model = OracleModel(rounded_weights(W), w.shape, w.lora_gamma, dtype=np.float32, kv_dtype="bf16")
    check_rows_against_oracle(model, P, toks, rows, 3e-2)


def test_1b_gqa_lossless_and_teacher_forced():
    w = workload("1b")
    W, dw = _weights("1b")
    P = make_prompts(w)
    _lossless(w, dw, P)
    _every_step_logits(w, dw, W, P)


def test_7b_lossless_and_teacher_forced():
    w = workload("7b")
    W, dw = _weights("7b")
    P = make_prompts(w)
    _lossless(w, dw, P)
    _every_step_logits(w, dw, W, P)


def test_7b_batch8_ragged_two_waves():
    w = workload("7b-b8")
    _, dw = _weights("7b")
    waves = [make_prompts(w, wave) for wave in range(2)]
    for P in waves:
        assert len({len(p) for p in P}) > 1
    cap = max(_capacity(w, P) for P in waves)
    ar = []
    eng = _engine(w, dw, cap)
    for P in waves:
        ar.append(eng.generate_ar(P, GEN))
    eng.close()
    # one context for both waves: the drafter's training carries over
    eng = _engine(w, dw, cap)
    for P, ref in zip(waves, ar):
        toks, mats, _, _ = eng.generate(P, GEN, update_every=w.update_every, hyper=w.update)
        for b in range(w.batch):
            assert toks[b] == list(ref[b]), b
        assert ((mats >= 0) & (mats <= w.k_spec)).all()
    st = eng.stats()
    eng.close()
    assert st["device_status"] == 0, st["device_flags"]
    assert st["updates"] >= 2


def test_7b_16k_prompt_lossless():
    w = workload("7b-16k")
    _, dw = _weights("7b")
    P = make_prompts(w)
    assert len(P[0]) == 16384
    _lossless(w, dw, P, n_gen=16)


def test_7b_update_gradients_on_logged_tuples():
    """One LoRA update at the 7B shape: dA, dB against the oracle's closed-form
    gradients on the GPU's own logged tuples (Sec. 3.4), within 1e-3 of the
    largest entry."""
    from oracle.update import grad_logits, head_logits, objective_weights, param_grads
    from workloads import UpdateHyper
    from gpu_helpers import logged_u
    from workloads.gen import bf16_round
    w = workload("7b")
    W, dw = _weights("7b")
    rng = np.random.default_rng(5)
    a0 = (rng.standard_normal(W.lora_a.shape) * 0.05).astype(np.float32)
    b_saved = dw.lora_b.clone()
    dw.lora_a.copy_(torch.from_numpy(a0))
    hyper = UpdateHyper(objective="dvi", lr=1e-3, t_warmup=0, t_ramp=0, w_ent=0.01, w_ce=0.05)
    P = make_prompts(w)
    eng = _engine(w, dw, _capacity(w, P))
    eng.generate(P, 10 ** 6, max_steps=w.update_every, log=True)
    eng.sync()
    V, d = w.shape.vocab, w.shape.d_model
    meta = eng.buffer("LOG_META", torch.int32).view(-1, 6).cpu().numpy()
    lg = eng.buffer("LOG_LOGITS", torch.float32).view(-1, V).cpu().numpy().astype(np.float64)
    lu = logged_u(eng, w)
    b0 = dw.lora_b.cpu().numpy().astype(np.float64)
    eng.update(hyper)
    eng.sync()
    ga = eng.buffer("GRAD_A", torch.float32).view(V, -1).cpu().numpy()
    gb = eng.buffer("GRAD_B", torch.float32).view(w.lora_rank, -1).cpu().numpy()
    st = eng.stats()
    eng.close()
    dw.lora_a.zero_()                 # the cached weights serve the other tests
    dw.lora_b.copy_(b_saved)
    assert st["device_status"] == 0, st["device_flags"]
    rows = np.nonzero(meta[:, 0])[0]
    assert len(rows) > 0
    w_s = bf16_round(W.draft_head).astype(np.float64)
    A = a0.astype(np.float64)
    Z = head_logits(lu[rows], w_s, A, b0, w.lora_gamma)
    G = grad_logits(Z, lg[rows], meta[rows, 1], meta[rows, 5], meta[rows, 2].astype(np.float64),
                    objective_weights(0, hyper), 0.0)
    ref = param_grads(G, lu[rows], A, b0, w.lora_gamma)
    for name, got in (("A", ga), ("B", gb)):
        rel = np.abs(got - ref[name]).max() / np.abs(ref[name]).max()
        assert rel < 1e-3, (name, rel)
