"""The persistent projection chain (runtime option `persistent`; here with the
draft phase on the per-kernel path, runtime option megakernel = 0).

With the option, a bf16 decode pass runs each layer's O, gate/up and down
projections and the next layer's QKV as one persistent launch.  Its CTAs
split every projection's weight stream into equal contiguous K ranges, and
the phase boundaries pass through release/acquire counters.  Checked through
the C-ABI:

* the chain is in effect (stats: persistent_ctas > 0);
* losslessness (Sec. 3.3): the DVI stream equals the GPU's own greedy
  autoregressive stream, with the drafter training online.  This runs on a
  small bf16 model whose phases have fewer K blocks than CTAs, on 1B (GQA)
  and on 7B, and with the bonus row;
* teacher-forced verify logits against the oracle within 3e-2 (float32 on
  the bf16-rounded weights, bf16 KV cache);
* the ragged 8-sequence batch (40 verify rows) over two prompt waves;
* the chain and the per-kernel path give the same verify logits up to
  summation order.
"""
import numpy as np
import pytest
import torch

from oracle import OracleModel
from workloads import workload, make_prompts
from gpu_helpers import engine_for, rounded_weights, teacher_forced_logits
from test_gpu_decode import _bf16_case
from test_gpu_full_size import GEN, _capacity, _weights

pytestmark = pytest.mark.gpu


def _engine(w, dw, max_seq_len, persistent=True):
    from paper_2510_05421_gb300 import DVIEngine
    return DVIEngine(w.shape, w.dtype, dw, batch=w.batch, k_spec=w.k_spec, split_k=w.split_k,
                     lora_rank=w.lora_rank, lora_gamma=w.lora_gamma, max_seq_len=max_seq_len,
                     log_steps=w.update_every, persistent=persistent, megakernel=False)


def _first_step_verify_logits(eng, w, P):
    eng.generate(P, 10 ** 6, max_steps=1, log=True)
    eng.sync()
    meta = eng.buffer("LOG_META", torch.int32).view(-1, 6).cpu().numpy()
    lg = eng.buffer("LOG_LOGITS", torch.float32).view(-1, w.shape.vocab).cpu().numpy()
    rows = [i for i in range(w.k_spec) if meta[i, 0]]
    assert rows and rows == list(range(len(rows)))
    return lg[rows], meta[rows]


def test_small_bf16_lossless_and_teacher_forced():
    w = _bf16_case()
    P = make_prompts(w)
    eng, W, _ = engine_for(w, persistent=True, megakernel=False)
    ar = eng.generate_ar(P, w.gen_tokens)[0]
    st = eng.stats()
    eng.close()
    assert st["persistent_ctas"] > 0
    eng, W, _ = engine_for(w, W=W, persistent=True, megakernel=False)
    toks, mats, _, _ = eng.generate(P, w.gen_tokens, update_every=w.update_every, hyper=w.update)
    st = eng.stats()
    eng.close()
    assert st["device_status"] == 0, st["device_flags"]
    assert st["updates"] >= 2
    assert toks[0] == list(ar)
    assert ((mats >= 0) & (mats <= w.k_spec)).all()
    eng, _, _ = engine_for(w, W=W, persistent=True, megakernel=False)
    lg, _ = _first_step_verify_logits(eng, w, P)
    eng.close()
    model = OracleModel(rounded_weights(W), w.shape, w.lora_gamma, kv_dtype="bf16")
    seq = np.concatenate([P[0], np.array(toks[0][:len(lg)], dtype=np.int32)])
    ref = teacher_forced_logits(model, seq)
    n0 = len(P[0])
    for i in range(len(lg)):
        err = np.abs(lg[i] - ref[n0 + i]).max()
        assert err < 3e-2, (i, err)


def test_small_bf16_bonus_lossless():
    w = _bf16_case()
    P = make_prompts(w)
    eng, W, _ = engine_for(w, persistent=True, megakernel=False)
    ar = eng.generate_ar(P, w.gen_tokens)[0]
    eng.close()
    eng, W, _ = engine_for(w, W=W, bonus=True, persistent=True, megakernel=False,
                           max_seq_len=len(P[0]) + 6 * w.gen_tokens + 16)
    toks, _, _, _ = eng.generate(P, w.gen_tokens, update_every=w.update_every, hyper=w.update)
    st = eng.stats()
    eng.close()
    assert st["device_status"] == 0, st["device_flags"]
    assert st["persistent_ctas"] > 0
    assert toks[0] == list(ar)


@pytest.mark.parametrize("name", ["1b", "7b"])
def test_full_size_lossless_teacher_forced_and_per_kernel_agreement(name):
    w = workload(name)
    W, dw = _weights(name)
    P = make_prompts(w)
    cap = _capacity(w, P)
    eng = _engine(w, dw, cap)
    ar = eng.generate_ar(P, GEN)
    eng.close()
    eng = _engine(w, dw, cap)
    toks, mats, _, _ = eng.generate(P, GEN, update_every=w.update_every, hyper=w.update)
    st = eng.stats()
    eng.close()
    assert st["device_status"] == 0, st["device_flags"]
    assert st["persistent_ctas"] > 0
    for b in range(len(P)):
        assert toks[b] == list(ar[b]), b
    assert ((mats >= 0) & (mats <= w.k_spec)).all()
    # first step: chain logits against the oracle and against the per-kernel path
    eng = _engine(w, dw, cap)
    lg, meta = _first_step_verify_logits(eng, w, P)
    eng.close()
    eng = _engine(w, dw, cap, persistent=False)
    lg0, meta0 = _first_step_verify_logits(eng, w, P)
    eng.close()
    n = min(len(lg), len(lg0))
    assert np.abs(lg[:n] - lg0[:n]).max() < 1e-2
    model = OracleModel(rounded_weights(W), w.shape, w.lora_gamma, dtype=np.float32, kv_dtype="bf16")
    seq = np.concatenate([P[0], np.array(toks[0][:len(lg)], dtype=np.int32)])
    ref = teacher_forced_logits(model, seq)
    n0 = len(P[0])
    for i in range(len(lg)):
        err = np.abs(lg[i] - ref[n0 + i]).max()
        assert err < 3e-2, (i, err)
        assert int(np.argmax(lg[i])) == int(meta[i, 5])


def test_7b_batch8_ragged_two_waves():
    w = workload("7b-b8")
    _, dw = _weights("7b")
    waves = [make_prompts(w, wave) for wave in range(2)]
    cap = max(_capacity(w, P) for P in waves)
    eng = _engine(w, dw, cap)
    ar = [eng.generate_ar(P, GEN) for P in waves]
    eng.close()
    eng = _engine(w, dw, cap)
    for P, ref in zip(waves, ar):
        toks, _, _, _ = eng.generate(P, GEN, update_every=w.update_every, hyper=w.update)
        for b in range(w.batch):
            assert toks[b] == list(ref[b]), b
    st = eng.stats()
    eng.close()
    assert st["device_status"] == 0, st["device_flags"]
    assert st["persistent_ctas"] > 0
