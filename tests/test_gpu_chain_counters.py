"""Completion-counter chaining of decode passes (runtime option `chain_counters`;
here with the draft phase on the per-kernel path, runtime option megakernel = 0).

With the option, consecutive projection, attention and head launches of a
bf16 draft pass, verify pass or AR step wait for a per-launch completion
counter (every CTA of the predecessor adds 1 with release semantics after its
last write; the successor polls with acquire semantics) instead of the
predecessor's whole grid.  The kernels and their arithmetic are unchanged, so
everything a step produces must be bit-identical to the default path.  Checked
through the C-ABI:

* the tiny bf16 model with online drafter updates and with the bonus row:
  committed tokens, accept lengths, logged verifier logits, logged drafter
  logits z and the LoRA factors after the updates are bitwise equal, and no
  wait timed out;
* the 1B GQA workload at full size: the same, plus the greedy AR stream;
* the DVI stream with chaining equals the GPU's greedy AR stream (Sec. 3.3).
"""
import numpy as np
import pytest
import torch

from workloads import workload, make_prompts
from gpu_helpers import engine_for
from test_gpu_decode import _bf16_case

pytestmark = pytest.mark.gpu


def _run(w, W, chain, bonus=False, steps=None):
    eng, W, dw = engine_for(w, W=W, chain_counters=chain, bonus=bonus, megakernel=False)
    P = make_prompts(w)
    toks, mats, _, _ = eng.generate(P, w.gen_tokens, update_every=w.update_every, hyper=w.update)
    # a last step with logging on and no update after it: the replay buffer
    # holds this step's verifier logits and drafter logits
    eng.generate(P, 10 ** 6, max_steps=1, log=True)
    eng.sync()
    st = eng.stats()
    out = dict(toks=toks, mats=np.asarray(mats),
               logits=eng.buffer("LOG_LOGITS", torch.float32).cpu().numpy().copy(),
               z=eng.buffer("Z", torch.float32).cpu().numpy().copy(),
               meta=eng.buffer("LOG_META", torch.int32).cpu().numpy().copy(),
               lora_a=dw.lora_a.cpu().numpy().copy(), lora_b=dw.lora_b.cpu().numpy().copy(), stats=st)
    eng.close()
    return out, W


def _same(a, b):
    assert a["stats"]["device_status"] == 0, a["stats"]["device_flags"]
    assert b["stats"]["device_status"] == 0, b["stats"]["device_flags"]
    assert a["toks"] == b["toks"]
    assert np.array_equal(a["mats"], b["mats"])
    assert np.array_equal(a["meta"], b["meta"])
    assert np.array_equal(a["logits"], b["logits"])
    assert np.array_equal(a["z"], b["z"])
    assert np.array_equal(a["lora_a"], b["lora_a"])
    assert np.array_equal(a["lora_b"], b["lora_b"])


@pytest.mark.parametrize("bonus", [False, True])
def test_small_bf16_bit_identical(bonus):
    w = _bf16_case()
    on, W = _run(w, None, True, bonus=bonus)
    off, _ = _run(w, W, False, bonus=bonus)
    assert on["stats"]["updates"] >= 2
    _same(on, off)


def test_1b_bit_identical_and_lossless():
    w = workload("1b").with_(gen_tokens=48)
    on, W = _run(w, None, True)
    off, _ = _run(w, W, False)
    _same(on, off)
    P = make_prompts(w)
    eng, _, _ = engine_for(w, W=W, chain_counters=True, megakernel=False)
    ar = eng.generate_ar(P, w.gen_tokens)
    st = eng.stats()
    eng.close()
    assert st["device_status"] == 0, st["device_flags"]
    for b in range(len(P)):
        assert on["toks"][b][:w.gen_tokens] == list(ar[b])[:w.gen_tokens]
