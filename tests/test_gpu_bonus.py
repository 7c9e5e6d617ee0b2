"""The bonus-row verify (K + 1 verify rows, m + 1 tokens committed every step).

Sec. 3.3 emits the verifier's correction y*_{n+m+1} after the accepted
prefix; with only the K drafted rows verified that token exists for m < K.
The bonus variant runs one more shallow pass on t~_K and verifies a
(K+1)-th row, so y*_{n+K+1} is also available at m = K.  Checked through
the C-ABI against the oracle's bonus run: committed tokens and accept
lengths bit-exact in f32 (with the drafter updating), the stream equal to
greedy AR, m = K and K + 1 commits when the drafter is the whole model, and
bf16 DVI == GPU AR.
"""
import numpy as np
import pytest

from oracle import OracleModel, dvi_generate, greedy_ar, DrafterUpdater
from workloads import workload, make_weights, make_prompts
from gpu_helpers import engine_for
from test_gpu_decode import _bf16_case

pytestmark = pytest.mark.gpu


def test_tiny_f32_bonus_matches_oracle():
    w = workload("tiny")
    W = make_weights(w)
    P = make_prompts(w)
    eng, _, _ = engine_for(w, W=W, bonus=True, max_seq_len=32 + 5 * w.gen_tokens + 16)
    toks, mats, _, _ = eng.generate(P, w.gen_tokens, update_every=w.update_every, hyper=w.update)
    st = eng.stats()
    eng.close()
    assert st["device_status"] == 0, st["device_flags"]
    m = OracleModel(W, w.shape, w.lora_gamma)
    res = dvi_generate(m, P, w.gen_tokens, w.split_k, w.k_spec, w.update_every, DrafterUpdater(m, w.update),
                       bonus=True)
    assert toks[0] == list(res.tokens[0])
    assert list(mats[:, 0]) == [s.m for s in res.steps]
    assert st["updates"] == len(res.updates)
    m2 = OracleModel(W, w.shape, w.lora_gamma)
    assert toks[0] == list(greedy_ar(m2, P[0], w.gen_tokens))


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_bonus_full_acceptance_commits_k_plus_one(dtype):
    w = workload("tiny").with_(dtype=dtype, split_k=4, gen_tokens=40, scaled_layers=(), scale=1.0)
    W = make_weights(w)
    W.lora_a[:] = 0.0
    eng, _, _ = engine_for(w, W=W, bonus=True)
    eng.generate(make_prompts(w), 1)          # prefill only
    for _ in range(4):
        ids, cnt, acc = eng.step()
        eng.sync()                             # the step ran on the engine's stream
        assert (acc.cpu().numpy() == w.k_spec).all()
        assert (cnt.cpu().numpy() == w.k_spec + 1).all()
    st = eng.stats()
    eng.close()
    assert st["device_status"] == 0, st["device_flags"]


def test_bf16_bonus_equals_gpu_ar():
    w = _bf16_case()
    P = make_prompts(w)
    eng, W, _ = engine_for(w)
    ar = eng.generate_ar(P, w.gen_tokens)[0]
    eng.close()
    eng, W, _ = engine_for(w, W=W, bonus=True, max_seq_len=len(P[0]) + 6 * w.gen_tokens + 16)
    toks, mats, _, _ = eng.generate(P, w.gen_tokens, update_every=w.update_every, hyper=w.update)
    st = eng.stats()
    eng.close()
    assert st["device_status"] == 0, st["device_flags"]
    assert toks[0] == list(ar)
