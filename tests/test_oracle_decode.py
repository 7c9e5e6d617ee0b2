"""Pins of the oracle's DVI loop (Sec. 3.1, Sec. 3.3).

* Losslessness: with a frozen verifier the committed stream equals greedy AR
  decoding of the full model, whatever the drafter proposes -- checked by
  brute force over seeds, split points k, block lengths K, the bonus-token
  variant and with online updates on.
* Bounds: 0 <= m <= K; each step commits min(m+1, K) tokens (m+1 with bonus).
* Full acceptance: with the drafter equal to the whole model (k = L,
  W^S = W^V, A = 0) every drafted token is accepted.
* Verify rows equal the AR logits at the same positions.
* Rewards per step are 1..1 then 0 at the first reject (Sec. 3.3).
"""
import numpy as np
import pytest

from oracle import OracleModel, greedy_ar, dvi_generate, DrafterUpdater
from oracle.decode import prefill
from workloads import make_weights, make_prompts, workload, tiny_shape, UpdateHyper

SMALL = tiny_shape(n_layers=4, d_model=64, n_heads=4, n_kv_heads=2, head_dim=16,
                   d_ffn=96, vocab=128)


def _setup(seed, shape=SMALL, scale=0.1, gen=24, plen=12, rank=4):
    w = workload("tiny").with_(shape=shape, weight_seed=seed, prompt_seed=100 + seed,
                               prompt_len=(plen, plen), gen_tokens=gen, lora_rank=rank,
                               scaled_layers=(3, 4), scale=scale)
    W = make_weights(w, threads=2)
    return w, W, make_prompts(w)


@pytest.mark.parametrize("seed", range(4))
@pytest.mark.parametrize("k", [1, 2, 3])
@pytest.mark.parametrize("K", [1, 3, 6])
def test_lossless_against_greedy_ar(seed, k, K):
    w, W, P = _setup(seed)
    m = OracleModel(W, w.shape, 1.0)
    ar = greedy_ar(m, P[0], w.gen_tokens)
    res = dvi_generate(m, P, w.gen_tokens, k, K)
    np.testing.assert_array_equal(res.tokens[0], ar)
    for s in res.steps:
        assert 0 <= s.m <= K
        assert len(s.committed) == min(s.m + 1, K)
        assert s.committed[:s.m] == s.drafts[:s.m]
        if s.m < K:
            assert s.committed[-1] == s.ystar[s.m] and s.drafts[s.m] != s.ystar[s.m]


@pytest.mark.parametrize("seed", range(3))
def test_lossless_with_bonus_and_updates(seed):
    w, W, P = _setup(seed, gen=40)
    for bonus in (False, True):
        m = OracleModel(W, w.shape, 1.0)
        ar = greedy_ar(m, P[0], w.gen_tokens)
        upd = DrafterUpdater(m, UpdateHyper(objective="dvi", lr=5e-2, t_warmup=1, t_ramp=2))
        res = dvi_generate(m, P, w.gen_tokens, 2, 4, update_every=2, updater=upd, bonus=bonus)
        np.testing.assert_array_equal(res.tokens[0], ar)
        assert len(res.updates) >= 2
        for s in res.steps:
            assert len(s.committed) == (s.m + 1 if bonus else min(s.m + 1, 4))


def test_lossless_batch_of_ragged_sequences():
    """Sequences stepped together share one buffer and drafter but stay lossless."""
    w, W, _ = _setup(3, gen=20)
    w = w.with_(batch=3, prompt_len=(5, 15))
    P = make_prompts(w)
    assert len({len(p) for p in P}) > 1
    m = OracleModel(W, w.shape, 1.0)
    refs = [greedy_ar(OracleModel(W, w.shape, 1.0), p, 20) for p in P]
    upd = DrafterUpdater(m, UpdateHyper(objective="kl", lr=1e-2))
    res = dvi_generate(m, P, 20, 2, 3, update_every=2, updater=upd)
    for b in range(3):
        np.testing.assert_array_equal(res.tokens[b], refs[b])


@pytest.mark.parametrize("K", [1, 4, 7])
def test_full_acceptance_when_drafter_is_whole_model(K):
    w, W, P = _setup(1, scale=1.0)
    W.lora_a[:] = 0.0
    W.draft_head[:] = W.lm_head
    m = OracleModel(W, w.shape, 1.0)
    L = w.shape.n_layers
    res = dvi_generate(m, P, w.gen_tokens, L, K)
    assert all(s.m == K for s in res.steps)
    np.testing.assert_array_equal(res.tokens[0], greedy_ar(m, P[0], w.gen_tokens))


def test_verify_rows_equal_ar_logits():
    w, W, P = _setup(2)
    m = OracleModel(W, w.shape, 1.0)
    ar, ar_logits, _ = greedy_ar(m, P[0], w.gen_tokens, return_logits=True)
    res = dvi_generate(m, P, w.gen_tokens, 2, 4, keep_logits=True)
    pos = 1                                   # index into ar: token after the prefill one
    for s in res.steps:
        for i in range(len(s.committed)):
            if pos + i >= len(ar):
                break
            if i <= s.m:
                np.testing.assert_allclose(s.verify_logits[i], ar_logits[pos + i],
                                           rtol=1e-10, atol=1e-10)
        pos += len(s.committed)


def test_reward_pattern_and_tuple_fields():
    w, W, P = _setup(0, gen=30)
    m = OracleModel(W, w.shape, 1.0)
    got = []

    class Rec:
        def update(self, tuples):
            got.append(list(tuples))
            return {}

    res = dvi_generate(m, P, w.gen_tokens, 2, 4, update_every=1, updater=Rec())
    assert len(got) == len(res.steps)
    for s, tup in zip(res.steps, got):
        rs = [t.r for t in tup]
        assert rs == [1] * s.m + ([0] if s.m < 4 else [])
        assert [t.i for t in tup] == list(range(1, len(tup) + 1))
        assert [t.a for t in tup] == s.drafts[:len(tup)]
        assert [t.ystar for t in tup] == s.ystar[:len(tup)]
        assert tup[0].prev_id != -1


def test_prefill_first_token_is_ar_first_token():
    w, W, P = _setup(5)
    m = OracleModel(W, w.shape, 1.0)
    tok, _ = prefill(m, m.new_cache(64), P[0])
    assert tok == greedy_ar(m, P[0], 3)[0]
