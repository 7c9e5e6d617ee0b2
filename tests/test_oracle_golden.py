"""The oracle still reproduces its stored tiny-workload run (tests/golden)."""
import json
import os

import numpy as np

from oracle import OracleModel, greedy_ar, dvi_generate, DrafterUpdater
from workloads import workload, make_weights, make_prompts

GOLD = os.path.join(os.path.dirname(__file__), "golden", "tiny_dvi.json")


def test_tiny_golden_run():
    g = json.load(open(GOLD))
    w = workload("tiny")
    W = make_weights(w, threads=4)
    P = make_prompts(w)
    assert [int(x) for x in P[0]] == g["prompt"]
    m = OracleModel(W, w.shape, w.lora_gamma)
    res = dvi_generate(m, P, w.gen_tokens, w.split_k, w.k_spec, w.update_every,
                       DrafterUpdater(m, w.update))
    assert g["ar_tokens"] == g["dvi_tokens"]                    # lossless
    assert [int(x) for x in res.tokens[0]] == g["dvi_tokens"]
    assert [s.m for s in res.steps] == g["accept_lengths"]
    np.testing.assert_allclose([u["loss"] for u in res.updates], g["update_losses"],
                               rtol=1e-9)
