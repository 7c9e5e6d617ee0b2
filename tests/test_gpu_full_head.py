"""Full-head drafter training (W^(S) itself, dW = G^T U) through the C-ABI.

The LoRA parameterisation is the paper's default (Sec. 3.2); training the
base projection W^(S) directly is the second parameterisation of the update
of Sec. 3.4.  Checked against the oracle:

* f32: the logged tuples, dL/dW^(S) within 1e-3 (relative to its largest
  entry), W^(S) after the Adam step, and the accept lengths of the next
  update period, which depend on the drafts of the updated head.
* bf16: the decode stays lossless while W^(S) trains (DVI == GPU greedy AR),
  dL/dW^(S) of one update against the oracle on the GPU's own logged tuples,
  and the bf16 head equals the rounding of the f32 master.
"""
import numpy as np
import pytest
import torch

from oracle import OracleModel, dvi_generate
from oracle.update import AdamState, adam_step, grad_logits, head_logits, objective_weights, param_grads
from workloads import workload, make_weights, make_prompts, UpdateHyper
from gpu_helpers import engine_for, logged_u, rounded_weights
from test_gpu_decode import Recorder, _bf16_case

pytestmark = pytest.mark.gpu


def _check_step(w_new, w_old, g_ref, lr):
    """W^(S) after one Adam step against the oracle's step from the same W and dW."""
    ref = w_old.astype(np.float64).copy()
    adam_step(ref, g_ref, AdamState(np.zeros_like(ref), np.zeros_like(ref)), lr, 0.9, 0.999, 1e-8)
    diff = np.abs(w_new - ref)
    # entries whose gradient is far above eps move by ~lr exactly; the rest by
    # at most lr whatever the rounding of their tiny gradient
    big = np.abs(g_ref) > 1e-4 * np.abs(g_ref).max()
    assert big.mean() > 0.5
    assert diff[big].max() < 1e-6, diff[big].max()
    assert diff.max() <= 2 * lr + 1e-6


@pytest.mark.parametrize("rank", [8, 0])
def test_tiny_f32_full_head_gradient_step_and_next_drafts(rank):
    w = workload("tiny").with_(lora_rank=rank)
    hyper = UpdateHyper(objective="dvi", lr=1e-3, t_warmup=0, t_ramp=0, w_ent=0.01, w_ce=0.05)
    W = make_weights(w)
    if rank:
        W.lora_a[:] = np.random.default_rng(11).standard_normal(W.lora_a.shape).astype(np.float32) * 0.05
    eng, _, dw = engine_for(w, W=W, head_mode=1)
    P = make_prompts(w)
    U = w.update_every
    w_before = dw.draft_head.cpu().numpy().copy()
    _, mats1, _, _ = eng.generate(P, 10 ** 6, max_steps=U, log=True)
    eng.sync()
    meta = eng.buffer("LOG_META", torch.int32).view(-1, 6).cpu().numpy()
    eng.update(hyper, keep_grad_w=True)
    eng.sync()
    gw = eng.buffer("GRAD_W", torch.float32).view(w.shape.vocab, -1).cpu().numpy()
    w_after = dw.draft_head.cpu().numpy().copy()
    st = eng.stats()
    assert st["device_status"] == 0, st["device_flags"]
    eng.close()

    m = OracleModel(W, w.shape, w.lora_gamma)
    rec = Recorder(m, hyper, full=True)
    res = dvi_generate(m, P, 10 ** 6, w.split_k, w.k_spec, U, rec, max_steps=2 * U)
    assert [s.m for s in res.steps[:U]] == list(mats1[:, 0])
    assert int(meta[:, 0].sum()) == len(rec.buffers[0])
    info = res.updates[0]
    np.testing.assert_allclose(st["last_loss"], info["loss"], rtol=1e-4, atol=1e-6)
    g_ref = info["grads"]["W_s"]
    rel = np.abs(gw - g_ref).max() / np.abs(g_ref).max()
    assert rel < 1e-3, rel
    _check_step(w_after, w_before, g_ref, hyper.lr)

    # a second period decoded with the trained head: same drafts, same m
    eng, _, dw = engine_for(w, W=W, head_mode=1)
    _, mats, _, _ = eng.generate(P, 10 ** 6, update_every=U, hyper=hyper, max_steps=2 * U, log=True)
    eng.close()
    assert [s.m for s in res.steps] == list(mats[:, 0])


def test_bf16_full_head_lossless_and_gradient():
    w = _bf16_case()
    P = make_prompts(w)
    eng, W, _ = engine_for(w)
    ar = eng.generate_ar(P, w.gen_tokens)[0]
    eng.close()

    eng, W, dw = engine_for(w, W=W, head_mode=1)
    toks, mats, _, _ = eng.generate(P, w.gen_tokens, update_every=w.update_every, hyper=w.update)
    st = eng.stats()
    assert st["device_status"] == 0, st["device_flags"]
    assert st["updates"] >= 2
    assert toks[0] == list(ar)
    eng.close()

    # one update on the GPU's own logged tuples against the oracle's dW
    hyper = UpdateHyper(objective="dvi", lr=1e-3, t_warmup=0, t_ramp=0, w_ent=0.01, w_ce=0.05)
    eng, W, dw = engine_for(w, W=W, head_mode=1)
    eng.generate(P, 10 ** 6, max_steps=w.update_every, log=True)
    eng.sync()
    V, d = w.shape.vocab, w.shape.d_model
    meta = eng.buffer("LOG_META", torch.int32).view(-1, 6).cpu().numpy()
    lg = eng.buffer("LOG_LOGITS", torch.float32).view(-1, V).cpu().numpy().astype(np.float64)
    lu = logged_u(eng, w)
    w_s = dw.draft_head.float().cpu().numpy().astype(np.float64)
    eng.update(hyper, keep_grad_w=True)
    eng.sync()
    gw = eng.buffer("GRAD_W", torch.float32).view(V, d).cpu().numpy()
    w_new = dw.draft_head.float().cpu().numpy()
    eng.close()
    rows = np.nonzero(meta[:, 0])[0]
    assert len(rows) > 0
    Wr = rounded_weights(W)
    Z = head_logits(lu[rows], w_s, Wr.lora_a.astype(np.float64), Wr.lora_b.astype(np.float64), w.lora_gamma)
    wts = objective_weights(0, hyper)
    G = grad_logits(Z, lg[rows], meta[rows, 1], meta[rows, 5], meta[rows, 2].astype(np.float64), wts, 0.0)
    g_ref = param_grads(G, lu[rows], None, None, w.lora_gamma, full=True)["W_s"]
    rel = np.abs(gw - g_ref).max() / np.abs(g_ref).max()
    assert rel < 1e-3, rel
    # the bf16 head moved by about lr per entry and is a bf16 rounding
    step = np.abs(w_new - w_s)
    assert np.median(step) > 0.25 * hyper.lr and step.max() < 4 * hyper.lr
    assert torch.equal(torch.from_numpy(w_new).bfloat16().float(), torch.from_numpy(w_new))
