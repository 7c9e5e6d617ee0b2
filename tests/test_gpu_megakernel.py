"""The draft-phase megakernel (runtime option `megakernel`).

With the option, one persistent launch runs the whole draft phase of a decode
step (every draft pass's k layers, the drafter head and its argmax, the
hand-off of h_k to the verify rows), and the greedy AR step runs its first k
layers through the same kernel.  Checked through the C-ABI:

* the kernel is in effect (stats: megakernel_ctas > 0) and no wait timed out
  (it is the default for eligible bf16 contexts; the per-kernel draft path,
  megakernel = 0, is checked the same way on the tiny model);
* losslessness (Sec. 3.3): the DVI stream equals the GPU's greedy AR stream
  bit for bit with the drafter training online: tiny bf16 (head_dim 128,
  eagerly and with graphs), the bonus row, head_dim 64 with GQA groups of 4
  and 8, two ragged sequences in one launch, the 1B and 7B workloads at full size,
  the 7B shape with a 16K-token prompt (64 key / value chunks per attention
  unit);
* the verifier logits of the first step's verify rows (whose inputs h_k the
  kernel computed) against the oracle's teacher-forced logits on the
  bf16-rounded weights with a bf16 KV cache, within 3e-2 (every logged row of
  8 steps for 1B);
* the drafter of the first draft pass against the oracle: the logged u =
  RMSNorm_final(h_k) and the logged drafter logits z = W^S u + gamma A (B u)
  within 3e-2 (Sec. 3.1 draft head).
"""
import numpy as np
import pytest
import torch

from oracle import OracleModel
from workloads import workload, make_weights, make_prompts, tiny_shape
from gpu_helpers import (engine_for, rounded_weights, teacher_forced_logits, logged_u, run_logged_steps,
                         check_rows_against_oracle)
from test_gpu_decode import _bf16_case

pytestmark = pytest.mark.gpu


def _lossless(w, W=None, max_seq_len=None, mk=True, **kw):
    P = make_prompts(w)
    eng, W, _ = engine_for(w, W=W, megakernel=mk, max_seq_len=max_seq_len, **kw)
    ar = eng.generate_ar(P, w.gen_tokens)
    st = eng.stats()
    eng.close()
    assert (st["megakernel_ctas"] > 0) == mk
    assert st["device_status"] == 0, st["device_flags"]
    eng, W, _ = engine_for(w, W=W, megakernel=mk, max_seq_len=max_seq_len, **kw)
    toks, mats, _, _ = eng.generate(P, w.gen_tokens, update_every=w.update_every, hyper=w.update)
    st = eng.stats()
    eng.close()
    assert st["device_status"] == 0, st["device_flags"]
    for b in range(len(P)):
        assert toks[b] == list(ar[b])[:w.gen_tokens], b
    assert ((mats >= 0) & (mats <= w.k_spec)).all()
    return W, P, st


def _first_step(w, W, P, max_seq_len=None, mk=True, **kw):
    """One logged step of a fresh engine: verify rows, z and u of the buffer."""
    eng, _, _ = engine_for(w, W=W, megakernel=mk, max_seq_len=max_seq_len, **kw)
    toks, _, _, _ = eng.generate(P, 10 ** 6, max_steps=1, log=True)
    eng.sync()
    V = w.shape.vocab
    meta = eng.buffer("LOG_META", torch.int32).view(-1, 6).cpu().numpy()
    lg = eng.buffer("LOG_LOGITS", torch.float32).view(-1, V).double().cpu().numpy()
    z = eng.buffer("Z", torch.float32).view(-1, V).double().cpu().numpy()
    u = logged_u(eng, w)
    st = eng.stats()
    eng.close()
    assert st["device_status"] == 0, st["device_flags"]
    return toks, meta, lg, z, u


def _check_first_step(w, W, P, tol=3e-2, **kw):
    toks, meta, lg, z, u = _first_step(w, W, P, **kw)
    model = OracleModel(rounded_weights(W), w.shape, w.lora_gamma, dtype=np.float32, kv_dtype="bf16")
    K, k = w.k_spec, w.split_k
    for b in range(len(P)):
        n0 = len(P[b])
        seq = np.concatenate([P[b], np.asarray(toks[b], dtype=np.int32)])
        ref = teacher_forced_logits(model, seq)
        rows = [i for i in range(K) if meta[b * K + i, 0]]
        assert rows and rows == list(range(len(rows)))
        for i in rows:
            err = np.abs(lg[b * K + i] - ref[n0 + i]).max()
            assert err < tol, (b, i, err)
        # the first draft pass reads the pending token at position n0
        cache = model.new_cache(n0 + 2)
        h = model.layers_range(0, k, model.embed(seq[:n0 + 1]), 0, cache)[n0]
        u_ref = model.final_norm(h[None])[0]
        z_ref = model.drafter_logits(h[None])[0]
        err_u = np.abs(u[b * K] - u_ref).max()
        err_z = np.abs(z[b * K] - z_ref).max()
        assert err_u < tol * max(1.0, np.abs(u_ref).max()), (b, err_u)
        assert err_z < tol, (b, err_z)


@pytest.mark.parametrize("graphs", [True, False])
def test_tiny_bf16_lossless_and_oracle(graphs):
    w = _bf16_case()
    W, P, st = _lossless(w, use_graphs=graphs)
    assert st["updates"] >= 2
    _check_first_step(w, W, P, use_graphs=graphs)


def test_tiny_bf16_per_kernel_draft_path():
    """The same checks with the draft phase one kernel per projection (megakernel = 0)."""
    w = _bf16_case()
    W, P, _ = _lossless(w, mk=False)
    _check_first_step(w, W, P, mk=False)


def test_tiny_bf16_bonus_lossless():
    w = _bf16_case()
    _lossless(w, bonus=True)


def test_head_dim_64_gqa4_lossless_and_oracle():
    shape = tiny_shape(n_layers=4, d_model=512, n_heads=8, n_kv_heads=2, head_dim=64, d_ffn=1408, vocab=4000)
    w = _bf16_case().with_(shape=shape)
    W, P, _ = _lossless(w)
    _check_first_step(w, W, P)


def test_head_dim_64_gqa8_lossless_and_oracle():
    """A GQA group of 8: the score and value MMAs take two head tiles (query
    heads 4..7 in A rows 8..15 and in o^T's second column tile)."""
    shape = tiny_shape(n_layers=4, d_model=1024, n_heads=16, n_kv_heads=2, head_dim=64, d_ffn=1408, vocab=4000)
    w = _bf16_case().with_(shape=shape)
    W, P, _ = _lossless(w)
    _check_first_step(w, W, P)


def test_two_ragged_sequences_lossless_and_oracle():
    w = _bf16_case().with_(batch=2, prompt_len=(9, 57), gen_tokens=40)
    P = make_prompts(w)
    assert len({len(p) for p in P}) == 2
    cap = max(len(p) for p in P) + w.k_spec * w.gen_tokens + 16
    W, P, _ = _lossless(w, max_seq_len=cap)
    _check_first_step(w, W, P, max_seq_len=cap)


def test_1b_full_size_lossless_and_every_step():
    w = workload("1b").with_(gen_tokens=24)
    W = make_weights(w)
    P = make_prompts(w)
    cap = max(len(p) for p in P) + w.gen_tokens * w.k_spec + 64
    _lossless(w, W=W, max_seq_len=cap)
    eng, _, _ = engine_for(w, W=W, megakernel=True, max_seq_len=cap)
    toks, rows = run_logged_steps(eng, P, 8, update_every=w.update_every, hyper=w.update)
    st = eng.stats()
    eng.close()
    assert st["device_status"] == 0, st["device_flags"]
    model = OracleModel(rounded_weights(W), w.shape, w.lora_gamma, dtype=np.float32, kv_dtype="bf16")
    check_rows_against_oracle(model, P, toks, rows, 3e-2)


def test_7b_full_size_lossless_and_first_step():
    w = workload("7b").with_(gen_tokens=16)
    W = make_weights(w)
    P = make_prompts(w)
    cap = max(len(p) for p in P) + w.gen_tokens * w.k_spec + 64
    _lossless(w, W=W, max_seq_len=cap)
    _check_first_step(w, W, P, max_seq_len=cap)


def test_7b_16k_context_lossless():
    w = workload("7b-16k").with_(gen_tokens=12)
    W = make_weights(w)
    P = make_prompts(w)
    assert len(P[0]) == 16384
    cap = len(P[0]) + w.gen_tokens * w.k_spec + 64
    _lossless(w, W=W, max_seq_len=cap)
