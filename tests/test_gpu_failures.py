"""Device-side failure reports (the status bits of dvi_get_stats), each
triggered from the host with inputs the kernels bound-check, so no kernel
faults, traps or waits:

* KV_FULL: a KV capacity too small for the run.  Rows that would fall past
  max_seq_len are not written (the prompt rows of every layer, sequence and
  head -- where an unchecked write would land -- stay as they were), and
  attention reads stay clamped to the capacity.
* NONFINITE: a NaN written into the LoRA factor A before the logged steps.
  The drafter logits of the buffer, and so the update's loss, are not
  finite: the update skips its parameter step (A and B unchanged), still
  advances the schedule's clock t and empties the buffer, and is not
  counted as applied.
* BAD_TOKEN: prompt ids outside [0, V); the embedding reads row 0 instead.
* LOG_FULL: more logged decode steps than the replay buffer holds; the
  extra step's tuples are dropped and the buffer's own rows stay intact.
"""
import numpy as np
import pytest
import torch

from workloads import workload, make_prompts
from gpu_helpers import engine_for

pytestmark = pytest.mark.gpu


def _dev(eng, p):
    return torch.from_numpy(np.ascontiguousarray(p, dtype=np.int32)).to(eng.device)


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_kv_full_is_flagged_and_no_row_spills(dtype):
    w = workload("tiny")
    s = w.shape
    P = make_prompts(w)
    n0, K = len(P[0]), w.k_spec
    cap = n0 + K + 1 + 3            # prefill accepts n + K + 1 <= capacity; a few steps overflow it
    eng, _, _ = engine_for(w, dtype=dtype, max_seq_len=cap)
    td = torch.bfloat16 if dtype == "bf16" else torch.float32
    eng.prefill(0, _dev(eng, P[0]))
    eng.sync()
    shape = (s.n_layers, 1, s.n_kv_heads, cap, s.head_dim)
    kc = eng.buffer("K_CACHE", td).view(shape)
    vc = eng.buffer("V_CACHE", td).view(shape)
    k0, v0 = kc[..., :n0, :].clone(), vc[..., :n0, :].clone()
    assert eng.stats()["device_status"] == 0
    for _ in range(4):
        eng.step()
    st = eng.stats()
    assert "KV_FULL" in st["device_flags"], st["device_flags"]
    assert eng.buffer("LENS", torch.int32)[0].item() >= cap
    assert torch.equal(kc[..., :n0, :], k0)
    assert torch.equal(vc[..., :n0, :], v0)
    eng.close()


def test_nan_in_lora_a_skips_the_update():
    w = workload("tiny")
    P = make_prompts(w)
    eng, _, dw = engine_for(w, dtype="f32")
    dw.lora_a[0, 0] = float("nan")          # injected from the host, before the logged steps
    torch.cuda.synchronize()
    eng.generate(P, 10 ** 6, max_steps=w.update_every, log=True)
    eng.sync()
    st0 = eng.stats()
    meta = eng.buffer("LOG_META", torch.int32).view(-1, 6)
    assert meta[:, 0].sum().item() > 0
    a0, b0 = dw.lora_a.clone(), dw.lora_b.clone()
    torch.cuda.synchronize()
    eng.update(w.update)
    st = eng.stats()
    assert "NONFINITE" in st["device_flags"], st["device_flags"]
    assert st["updates"] == st0["updates"]                 # not applied
    assert st["update_t"] == st0["update_t"] + 1           # the clock still advances
    assert torch.equal(torch.isnan(dw.lora_a), torch.isnan(a0))
    assert torch.equal(torch.nan_to_num(dw.lora_a), torch.nan_to_num(a0))
    assert torch.equal(dw.lora_b, b0)
    assert meta[:, 0].sum().item() == 0                    # buffer emptied
    eng.close()


@pytest.mark.parametrize("bad", [1024, -1])
def test_out_of_range_prompt_id_is_flagged(bad):
    w = workload("tiny")
    P = make_prompts(w)
    eng, _, _ = engine_for(w, dtype="bf16")
    p = P[0].copy()
    p[5] = bad                              # vocabulary is 1024
    eng.prefill(0, _dev(eng, p))
    st = eng.stats()
    assert "BAD_TOKEN" in st["device_flags"], st["device_flags"]
    eng.close()


def test_replay_buffer_overflow_is_flagged():
    w = workload("tiny")
    P = make_prompts(w)
    eng, _, _ = engine_for(w, dtype="f32", log_steps=2)
    eng.prefill(0, _dev(eng, P[0]))
    eng.log(True)
    for _ in range(2):
        eng.step()
    eng.sync()
    meta2 = eng.buffer("LOG_META", torch.int32).clone()
    lg2 = eng.buffer("LOG_LOGITS", torch.float32).clone()
    assert eng.stats()["device_status"] == 0
    eng.step()                              # a third logged step: no room
    st = eng.stats()
    assert "LOG_FULL" in st["device_flags"], st["device_flags"]
    assert torch.equal(eng.buffer("LOG_META", torch.int32), meta2)
    assert torch.equal(eng.buffer("LOG_LOGITS", torch.float32), lg2)
    eng.close()
