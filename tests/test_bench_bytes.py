"""bench.py's byte model: the algorithmic HBM bytes behind every roofline
fraction it reports, checked on the CPU against sizes fixed independently
of the formula (the parameter counts of the Llama shapes, the per-pass
totals worked out for the 7B workload, the committed ncu traffic).
"""
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402
from workloads import workload  # noqa: E402


def test_layer_head_and_kv_row_sizes():
    s7 = workload("7b").shape
    # Llama-2-7B block: 4 d^2 attention + 3 d F FFN parameters, bf16
    assert bench.layer_bytes(s7, 2) == (4 * 4096 ** 2 + 3 * 4096 * 11008) * 2 == 404_750_336
    # K and V rows of one position: 32 heads x 128 dims x 2 tensors, bf16
    assert bench.kv_row_bytes(s7, 2) == 16_384
    s1 = workload("1b").shape
    # 1B GQA block: q and o 2048 x 2048, k and v 1024 x 2048, FFN 3 x 2048 x 5632
    assert bench.layer_bytes(s1, 2) == (2 * 2048 * 2048 + 2 * 1024 * 2048 + 3 * 2048 * 5632) * 2 == 94_371_840
    assert bench.kv_row_bytes(s1, 2) == 2 * 8 * 128 * 2


def test_step_bytes_of_the_7b_workload():
    w = workload("7b")
    draft, verify = bench.step_bytes(w, [1280])
    # verify: 30 deep layers (404.8 MB each), the LM head (262.1 MB) and
    # 30 x 1285 attended K/V rows of 16 KB: about 13.04 GB
    assert verify == 30 * 404_750_336 + 32000 * 4096 * 2 + 30 * 1285 * 16_384
    assert verify == pytest.approx(13.036e9, rel=1e-3)
    # draft: 5 passes of 2 layers + the drafter head (+ the f32 LoRA factors)
    # and the shallow K/V rows: about 5.57 GB
    assert draft == pytest.approx(5.57e9, rel=2e-3)
    # more context only adds K/V rows
    d2, v2 = bench.step_bytes(w, [1280 + 64])
    assert v2 - verify == 30 * 64 * 16_384
    assert d2 - draft == 5 * 2 * 64 * 16_384


def test_batch_adds_kv_rows_not_weights():
    w = workload("7b-b8")
    d1, v1 = bench.step_bytes(w, [1000])
    d8, v8 = bench.step_bytes(w, [1000] * 8)
    assert v8 - v1 == 7 * 30 * 1005 * 16_384
    assert d8 - d1 == 7 * sum(2 * (1000 + j + 1) * 16_384 for j in range(5))


def test_prefill_bytes_of_a_1024_token_prompt():
    w = workload("7b")
    # eight 128-row chunks each stream every layer's weights; each chunk
    # reads its prefix's K/V rows and writes its own; one LM-head row
    weights = 8 * 32 * 404_750_336
    kv = 32 * 16_384 * sum(c0 + 128 + 128 for c0 in range(0, 1024, 128))
    assert bench.prefill_bytes(w, 1024, 128) == weights + kv + 32000 * 4096 * 2 == 106_831_020_032


def test_committed_ncu_traffic_is_the_algorithmic_bytes():
    """The ncu DRAM counts of the verify pass (profiles/) stay within 1 % of
    the byte model: no operand is re-read from DRAM."""
    w = workload("7b")
    n = [1300.0]
    _, verify = bench.step_bytes(w, n)
    t = bench.measured_traffic(w, n)
    assert t is not None
    assert 1.0 <= t / verify < 1.01
    tp = bench.measured_traffic(w, n, persistent=True)
    assert tp is not None and 1.0 <= tp / verify < 1.04
    # another shape has no capture
    assert bench.measured_traffic(workload("1b"), n) is None


def test_prefill_flops_and_bound():
    w = workload("7b")
    # 2 FLOPs per weight per token over 32 layers of 202,375,168 weights,
    # causal attention's two products (32 heads x 128, 1024 x 1025 / 2
    # attended pairs per layer), the LM head on one row
    expect = 32 * (2 * 202_375_168 * 1024 + 4 * 32 * 128 * (1024 * 1025 // 2)) + 2 * 32000 * 4096
    assert bench.prefill_flops(w, 1024) == expect
    assert expect == pytest.approx(13.54e12, rel=1e-3)
    pk = {"hbm_gbs": 6785.5, "bf16_tflops": 1884.7}
    # the algorithm reads every weight once: 13.5 TFLOP against ~14.3 GB is
    # far above the ridge, so the tensor pipe bounds it whatever the passes
    alg = bench.prefill_alg_bytes(w, 1024)
    assert alg == 32 * 404_750_336 + 32000 * 4096 * 2 + 32 * 16_384 * 2 * 1024
    r = bench.prefill_roofline(expect, alg, 72.0, pk, traffic=bench.prefill_bytes(w, 1024, 128))
    assert r["bound"] == "tensor" and r["unit"] == "TFLOP/s"
    assert r["frac"] == pytest.approx(expect / 0.072 / 1e12 / 1884.7)
    assert r["traffic_model"] == 106_831_020_032
    # a short prompt is bound by its bytes
    r = bench.prefill_roofline(bench.prefill_flops(w, 16), bench.prefill_alg_bytes(w, 16), 5.0, pk)
    assert r["bound"] == "hbm"


def test_update_bytes_of_the_7b_workload():
    w = workload("7b")
    # 20 rows: logged z and verifier logits (2 x 20 x 32000 x 4 B), u as two
    # bf16 planes (20 x 4096 x 4 B), and A [32000 x 16], B [16 x 4096] f32
    # with their Adam moments read and written and the gradient written
    expect = 2 * 20 * 32000 * 4 + 20 * 4096 * 4 + 7 * (32000 + 4096) * 16 * 4
    assert bench.update_bytes(w, 20) == expect
    assert expect == pytest.approx(21.6e6, rel=1e-2)
