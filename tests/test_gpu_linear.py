"""The projection kernel through the C-ABI (dvi_linear): tcgen05/TMA for bf16,
FP32 FMA for f32, against a float64 matmul of the (bf16-rounded) weights and
the f32 input -- the bf16 kernel carries the input as a bf16 pair hi + lo, so
only the weights are rounded -- over shapes spanning several 128-row tiles,
split-K and ragged tails.
Also: bitwise determinism, and a row's result does not depend on how many
rows share the launch (what makes the verify pass agree bit for bit with AR
decoding)."""
import numpy as np
import pytest
import torch

from workloads import workload
from workloads.gen import bf16_round
from gpu_helpers import engine_for

pytestmark = pytest.mark.gpu

SHAPES = [(128, 64, 1), (256, 256, 5), (384, 4096, 16), (1000, 512, 17), (4096, 4096, 40),
          (512, 11008, 5), (32000, 4096, 1), (640, 2048, 128), (256, 1024, 256), (12288, 4096, 5)]


@pytest.fixture(scope="module", params=["bf16", "f32"])
def eng(request):
    w = workload("tiny")
    e, _, _ = engine_for(w, dtype=request.param, use_graphs=False)
    yield e
    e.close()


def _case(n_out, k, m, dtype, seed):
    g = np.random.default_rng(seed)
    W = (g.standard_normal((n_out, k)) * 0.02).astype(np.float32)
    X = g.standard_normal((m, k)).astype(np.float32)
    td = torch.bfloat16 if dtype == "bf16" else torch.float32
    Wd = torch.from_numpy(W).cuda().to(td)
    Xd = torch.from_numpy(X).cuda()
    if dtype == "bf16":
        W = bf16_round(W)
    ref = X.astype(np.float64) @ W.astype(np.float64).T
    return Wd, Xd, ref


@pytest.mark.parametrize("shape", SHAPES)
def test_linear_matches_float64(eng, shape):
    n_out, k, m = shape
    Wd, Xd, ref = _case(n_out, k, m, eng.dtype, hash(shape) % 1000)
    y = eng.linear(Wd, Xd)
    torch.cuda.synchronize()
    y = y.cpu().numpy().astype(np.float64)
    scale = np.abs(ref).max()
    err = np.abs(y - ref).max() / scale
    assert err < (2e-5 if eng.dtype == "f32" else 1e-4), err
    assert eng.stats()["device_status"] == 0


def test_linear_deterministic_and_row_independent(eng):
    Wd, Xd, _ = _case(4096, 4096, 40, eng.dtype, 7)
    y1 = eng.linear(Wd, Xd)
    y2 = eng.linear(Wd, Xd)
    y_one = eng.linear(Wd, Xd[:1].contiguous())
    y_five = eng.linear(Wd, Xd[:5].contiguous())
    torch.cuda.synchronize()
    assert torch.equal(y1, y2)
    assert torch.equal(y_one[0], y1[0])
    assert torch.equal(y_five, y1[:5])
