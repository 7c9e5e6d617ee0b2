"""dvi_linear_noalloc: the projection for callers that cannot allocate.

Some callers must not allocate device memory: code that runs inside
another framework's memory pool or under a fixed device-memory budget, or a
plug-in that is handed only its input and output buffers.  The entry point
keeps its split-K scratch in a fixed array inside the library.  Through the
C-ABI this checks two calls in a row (the second one reuses the scratch the
first left behind) against a float64 matmul of the bf16-rounded (or f32)
weights and the f32 input, within the projection tests' tolerance, and that
a shape larger than the fixed scratch is refused without running.
Collected last on purpose: it runs after every other test in a session,
and passes alone in a fresh process too.
"""
import numpy as np
import pytest
import torch

from workloads.gen import bf16_round

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("dtype,tol", [("bf16", 1e-4), ("f32", 2e-5)])
def test_noalloc_matches_float64_twice(dtype, tol):
    from paper_2510_05421_gb300.dvi import linear_noalloc
    g = np.random.default_rng(5)
    td = torch.bfloat16 if dtype == "bf16" else torch.float32
    # (4096 x 4096, 16 rows) splits K over a cluster (bf16) or the scratch (f32)
    for n_out, k_in, m in ((4096, 4096, 16), (1000, 512, 5), (2048, 1024, 40)):
        W = (g.standard_normal((n_out, k_in)) * 0.02).astype(np.float32)
        X = g.standard_normal((m, k_in)).astype(np.float32)
        w = torch.from_numpy(W).cuda().to(td)
        x = torch.from_numpy(X).cuda()
        Wr = bf16_round(W) if dtype == "bf16" else W
        ref = X.astype(np.float64) @ Wr.astype(np.float64).T
        scale = np.abs(ref).max()
        outs = []
        for _ in range(2):
            y = torch.full((m, n_out), float("nan"), dtype=torch.float32, device="cuda")
            assert linear_noalloc(w, x, y) == 0
            torch.cuda.synchronize()
            got = y.cpu().numpy().astype(np.float64)
            assert np.abs(got - ref).max() <= tol * scale, (n_out, k_in, m)
            outs.append(got)
        assert np.array_equal(outs[0], outs[1])


def test_noalloc_rejects_shapes_beyond_its_scratch():
    from paper_2510_05421_gb300.dvi import linear_noalloc
    # f32 path: 32 tiles x 16 row tiles x several K-splits x 128 x 16 partial
    # sums > the 2^21-float scratch
    w = torch.zeros(4096, 11008, dtype=torch.float32, device="cuda")
    x = torch.zeros(256, 11008, dtype=torch.float32, device="cuda")
    y = torch.zeros(256, 4096, dtype=torch.float32, device="cuda")
    assert linear_noalloc(w, x, y) == -2
