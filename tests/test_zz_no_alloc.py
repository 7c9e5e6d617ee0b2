"""dvi_linear_noalloc: the projection for callers that cannot allocate.

Some callers must not allocate device memory (they run inside another
framework's memory pool or a fixed budget, or only receive their input and
output buffers).  The entry point keeps its split-K scratch in a fixed array
inside the library; this checks, through the C-ABI, that two calls in a row
give the same result as dvi_linear (which uses a context's workspace),
within the projection tests' tolerance, and that a shape larger than the
fixed scratch is refused without running.  Collected last on purpose.
"""
import numpy as np
import pytest
import torch

from workloads import workload
from gpu_helpers import engine_for

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("dtype,tol", [("bf16", 1e-4), ("f32", 2e-5)])
def test_noalloc_matches_linear_twice(dtype, tol):
    from paper_2510_05421_gb300.dvi import linear_noalloc
    eng, _, _ = engine_for(workload("tiny"), dtype=dtype, use_graphs=False)
    g = np.random.default_rng(5)
    td = torch.bfloat16 if dtype == "bf16" else torch.float32
    for n_out, k_in, m in ((4096, 4096, 16), (1000, 512, 5)):
        w = torch.from_numpy((g.standard_normal((n_out, k_in)) * 0.02).astype(np.float32)).cuda().to(td)
        x = torch.from_numpy(g.standard_normal((m, k_in)).astype(np.float32)).cuda()
        ref = eng.linear(w, x)
        torch.cuda.synchronize()
        scale = ref.abs().max().item()
        for _ in range(2):
            y = torch.full((m, n_out), float("nan"), dtype=torch.float32, device="cuda")
            assert linear_noalloc(w, x, y) == 0
            torch.cuda.synchronize()
            assert (y - ref).abs().max().item() <= tol * scale
    eng.close()


def test_noalloc_rejects_shapes_beyond_its_scratch():
    from paper_2510_05421_gb300.dvi import linear_noalloc
    # f32 path: 32 tiles x 16 row tiles x several K-splits x 128 x 16 partial
    # sums > the 2^21-float scratch
    w = torch.zeros(4096, 11008, dtype=torch.float32, device="cuda")
    x = torch.zeros(256, 11008, dtype=torch.float32, device="cuda")
    y = torch.zeros(256, 4096, dtype=torch.float32, device="cuda")
    assert linear_noalloc(w, x, y) == -2
