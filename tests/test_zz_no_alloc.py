"""jf_op_gemm_noalloc: the projection GEMM for callers that cannot allocate device memory.

Some callers cannot obtain device memory for a workspace -- code running inside a device-memory
allocator's own hooks, or a process whose device memory another pool has reserved entirely. For
them the library keeps the GEMM's split-K scratch in one fixed device array. This file is collected
last on purpose, so that a run stopping at its first failure has already run every other test; it
must pass on its own in a fresh process as well as after the rest of the suite.
"""
import numpy as np
import pytest

from paper_2512_14681_gb300 import inputs as I
from tests.parity import need_gpu

pytestmark = pytest.mark.gpu

# the GEMM tests' tolerance: fp32 accumulation of bf16 products
TOL_PER_K = 4e-7


def _bf16(torch, a):
    return torch.from_numpy(a).to(torch.bfloat16).cuda()


def test_noalloc_gemm_matches_workspace_gemm_on_consecutive_calls():
    torch = need_gpu()
    from paper_2512_14681_gb300 import _lib as J
    from paper_2512_14681_gb300.jacobi import op_gemm, op_gemm_noalloc

    # two calls in a row with different shapes and split counts share the fixed scratch
    cases = [(3584, 3584, 32, 5, 11), (4608, 3584, 16, 0, 12)]
    for N, K, M, splits, seed in cases:
        W = _bf16(torch, I.random_array((N, K), seed=seed, scale=0.5))
        X = _bf16(torch, I.random_array((M, K), seed=seed + 100, scale=0.5))
        y_ref, e_ref, _ = op_gemm(W, X, k_splits=splits)
        y, e, status = op_gemm_noalloc(W, X, k_splits=splits)
        assert status == J.JF_OK
        torch.cuda.synchronize()
        assert int(e.item()) == 0 and int(e_ref.item()) == 0
        diff = (y - y_ref).abs().max().item()
        assert diff <= TOL_PER_K * K + 1e-5, f"N={N} K={K} M={M}: max diff {diff}"


def test_noalloc_gemm_refuses_shapes_beyond_its_scratch():
    torch = need_gpu()
    from paper_2512_14681_gb300 import _lib as J
    from paper_2512_14681_gb300.jacobi import op_gemm_noalloc

    # 7B down projection at 256 rows with 8 splits needs far more than the fixed 8 MiB
    W = torch.zeros((3584, 18944), dtype=torch.bfloat16, device="cuda")
    X = torch.zeros((256, 18944), dtype=torch.bfloat16, device="cuda")
    _, _, status = op_gemm_noalloc(W, X, k_splits=8)
    assert status == J.JF_ECAPACITY
