"""Projection GEMM (tcgen05 bf16 and CUDA-core fp32) through jf_op_gemm vs the oracle's fp64 linear.

The weight-streaming projections are the matrix products of the forward pass of Eq. 3. Inputs
are bf16 values; the oracle multiplies the same values in fp64, so the only difference is the
kernel's fp32 accumulation (error below ~K * 2^-24 * |products|).
"""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2512_14681_gb300 import inputs as I
from tests.parity import need_gpu

pytestmark = pytest.mark.gpu


def _bf16(torch, a):
    return torch.from_numpy(a).to(torch.bfloat16).cuda()


def _token_tile(M):
    """The token-tile width the library picks: the narrowest that holds M rows (32 at the least); above
    256 rows the narrowest of 128, 160, 256 that needs no more tiles than 256-wide ones."""
    for b in (32, 64, 128, 160, 256):
        if M <= b:
            return b
    tiles = -(-M // 256)
    return next(b for b in (128, 160, 256) if -(-M // b) == tiles)


@pytest.mark.parametrize(
    "N,K,M,splits",
    [
        (128, 64, 1, 1),        # one tile, one stage
        (300, 512, 7, 0),       # ragged N (TMA zero fill) and ragged M
        (1024, 3584, 32, 0),    # 7B-width K, default split
        (4608, 3584, 32, 4),    # 7B QKV shape, split-K 4
        (3584, 18944, 16, 0),   # 7B down projection shape
        (640, 1024, 33, 3),     # M just above a token tile
        (512, 2048, 160, 0),    # multi-block + candidate width
        (384, 1536, 300, 2),    # token tiling (M > 256: 2 tiles of 160) with split-K
        (512, 1024, 384, 0),    # 2 token tiles of 256, the second one half full
        (640, 2048, 600, 2),    # 3 token tiles of 256, split-K
        (1000, 520, 256, 0),    # K not a multiple of 64
    ],
)
def test_gemm_bf16_matches_oracle(N, K, M, splits):
    torch = need_gpu()
    from paper_2512_14681_gb300.jacobi import op_gemm

    W = I.random_array((N, K), seed=N + K, scale=0.5)
    X = I.random_array((M, K), seed=M + 7, scale=0.5)
    Wt, Xt = _bf16(torch, W), _bf16(torch, X)
    Y, err, ws = op_gemm(Wt, Xt, k_splits=splits)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    Wd = Wt.float().cpu().numpy().astype(np.float64)
    Xd = Xt.float().cpu().numpy().astype(np.float64)
    ref = O.linear(Xd, Wd)
    got = Y.cpu().numpy().astype(np.float64)
    tol = 4e-7 * K + 1e-5
    diff = np.abs(got - ref)
    assert diff.max() <= tol, f"max abs diff {diff.max()} (tol {tol})"
    # split-K tickets (the workspace's last bytes) are left at zero for the next launch
    bn = _token_tile(M)
    n_counters = ((N + 127) // 128) * ((M + bn - 1) // bn)
    nbytes = (n_counters * 4 + 255) // 256 * 256
    assert int(torch.count_nonzero(ws[-nbytes:]).item()) == 0


def test_gemm_bf16_repeat_launches_are_deterministic():
    torch = need_gpu()
    from paper_2512_14681_gb300.jacobi import op_gemm

    W = _bf16(torch, I.random_array((3584, 3584), seed=1, scale=0.5))
    X = _bf16(torch, I.random_array((32, 3584), seed=2, scale=0.5))
    a, _, _ = op_gemm(W, X, k_splits=5)
    b, _, _ = op_gemm(W, X, k_splits=5)
    torch.cuda.synchronize()
    assert torch.equal(a, b)
    # a row's result does not depend on the other rows in flight
    c, _, _ = op_gemm(W, X[:1].contiguous(), k_splits=5)
    torch.cuda.synchronize()
    assert torch.equal(c[0], a[0])


def test_gemm_f32_matches_oracle():
    torch = need_gpu()
    from paper_2512_14681_gb300.jacobi import op_gemm

    W = I.random_array((300, 256), seed=3, scale=0.5)
    X = I.random_array((40, 256), seed=4, scale=0.5)
    Y, err, _ = op_gemm(torch.from_numpy(W).cuda(), torch.from_numpy(X).cuda())
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    ref = O.linear(X.astype(np.float64), W.astype(np.float64))
    assert np.abs(Y.cpu().numpy() - ref).max() < 1e-4
