"""tvl_gemm (tcgen05, bf16x3 split, fp32 accumulation) against the double
oracle's GEMV, row by row, and exactly on integer-valued operands."""
import numpy as np
import pytest

import oracle
from helpers import gemv_bound
from paper_2601_03324_gb300 import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def tvl():
    from paper_2601_03324_gb300 import tvl as t
    return t


def run(tvl, W, X):
    n, K = X.shape
    M = W.shape[0]
    dW, dX = torch.from_numpy(W).cuda(), torch.from_numpy(X).cuda()
    dY = torch.full((n, M), float("nan"), device="cuda")
    s = torch.cuda.Stream()
    tvl.tvl_gemm(dW.data_ptr(), dX.data_ptr(), dY.data_ptr(), n, M, K, s.cuda_stream)
    assert tvl.tvl_gemm_status(s.cuda_stream) == tvl.OK
    return dY.cpu().numpy()


@pytest.mark.parametrize("shape", [(1, 1, 8), (5, 7, 64), (128, 128, 64), (130, 200, 136),
                                   (3, 129, 4096), (257, 384, 72)],
                         ids=lambda s: "x".join(map(str, s)))
def test_gemm_integer_operands_are_exact(tvl, shape):
    # integers of at most 8 significant bits are bf16 values (lo part 0), and
    # every partial sum stays an integer below 2^24: the result is exact
    n, M, K = shape
    rng = np.random.default_rng(sum(shape))
    W = rng.integers(-15, 16, size=(M, K)).astype(np.float32)
    X = rng.integers(-15, 16, size=(n, K)).astype(np.float32)
    Y = run(tvl, W, X)
    ref = (X.astype(np.int64) @ W.astype(np.int64).T).astype(np.float32)
    assert np.array_equal(Y, ref)


@pytest.mark.parametrize("shape", [(7, 96, 64), (130, 200, 136), (256, 768, 768),
                                   (896, 2304, 768), (37, 300, 4104), (64, 768, 2048),
                                   (512, 1000, 4096)],
                         ids=lambda s: "x".join(map(str, s)))
def test_gemm_matches_the_oracle_gemv_within_its_bound(tvl, shape):
    n, M, K = shape
    W = synth.normal((M, K), 1, 90 + n % 7, 0.0, 0.02)
    X = synth.normal((n, K), 1, 91 + M % 7, 0.0, 1.0)
    Y = run(tvl, W, X)
    rows = range(n) if n * M * K <= 4e7 else np.linspace(0, n - 1, 24).astype(int)
    for i in rows:
        y = oracle.gemv(W, X[i])
        assert np.all(np.abs(Y[i] - y) <= gemv_bound(W, X[i])), (i, float(np.abs(Y[i] - y).max()))


def test_gemm_rejects_bad_shapes(tvl):
    d = torch.zeros(64, device="cuda")
    p = d.data_ptr()
    with pytest.raises(tvl.TvlError) as e:
        tvl.tvl_gemm(p, p, p, 1, 1, 12, 0)  # K % 8 != 0
    assert e.value.status == tvl.E_UNSUPPORTED
    with pytest.raises(tvl.TvlError) as e:
        tvl.tvl_gemm(p, p, p, 0, 1, 8, 0)
    assert e.value.status == tvl.E_INVAL
