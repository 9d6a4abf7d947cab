"""tvl_gemv on the GPU vs the double-accumulator oracle (paper §6.1)."""
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


def run(tvl, W, x, stream=None, w_offset=0):
    M, K = W.shape
    if w_offset:
        base = torch.empty(M * K + w_offset, device="cuda")
        base[w_offset:] = torch.from_numpy(W.ravel()).cuda()
        dW = base[w_offset:]
    else:
        dW = torch.from_numpy(W).cuda()
    dx = torch.from_numpy(x).cuda()
    dy = torch.full((M,), float("nan"), device="cuda")
    s = stream if stream is not None else torch.cuda.current_stream()
    tvl.tvl_gemv(dW.data_ptr(), dx.data_ptr(), dy.data_ptr(), M, K, s.cuda_stream)
    s.synchronize()
    return dy.cpu().numpy()


# the sweep shapes of the paper's model family, plus ragged and degenerate ones
SHAPES = list(synth.GEMV_SHAPES) + [(1, 4), (1, 16384), (5, 4096), (300, 288), (4097, 36),
                                    (2, 8196), (129, 8192 + 128)]
ODD = [(7, 13), (1, 1), (33, 4097), (3, 20000), (1000, 3)]


@pytest.mark.parametrize("shape", SHAPES + ODD, ids=lambda s: f"{s[0]}x{s[1]}")
def test_gemv_matches_oracle(tvl, shape):
    i = (SHAPES + ODD).index(shape)
    W, x = synth.gemv_operands(*shape, i)
    y = run(tvl, W, x)
    y_ref = oracle.gemv(W, x)
    assert np.all(np.abs(y - y_ref) <= gemv_bound(W, x)), float(np.abs(y - y_ref).max())


def test_gemv_is_bitwise_deterministic_across_calls_and_streams(tvl):
    for shape in ((768, 768), (768, 2048), (5, 4096), (4096, 11008)):
        W, x = synth.gemv_operands(*shape, 3)
        a = run(tvl, W, x)
        b = run(tvl, W, x, stream=torch.cuda.Stream())
        c = run(tvl, W, x)
        assert np.array_equal(a, b) and np.array_equal(a, c)


def test_gemv_unaligned_weights_take_the_plain_path(tvl):
    W, x = synth.gemv_operands(96, 256, 4)
    y = run(tvl, W, x, w_offset=1)  # W 4 bytes off a 16-byte boundary
    assert np.all(np.abs(y - oracle.gemv(W, x)) <= gemv_bound(W, x))


def test_gemv_identity_is_exact(tvl):
    K = 1024
    x = synth.normal((K,), 5, 0)
    y = run(tvl, np.eye(K, dtype=np.float32), x)
    assert np.array_equal(y, x)


def test_gemv_rejects_bad_sizes(tvl):
    with pytest.raises(tvl.TvlError) as e:
        tvl.tvl_gemv(16, 16, 16, 0, 4)
    assert e.value.status == tvl.E_INVAL
