"""tvl_gemv_noalloc (split-K scratch in a static module array, nothing
allocated) against tvl_gemv on the GPU. This file is collected last, so it
runs both after every other test and, with -k or by path, alone."""
import numpy as np
import pytest

from helpers import gemv_bound
from paper_2601_03324_gb300 import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

# split along K (S > 1), one row per CTA or more (S = 1), ragged and
# unaligned-K shapes that take the per-row kernel
SHAPES = [(768, 768), (2048, 768), (768, 2048), (5, 4096), (64, 8192), (100, 2048),
          (300, 288), (4096, 11008), (32000, 768), (7, 13), (33, 4097)]


@pytest.fixture(scope="module")
def tvl():
    from paper_2601_03324_gb300 import tvl as t
    return t


@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: f"{s[0]}x{s[1]}")
def test_noalloc_matches_tvl_gemv_on_two_consecutive_calls(tvl, shape):
    """Same kernel, same split, partials summed in the same order: the output
    equals tvl_gemv's bit for bit, on two calls in a row (the second finds the
    counters the first left), and lies within the GEMV bound of the oracle."""
    import oracle
    M, K = shape
    W, x = synth.gemv_operands(M, K, 11)
    dW, dx = torch.from_numpy(W).cuda(), torch.from_numpy(x).cuda()
    s = torch.cuda.Stream()
    ref = torch.full((M,), float("nan"), device="cuda")
    tvl.tvl_gemv(dW.data_ptr(), dx.data_ptr(), ref.data_ptr(), M, K, s.cuda_stream)
    s.synchronize()
    y_ref = ref.cpu().numpy()
    truth = oracle.gemv(W, x)
    bound = gemv_bound(W, x)
    for _ in range(2):
        y = torch.full((M,), float("nan"), device="cuda")
        tvl.tvl_gemv_noalloc(dW.data_ptr(), dx.data_ptr(), y.data_ptr(), M, K, s.cuda_stream)
        s.synchronize()
        got = y.cpu().numpy()
        assert np.array_equal(got, y_ref)
        assert np.all(np.abs(got - truth) <= bound), float(np.abs(got - truth).max())
    assert tvl.tvl_gemv_status(s.cuda_stream) == tvl.OK


def test_noalloc_allocates_no_device_memory(tvl):
    """After the first call on the device (the one-time setup), further calls
    leave the device's free memory and the library's allocation count as they
    were."""
    M, K = 64, 8192  # fewer rows than SMs: split along K, the static scratch is in use
    W, x = synth.gemv_operands(M, K, 12)
    dW, dx = torch.from_numpy(W).cuda(), torch.from_numpy(x).cuda()
    y = torch.empty(M, device="cuda")
    s = torch.cuda.Stream()
    tvl.tvl_gemv_noalloc(dW.data_ptr(), dx.data_ptr(), y.data_ptr(), M, K, s.cuda_stream)
    s.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    live0 = tvl.lib.tvl_debug_live_allocations()
    for _ in range(5):
        tvl.tvl_gemv_noalloc(dW.data_ptr(), dx.data_ptr(), y.data_ptr(), M, K, s.cuda_stream)
    s.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0
    assert tvl.lib.tvl_debug_live_allocations() == live0


def test_noalloc_rejects_bad_arguments(tvl):
    with pytest.raises(tvl.TvlError):
        tvl.tvl_gemv_noalloc(0, 0, 0, 4, 4, 0)
    d = torch.zeros(16, device="cuda")
    with pytest.raises(tvl.TvlError):
        tvl.tvl_gemv_noalloc(d.data_ptr(), d.data_ptr(), d.data_ptr(), 0, 4, 0)
