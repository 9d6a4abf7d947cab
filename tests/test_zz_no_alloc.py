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
SHAPES = [(768, 768), (2048, 768), (768, 2048), (5, 4096), (300, 288), (4096, 11008),
          (32000, 768), (7, 13), (33, 4097)]


@pytest.fixture(scope="module")
def tvl():
    from paper_2601_03324_gb300 import tvl as t
    return t


@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: f"{s[0]}x{s[1]}")
def test_noalloc_matches_tvl_gemv_on_two_consecutive_calls(tvl, shape):
    M, K = shape
    W, x = synth.gemv_operands(M, K, 11)
    dW, dx = torch.from_numpy(W).cuda(), torch.from_numpy(x).cuda()
    s = torch.cuda.Stream()
    ref = torch.full((M,), float("nan"), device="cuda")
    tvl.tvl_gemv(dW.data_ptr(), dx.data_ptr(), ref.data_ptr(), M, K, s.cuda_stream)
    s.synchronize()
    y_ref = ref.cpu().numpy()
    bound = gemv_bound(W, x)
    outs = []
    for _ in range(2):  # the counters must be back at zero for the second call
        y = torch.full((M,), float("nan"), device="cuda")
        tvl.tvl_gemv_noalloc(dW.data_ptr(), dx.data_ptr(), y.data_ptr(), M, K, s.cuda_stream)
        s.synchronize()
        outs.append(y.cpu().numpy())
    for y in outs:
        assert np.all(np.isfinite(y))
        assert np.all(np.abs(y - y_ref) <= bound), float(np.abs(y - y_ref).max())


def test_noalloc_rejects_bad_arguments(tvl):
    with pytest.raises(tvl.TvlError):
        tvl.tvl_gemv_noalloc(0, 0, 0, 4, 4, 0)
    d = torch.zeros(16, device="cuda")
    with pytest.raises(tvl.TvlError):
        tvl.tvl_gemv_noalloc(d.data_ptr(), d.data_ptr(), d.data_ptr(), 0, 4, 0)
