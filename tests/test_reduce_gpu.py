"""GPU parity of the memory-bound operators of Table 2 (min/max reduction,
2-D max / average pooling) against the CPU oracle."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_09905_gb300 import qx

from gpu_util import build_once

pytestmark = pytest.mark.gpu

DT = {qx.I16: torch.int16, qx.I32: torch.int32, qx.F32: torch.float32}


@pytest.fixture(scope="module", autouse=True)
def _built():
    build_once()


def _data(shape, dtype, seed, lo=None, hi=None):
    g = torch.Generator().manual_seed(seed)
    if dtype == qx.F32:
        return torch.randn(shape, generator=g)
    info = torch.iinfo(DT[dtype])
    lo = info.min if lo is None else lo
    hi = info.max if hi is None else hi
    return torch.randint(lo, hi + 1, shape, generator=g, dtype=torch.int64).to(DT[dtype])


@pytest.mark.parametrize("dtype", [qx.I16, qx.I32, qx.F32])
@pytest.mark.parametrize("n", [1, 7, 1023, 1 << 20, (1 << 24) + 5])
def test_minmax(dtype, n):
    x = _data((n,), dtype, seed=n + dtype)
    with qx.Plan(qx.minmax_desc(n, dtype)) as plan:
        out = plan.minmax(x.cuda())
        out2 = plan.minmax(x.cuda())         # the arrival counter rearms itself
        torch.cuda.synchronize()
        assert plan.status() == qx.OK
    lo, hi = oracle.minmax(x)
    assert (out.cpu().tolist(), out2.cpu().tolist()) == ([lo, hi], [lo, hi])


def test_minmax_unaligned_and_extremes():
    x = _data((100003,), qx.I32, seed=3)
    x[77] = -2**31
    x[50000] = 2**31 - 1
    xs = x.cuda()[1:]                         # 4-byte aligned, not 16-byte aligned
    with qx.Plan(qx.minmax_desc(xs.numel(), qx.I32)) as plan:
        out = plan.minmax(xs)
        torch.cuda.synchronize()
    assert out.cpu().tolist() == list(oracle.minmax(x[1:]))


@pytest.mark.parametrize("dtype", [qx.I16, qx.I32, qx.F32])
@pytest.mark.parametrize("mode", ["max", "avg"])
@pytest.mark.parametrize("shape,k,s", [((32, 128, 112, 112), 2, 2), ((2, 3, 9, 7), 2, 2),
                                       ((1, 4, 17, 21), 3, 2), ((3, 2, 8, 8), 2, 1),
                                       ((2, 5, 10, 16), 2, 2)])
def test_pool2d(dtype, mode, shape, k, s):
    lo, hi = (-1000, 1000) if dtype != qx.F32 else (None, None)
    x = _data(shape, dtype, seed=sum(shape) + k + s, lo=lo, hi=hi)
    n, c, h, w = shape
    with qx.Plan(qx.pool_desc(n, c, h, w, k, k, s, mode, dtype)) as plan:
        y = plan.pool2d(x.cuda())
        torch.cuda.synchronize()
        assert plan.status() == qx.OK
    ref = oracle.pool2d(x, k, k, s, mode)
    got = y.cpu().numpy().astype(np.float64 if dtype == qx.F32 else np.int64)
    if dtype == qx.F32 and mode == "avg":
        # FP32 mean of k*k terms against the float64 mean
        mag = oracle.pool2d(np.abs(x.numpy()), k, k, s, "avg")
        assert (np.abs(got - ref) <= 1e-6 * mag + 1e-30).all()
    else:
        assert np.array_equal(got, ref)


def test_pool_argument_errors():
    with pytest.raises(qx.QxError):
        qx.Plan(qx.pool_desc(1, 1, 1, 4, 2, 2, 2))            # window taller than the image
    with qx.Plan(qx.pool_desc(1, 2, 4, 4)) as plan:
        lib = qx.load()
        x = torch.zeros((1, 2, 4, 4), dtype=torch.int32, device="cuda")
        assert lib.qx_minmax(plan.handle, x.data_ptr(), x.data_ptr(), None) == qx.ERR_INVALID_ARG
        assert lib.qx_pool2d(plan.handle, None, x.data_ptr(), None) == qx.ERR_INVALID_ARG


@pytest.mark.parametrize("dtype,n", [(qx.I32, 1 << 28), (qx.I16, 1 << 29)])
def test_minmax_benchmark_sizes(dtype, n):
    # the benchmarked 1 GiB inputs, in the benchmark's launch configuration
    x = _data((n,), dtype, seed=5)
    with qx.Plan(qx.minmax_desc(n, dtype)) as plan:
        out = plan.minmax(x.cuda())
        torch.cuda.synchronize()
        assert plan.status() == qx.OK
    assert out.cpu().tolist() == list(oracle.minmax(x))
