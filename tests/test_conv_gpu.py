"""GPU parity of the GEMM-backed Conv2D (Table 2 Conv2D rows; lowering done on
load by TMA im2col) against the CPU oracle's direct convolution, bit for bit."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_09905_gb300 import inputs, qx

from gpu_util import assert_exact, build_once, wrap32

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    build_once()


def conv_gpu(x, w, stride, pad, rx, rw, dtype=qx.I16, flags=0):
    n, c, h, wd = x.shape
    k, _, r, s = w.shape
    with qx.Plan(qx.conv_desc(n, c, h, wd, k, r, s, stride, pad, rx, rw, dtype=dtype,
                              flags=flags)) as plan:
        y = plan.conv2d(x.cuda(), w.cuda())
        torch.cuda.synchronize()
        st = plan.status()
        info = plan.info()
    return y.cpu().numpy().astype(np.int64), st, info


def test_conv_workload_int16():
    """8 x 64 x 56 x 56 input, 128 x 64 x 3 x 3 weights, stride 1, pad 1."""
    x, w = inputs.conv_case(8, 64, 56, 56, 128, 3, 3, -255, 255, seed=0)
    ref = oracle.conv2d(x, w, 1, 1)
    got, st, info = conv_gpu(x, w, 1, 1, (-255, 255), (-255, 255))
    assert st == qx.OK
    assert_exact(got, ref, f"conv workload {info}")


def test_conv_workload_int32():
    x, w = inputs.conv_case(8, 64, 56, 56, 128, 3, 3, -255, 255, seed=1, dtype=torch.int32)
    ref = oracle.conv2d(x, w, 1, 1)
    got, st, _ = conv_gpu(x, w, 1, 1, (-255, 255), (-255, 255), dtype=qx.I32)
    assert st == qx.OK
    assert_exact(got, ref, "conv int32")


@pytest.mark.parametrize("shape,stride,pad", [
    ((1, 3, 7, 9, 5, 3, 3), 1, 1),
    ((2, 64, 16, 16, 64, 3, 3), 1, 1),
    ((3, 130, 9, 11, 200, 3, 3), 1, 1),
    ((2, 16, 12, 10, 24, 1, 1), 1, 0),
    ((1, 8, 13, 12, 16, 5, 3), 1, 2),
    ((2, 32, 15, 15, 40, 3, 3), 1, 0),
    ((1, 64, 30, 30, 64, 3, 3), 2, 1),
    ((2, 16, 17, 13, 32, 3, 3), 2, 0),
])
def test_conv_shapes(shape, stride, pad):
    n, c, h, wd, k, r, s = shape
    x, w = inputs.conv_case(n, c, h, wd, k, r, s, -255, 255, seed=sum(shape) + stride)
    ref = oracle.conv2d(x, w, stride, pad)
    got, st, info = conv_gpu(x, w, stride, pad, (-255, 255), (-255, 255))
    assert st == qx.OK
    assert_exact(got, ref, f"conv {shape} stride {stride} pad {pad} {info}")


def test_conv_all_ones_borders():
    x = torch.ones((1, 64, 8, 8), dtype=torch.int16)
    w = torch.ones((64, 64, 3, 3), dtype=torch.int16)
    got, st, _ = conv_gpu(x, w, 1, 1, (0, 1), (0, 1))
    assert st == qx.OK
    exp = np.full((8, 8), 9 * 64)
    exp[0, :] = exp[-1, :] = exp[:, 0] = exp[:, -1] = 6 * 64
    exp[0, 0] = exp[0, -1] = exp[-1, 0] = exp[-1, -1] = 4 * 64
    assert (got[0] == exp).all()


@pytest.mark.parametrize("rx,rw", [((-20000, 20000), (-255, 255)),
                                   ((-255, 255), (-30000, 30000)),
                                   ((-2**20, 2**20), (-2**11, 2**11))])
def test_conv_limb_schemes_int32(rx, rw):
    n, c, h, wd, k, r, s = 2, 16, 9, 9, 24, 3, 3
    g = torch.Generator().manual_seed(rx[1] % 1000)
    x = torch.randint(rx[0], rx[1] + 1, (n, c, h, wd), generator=g, dtype=torch.int32)
    w = torch.randint(rw[0], rw[1] + 1, (k, c, r, s), generator=g, dtype=torch.int32)
    ref = oracle.conv2d(x, w, 1, 1)
    got, st, info = conv_gpu(x, w, 1, 1, rx, rw, dtype=qx.I32)
    assert st == qx.OK
    assert info[0]["mma_per_kstep"] > 1
    assert_exact(got, wrap32(ref), f"conv limbs {info}")


def test_conv_range_check():
    x, w = inputs.conv_case(1, 8, 6, 6, 8, 3, 3, -10, 10, seed=2)
    w[3, 2, 1, 1] = -11
    _, st, _ = conv_gpu(x, w, 1, 1, (-10, 10), (-10, 10), flags=qx.FLAG_CHECK_RANGES)
    assert st == qx.ERR_CONTRACT


# ------------------------------------------------------------ FP32 (3xTF32)
def conv_gpu_f32(x, w, stride, pad):
    n, c, h, wd = x.shape
    k, _, r, s = w.shape
    with qx.Plan(qx.conv_desc(n, c, h, wd, k, r, s, stride, pad, (0, 0), (0, 0),
                              dtype=qx.F32)) as plan:
        y = plan.conv2d(x.cuda(), w.cuda())
        torch.cuda.synchronize()
        st = plan.status()
    return y.cpu().numpy().astype(np.float64), st


def assert_within_tolerance(got, ref, mag, what):
    """max |err| <= 1e-5 * sum_k |a_k||b_k| for every output element."""
    err = np.abs(got - ref)
    worst = float((err / np.maximum(mag, 1e-300)).max())
    assert (err <= 1e-5 * mag).all(), f"{what}: worst err / sum|a||b| = {worst:.3e}"
    return worst


def test_conv_workload_f32():
    x, w = inputs.conv_case_f32(8, 64, 56, 56, 128, 3, 3, seed=0)
    got, st = conv_gpu_f32(x, w, 1, 1)
    assert st == qx.OK
    ref = oracle.conv2d_f64(x, w, 1, 1)
    mag = oracle.conv2d_absref(x, w, 1, 1)
    assert_within_tolerance(got, ref, mag, "conv fp32 workload")


@pytest.mark.parametrize("shape,stride,pad", [((1, 3, 7, 9, 5, 3, 3), 1, 1),
                                              ((3, 130, 9, 11, 200, 3, 3), 1, 1),
                                              ((2, 16, 12, 10, 24, 1, 1), 1, 0),
                                              ((1, 64, 30, 30, 64, 3, 3), 2, 1)])
def test_conv_shapes_f32(shape, stride, pad):
    n, c, h, wd, k, r, s = shape
    x, w = inputs.conv_case_f32(n, c, h, wd, k, r, s, seed=sum(shape))
    got, st = conv_gpu_f32(x, w, stride, pad)
    assert st == qx.OK
    assert_within_tolerance(got, oracle.conv2d_f64(x, w, stride, pad),
                            oracle.conv2d_absref(x, w, stride, pad), f"conv fp32 {shape}")


def test_conv_f32_integer_values_exact():
    # integers of at most 11 significant bits are TF32-exact, so the result is exact
    x, w = inputs.conv_case(2, 32, 10, 10, 16, 3, 3, -100, 100, seed=4)   # 288 * 100^2 < 2^24
    got, st = conv_gpu_f32(x.float(), w.float(), 1, 1)
    assert st == qx.OK
    assert (got == oracle.conv2d(x, w, 1, 1)).all()


# ------------------------------------- few input channels (explicit patches)
@pytest.mark.parametrize("shape,stride,pad", [
    ((64, 1, 32, 32, 6, 5, 5), 1, 0),         # LeNet conv1
    ((64, 6, 14, 14, 16, 5, 5), 1, 0),        # LeNet conv2
    ((3, 31, 9, 9, 33, 3, 3), 1, 1),
    ((2, 2, 11, 7, 130, 3, 2), 2, 1),
    ((3, 3, 10, 13, 8, 5, 5), 1, 2),          # halo wider than one tap
    ((2, 16, 60, 60, 24, 3, 3), 1, 1),        # image too large to stage: gather path
    ((1, 4, 9, 9, 7, 4, 2), 3, 0),            # stride 3: unused edge rows and columns
])
def test_conv_explicit_patches(shape, stride, pad):
    n, c, h, wd, k, r, s = shape
    x, w = inputs.conv_case(n, c, h, wd, k, r, s, -255, 255, seed=sum(shape) + stride, dtype=torch.int32)
    ref = oracle.conv2d(x, w, stride, pad)
    got, st, info = conv_gpu(x, w, stride, pad, (-255, 255), (-255, 255), dtype=qx.I32)
    assert st == qx.OK
    assert_exact(got, ref, f"conv {shape} s{stride} p{pad} {info}")


@pytest.mark.parametrize("h", [14, 60])   # staged image, gather path
def test_conv_explicit_patches_range_check(h):
    x, w = inputs.conv_case(2, 6, h, h, 16, 5, 5, 0, 255, seed=h, dtype=torch.int32)
    x[1, 3, h // 2, h // 3] = 256
    _, st, _ = conv_gpu(x, w, 1, 0, (0, 255), (-255, 255), dtype=qx.I32, flags=qx.FLAG_CHECK_RANGES)
    assert st == qx.ERR_CONTRACT
    x[1, 3, h // 2, h // 3] = 255
    got, st, _ = conv_gpu(x, w, 1, 0, (0, 255), (-255, 255), dtype=qx.I32, flags=qx.FLAG_CHECK_RANGES)
    assert st == qx.OK
    assert_exact(got, oracle.conv2d(x, w, 1, 0), "conv patches in range")


def test_conv_explicit_patches_int16():
    x, w = inputs.conv_case(5, 3, 21, 19, 12, 5, 5, -255, 255, seed=3)
    got, st, info = conv_gpu(x, w, 1, 2, (-255, 255), (-255, 255))
    assert st == qx.OK
    assert_exact(got, oracle.conv2d(x, w, 1, 2), f"conv int16 patches {info}")


# --------------------------------- 2 x 2 pooling in the conv's epilogue
@pytest.mark.parametrize("shape,stride,pad,mode,requant", [
    ((64, 1, 32, 32, 6, 5, 5), 1, 0, "max", (4, 255)),        # LeNet conv1 + pool
    ((64, 6, 14, 14, 16, 5, 5), 1, 0, "avg", (5, 255)),       # LeNet conv2 + pool
    ((3, 3, 10, 12, 20, 3, 3), 1, 1, "avg", None),            # negative sums: floor
    ((2, 4, 15, 15, 9, 3, 3), 2, 1, "max", None),
    ((5, 2, 9, 9, 130, 2, 2), 1, 0, "max", (3, 100)),         # two N-side tiles
    ((2, 1, 64, 64, 8, 3, 3), 1, 0, "avg", (2, 255)),         # largest staged image (48208 B)
])
def test_conv_pooled_output(shape, stride, pad, mode, requant):
    n, c, h, wd, k, r, s = shape
    x, w = inputs.conv_case(n, c, h, wd, k, r, s, -255, 255, seed=sum(shape), dtype=torch.int32)
    flags = qx.FLAG_POOL2_MAX if mode == "max" else qx.FLAG_POOL2_AVG
    desc = qx.conv_desc(n, c, h, wd, k, r, s, stride, pad, (-255, 255), (-255, 255), dtype=qx.I32,
                        flags=flags, requant=requant)
    with qx.Plan(desc) as plan:
        y = plan.conv2d(x.cuda(), w.cuda())
        torch.cuda.synchronize()
        assert plan.status() == qx.OK
    full = oracle.conv2d(x, w, stride, pad)
    if requant is not None:
        full = oracle.requant(full, *requant)
    want = oracle.pool2d(wrap32(full), 2, 2, 2, mode)
    assert y.shape == (n, k, want.shape[2], want.shape[3])
    assert_exact(y.cpu().numpy().astype(np.int64), want, f"pooled conv {shape} {mode} {requant}")


# ------------------------------------------------ ReLU-requantize epilogue
@pytest.mark.parametrize("c", [6, 64])      # explicit patches and im2col-on-load
def test_conv_requant_epilogue(c):
    x, w = inputs.conv_case(4, c, 12, 12, 20, 3, 3, -255, 255, seed=c, dtype=torch.int32)
    desc = qx.conv_desc(4, c, 12, 12, 20, 3, 3, 1, 1, (-255, 255), (-255, 255), dtype=qx.I32,
                        requant=(9, 1000))
    with qx.Plan(desc) as plan:
        y = plan.conv2d(x.cuda(), w.cuda())
        torch.cuda.synchronize()
        assert plan.status() == qx.OK
    want = oracle.requant(oracle.conv2d(x, w, 1, 1), 9, 1000)
    assert 0 < (want == 1000).sum() < want.size and (want == 0).any()   # both clamps exercised
    assert_exact(y.cpu().numpy().astype(np.int64), want, f"conv requant c={c}")


# ----------------------------------------------- seeded random shape sweep
@pytest.mark.parametrize("seed", range(3))
def test_conv_random_shapes(seed):
    """Random shapes through both lowerings (explicit patches below 32 input
    channels, im2col on load above), int16 and int32, with the pooled epilogue
    whenever P and Q come out even on the patch path; bit-exact against the
    oracle."""
    rng = np.random.default_rng(900 + seed)
    for _ in range(6):
        c = int(rng.choice([1, 2, 5, 17, 31, 40, 70]))
        n, k = int(rng.integers(1, 4)), int(rng.integers(1, 70))
        r, s = (int(v) for v in rng.integers(1, 6, size=2))
        stride, pad = int(rng.integers(1, 4)), int(rng.integers(0, 3))
        h = int(rng.integers(max(1, r - 2 * pad), 21))
        w = int(rng.integers(max(1, s - 2 * pad), 21))
        dt = torch.int16 if rng.integers(0, 2) else torch.int32
        lim = 255
        x, wt = inputs.conv_case(n, c, h, w, k, r, s, -lim, lim, seed=int(rng.integers(1 << 30)), dtype=dt)
        qdt = qx.I16 if dt == torch.int16 else qx.I32
        full = oracle.conv2d(x, wt, stride, pad)
        P, Q = full.shape[2], full.shape[3]
        pool = c < 32 and P % 2 == 0 and Q % 2 == 0 and rng.integers(0, 2) == 1
        flags = qx.FLAG_POOL2_MAX if pool else 0
        try:
            plan = qx.Plan(qx.conv_desc(n, c, h, w, k, r, s, stride, pad, (-lim, lim), (-lim, lim),
                                        dtype=qdt, flags=flags))
        except qx.QxError as e:
            assert pool and e.status == qx.ERR_UNSUPPORTED     # image too large to stage
            continue
        with plan:
            y = plan.conv2d(x.cuda(), wt.cuda())
            torch.cuda.synchronize()
            assert plan.status() == qx.OK
        want = oracle.pool2d(full, 2, 2, 2, "max") if pool else full
        assert_exact(y.cpu().numpy().astype(np.int64), want,
                     f"conv n{n} c{c} {h}x{w} k{k} {r}x{s} s{stride} p{pad} {dt} pool={pool}")
