"""GPU parity of the exact integer GEMMs (Table 1: packed INT16-in/INT32-acc
and INT32 operands) against the CPU oracle, bit for bit."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_09905_gb300 import inputs, qx

from gpu_util import assert_exact, build_once, gemm_gpu, wrap32

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    build_once()


def _case(M, N, K, lo, hi, seed, dtype=torch.int16):
    A, B = inputs.gemm_case(M, N, K, lo, hi, seed, dtype)
    ref, worst = oracle.gemm(A, B)
    return A, B, ref, worst


# the Table 1 sweep and the skinny attention-like shape, INT16 operands
@pytest.mark.parametrize("M,N,K", [(256, 256, 256), (512, 512, 512), (768, 768, 768),
                                   (1024, 1024, 1024), (2048, 2048, 2048), (4096, 64, 1024)])
def test_table1_shapes_int16(M, N, K):
    A, B, ref, worst = _case(M, N, K, -1023, 1023, seed=M + N + K)
    assert worst <= 2**31 - 1
    got, st, info = gemm_gpu(A, B, (-1023, 1023), (-1023, 1023))
    assert st == qx.OK
    assert_exact(got, ref, f"gemm {M}x{N}x{K} scheme {info}")


# the same values stored as INT32 operands through the INT32 path
@pytest.mark.parametrize("M,N,K", [(256, 256, 256), (1024, 1024, 1024)])
def test_table1_shapes_int32(M, N, K):
    A, B, ref, _ = _case(M, N, K, -1023, 1023, seed=7 + K, dtype=torch.int32)
    got, st, _ = gemm_gpu(A, B, (-1023, 1023), (-1023, 1023), dtype=qx.I32)
    assert st == qx.OK
    assert_exact(got, ref, "int32 gemm")


@pytest.mark.parametrize("M,N,K", [(1, 1, 1), (7, 13, 5), (129, 257, 65), (300, 200, 1000),
                                   (200, 300, 77), (130, 1, 513), (1, 333, 129), (383, 129, 1)])
def test_ragged_shapes(M, N, K):
    A, B, ref, _ = _case(M, N, K, -1023, 1023, seed=M * 7 + N * 3 + K)
    got, st, info = gemm_gpu(A, B, (-1023, 1023), (-1023, 1023))
    assert st == qx.OK
    assert_exact(got, ref, f"ragged {M}x{N}x{K} {info}")


@pytest.mark.parametrize("a,b", [(1023, 1023), (-1023, 1023), (-1023, -1023), (1008, -1023)])
def test_contract_edge_constant(a, b):
    # constant operands drive every FP32 partial sum to the planner's bound
    M, N, K = 256, 384, 2048
    A = torch.full((M, K), a, dtype=torch.int16)
    B = torch.full((K, N), b, dtype=torch.int16)
    got, st, info = gemm_gpu(A, B, (-1023, 1023), (-1023, 1023))
    assert st == qx.OK
    assert info[0]["acc_bound"] > 0.99 * 2**24 or info[0]["acc_bound"] > 12_000_000
    assert (got == K * a * b).all(), f"constant {a}*{b}: {np.unique(got)[:4]} scheme {info}"


def test_contract_edge_digit_extremes():
    # values whose low digit is -2^(s-1) or whose high digit is extreme, mixed signs
    M, N, K = 128, 256, 1024
    g = torch.Generator().manual_seed(3)
    choices = torch.tensor([1023, -1023, 1008, -1008, 16, -16, 48, -1024 + 1], dtype=torch.int16)
    A = choices[torch.randint(0, len(choices), (M, K), generator=g)]
    B = torch.where(torch.rand(K, N, generator=g) < 0.5, 1023, -1023).to(torch.int16)
    ref, _ = oracle.gemm(A, B)
    got, st, info = gemm_gpu(A, B, (-1023, 1023), (-1023, 1023))
    assert st == qx.OK
    assert_exact(got, ref, f"digit extremes {info}")


# every kernel instance (N-side limbs x M-side limbs) through ranges that need it
@pytest.mark.parametrize("ra,rb,K,want", [
    ((-100, 100), (-100, 100), 300, (1, 1)),
    ((-1023, 1023), (-1023, 1023), 200, (2, 1)),
    ((-10, 10), (-30000, 30000), 100, (1, 2)),
    ((-32767, 32767), (-32767, 32767), 64, (2, 2)),
    ((-2**20, 2**20), (-2048, 2048), 70, (3, 1)),
    ((-2**26, 2**26), (-2048, 2048), 70, (4, 1)),
    ((-2**26, 2**26), (-2**15, 2**15), 70, (4, 2)),
])
def test_every_limb_scheme_int32(ra, rb, K, want):
    info = qx.query(qx.gemm_desc(200, 150, K, ra, rb, dtype=qx.I32))[0]
    assert (info["limbs_a"], info["limbs_b"]) == want
    g = torch.Generator().manual_seed(K)
    A = torch.randint(ra[0], ra[1] + 1, (200, K), generator=g, dtype=torch.int32)
    B = torch.randint(rb[0], rb[1] + 1, (K, 150), generator=g, dtype=torch.int32)
    A[0, :] = ra[1]
    B[:, 0] = rb[1]
    ref, _ = oracle.gemm(A, B)
    got, st, _ = gemm_gpu(A, B, ra, rb, dtype=qx.I32)
    assert st == qx.OK
    assert_exact(got, wrap32(ref), f"scheme {want}")   # exact modulo 2^32


def test_full_int16_range_small_k():
    A, B, ref, worst = _case(96, 160, 2, -32768, 32767, seed=5)
    assert worst < 2**31
    got, st, info = gemm_gpu(A, B, (-32768, 32767), (-32768, 32767))
    assert st == qx.OK
    assert_exact(got, ref, f"full range {info}")


def test_k_zero_gives_zeros():
    A = torch.zeros((5, 0), dtype=torch.int16)
    B = torch.zeros((0, 7), dtype=torch.int16)
    got, st, _ = gemm_gpu(A, B, (-1, 1), (-1, 1))
    assert st == qx.OK and (got == 0).all() and got.shape == (5, 7)


def test_plan_reuse_and_side_stream():
    M, N, K = 300, 260, 700
    plan = qx.Plan(qx.gemm_desc(M, N, K, (-1023, 1023), (-1023, 1023)))
    s = torch.cuda.Stream()
    for seed in (1, 2, 3):
        A, B, ref, _ = _case(M, N, K, -1023, 1023, seed)
        with torch.cuda.stream(s):
            C = plan.gemm_i16_i32(A.cuda(), B.cuda())
        s.synchronize()
        assert_exact(C.cpu().numpy().astype(np.int64), ref, f"reuse {seed}")
    assert plan.status() == qx.OK
    plan.close()


def test_leading_dimensions():
    M, N, K = 70, 90, 110
    lda, ldb, ldc = 128, 96, 104
    g = torch.Generator().manual_seed(9)
    Af = torch.randint(-1023, 1024, (M, lda), generator=g, dtype=torch.int16)
    Bf = torch.randint(-1023, 1024, (K, ldb), generator=g, dtype=torch.int16)
    ref, _ = oracle.gemm(Af[:, :K], Bf[:, :N])
    with qx.Plan(qx.gemm_desc(M, N, K, (-1023, 1023), (-1023, 1023), lda=lda, ldb=ldb, ldc=ldc)) as p:
        C = torch.full((M, ldc), -7, dtype=torch.int32, device="cuda")
        p.gemm_i16_i32(Af.cuda(), Bf.cuda(), C)
        torch.cuda.synchronize()
    C = C.cpu().numpy().astype(np.int64)
    assert_exact(C[:, :N], ref, "ld")
    assert (C[:, N:] == -7).all()          # padding columns untouched


def test_range_check_flags_contract_violation():
    M = N = K = 128
    A, B = inputs.gemm_case(M, N, K, -100, 100, seed=1)
    A[5, 7] = 101
    got, st, _ = gemm_gpu(A, B, (-100, 100), (-100, 100), flags=qx.FLAG_CHECK_RANGES)
    assert st == qx.ERR_CONTRACT
    A[5, 7] = 100
    got, st, _ = gemm_gpu(A, B, (-100, 100), (-100, 100), flags=qx.FLAG_CHECK_RANGES)
    assert st == qx.OK
    assert_exact(got, oracle.gemm(A, B)[0], "checked")


def test_argument_errors_return_before_launch():
    plan = qx.Plan(qx.gemm_desc(64, 64, 64, (-5, 5), (-5, 5)))
    A = torch.zeros((64, 64), dtype=torch.int16, device="cuda")
    with pytest.raises(ValueError):
        plan.gemm_i16_i32(A, A.to(torch.int32))
    lib = qx.load()
    assert lib.qx_gemm_i16_i32(plan.handle, None, A.data_ptr(), A.data_ptr(), None) == qx.ERR_INVALID_ARG
    assert lib.qx_gemm_i16_i32(plan.handle, A.data_ptr() + 2, A.data_ptr(), A.data_ptr(),
                               None) == qx.ERR_UNSUPPORTED
    assert lib.qx_gemm_i32(plan.handle, A.data_ptr(), A.data_ptr(), A.data_ptr(), None) == qx.ERR_INVALID_ARG
    assert lib.qx_conv2d_gemm(plan.handle, A.data_ptr(), A.data_ptr(), A.data_ptr(), None) == qx.ERR_INVALID_ARG
    plan.close()


def test_gemm_8192_sampled_rows_and_freivalds():
    """The 8192^3 INT16 GEMM (values in [-500, 500]) in the bench's launch
    configuration: 48 sampled rows against the oracle, and the whole result
    through Freivalds' check A (B x) == C x with random +-1 vectors."""
    M = N = K = 8192
    A, B = inputs.gemm_case(M, N, K, -500, 500, seed=0)
    got, st, info = gemm_gpu(A, B, (-500, 500), (-500, 500))
    assert st == qx.OK and info[0]["n_chunks"] == 4
    rows = np.random.default_rng(0).choice(M, size=48, replace=False)
    rows = np.concatenate([[0, M - 1], rows])
    ref_rows, _ = oracle.gemm(A[rows], B)
    assert_exact(got[rows], ref_rows, "8192 sampled rows")
    a = A.numpy().astype(np.int64)
    b = B.numpy().astype(np.int64)
    rng = np.random.default_rng(1)
    for _ in range(4):
        x = rng.choice([-1, 1], size=(N, 2)).astype(np.int64)
        assert (a @ (b @ x) == got @ x).all()


def test_full_smul24_operand_range_int32():
    """INT32 operands over the whole 24-bit signed range of the smul24 contract
    (|a|, |b| < 2^23): four digits of A times two of B; the product is exact
    modulo 2^32 (it leaves int32, so the oracle's value is reduced the same way)."""
    r = (-(2**23 - 1), 2**23 - 1)
    info = qx.query(qx.gemm_desc(130, 140, 300, r, r, dtype=qx.I32))[0]
    assert (info["limbs_a"], info["limbs_b"]) == (4, 2)
    g = torch.Generator().manual_seed(23)
    A = torch.randint(r[0], r[1] + 1, (130, 300), generator=g, dtype=torch.int32)
    B = torch.randint(r[0], r[1] + 1, (300, 140), generator=g, dtype=torch.int32)
    A[0, :] = r[1]
    A[1, :] = r[0]
    B[:, 0] = r[1]
    ref, _ = oracle.gemm(A, B)
    got, st, _ = gemm_gpu(A, B, r, r, dtype=qx.I32)
    assert st == qx.OK
    assert_exact(got, wrap32(ref), "smul24 range")


def test_gemm_requant_epilogue():
    A, B = inputs.gemm_case(300, 130, 200, -255, 255, seed=61, dtype=torch.int32)
    desc = qx.gemm_desc(300, 130, 200, (-255, 255), (-255, 255), dtype=qx.I32, requant=(8, 5000))
    with qx.Plan(desc) as plan:
        C = plan.gemm_i32(A.cuda(), B.cuda())
        torch.cuda.synchronize()
        assert plan.status() == qx.OK
    want = oracle.requant(oracle.gemm(A, B)[0], 8, 5000)
    assert (want == 5000).any() and (want == 0).any()
    assert_exact(C.cpu().numpy().astype(np.int64), want, "gemm requant")


def test_int8_mma_peak_measurement():
    # the measurement utility behind the INT8-limb roofline: a positive rate,
    # and argument errors returned without work
    tops = qx.measure_int8_mma_peak(0)
    assert 1.0 < tops < 1e5
    assert qx.load().qx_measure_int8_mma_peak(0, None) == qx.ERR_INVALID_ARG


# Narrow outputs exercise the short-tile paths of the limb kernel: the N side
# (rows of C) in one tile loaded once per CTA when its k-blocks fit the stage
# ring, the last k-block's empty K sub-steps skipped, and the two epilogue
# warps of a lane quarter taking alternate tiles when every row of C falls in
# the first half of the tile -- with one FP32 chunk per tile or several.
@pytest.mark.parametrize("M,N,K,lim,dtype", [
    (6, 1000, 40, 255, torch.int16),        # resident N side, 3 of 4 sub-steps, one chunk
    (8, 4096, 100, 1023, torch.int16),      # 2 k-blocks, tail of 3 sub-steps
    (20, 777, 5000, 2000, torch.int32),     # many chunks, N side re-loaded per tile
    (40, 300, 130, 255, torch.int32),       # rows past the first half: no alternation
    (33, 2000, 17, 7, torch.int32),         # one sub-step of one k-block
])
def test_narrow_outputs(M, N, K, lim, dtype):
    A, B, ref, _ = _case(M, N, K, -lim, lim, seed=M * 7 + K, dtype=dtype)
    dt = qx.I16 if dtype == torch.int16 else qx.I32
    got, st, info = gemm_gpu(A, B, (-lim, lim), (-lim, lim), dtype=dt, path="prepass")
    assert st == qx.OK
    if (M, N, K) == (20, 777, 5000):
        assert info[0]["n_chunks"] > 1
    assert_exact(got, wrap32(ref), f"narrow GEMM {M}x{N}x{K} {info}")
