"""GPU parity of the fused-conversion GEMM (operands split into FP16 limbs
inside the tensor-core kernel, one launch) against the CPU oracle, bit for
bit, and against the two-kernel pre-pass path on the same inputs."""
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


# Table 1 sizes through the fused kernel; 2048^3 has more tiles than SMs, so
# CTAs loop over tiles and their warps alternate conversion and epilogue
@pytest.mark.parametrize("M,N,K", [(256, 256, 256), (512, 512, 512), (768, 768, 768),
                                   (1024, 1024, 1024), (2048, 2048, 2048), (4096, 64, 1024)])
@pytest.mark.parametrize("dtype", [torch.int16, torch.int32])
def test_table1_shapes_fused(M, N, K, dtype):
    A, B = inputs.gemm_case(M, N, K, -1023, 1023, seed=M + 2 * N + K, dtype=dtype)
    ref, _ = oracle.gemm(A, B)
    got, st, info = gemm_gpu(A, B, (-1023, 1023), (-1023, 1023),
                             dtype=qx.I16 if dtype == torch.int16 else qx.I32, path="fused")
    assert st == qx.OK
    assert_exact(got, ref, f"fused {M}x{N}x{K} {dtype} {info}")


# ragged M, N and K with rows padded to 16 bytes: partial tiles, partial
# 8-element groups at the row ends (zero-filled copies) and a K tail
@pytest.mark.parametrize("M,N,K", [(1, 1, 1), (7, 13, 5), (129, 257, 65), (300, 200, 1000),
                                   (200, 300, 77), (130, 1, 513), (1, 333, 129), (383, 129, 1)])
def test_ragged_shapes_fused(M, N, K):
    lda, ldb = (K + 7) // 8 * 8, (N + 7) // 8 * 8
    g = torch.Generator().manual_seed(M * 5 + N * 3 + K)
    Af = torch.randint(-1023, 1024, (M, lda), generator=g, dtype=torch.int16)
    Bf = torch.randint(-1023, 1024, (K, ldb), generator=g, dtype=torch.int16)
    ref, _ = oracle.gemm(Af[:, :K], Bf[:, :N])
    desc = qx.gemm_desc(M, N, K, (-1023, 1023), (-1023, 1023), lda=lda, ldb=ldb,
                        flags=qx.FLAG_FUSED_CONVERT)
    with qx.Plan(desc) as p:
        assert p.fused
        C = p.gemm_i16_i32(Af.cuda(), Bf.cuda())
        torch.cuda.synchronize()
        assert p.status() == qx.OK
    assert_exact(C.cpu().numpy().astype(np.int64), ref, f"ragged fused {M}x{N}x{K}")


# every kernel instance (N-side limbs x M-side limbs), INT32 operands; the
# (2, 2) and (4, 2) instances hold one raw k-block at a time
@pytest.mark.parametrize("ra,rb,K,want", [
    ((-100, 100), (-100, 100), 304, (1, 1)),
    ((-1023, 1023), (-1023, 1023), 200, (2, 1)),
    ((-10, 10), (-30000, 30000), 104, (1, 2)),
    ((-32767, 32767), (-32767, 32767), 64, (2, 2)),
    ((-2**20, 2**20), (-2048, 2048), 72, (3, 1)),
    ((-2**26, 2**26), (-2048, 2048), 72, (4, 1)),
    ((-2**26, 2**26), (-2**15, 2**15), 72, (4, 2)),
])
def test_every_limb_scheme_fused(ra, rb, K, want):
    info = qx.query(qx.gemm_desc(200, 152, K, ra, rb, dtype=qx.I32))[0]
    assert (info["limbs_a"], info["limbs_b"]) == want
    g = torch.Generator().manual_seed(K + 1)
    A = torch.randint(ra[0], ra[1] + 1, (200, K), generator=g, dtype=torch.int32)
    B = torch.randint(rb[0], rb[1] + 1, (K, 152), generator=g, dtype=torch.int32)
    A[0, :] = ra[1]
    A[1, :] = ra[0]
    B[:, 0] = rb[1]
    B[:, 1] = rb[0]
    ref, _ = oracle.gemm(A, B)
    got, st, _ = gemm_gpu(A, B, ra, rb, dtype=qx.I32, path="fused")
    assert st == qx.OK
    assert_exact(got, wrap32(ref), f"fused scheme {want}")


def test_full_smul24_range_fused():
    r = (-(2**23 - 1), 2**23 - 1)
    g = torch.Generator().manual_seed(24)
    A = torch.randint(r[0], r[1] + 1, (136, 96), generator=g, dtype=torch.int32)
    B = torch.randint(r[0], r[1] + 1, (96, 120), generator=g, dtype=torch.int32)
    ref, _ = oracle.gemm(A, B)
    got, st, info = gemm_gpu(A, B, r, r, dtype=qx.I32, path="fused")
    assert st == qx.OK
    assert_exact(got, wrap32(ref), f"smul24 fused {info}")


@pytest.mark.parametrize("a,b", [(1023, 1023), (-1023, 1023), (1008, -1023)])
def test_contract_edge_constant_fused(a, b):
    # K = 2048: several FP32 chunks per tile, each driven to the planner's bound
    M, N, K = 256, 384, 2048
    A = torch.full((M, K), a, dtype=torch.int16)
    B = torch.full((K, N), b, dtype=torch.int16)
    got, st, info = gemm_gpu(A, B, (-1023, 1023), (-1023, 1023), path="fused")
    assert st == qx.OK
    assert info[0]["n_chunks"] > 1
    assert (got == K * a * b).all(), f"constant {a}*{b}: {np.unique(got)[:4]} scheme {info}"


def test_fused_equals_prepass_bitwise():
    # both paths on the same plan shape and inputs, exact modulo 2^32 even
    # when the true product leaves int32 (ranges that allow it)
    M, N, K = 384, 264, 520
    g = torch.Generator().manual_seed(77)
    A = torch.randint(-30000, 30001, (M, K), generator=g, dtype=torch.int32)
    B = torch.randint(-30000, 30001, (K, N), generator=g, dtype=torch.int32)
    f, st1, _ = gemm_gpu(A, B, (-30000, 30000), (-30000, 30000), dtype=qx.I32, path="fused")
    p, st2, _ = gemm_gpu(A, B, (-30000, 30000), (-30000, 30000), dtype=qx.I32, path="prepass")
    assert st1 == st2 == qx.OK
    assert np.array_equal(f, p)
    assert_exact(f, wrap32(oracle.gemm(A, B)[0]), "fused vs oracle")


def test_range_check_fused():
    A, B = inputs.gemm_case(136, 128, 128, -100, 100, seed=3)
    B[70, 9] = -101
    _, st, _ = gemm_gpu(A, B, (-100, 100), (-100, 100), flags=qx.FLAG_CHECK_RANGES, path="fused")
    assert st == qx.ERR_CONTRACT
    B[70, 9] = -100
    A[135, 127] = 101
    _, st, _ = gemm_gpu(A, B, (-100, 100), (-100, 100), flags=qx.FLAG_CHECK_RANGES, path="fused")
    assert st == qx.ERR_CONTRACT
    A[135, 127] = 100
    got, st, _ = gemm_gpu(A, B, (-100, 100), (-100, 100), flags=qx.FLAG_CHECK_RANGES, path="fused")
    assert st == qx.OK
    assert_exact(got, oracle.gemm(A, B)[0], "checked fused")


def test_requant_epilogue_fused():
    M, N, K = 200, 120, 400
    A, B = inputs.gemm_case(M, N, K, 0, 255, seed=12, dtype=torch.int32)
    B = B - 128
    ref, _ = oracle.gemm(A, B)
    want = oracle.requant(ref, 9, 255)
    desc = qx.gemm_desc(M, N, K, (0, 255), (-128, 127), dtype=qx.I32, requant=(9, 255),
                        flags=qx.FLAG_FUSED_CONVERT)
    with qx.Plan(desc) as p:
        assert p.fused
        C = p.gemm_i32(A.cuda(), B.cuda())
        torch.cuda.synchronize()
        assert p.status() == qx.OK
    assert_exact(C.cpu().numpy().astype(np.int64), want, "requant fused")


def test_path_choice():
    # the pre-pass path unless the fused one is asked for
    d = lambda flags: qx.gemm_desc(256, 256, 256, (-1023, 1023), (-1023, 1023), flags=flags)
    plans = [qx.Plan(d(0)), qx.Plan(d(qx.FLAG_PREPASS)), qx.Plan(d(qx.FLAG_FUSED_CONVERT))]
    try:
        assert [p.fused for p in plans] == [False, False, True]
    finally:
        for p in plans:
            p.close()


def test_fused_flag_rejects_unaligned_rows():
    with pytest.raises(qx.QxError) as e:
        qx.Plan(qx.gemm_desc(64, 64, 63, (-5, 5), (-5, 5), flags=qx.FLAG_FUSED_CONVERT))
    assert e.value.status == qx.ERR_UNSUPPORTED


def test_pack_and_run_packed_on_a_fused_plan():
    # the split calls keep the two-kernel path and give the same bits
    A, B = inputs.gemm_case(256, 256, 256, -1023, 1023, seed=4)
    ref, _ = oracle.gemm(A, B)
    with qx.Plan(qx.gemm_desc(256, 256, 256, (-1023, 1023), (-1023, 1023),
                              flags=qx.FLAG_FUSED_CONVERT)) as p:
        assert p.fused
        C = torch.empty((256, 256), dtype=torch.int32, device="cuda")
        p.pack(A.cuda(), B.cuda())
        p.run_packed(C)
        torch.cuda.synchronize()
        assert p.status() == qx.OK
    assert_exact(C.cpu().numpy().astype(np.int64), ref, "split calls")


def test_fused_in_cuda_graph_back_to_back():
    M, N, K = 512, 512, 512
    A, B = inputs.gemm_case(M, N, K, -1023, 1023, seed=8)
    ref, _ = oracle.gemm(A, B)
    dA, dB = A.cuda(), B.cuda()
    C = torch.empty((M, N), dtype=torch.int32, device="cuda")
    with qx.Plan(qx.gemm_desc(M, N, K, (-1023, 1023), (-1023, 1023), flags=qx.FLAG_FUSED_CONVERT)) as p:
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            p.gemm_i16_i32(dA, dB, C)
        s.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            for _ in range(4):
                p.gemm_i16_i32(dA, dB, C)
        C.zero_()
        g.replay()
        torch.cuda.synchronize()
        assert p.status() == qx.OK
    assert_exact(C.cpu().numpy().astype(np.int64), ref, "graph")
