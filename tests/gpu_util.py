"""Helpers shared by the GPU parity tests (test-side marshalling only)."""
import numpy as np
import torch

import oracle
from paper_2606_09905_gb300 import qx


def build_once():
    from paper_2606_09905_gb300 import _build
    _build.build()
    qx.load()


def wrap32(x: np.ndarray) -> np.ndarray:
    """Exact integers reduced to int32 two's complement (the result modulo 2^32)."""
    return ((x.astype(np.int64) + 2**31) % 2**32 - 2**31).astype(np.int64)


PATH_FLAGS = {None: 0, "fused": qx.FLAG_FUSED_CONVERT, "prepass": qx.FLAG_PREPASS}


def gemm_gpu(A, B, range_a, range_b, dtype=qx.I16, flags=0, stream=None, path=None):
    """C = A B through one plan; `path` forces the fused or the pre-pass GEMM."""
    M, K = A.shape
    N = B.shape[1]
    flags |= PATH_FLAGS[path]
    with qx.Plan(qx.gemm_desc(M, N, K, range_a, range_b, dtype=dtype, flags=flags)) as plan:
        if path is not None:
            assert plan.fused == (path == "fused")
        fn = plan.gemm_i16_i32 if dtype == qx.I16 else plan.gemm_i32
        C = fn(A.cuda(), B.cuda(), stream=stream)
        torch.cuda.synchronize()
        st = plan.status()
        info = plan.info()
    return C.cpu().numpy().astype(np.int64), st, info


def assert_exact(got: np.ndarray, ref: np.ndarray, what: str = ""):
    if not np.array_equal(got, ref):
        bad = np.argwhere(got != ref)
        i = tuple(bad[0])
        raise AssertionError(f"{what}: {len(bad)} of {ref.size} elements differ; first at {i}: "
                             f"got {got[i]}, expected {ref[i]}")


def oracle_gemm_exact(A, B):
    C, _ = oracle.gemm(A, B)
    return C
