"""GPU parity of the attention core O = (Q K^T) V (Table 2 attention rows; no
softmax, no scale) against the CPU oracle, bit for bit."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_09905_gb300 import inputs, qx

from gpu_util import assert_exact, build_once

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    build_once()


def attn_gpu(Q, K, V, rq, rk, rv, dtype=qx.I16, flags=0):
    L, d = Q.shape
    with qx.Plan(qx.attn_desc(L, d, rq, rk, rv, dtype=dtype, flags=flags)) as plan:
        O = plan.attn(Q.cuda(), K.cuda(), V.cuda())
        torch.cuda.synchronize()
        st = plan.status()
        info = plan.info()
    return O.cpu().numpy().astype(np.int64), st, info


def test_attn_workload_int16():
    Q, K, V = inputs.attn_case(1024, 64, -7, 7, seed=0)
    ref, _, worst = oracle.attn(Q, K, V)
    assert worst <= 3136
    got, st, info = attn_gpu(Q, K, V, (-7, 7), (-7, 7), (-7, 7))
    assert st == qx.OK
    assert_exact(got, ref, f"attn workload {info}")


def test_attn_workload_int32():
    Q, K, V = inputs.attn_case(1024, 64, -7, 7, seed=1, dtype=torch.int32)
    ref, _, _ = oracle.attn(Q, K, V)
    got, st, _ = attn_gpu(Q, K, V, (-7, 7), (-7, 7), (-7, 7), dtype=qx.I32)
    assert st == qx.OK
    assert_exact(got, ref, "attn int32")


@pytest.mark.parametrize("L,d", [(1, 64), (100, 64), (1000, 32), (300, 128), (129, 8),
                                 (4096, 64), (640, 96)])
def test_attn_shapes(L, d):
    Q, K, V = inputs.attn_case(L, d, -7, 7, seed=L + d)
    ref, _, _ = oracle.attn(Q, K, V)
    got, st, info = attn_gpu(Q, K, V, (-7, 7), (-7, 7), (-7, 7))
    assert st == qx.OK
    assert_exact(got, ref, f"attn L={L} d={d} {info}")


def test_attn_extremes():
    L, d = 512, 64
    Q = torch.full((L, d), 7, dtype=torch.int16)
    K = torch.full((L, d), -7, dtype=torch.int16)
    V = torch.full((L, d), 7, dtype=torch.int16)
    got, st, _ = attn_gpu(Q, K, V, (-7, 7), (-7, 7), (-7, 7))
    assert st == qx.OK
    assert (got == -3136 * 7 * L).all()


def test_attn_identity_reassociation():
    # (Q K^T) V = Q (K^T V) exactly, with wider value ranges
    L, d = 256, 64
    g = torch.Generator().manual_seed(4)
    Q = torch.randint(-40, 41, (L, d), generator=g, dtype=torch.int16)
    K = torch.randint(-40, 41, (L, d), generator=g, dtype=torch.int16)
    V = torch.randint(-30, 31, (L, d), generator=g, dtype=torch.int16)
    got, st, info = attn_gpu(Q, K, V, (-40, 40), (-40, 40), (-30, 30))
    assert st == qx.OK
    q, k, v = (t.numpy().astype(np.int64) for t in (Q, K, V))
    assert_exact(got, q @ (k.T @ v), f"reassociation {info}")
