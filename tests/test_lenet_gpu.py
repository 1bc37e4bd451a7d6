"""GPU parity of the LeNet-shaped INT32 pipeline (Results: CNN performance)
against the oracle's composition of conv2d, requant, pool2d and gemm, bit
for bit."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_09905_gb300 import inputs, qx

from gpu_util import assert_exact, build_once

pytestmark = pytest.mark.gpu

SHIFTS = (4, 5, 5, 5)
ACT_HI = 255
W_RANGES = [(-7, 7)] * 5


@pytest.fixture(scope="module", autouse=True)
def _built():
    build_once()


def lenet_gpu(x, ws, avg=False, shifts=SHIFTS, act_hi=ACT_HI, range_x=(0, 255), ranges_w=W_RANGES):
    with qx.Lenet(x.shape[0], range_x, ranges_w, shifts, act_hi, avg_pool=avg) as net:
        logits = net.forward(x.cuda(), [w.cuda() for w in ws])
        torch.cuda.synchronize()
        st = net.status()
    return logits.cpu().numpy().astype(np.int64), st


@pytest.mark.parametrize("batch", [1, 7, 64, 300])
def test_lenet_matches_oracle(batch):
    x, *ws = inputs.lenet_case(batch, seed=batch)
    want = oracle.lenet(x, *ws, SHIFTS, ACT_HI)
    got, st = lenet_gpu(x, ws)
    assert st == qx.OK
    assert_exact(got, want, f"lenet batch {batch}")


def test_lenet_average_pooling():
    x, *ws = inputs.lenet_case(33, seed=3)
    want = oracle.lenet(x, *ws, SHIFTS, ACT_HI, pool="avg")
    got, st = lenet_gpu(x, ws, avg=True)
    assert st == qx.OK
    assert_exact(got, want, "lenet, average pooling")


def test_lenet_pass_through_network():
    # the same centre-tap / identity network the oracle is pinned with
    x = torch.randint(0, 100, (3, 1, 32, 32), generator=torch.Generator().manual_seed(6), dtype=torch.int32)
    w1 = torch.zeros((6, 1, 5, 5), dtype=torch.int32); w1[0, 0, 2, 2] = 1
    w2 = torch.zeros((16, 6, 5, 5), dtype=torch.int32); w2[0, 0, 2, 2] = 1
    w3 = torch.zeros((400, 120), dtype=torch.int32); w3[torch.arange(120), torch.arange(120)] = 1
    w4 = torch.zeros((120, 84), dtype=torch.int32); w4[torch.arange(84), torch.arange(84)] = 1
    w5 = torch.ones((84, 10), dtype=torch.int32)
    got, st = lenet_gpu(x, [w1, w2, w3, w4, w5], shifts=(0, 0, 0, 0), act_hi=10**6,
                        range_x=(0, 99), ranges_w=[(0, 1)] * 5)
    assert st == qx.OK
    m = x.numpy()[:, 0, 2:30, 2:30].reshape(3, 14, 2, 14, 2).max(axis=(2, 4))
    m = m[:, 2:12, 2:12].reshape(3, 5, 2, 5, 2).max(axis=(2, 4))
    assert (got == m.reshape(3, -1).sum(axis=1)[:, None]).all()


def test_lenet_rejects_a_range_that_could_overflow():
    with pytest.raises(qx.QxError) as e:
        qx.Lenet(4, (0, 255), [(-7, 7), (-2**20, 2**20), (-7, 7), (-7, 7), (-7, 7)], SHIFTS, ACT_HI)
    assert e.value.status == qx.ERR_CONTRACT


def test_lenet_batch_4096_sampled():
    # the benchmarked batch: every logit on the GPU, the oracle on a spread of
    # images (each image's logits depend on that image alone)
    x, *ws = inputs.lenet_case(4096, seed=4096)
    got, st = lenet_gpu(x, ws)
    assert st == qx.OK
    idx = np.array([0, 1, 511, 1024, 2047, 2048, 3000, 4094, 4095])
    want = oracle.lenet(x[torch.from_numpy(idx)], *ws, SHIFTS, ACT_HI)
    assert_exact(got[idx], want, "lenet batch 4096, sampled images")
