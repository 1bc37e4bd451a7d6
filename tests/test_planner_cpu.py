"""The host planner's exactness guarantee, checked against arithmetic done
here rather than against the planner's own bookkeeping.

For every scheme the planner returns, the Methodology's exactness argument
needs three facts: (1) every admissible operand value splits into the
declared number of balanced base-2^s digits, each an exact FP16 integer
(|digit| <= 2048), and the digits recombine to the value; (2) no FP32
partial sum over one chunk can reach 2^24, i.e. chunk_k x max|digit_a| x
max|digit_b| <= 2^24; (3) the chunks cover K and the recombination weights
fit the int32 result.  The digit bounds are measured here by splitting every
value of the range (small ranges) or its extremes plus a seeded sample
(large ranges), so a planner that under-counts a top digit, over-sizes a
chunk or drops a limb fails.  Host-only: no device is touched."""
import numpy as np
import pytest

from paper_2606_09905_gb300 import qx

ACC_LIMIT = 2**24
FP16_EXACT = 2048


@pytest.fixture(scope="module", autouse=True)
def lib():
    from paper_2606_09905_gb300 import _build
    _build.build()
    return qx.load()


def balanced_digits(x: np.ndarray, limbs: int, shift: int) -> list[np.ndarray]:
    """Digits d_0..d_{limbs-1} with x = sum d_i 2^(i*shift); every digit but
    the top one lies in [-2^(shift-1), 2^(shift-1))."""
    x = x.astype(np.int64).copy()
    if limbs == 1:
        return [x]
    base = np.int64(1) << np.int64(shift)
    half = base // 2
    out = []
    for _ in range(limbs - 1):
        d = np.mod(x + half, base) - half
        out.append(d)
        x = (x - d) // base
    out.append(x)
    return out


def values_of(lo: int, hi: int, rng: np.random.Generator) -> np.ndarray:
    if hi - lo <= 200_000:
        return np.arange(lo, hi + 1, dtype=np.int64)
    sample = rng.integers(lo, hi, size=20_000, endpoint=True, dtype=np.int64)
    edges = np.array([lo, lo + 1, hi - 1, hi, 0, -1, 1], dtype=np.int64)
    edges = edges[(edges >= lo) & (edges <= hi)]
    return np.concatenate([sample, edges])


def max_digit(lo: int, hi: int, limbs: int, shift: int, rng) -> int:
    """Largest |digit| over the range; asserts the digits recombine exactly."""
    x = values_of(lo, hi, rng)
    ds = balanced_digits(x, limbs, shift)
    back = sum(d * (np.int64(1) << np.int64(i * shift)) for i, d in enumerate(ds))
    assert np.array_equal(back, x), (lo, hi, limbs, shift)
    # The top digit is monotone in x, so the range ends bound it even when
    # only a sample of the interior was split.
    top = balanced_digits(np.array([lo, hi], dtype=np.int64), limbs, shift)[-1]
    m = max(int(np.abs(d).max()) for d in ds)
    return max(m, int(np.abs(top).max()))


def check_contraction(s: dict, range_a, range_b, K: int, rng):
    la, sa, lb, sb = s["limbs_a"], s["shift_a"], s["limbs_b"], s["shift_b"]
    assert 1 <= la <= 4 and 1 <= lb <= 2
    if la > 1:
        assert 1 <= sa <= 12
    if lb > 1:
        assert 1 <= sb <= 12
    da = max_digit(*range_a, la, sa, rng)
    db = max_digit(*range_b, lb, sb, rng)
    assert da <= FP16_EXACT and db <= FP16_EXACT, (s, da, db)
    per = max(1, da * db)
    assert s["chunk_k"] % 64 == 0
    assert s["chunk_k"] * per <= ACC_LIMIT, (s, da, db)
    assert s["acc_bound"] >= s["chunk_k"] * per     # the recorded bound is not optimistic
    assert s["acc_bound"] <= ACC_LIMIT
    assert s["k"] == K
    if K > 0:
        assert s["n_chunks"] * s["chunk_k"] >= K
        assert (s["n_chunks"] - 1) * s["chunk_k"] < K          # no empty chunk
    assert (la - 1) * (sa if la > 1 else 0) + (lb - 1) * (sb if lb > 1 else 0) <= 31
    assert s["mma_per_kstep"] == la * lb


def random_range(rng, mag_max: int):
    kind = rng.integers(0, 4)
    m = int(rng.integers(1, mag_max + 1))
    if kind == 0:
        return (-m, m)
    if kind == 1:
        return (0, m)
    if kind == 2:
        return (-m, int(rng.integers(-m, m + 1)))
    lo = int(rng.integers(-m, m + 1))
    return (lo, int(rng.integers(lo, m + 1)))


@pytest.mark.parametrize("seed", range(6))
def test_gemm_i16_schemes_are_exact(seed):
    rng = np.random.default_rng(1000 + seed)
    for _ in range(12):
        ra, rb = random_range(rng, 32767), random_range(rng, 32767)
        K = int(rng.choice([1, 63, 64, 65, 1000, 4096, 8192, 65536]))
        s = qx.query(qx.gemm_desc(128, 128, K, ra, rb))
        assert len(s) == 1
        check_contraction(s[0], ra, rb, K, rng)


@pytest.mark.parametrize("seed", range(4))
def test_gemm_i32_schemes_are_exact_or_refused(seed):
    rng = np.random.default_rng(2000 + seed)
    accepted = 0
    for _ in range(16):
        ra, rb = random_range(rng, 2**int(rng.integers(4, 31)) - 1), random_range(rng, 2**int(rng.integers(4, 31)) - 1)
        K = int(rng.choice([64, 777, 4096]))
        try:
            s = qx.query(qx.gemm_desc(64, 64, K, ra, rb, dtype=qx.I32))
        except qx.QxError as e:
            assert e.status == qx.ERR_CONTRACT
            # with max|b| < 2^11 (one digit) and max|a| < 2^23 (four 8-bit
            # digits, each |d| <= 128) a 64-term chunk stays below 2^24, so
            # a refusal is only allowed outside that box
            ma, mb = max(map(abs, ra)), max(map(abs, rb))
            assert ma >= 2**23 or mb >= 2**11, (ra, rb)
            continue
        accepted += 1
        check_contraction(s[0], ra, rb, K, rng)
    assert accepted > 0


def test_gemm_full_int16_range_every_value():
    """The full INT16 contract, every one of the 65536 values split."""
    rng = np.random.default_rng(7)
    full = (-32768, 32767)
    for K in (64, 8192, 2**20):
        s = qx.query(qx.gemm_desc(256, 256, K, full, full))[0]
        check_contraction(s, full, full, K, rng)


def test_single_digit_when_one_chunk_covers_k():
    """When max|a| max|b| K <= 2^24 the plain products need neither a digit
    split nor a second chunk, and no other scheme can do less work."""
    for m, K in ((1, 2**20), (7, 4096), (64, 4096), (181, 512)):
        assert m * m * K <= ACC_LIMIT
        s = qx.query(qx.gemm_desc(64, 64, K, (-m, m), (-m, m)))[0]
        assert s["mma_per_kstep"] == 1 and s["n_chunks"] == 1, (m, K, s)


@pytest.mark.parametrize("seed", range(3))
def test_conv_schemes_are_exact(seed):
    rng = np.random.default_rng(3000 + seed)
    for _ in range(8):
        rx, rw = random_range(rng, 32767), random_range(rng, 32767)
        c = int(rng.choice([1, 3, 16, 64, 100]))
        r = int(rng.choice([1, 3, 5]))
        try:
            s = qx.query(qx.conv_desc(2, c, 16, 16, 32, r, r, 1, r // 2, rx, rw))
        except qx.QxError as e:
            # the x side is limited to two digits by the im2col path
            assert e.status == qx.ERR_UNSUPPORTED
            continue
        assert len(s) == 1
        # N side = weights, M side = the input image
        check_contraction(s[0], rw, rx, s[0]["k"], rng)
        assert s[0]["k"] >= c * r * r


@pytest.mark.parametrize("seed", range(3))
def test_attention_schemes_are_exact(seed):
    rng = np.random.default_rng(4000 + seed)
    done = 0
    for _ in range(20):
        L = int(rng.choice([64, 200, 1024, 4096]))
        d = int(rng.choice([16, 64, 128]))
        rq, rk, rv = (random_range(rng, int(rng.integers(1, 64))) for _ in range(3))
        # d max|Q| max|K| <= 128 * 63 * 63 < 2^24: always plannable
        s0, s1 = qx.query(qx.attn_desc(L, d, rq, rk, rv))
        done += 1
        qm, km, vm = (max(map(abs, r)) for r in (rq, rk, rv))
        smax = d * qm * km
        # S = Q K^T: one digit per side, all d terms in one FP32 sum
        assert s0["limbs_a"] == 1 and s0["limbs_b"] == 1
        assert s0["acc_bound"] >= smax and smax <= ACC_LIMIT
        # O = S V: S in balanced digits over [-smax, smax], V whole
        la, sh = s1["limbs_a"], s1["shift_a"]
        dS = max_digit(-smax, smax, la, sh, rng)
        assert dS <= FP16_EXACT and vm <= FP16_EXACT
        assert s1["chunk_k"] * max(1, dS * vm) <= ACC_LIMIT
        assert s1["n_chunks"] * s1["chunk_k"] >= L
    assert done > 0
