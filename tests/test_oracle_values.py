"""Pins of the oracle's value maps against closed forms, library routines,
exhaustive enumeration and distribution tests.

Value maps are this library's reading of "synthesize test inputs with standard
numerical methods" (CUDA-Harness Sec. 4.2.1); the broad-range requirement
(a Gaussian with mean 5 and standard deviation 10 is the paper's example) is
why the normal map takes an arbitrary mean and scale.
"""
import math

import numpy as np
import pytest
import torch
from scipy import stats

# ---------------------------------------------------------------------------
# fp32 -> bf16 / fp16, round to nearest even
# ---------------------------------------------------------------------------


def _bf16_patterns():
    hi = np.arange(1 << 16, dtype=np.uint32) << 16
    lows = np.array([0, 1, 0x7FFF, 0x8000, 0x8001, 0xFFFF, 0x4000, 0xC000], dtype=np.uint32)
    rng = np.random.default_rng(1)
    rnd = rng.integers(0, 1 << 16, size=8, dtype=np.uint32)
    return (hi[:, None] | np.concatenate([lows, rnd])[None, :]).ravel()


def test_bf16_rounding_matches_torch(oracle):
    # every bf16 high half with the low halves that decide the rounding
    # (below, at and above the tie, odd and even), against torch's conversion
    u = _bf16_patterns()
    x = u.view(np.float32)
    got = oracle.f32_to_bf16(x)
    want = torch.from_numpy(x.copy()).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    nan = np.isnan(x)
    assert np.array_equal(got[~nan], want[~nan])
    assert np.all(got[nan] == 0x7FC0)


def _f16_patterns():
    # all binary16 values, their midpoints to the next value (the ties) and
    # one fp32 ulp either side of each midpoint, plus random fp32 patterns
    h = np.arange(0x7C00, dtype=np.uint16)  # non-negative finite binary16
    v = h.view(np.float16).astype(np.float64)
    nxt = np.append(v[1:], 65536.0)
    mid = ((v + nxt) / 2).astype(np.float32)  # exact in fp32
    mid_u = mid.view(np.uint32)
    cand = np.concatenate([v.astype(np.float32).view(np.uint32), mid_u, mid_u + 1, mid_u - 1])
    rng = np.random.default_rng(2)
    cand = np.concatenate([cand, rng.integers(0, 1 << 32, size=1 << 20, dtype=np.uint64).astype(np.uint32),
                           np.array([0x477FF000, 0x477FEFFF, 0x477FF001, 0x7F7FFFFF, 0x00000001, 0x33000000,
                                     0x33000001, 0x32FFFFFF, 0x387FC000, 0x38800000], dtype=np.uint32)])
    cand = np.concatenate([cand, cand | np.uint32(0x80000000)])
    return cand


def test_f16_rounding_matches_numpy(oracle):
    u = _f16_patterns()
    x = u.view(np.float32)
    got = oracle.f32_to_f16(x)
    with np.errstate(over="ignore"):
        want = x.astype(np.float16).view(np.uint16)
    nan = np.isnan(x)
    assert np.array_equal(got[~nan], want[~nan])
    assert np.all(got[nan] == 0x7E00)


def test_16bit_widening_exhaustive(oracle):
    h = np.arange(1 << 16, dtype=np.uint16)
    bf = np.array([oracle.bf16_to_f32(int(v)) for v in h[::7]], dtype=np.float32)
    want_bf = torch.from_numpy(h[::7].view(np.int16).copy()).view(torch.bfloat16).float().numpy()
    assert np.array_equal(bf.view(np.uint32)[~np.isnan(bf)], want_bf.view(np.uint32)[~np.isnan(want_bf)])
    assert np.array_equal(np.isnan(bf), np.isnan(want_bf))
    f = np.array([oracle.f16_to_f32(int(v)) for v in h[::5]], dtype=np.float32)
    want_f = h[::5].view(np.float16).astype(np.float32)
    nn = ~np.isnan(want_f)
    assert np.array_equal(f[nn].view(np.uint32), want_f[nn].view(np.uint32))
    assert np.array_equal(np.isnan(f), np.isnan(want_f))


# ---------------------------------------------------------------------------
# uniform map
# ---------------------------------------------------------------------------


def test_uniform_minus1_1_exhaustive_closed_form(oracle):
    # U[-1,1): b - a = 2, 2 * m 2^-24 = m 2^-23 and -1 + m 2^-23 are exact in
    # fp32, so every one of the 2^24 outputs equals the rational -1 + m/2^23
    for c in range(16):  # 2^20 words at a time
        m = np.arange(c << 20, (c + 1) << 20, dtype=np.uint32)
        x = oracle.uniform_map(-1.0, 1.0, m << np.uint32(8))
        assert np.array_equal(x.astype(np.float64), -1.0 + m.astype(np.float64) / 2.0**23)


def test_uniform_wide_range_exhaustive(oracle):
    # U[-100,100): x(0) = a, monotone in m, x < b, and two fp32 roundings
    # keep every output within 2^-16 of a + (b-a) m / 2^24
    prev = -np.inf
    for c in range(16):  # 2^20 words at a time
        m = np.arange(c << 20, (c + 1) << 20, dtype=np.uint32)
        x = oracle.uniform_map(-100.0, 100.0, m << np.uint32(8)).astype(np.float64)
        exact = -100.0 + 200.0 * m.astype(np.float64) / 2.0**24
        if c == 0:
            assert x[0] == -100.0
        assert x[0] >= prev and np.all(np.diff(x) >= 0)
        prev = x[-1]
        assert x.max() < 100.0
        assert np.max(np.abs(x - exact)) <= 2.0**-16


def test_uniform_ignores_low_byte(oracle):
    rng = np.random.default_rng(3)
    w = rng.integers(0, 1 << 32, size=4096, dtype=np.uint64).astype(np.uint32)
    assert np.array_equal(oracle.uniform_map(-3.0, 5.0, w), oracle.uniform_map(-3.0, 5.0, w & np.uint32(0xFFFFFF00)))


# ---------------------------------------------------------------------------
# Box-Muller normals
# ---------------------------------------------------------------------------


def _bm(oracle, wa, wb):
    z = oracle.box_muller(np.array([wa, wb], dtype=np.uint32))
    return float(z[0]), float(z[1])


def test_box_muller_axis_angles_exact(oracle):
    wa = 123456 << 8
    r = math.sqrt(-2.0 * math.log((123456 + 1) * 2.0**-24))
    z0, z1 = _bm(oracle, wa, 0)            # angle 0
    assert z1 == 0.0 and z0 == np.float32(r)
    z0, z1 = _bm(oracle, wa, (1 << 22) << 8)   # quarter turn
    assert z0 == 0.0 and z1 == np.float32(r)
    z0, z1 = _bm(oracle, wa, (1 << 23) << 8)   # half turn
    assert z1 == 0.0 and z0 == np.float32(-r)
    z0, z1 = _bm(oracle, wa, (3 << 22) << 8)   # three quarters
    assert z0 == 0.0 and z1 == np.float32(-r)


def test_box_muller_u1_one_gives_zero(oracle):
    z0, z1 = _bm(oracle, 0xFFFFFFFF, 0x12345678)
    assert z0 == 0.0 and z1 == 0.0


def test_box_muller_against_full_angle_library_cos_sin(oracle):
    # numpy's cos/sin of the unreduced angle 2 pi m / 2^24: agrees to fp32
    # rounding, which catches any quarter-turn or sign slip in the reduction
    rng = np.random.default_rng(4)
    w = rng.integers(0, 1 << 32, size=2 * 200000, dtype=np.uint64).astype(np.uint32)
    z = oracle.box_muller(w).astype(np.float64)
    u1 = ((w[0::2] >> 8).astype(np.float64) + 1.0) * 2.0**-24
    th = 2 * np.pi * (w[1::2] >> 8).astype(np.float64) / 2.0**24
    r = np.sqrt(-2.0 * np.log(u1))
    for got, want in ((z[0::2], r * np.cos(th)), (z[1::2], r * np.sin(th))):
        err = np.abs(got - want)
        assert np.all(err <= 2.0**-23 * np.maximum(np.abs(want), 2.0**-20) + 1e-12)
    # radius identity z0^2 + z1^2 = -2 ln u1
    rr = z[0::2] ** 2 + z[1::2] ** 2
    assert np.all(np.abs(rr - r * r) <= 4e-7 * r * r + 1e-30)


def test_box_muller_distribution(oracle):
    # 2^21 samples from consecutive Philox VALUE blocks: KS against N(0,1),
    # moments inside 5 sigma
    words = np.array([oracle.draw(11, 0, "value", b) for b in range(1 << 14)], dtype=np.uint32).ravel()
    rng = np.random.default_rng(5)
    words = np.concatenate([words, rng.integers(0, 1 << 32, size=(1 << 21) - words.size,
                                                dtype=np.uint64).astype(np.uint32)])
    z = oracle.box_muller(words).astype(np.float64)
    n = z.size
    assert stats.kstest(z, "norm").pvalue > 1e-4
    assert abs(z.mean()) < 5 / math.sqrt(n)
    assert abs(z.var() - 1) < 5 * math.sqrt(2.0 / n)
    assert np.max(np.abs(z)) <= math.sqrt(48 * math.log(2)) + 1e-6


# ---------------------------------------------------------------------------
# integer ranges
# ---------------------------------------------------------------------------


@pytest.mark.parametrize("r", [3, 201])
def test_int_range_bucket_counts_exhaustive(oracle, r):
    # multiply-high of all 2^32 words: every bucket holds floor or ceil(2^32/r)
    c = oracle.int_range_histogram(r)
    assert int(c.sum()) == 1 << 32
    lo, hi = (1 << 32) // r, -(-(1 << 32) // r)
    assert set(np.unique(c).tolist()) <= {lo, hi}


def test_int_range_endpoints(oracle):
    for lo, hi in ((-100, 100), (0, 0), (-(2**31), 2**31 - 1), (0, 2**32 - 1), (5, 6)):
        r = hi - lo + 1
        assert oracle.int_range_map32(lo, r, 0) == lo
        assert oracle.int_range_map32(lo, r, 0xFFFFFFFF) == hi
    # full 32-bit range: the identity on the word
    assert oracle.int_range_map32(0, 1 << 32, 0xDEADBEEF) == 0xDEADBEEF


# ---------------------------------------------------------------------------
# permutation bijection and exact-count strata
# ---------------------------------------------------------------------------


@pytest.mark.parametrize("N", [1, 2, 3, 1000, 4096, 1000003, 1 << 20])
def test_permutation_is_bijection(oracle, N):
    v = oracle.perm_values(N, 5, 0, 0, N)
    assert v.max() < N
    assert np.unique(v).size == N


def test_permutation_outside_domain_is_zero(oracle):
    # the ragged last quantum evaluates indices >= N; with N = 5 (3-bit space),
    # seed 3, stream 3, indices 5 and 7 are fixed points of the round map, so a
    # walk from them would never return to [0, N): both sides return 0 there
    assert [oracle.perm_value(5, 3, 3, g) for g in (5, 6, 7, 1 << 40)] == [0, 0, 0, 0]
    assert sorted(oracle.perm_value(5, 3, 3, g) for g in range(5)) == list(range(5))


def test_permutation_depends_on_seed_and_stream(oracle):
    a = oracle.perm_values(1 << 16, 5, 0, 0, 1 << 16)
    b = oracle.perm_values(1 << 16, 6, 0, 0, 1 << 16)
    c = oracle.perm_values(1 << 16, 5, 1, 0, 1 << 16)
    assert (a != b).mean() > 0.99 and (a != c).mean() > 0.99
    # no fixed ordering left: correlation with the identity is small
    assert abs(np.corrcoef(a.astype(np.float64), np.arange(a.size))[0, 1]) < 0.05


@pytest.mark.parametrize("N,k", [(10, 10), (10, 1), (1000, 3), (1 << 20, 34), (12345, 1000), (7, 2)])
def test_strata_distinct_and_inside(oracle, N, k):
    idx = [oracle.stratum_index(N, k, 9, 2, s) for s in range(k)]
    assert len(set(idx)) == k
    for s, i in enumerate(idx):
        assert (s * N) // k <= i < ((s + 1) * N) // k
    if N == k:
        assert idx == list(range(N))
