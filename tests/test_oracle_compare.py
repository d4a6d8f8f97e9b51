"""Pins of the oracle's functional validation (Eq. 1, CUDA-Harness Sec. 4.2.1)
and progressive validation (Sec. 4.2.2).

Pins: hand-computed verdicts (tests/golden/compare_cases.txt), numpy's
`isclose` as an independent implementation of the same rule on float32 data,
exact Python-integer arithmetic for the integer statistics, closed forms for
RMS, and invariants (identical buffers, monotonicity in the tolerances, a
single flipped element found at its index).
"""
import math

import numpy as np
import pytest

import workloads as W
from golden_cases import case_arrays, load_compare_cases

CASES = load_compare_cases()


@pytest.mark.parametrize("c", CASES, ids=[f"{c['dtype']}-{c['x']:x}-{c['y']:x}-{i}" for i, c in enumerate(CASES)])
def test_golden_single_element(oracle, c):
    cand, ref = case_arrays(c)
    r = oracle.compare([W.Pair(c["dtype"], 1, 0, 0, c["atol"], c["rtol"], c["equal_nan"])], cand, ref)[0]
    assert r["pass"] == c["match"]
    assert r["mismatches"] == 1 - c["match"]
    assert r["first_mismatch"] == (-1 if c["match"] else 0)
    assert r["nan_disagree"] == c["nan_disagree"]
    assert r["inf_disagree"] == c["inf_disagree"]
    assert r["max_abs_u64"] == c["max_abs_u64"]


def _as_f32(dtype, b):
    if dtype == "f32":
        return b.view(np.float32)
    if dtype == "f16":
        return b.view(np.float16).astype(np.float32)
    return (b.view(np.uint16).astype(np.uint32) << 16).view(np.float32)


@pytest.mark.parametrize("dtype", ["f32", "f16", "bf16"])
@pytest.mark.parametrize("atol,rtol", [(1e-3, 1e-3), (0.0, 0.0), (1e-2, 0.0), (0.0, 1e-2), (1e-5, 1e-5)])
def test_float_compare_matches_numpy_isclose(oracle, dtype, atol, rtol):
    n = 200003
    cand, ref = W.random_pair_arrays(dtype, n, seed=17, scale=3.0, mismatch_frac=5e-3, nonfinite_frac=2e-3)
    r = oracle.compare([W.Pair(dtype, n, 0, 0, atol, rtol, True)], cand, ref)[0]
    x, y = _as_f32(dtype, cand), _as_f32(dtype, ref)
    with np.errstate(all="ignore"):
        ok = np.isclose(x, y, rtol=np.float32(rtol), atol=np.float32(atol), equal_nan=True)
        bad = ~ok
        assert r["mismatches"] == int(bad.sum())
        assert r["first_mismatch"] == (int(np.argmax(bad)) if bad.any() else -1)
        xn, yn = np.isnan(x), np.isnan(y)
        assert r["nan_disagree"] == int((xn != yn).sum())
        inf_any = (np.isinf(x) | np.isinf(y)) & ~xn & ~yn & (x != y)
        assert r["inf_disagree"] == int(inf_any.sum())
        fin = np.isfinite(x) & np.isfinite(y)
        d = np.abs(x[fin] - y[fin])  # float32 arithmetic
        assert r["n_finite"] == int(fin.sum())
        assert r["max_abs"] == float(d.max())
        yf = np.abs(y[fin])
        nz = yf != 0
        assert r["max_rel"] == float((d[nz] / yf[nz]).max())
        want_rms = math.sqrt(math.fsum((d.astype(np.float64) ** 2).tolist()) / d.size)
        assert r["rms"] == pytest.approx(want_rms, rel=1e-12)


@pytest.mark.parametrize("dtype", ["i32", "i64", "u32"])
def test_integer_compare_exact_against_python_ints(oracle, dtype):
    n = 50021
    cand, ref = W.random_pair_arrays(dtype, n, seed=23, mismatch_frac=1e-2, nonfinite_frac=1e-3)
    r = oracle.compare([W.Pair(dtype, n, 0, 0)], cand, ref)[0]
    npt = {"i32": np.int32, "i64": np.int64, "u32": np.uint32}[dtype]
    xs = [int(v) for v in cand.view(npt)]
    ys = [int(v) for v in ref.view(npt)]
    diffs = [abs(a - b) for a, b in zip(xs, ys)]
    bad = [i for i, (a, b) in enumerate(zip(xs, ys)) if a != b]
    assert r["mismatches"] == len(bad)
    assert r["first_mismatch"] == (bad[0] if bad else -1)
    assert r["max_abs_u64"] == max(diffs)
    assert r["n_finite"] == n
    assert r["rms"] == pytest.approx(math.sqrt(math.fsum(float(d) ** 2 for d in diffs) / n), rel=1e-12)


def test_identical_buffers_never_mismatch(oracle):
    for dt in ("f32", "f16", "bf16", "i32", "i64", "u32"):
        cand, ref = W.random_pair_arrays(dt, 10007, seed=5)
        r = oracle.compare([W.Pair(dt, 10007, 0, 0, 0.0, 0.0, True)], ref, ref)[0]
        assert r["pass"] == 1 and r["mismatches"] == 0 and r["max_abs"] == 0.0 and r["rms"] == 0.0


def test_mismatches_monotone_in_tolerances(oracle):
    cand, ref = W.random_pair_arrays("f32", 100003, seed=7, scale=50.0, mismatch_frac=0.2)
    prev = None
    for t in (0.0, 1e-7, 1e-6, 1e-5, 1e-4, 1e-3, 1e-2, 1e-1, 1.0, 10.0):
        for atol, rtol in ((t, 0.0), (0.0, t), (t, t)):
            m = oracle.compare([W.Pair("f32", 100003, 0, 0, atol, rtol)], cand, ref)[0]["mismatches"]
            if (atol, rtol) == (t, t):
                assert prev is None or m <= prev
                prev = m


def test_single_flipped_element_found_at_its_index(oracle):
    n = 1000
    base = np.linspace(-5, 5, n, dtype=np.float32)
    ref = base.view(np.uint8)
    pairs, cands = [], []
    for i in range(n):
        c = base.copy()
        c[i] = c[i] + np.float32(1.0)
        cands.append(c)
        pairs.append(W.Pair("f32", n, 4 * n * i, 0, 1e-3, 1e-3))
    cand = np.concatenate(cands).view(np.uint8)
    res = oracle.compare(pairs, cand, ref)
    for i, r in enumerate(res):
        assert r["mismatches"] == 1 and r["first_mismatch"] == i


def test_rms_closed_form(oracle):
    # d = 0.5 at every element: rms = 0.5, max_abs = 0.5, max_rel = 0.5/1
    n = 4099
    ref = np.ones(n, dtype=np.float32)
    cand = np.full(n, 1.5, dtype=np.float32)
    r = oracle.compare([W.Pair("f32", n, 0, 0, 1.0, 0.0)], cand.view(np.uint8), ref.view(np.uint8))[0]
    assert r["rms"] == 0.5 and r["max_abs"] == 0.5 and r["max_rel"] == 0.5 and r["pass"] == 1


def test_empty_pair(oracle):
    r = oracle.compare([W.Pair("f32", 0, 0, 0, 0.0, 0.0)], np.zeros(16, np.uint8), np.zeros(16, np.uint8))[0]
    assert r["pass"] == 1 and r["first_mismatch"] == -1 and r["mismatches"] == 0 and r["rms"] == 0.0


def test_out_of_bounds_pair_rejected(oracle):
    with pytest.raises(ValueError):
        oracle.compare([W.Pair("f32", 5, 0, 0)], np.zeros(16, np.uint8), np.zeros(16, np.uint8))


def test_progressive_stops_at_first_failure(oracle):
    # stages 0,1 pass, stage 2 fails, stage 3 would fail too but is not run
    n = 64
    ref = np.zeros(4 * n, dtype=np.float32)
    cand = ref.copy()
    cand[2 * n + 5] = 1.0
    cand[3 * n + 1] = 1.0
    stages = [W.Pair("f32", n, 4 * n * s, 4 * n * s, 1e-3, 1e-3) for s in range(4)]
    res, ff = oracle.progressive(stages, cand.view(np.uint8), ref.view(np.uint8))
    assert ff == 2
    assert [r["state"] for r in res] == [1, 1, 1, 2]
    assert [r["pass"] for r in res] == [1, 1, 0, 0]
    assert res[2]["first_mismatch"] == 5
    assert res[3]["mismatches"] == 0  # not run
    res, ff = oracle.progressive(stages[:2], cand.view(np.uint8), ref.view(np.uint8))
    assert ff == -1
