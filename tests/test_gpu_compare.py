"""GPU parity of verify_compare (Eq. 1 per segment, CUDA-Harness Sec. 4.2.1)
against the CPU oracle on identical bytes.  Inputs come from the oracle or
from the neutral seeded generator in workloads.py, never from the CUDA path.

Bar: every integer field (counts, first-mismatch index, max |x-y| of
integers), the fp32 max |x-y| and max |x-y|/|y| (both exact: the same fp32
operations on both sides) bit-exact; RMS within 1e-6 relative.
"""
import numpy as np
import pytest

import oracle
import paper_2609_00058_gb300 as sv
import workloads as W
from golden_cases import case_arrays, load_compare_cases
from gpu_util import assert_results_match, device, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    return device()


def run_both(dev, pairs, cand, ref):
    got = sv.decode_results(sv.compare(pairs, to_dev(cand, dev), to_dev(ref, dev)), len(pairs))
    want = oracle.compare(pairs, cand, ref)
    return got, want


def test_golden_cases_on_gpu(dev):
    cases = load_compare_cases()
    # all hand-computed single-element cases in one call (more than the inline
    # table holds: exercises the uploaded table and the dtype grouping)
    cands, refs, pairs = [], [], []
    off = 0
    for c in cases:
        cb, rb = case_arrays(c)
        cands.append(np.pad(cb, (0, 16 - cb.size)))
        refs.append(np.pad(rb, (0, 16 - rb.size)))
        pairs.append(W.Pair(c["dtype"], 1, off, off, c["atol"], c["rtol"], c["equal_nan"]))
        off += 16
    cand, ref = np.concatenate(cands), np.concatenate(refs)
    got = sv.decode_results(sv.compare(pairs, to_dev(cand, dev), to_dev(ref, dev)), len(pairs))
    for c, g in zip(cases, got):
        assert g["pass"] == c["match"], c
        assert g["nan_disagree"] == c["nan_disagree"] and g["inf_disagree"] == c["inf_disagree"], c
        assert g["max_abs_u64"] == c["max_abs_u64"], c
        assert g["first_mismatch"] == (-1 if c["match"] else 0)


# sizes spanning several 16 KiB tiles with ragged tails, plus tiny ones
SIZES = [1, 3, 7, 8, 4095, 4096 * 3 + 5, 65536 + 1, 300007]


@pytest.mark.parametrize("dtype", ["f32", "f16", "bf16", "i32", "i64", "u32"])
@pytest.mark.parametrize("n", SIZES)
def test_random_pairs_match_oracle(dev, dtype, n):
    cand, ref = W.random_pair_arrays(dtype, n, seed=1000 + n, scale=5.0, mismatch_frac=2e-3, nonfinite_frac=1e-3)
    pairs = [W.Pair(dtype, n, 0, 0, 1e-3, 1e-3)]
    got, want = run_both(dev, pairs, cand, ref)
    assert_results_match(got, want, "%s n=%d" % (dtype, n))


@pytest.mark.parametrize("atol,rtol,eqnan", [(0.0, 0.0, True), (1e-5, 1e-5, False), (1e-2, 0.0, True),
                                             (0.0, 0.5, True), (3.0, 3.0, False)])
def test_tolerances_and_nan_flag(dev, atol, rtol, eqnan):
    n = 100003
    cand, ref = W.random_pair_arrays("f32", n, seed=77, scale=100.0, mismatch_frac=1e-2, nonfinite_frac=5e-3)
    pairs = [W.Pair("f32", n, 0, 0, atol, rtol, eqnan)]
    got, want = run_both(dev, pairs, cand, ref)
    assert_results_match(got, want)


def _segments(n_pairs, seed):
    rng = np.random.default_rng(seed)
    dts = ["f32", "f16", "bf16", "i32", "i64", "u32"]
    ar = W.Arena()
    specs = []
    for i in range(n_pairs):
        dt = dts[rng.integers(0, len(dts))]
        n = int(rng.choice([0, 1, 5, 17, 1000, 4096, 8193, 50000]))
        specs.append((dt, n, ar.take(max(n, 1) * W.DTYPE_BYTES[dt])))
    cand = np.zeros(ar.size, np.uint8)
    ref = np.zeros(ar.size, np.uint8)
    pairs = []
    for i, (dt, n, off) in enumerate(specs):
        if n:
            c, r = W.random_pair_arrays(dt, n, seed=seed * 1000 + i, mismatch_frac=5e-3)
            cand[off:off + c.size] = c
            ref[off:off + r.size] = r
        pairs.append(W.Pair(dt, n, off, off, 1e-3, 1e-3))
    return pairs, cand, ref


@pytest.mark.parametrize("n_pairs,seed", [(1, 1), (5, 2), (8, 3), (9, 4), (64, 5), (200, 7), (700, 6)])
def test_many_segments_mixed_dtypes(dev, n_pairs, seed):
    pairs, cand, ref = _segments(n_pairs, seed)
    got, want = run_both(dev, pairs, cand, ref)
    assert_results_match(got, want, "segments")


def test_separate_candidate_and_reference_buffers(dev):
    n = 40000
    cand, ref = W.random_pair_arrays("bf16", n, seed=9)
    # candidate at an offset inside a larger buffer, reference at 0 of its own
    big = np.zeros(cand.size + 4096, np.uint8)
    big[4096:] = cand
    pairs = [W.Pair("bf16", n, 4096, 0, 1e-2, 1e-2)]
    got = sv.decode_results(sv.compare(pairs, to_dev(big, dev), to_dev(ref, dev)), 1)
    want = oracle.compare(pairs, big, ref)
    assert_results_match(got, want)


def test_identical_buffers_and_flipped_element(dev):
    n = 1000
    base = np.linspace(-5, 5, n, dtype=np.float32)
    cands = []
    pairs = []
    for i in range(0, n, 37):
        c = base.copy()
        c[i] += np.float32(1.0)
        cands.append(c)
        pairs.append(W.Pair("f32", n, 4 * n * len(pairs), 0, 1e-3, 1e-3))
    cand = np.concatenate(cands).view(np.uint8)
    got = sv.decode_results(sv.compare(pairs, to_dev(cand, dev), to_dev(base.view(np.uint8), dev)), len(pairs))
    for k, g in enumerate(got):
        assert g["mismatches"] == 1 and g["first_mismatch"] == 37 * k
    same = sv.decode_results(sv.compare([W.Pair("f32", n, 0, 0)], to_dev(base, dev), to_dev(base, dev)), 1)[0]
    assert same["pass"] == 1 and same["rms"] == 0.0 and same["max_abs"] == 0.0


def test_large_dynamic_range_rms(dev):
    # differences near 1e-30 and 1e30: the fp32 fast path must not underflow
    # or overflow the sum of squares
    n = 20000
    rng = np.random.default_rng(3)
    ref = rng.standard_normal(n).astype(np.float32)
    for scale in (1e-30, 1e30, 1e-42):
        cand = (ref + np.float32(scale) * rng.standard_normal(n).astype(np.float32)).astype(np.float32)
        cand[::7] = ref[::7] + np.float32(scale)
        pairs = [W.Pair("f32", n, 0, 0, 0.0, 0.0)]
        got, want = run_both(dev, pairs, cand.view(np.uint8), ref.view(np.uint8))
        assert_results_match(got, want, "scale %g" % scale)
    huge = np.full(n, 3e38, np.float32)
    got, want = run_both(dev, [W.Pair("f32", n, 0, 0, 0.0, 0.0)], (-huge).view(np.uint8), huge.view(np.uint8))
    assert_results_match(got, want, "overflow")


def test_repeated_calls_are_deterministic(dev):
    n = 1 << 20
    cand, ref = W.random_pair_arrays("f32", n, seed=5)
    c, r = to_dev(cand, dev), to_dev(ref, dev)
    a = sv.decode_results(sv.compare([W.Pair("f32", n, 0, 0, 1e-3, 1e-3)], c, r), 1)[0]
    for _ in range(3):
        assert sv.decode_results(sv.compare([W.Pair("f32", n, 0, 0, 1e-3, 1e-3)], c, r), 1)[0] == a


@pytest.mark.parametrize("n_pairs,seed", [(3, 11), (9, 12), (200, 13)])
def test_compare_plan_matches_oracle_for_several_candidates(dev, n_pairs, seed):
    """One plan, three candidates (the original and two edited copies): every
    planned verdict equals the oracle's, and the unplanned call's."""
    pairs, cand, ref = _segments(n_pairs, seed)
    d_ref = to_dev(ref, dev)
    plan = sv.ComparePlan(pairs, cand.size, ref.size, device=dev)
    rng = np.random.default_rng(seed)
    for k in range(3):
        c = cand.copy()
        if k:
            c[rng.choice(c.size, 50, replace=False)] ^= np.uint8(1 << k)
        d_c = to_dev(c, dev)
        got = sv.decode_results(plan(d_c, d_ref), n_pairs)
        assert_results_match(got, oracle.compare(pairs, c, ref), "plan candidate %d" % k)
        assert_results_match(got, sv.decode_results(sv.compare(pairs, d_c, d_ref), n_pairs), "plan vs call")
