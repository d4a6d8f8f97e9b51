"""The oracle's multi-threaded drivers against its single-threaded functions.

The drivers only cut specs and pairs into element chunks and combine the
chunk verdicts in chunk order; generation is a function of the logical index
(Sec. 4.2.1), so the threaded bytes must equal the single-threaded bytes, and
every integer field of a verdict (Eq. 1) must be identical.  RMS may differ
only by the order of its fp64 sum.
"""
import numpy as np
import pytest

import workloads as W

THREADS = (2, 3, 8)


def _same_results(a, b, rms_rel=1e-12):
    assert len(a) == len(b)
    for x, y in zip(a, b):
        for k in ("mismatches", "nan_disagree", "inf_disagree", "n_finite", "first_mismatch", "max_abs_u64",
                  "max_abs", "max_rel", "pass", "state"):
            assert x[k] == y[k], (k, x, y)
        assert x["rms"] == pytest.approx(y["rms"], rel=rms_rel, abs=0.0)


def _small_workloads():
    return [
        W.single_fp32_pair(1 << 18),
        W.progressive_ladder((10, 14, 18, 19), deviate_stage=2, special_rate=1e-3),
        W.segmented_cases(200),
        W.dotlike_bf16_pair(rows=64, cols=256, k=12),
        W.int64_permutation_pair(1 << 18, swaps=17),
    ]


@pytest.mark.parametrize("threads", THREADS)
def test_threaded_generation_writes_the_same_bytes(oracle, threads):
    for wl in _small_workloads():
        one = np.zeros(wl.arena_bytes, np.uint8)
        many = np.zeros(wl.arena_bytes, np.uint8)
        for call in wl.gen_calls:
            oracle.generate(call, one)
            oracle.generate(call, many, threads=threads)
        assert np.array_equal(one, many), wl.name


def test_threaded_generation_of_chunked_specs(oracle):
    """A spec that is itself a chunk of a longer logical array (elem_offset,
    logical_n) with exact-count edits near the chunk edges."""
    n, N = 100_000, 300_000
    spec = W.GenSpec("f32", "normal", n, seed=9, stream=4, ref_offset=0, cand_offset=4 * n + 256,
                     elem_offset=100_000, logical_n=N, p0=5.0, p1=10.0, specials=("nan", "dup", "denorm"),
                     special_rate=3e-3, pelem=W.Perturb("rate_add_pm", stream=5, rate=1e-2, value=0.5),
                     pcount=W.Perturb("swap_pairs", stream=6, count=40))
    size = 8 * n + 512
    one, many = np.zeros(size, np.uint8), np.zeros(size, np.uint8)
    oracle.generate([spec], one)
    oracle.generate([spec], many, threads=5)
    assert np.array_equal(one, many)


@pytest.mark.parametrize("dtype", ["f32", "f16", "bf16", "i32", "i64", "u32"])
def test_threaded_compare_equals_single(oracle, dtype):
    ar = W.Arena()
    sizes = [0, 1, 7, 1000, 65_537, 300_001]
    placed = [(n, ar.take(max(n, 1) * W.DTYPE_BYTES[dtype])) for n in sizes]
    cand, ref = np.zeros(ar.size, np.uint8), np.zeros(ar.size, np.uint8)
    pairs = []
    for i, (n, off) in enumerate(placed):
        if n:
            c, r = W.random_pair_arrays(dtype, n, seed=70 + i, mismatch_frac=2e-3, nonfinite_frac=2e-3)
            cand[off:off + c.size], ref[off:off + r.size] = c, r
        pairs.append(W.Pair(dtype, n, off, off, 1e-3, 1e-3))
    want = oracle.compare(pairs, cand, ref)
    for t in THREADS:
        _same_results(oracle.compare(pairs, cand, ref, threads=t), want)


def test_threaded_compare_first_mismatch_in_a_later_chunk(oracle):
    """One pair cut into many chunks with its only mismatches far from the
    start: the first mismatch comes from the first chunk that has one."""
    n = 1 << 20
    ref = np.arange(n, dtype=np.int64)
    cand = ref.copy()
    cand[[777_777, 900_001]] += 5
    pair = [W.Pair("i64", n, 0, 0)]
    want = oracle.compare(pair, cand.view(np.uint8), ref.view(np.uint8))
    got = oracle.compare(pair, cand.view(np.uint8), ref.view(np.uint8), threads=8)
    _same_results(got, want)
    assert got[0]["first_mismatch"] == 777_777 and got[0]["mismatches"] == 2


def test_threaded_sums_add_up(oracle):
    """The single-threaded sum of squares is the sum the rms is taken from."""
    c, r = W.random_pair_arrays("f32", 50_000, seed=5)
    res, sums = oracle.compare_sums([W.Pair("f32", 50_000, 0, 0, 1e-3, 1e-3)], c, r)
    assert res[0]["rms"] == pytest.approx(np.sqrt(sums[0] / res[0]["n_finite"]), rel=1e-15)


def test_threaded_progressive_equals_single(oracle):
    wl = W.progressive_ladder((10, 14, 18, 19), deviate_stage=2, special_rate=1e-3)
    arena = np.zeros(wl.arena_bytes, np.uint8)
    oracle.generate(wl.gen_calls[0], arena)
    want, ff = oracle.progressive(wl.pairs, arena, arena)
    got, ff_t = oracle.progressive(wl.pairs, arena, arena, threads=4)
    assert ff == ff_t == 2
    _same_results(got, want)


def test_threaded_drivers_refuse_what_the_single_ones_refuse(oracle):
    bad = [W.Pair("f32", 100, 0, 0, -1.0, 0.0)]
    buf = np.zeros(4096, np.uint8)
    with pytest.raises(ValueError):
        oracle.compare(bad, buf, buf, threads=4)
    with pytest.raises(ValueError):
        oracle.progressive(bad, buf, buf, threads=4)
    with pytest.raises(ValueError):
        oracle.generate([W.GenSpec("i32", "uniform", 16, ref_offset=0)], buf, threads=4)
