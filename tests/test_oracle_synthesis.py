"""Pins of the oracle's test-data synthesis (CUDA-Harness Sec. 4.2.1) and of the
workload-level verdicts (Eq. 1, Sec. 4.2.2).

Pins: chunked generation equals whole generation; the per-index evaluation
equals the bulk generator; injection and perturbation counts follow their
definitions (binomial confidence bands, exact counts, multiset equality for
swaps); 16-bit outputs are the round-to-nearest-even of the fp32 stream (via
torch/numpy conversions); the dot-like values equal exact sums on
integer-valued factors and numpy's fp64 matmul within the fp32 error bound;
and the workloads' verdicts have closed forms (the ladder fails at the
deviating stage, exactly the perturbed segments fail).
"""
import math

import numpy as np
import pytest
import torch

import workloads as W

NPT = {"f32": np.float32, "f16": np.float16, "i32": np.int32, "i64": np.int64, "u32": np.uint32,
       "bf16": np.uint16}


def _gen(oracle, specs, size):
    arena = np.zeros(size, dtype=np.uint8)
    oracle.generate(specs, arena)
    return arena


def _view(arena, off, dtype, n):
    b = arena[off: off + n * W.DTYPE_BYTES[dtype]]
    return b.view(NPT[dtype])


def _bf16_f32(u16):
    return (u16.astype(np.uint32) << 16).view(np.float32)


ALL_SPECS = [
    dict(dtype="f32", dist="uniform", p0=-1.0, p1=1.0),
    dict(dtype="f16", dist="uniform", p0=-100.0, p1=100.0),
    dict(dtype="bf16", dist="uniform", p0=-100.0, p1=100.0),
    dict(dtype="f32", dist="normal", p0=5.0, p1=10.0, specials=("nan", "pinf", "ninf", "denorm", "zero", "dup"),
         special_rate=0.05),
    dict(dtype="bf16", dist="normal", p0=0.0, p1=1.0, specials=("nan", "denorm"), special_rate=0.02),
    dict(dtype="f16", dist="normal", p0=0.0, p1=3.0),
    dict(dtype="i32", dist="int_range", i0=-100, i1=100, specials=("zero", "imin", "imax", "dup"), special_rate=0.03),
    dict(dtype="u32", dist="int_range", i0=0, i1=2**32 - 1),
    dict(dtype="i64", dist="int_range", i0=-(2**62), i1=2**62),
    dict(dtype="i64", dist="int_range", i0=-(2**63), i1=2**63 - 1),
    dict(dtype="i64", dist="permutation", specials=("dup", "zero", "imin", "imax"), special_rate=0.01),
    dict(dtype="i32", dist="permutation"),
    dict(dtype="u32", dist="raw_bits"),
    dict(dtype="bf16", dist="raw_bits"),
    dict(dtype="i64", dist="raw_bits"),
    dict(dtype="f32", dist="constant", p0=2.5),
    dict(dtype="i64", dist="constant", i0=-7),
]
PERTS = [
    (W.Perturb(), W.Perturb()),
    (W.Perturb("rate_add_pm", stream=3, rate=0.05, value=0.25, ivalue=3), W.Perturb()),
    (W.Perturb(), W.Perturb("count_set", stream=4, count=7, value=float("nan"), ivalue=-1)),
    (W.Perturb("rate_add_pm", stream=3, rate=0.02, value=1e-3, ivalue=1),
     W.Perturb("swap_pairs", stream=5, count=5)),
    (W.Perturb(), W.Perturb("count_add", stream=6, count=3, value=1e-2, ivalue=2)),
]


def _spec(kw, n, pelem, pcount, ref, cand, **extra):
    d = dict(kw)
    d.update(extra)
    return W.GenSpec(n=n, seed=1234, stream=9, ref_offset=ref, cand_offset=cand, pelem=pelem, pcount=pcount, **d)


@pytest.mark.parametrize("ki", range(len(ALL_SPECS)))
@pytest.mark.parametrize("pi", range(len(PERTS)))
def test_value_at_matches_bulk_and_chunks_match_whole(oracle, ki, pi):
    kw = ALL_SPECS[ki]
    pelem, pcount = PERTS[pi]
    if kw["dtype"] not in W.FLOAT_DTYPES and pelem.kind == "rel_noise":
        pytest.skip("rel_noise is float-only")
    n = 1003
    sz = W.DTYPE_BYTES[kw["dtype"]]
    whole = _spec(kw, n, pelem, pcount, 0, 8192)
    a = _gen(oracle, [whole], 16384)
    # per-index evaluation, both roles
    for role, off in ((0, 0), (1, 8192)):
        got = a[off: off + n * sz]
        want = np.array([oracle.value_at(whole, a, g, role) for g in range(n)], dtype=np.uint64)
        assert np.array_equal(np.frombuffer(got.tobytes() + b"\0" * 0, dtype={2: np.uint16, 4: np.uint32,
                                                                              8: np.uint64}[sz]).astype(np.uint64),
                              want)
    # the same logical array generated as 4 chunks (elem_offset multiple of 4)
    cuts = [0, 256, 512, 900, n]
    chunks = []
    for c0, c1 in zip(cuts[:-1], cuts[1:]):
        chunks.append(_spec(kw, c1 - c0, pelem, pcount, c0 * sz, 8192 + c0 * sz, elem_offset=c0, logical_n=n))
    b = _gen(oracle, chunks, 16384)
    assert np.array_equal(a, b)


def test_specials_rate_and_kinds(oracle):
    n = 200000
    s = W.GenSpec("f32", "normal", n, seed=3, stream=1, ref_offset=0, p0=0.0, p1=1.0,
                  specials=("nan", "pinf", "ninf", "denorm"), special_rate=0.01)
    a = _gen(oracle, [s], 4 * n)
    x = _view(a, 0, "f32", n)
    u = x.view(np.uint32)
    nan, pinf, ninf = np.isnan(x), x == np.inf, x == -np.inf
    den = ((u & 0x7F800000) == 0) & ((u & 0x7FFFFF) != 0)
    counts = np.array([nan.sum(), pinf.sum(), ninf.sum(), den.sum()])
    tot = counts.sum()
    # binomial(n, 0.01): sd ~ 44.5; 5 sd band
    assert abs(tot - 0.01 * n) < 5 * math.sqrt(n * 0.01 * 0.99)
    # each kind ~ 1/4 of the specials (chi-square, 3 dof, p > 1e-4)
    chi = ((counts - tot / 4) ** 2 / (tot / 4)).sum()
    assert chi < 21.1
    assert np.all(u[nan] == 0x7FC00000)


@pytest.mark.parametrize("rate", [1e-4, 1.0 / 256, 0.01, 0.3, 1.0])
def test_special_rate_is_binomial(oracle, rate):
    # the count of selected elements is binomial(n, rate); rate 1 selects all
    n = 1 << 18
    s = W.GenSpec("f32", "uniform", n, seed=5, stream=3, ref_offset=0, p0=-1.0, p1=1.0, specials=("nan",),
                  special_rate=rate)
    x = _view(_gen(oracle, [s], 4 * n), 0, "f32", n)
    k = int(np.isnan(x).sum())
    if rate == 1.0:
        assert k == n
    else:
        assert abs(k - rate * n) < 5 * math.sqrt(n * rate * (1 - rate)) + 1


@pytest.mark.parametrize("dist", ["uniform", "normal"])
def test_special_selection_is_independent_of_the_value(oracle, dist):
    # the selection draws from its own purpose: the base values at selected
    # positions follow the same law as all base values (two-sample KS)
    from scipy import stats
    n = 1 << 18
    kw = dict(p0=-1.0, p1=1.0) if dist == "uniform" else dict(p0=0.0, p1=1.0)
    base = W.GenSpec("f32", dist, n, seed=11, stream=4, ref_offset=0, **kw)
    a = _view(_gen(oracle, [base], 4 * n), 0, "f32", n)
    b = _view(_gen(oracle, [base.replace(specials=("nan",), special_rate=0.02)], 4 * n), 0, "f32", n)
    sel = np.isnan(b)
    assert abs(sel.sum() - 0.02 * n) < 5 * math.sqrt(n * 0.02 * 0.98)
    assert stats.ks_2samp(a[sel], a[~sel]).pvalue > 1e-4
    assert np.array_equal(a[~sel], b[~sel])


def test_special_selection_word_layout(oracle):
    # the documented selection: element g is special iff word g%4 of its
    # SPECIAL_SEL block g/4 is below floor(rate 2^32)
    n = 4096
    rate = 0.05
    s = W.GenSpec("f32", "uniform", n, seed=21, stream=6, ref_offset=0, p0=0.0, p1=1.0, specials=("nan",),
                  special_rate=rate)
    x = _view(_gen(oracle, [s], 4 * n), 0, "f32", n)
    thr = math.floor(rate * 2 ** 32)
    want = np.zeros(n, bool)
    for b in range(n // 4):
        w = oracle.draw(21, 6, "special_sel", b)
        for j in range(4):
            want[4 * b + j] = w[j] < thr
    assert np.array_equal(np.isnan(x), want)


def test_special_selection_does_not_move_base_values(oracle):
    # each purpose draws from its own stream: changing the rate keeps the
    # non-special elements bit-identical
    n = 50000
    base = W.GenSpec("f32", "uniform", n, seed=8, stream=2, ref_offset=0, p0=-1.0, p1=1.0)
    a = _view(_gen(oracle, [base], 4 * n), 0, "f32", n)
    b = _view(_gen(oracle, [base.replace(specials=("nan",), special_rate=0.1)], 4 * n), 0, "f32", n)
    keep = ~np.isnan(b)
    assert 0.08 * n < (~keep).sum() < 0.12 * n
    assert np.array_equal(a[keep], b[keep])


def test_dup_copies_a_base_value(oracle):
    n = 4096
    base = W.GenSpec("i64", "permutation", n, seed=2, stream=0, ref_offset=0)
    a = _view(_gen(oracle, [base], 8 * n), 0, "i64", n)
    assert np.array_equal(np.sort(a), np.arange(n))
    d = _view(_gen(oracle, [base.replace(specials=("dup",), special_rate=0.2)], 8 * n), 0, "i64", n)
    changed = d != a
    assert 0.1 * n < changed.sum() < 0.3 * n
    assert np.all((d >= 0) & (d < n))  # every value is some base value
    assert np.unique(d).size < n


def test_count_set_and_swap_structure(oracle):
    n = 100000
    s = W.GenSpec("f32", "uniform", n, seed=1, stream=0, ref_offset=0, cand_offset=4 * n, p0=-1.0, p1=1.0,
                  pcount=W.Perturb("count_set", stream=2, count=3, value=float("nan")))
    a = _gen(oracle, [s], 8 * n)
    ref, cand = _view(a, 0, "f32", n), _view(a, 4 * n, "f32", n)
    assert np.isnan(cand).sum() == 3 and not np.isnan(ref).any()
    diff = np.nonzero(cand.view(np.uint32) != ref.view(np.uint32))[0]
    assert diff.size == 3
    for st, i in enumerate(diff):
        assert (st * n) // 3 <= i < ((st + 1) * n) // 3
    # swaps: the candidate is a rearrangement of the reference
    s2 = W.GenSpec("i64", "permutation", n, seed=5, stream=0, ref_offset=0, cand_offset=8 * n,
                   pcount=W.Perturb("swap_pairs", stream=1, count=17))
    a2 = _gen(oracle, [s2], 16 * n)
    r2, c2 = _view(a2, 0, "i64", n), _view(a2, 8 * n, "i64", n)
    assert np.array_equal(np.sort(r2), np.sort(c2))
    d2 = np.nonzero(r2 != c2)[0]
    assert d2.size == 34
    for t in range(17):
        i, j = d2[2 * t], d2[2 * t + 1]
        assert r2[i] == c2[j] and r2[j] == c2[i]


def test_rate_add_pm_fraction_and_size(oracle):
    n = 200000
    s = W.GenSpec("f32", "constant", n, seed=4, stream=0, ref_offset=0, cand_offset=4 * n, p0=1.0,
                  pelem=W.Perturb("rate_add_pm", stream=7, rate=1e-2, value=0.5))
    a = _gen(oracle, [s], 8 * n)
    ref, cand = _view(a, 0, "f32", n), _view(a, 4 * n, "f32", n)
    assert np.all(ref == 1.0)
    ch = cand != 1.0
    assert abs(ch.sum() - 0.01 * n) < 5 * math.sqrt(n * 0.01)
    assert set(np.unique(cand[ch]).tolist()) <= {0.5, 1.5}
    assert abs((cand[ch] == 1.5).mean() - 0.5) < 0.05


def test_rel_noise_scale(oracle):
    n = 100000
    s = W.GenSpec("f32", "uniform", n, seed=4, stream=0, ref_offset=0, cand_offset=4 * n, p0=1.0, p1=10.0,
                  pelem=W.Perturb("rel_noise", stream=8, value=2.0 ** -9))
    a = _gen(oracle, [s], 8 * n)
    ref, cand = _view(a, 0, "f32", n).astype(np.float64), _view(a, 4 * n, "f32", n).astype(np.float64)
    z = (cand - ref) / (ref * 2.0 ** -9)
    assert abs(z.mean()) < 5 / math.sqrt(n)
    assert abs(z.std() - 1.0) < 0.02


@pytest.mark.parametrize("dtype", ["f16", "bf16"])
@pytest.mark.parametrize("dist,p0,p1", [("uniform", -100.0, 100.0), ("normal", 5.0, 10.0)])
def test_16bit_outputs_round_the_fp32_stream(oracle, dtype, dist, p0, p1):
    n = 65536
    s32 = W.GenSpec("f32", dist, n, seed=6, stream=3, ref_offset=0, p0=p0, p1=p1)
    s16 = s32.replace(dtype=dtype)
    x32 = _view(_gen(oracle, [s32], 4 * n), 0, "f32", n)
    h = _gen(oracle, [s16], 2 * n)[: 2 * n].view(np.uint16)
    if dtype == "f16":
        want = x32.astype(np.float16).view(np.uint16)
    else:
        want = torch.from_numpy(x32.copy()).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(h, want)


def test_normal_broad_range(oracle):
    # the paper's broad-range example: mean 5, standard deviation 10
    n = 1 << 18
    s = W.GenSpec("f32", "normal", n, seed=7, stream=0, ref_offset=0, p0=5.0, p1=10.0)
    x = _view(_gen(oracle, [s], 4 * n), 0, "f32", n).astype(np.float64)
    assert abs(x.mean() - 5.0) < 5 * 10 / math.sqrt(n)
    assert abs(x.std() - 10.0) < 0.1


def test_int_range_covers_small_range(oracle):
    n = 40000
    s = W.GenSpec("i32", "int_range", n, seed=3, stream=0, ref_offset=0, i0=-100, i1=100)
    x = _view(_gen(oracle, [s], 4 * n), 0, "i32", n)
    assert x.min() == -100 and x.max() == 100 and np.unique(x).size == 201


def test_dotlike_exact_on_integer_factors(oracle):
    # A = 0.5, B = 2 everywhere: every sum is exactly K; with K = 64 the bf16
    # value 64 is exact too
    rows, cols, k = 8, 12, 64
    ar = W.Arena()
    ao, bo = ar.take(4 * rows * k), ar.take(4 * k * cols)
    ro = ar.take(2 * rows * cols)
    specs = [W.GenSpec("f32", "constant", rows * k, ref_offset=ao, p0=0.5),
             W.GenSpec("f32", "constant", k * cols, ref_offset=bo, p0=2.0)]
    a = _gen(oracle, specs, ar.size)
    d = W.GenSpec("bf16", "dotlike", rows * cols, ref_offset=ro, rows=rows, cols=cols, dot_k=k, a_offset=ao,
                  b_offset=bo)
    oracle.generate([d], a)
    assert np.all(_bf16_f32(_view(a, ro, "bf16", rows * cols)) == 64.0)


def test_dotlike_against_numpy_matmul(oracle):
    wl = W.dotlike_bf16_pair(rows=96, cols=128, k=64)
    a, _, _ = oracle.run_workload(wl)
    fa, fb = wl.gen_calls[0]
    d = wl.gen_calls[1][0]
    A = _view(a, fa.ref_offset, "f32", 96 * 64).reshape(96, 64).astype(np.float64)
    B = _view(a, fb.ref_offset, "f32", 64 * 128).reshape(64, 128).astype(np.float64)
    exact = A @ B
    absprod = np.abs(A) @ np.abs(B)
    ref = _bf16_f32(_view(a, d.ref_offset, "bf16", 96 * 128)).reshape(96, 128).astype(np.float64)
    # 64 fused steps in fp32 (error <= 64 u sum|a b|), then one bf16 rounding
    bound = 64 * 2.0 ** -24 * absprod + np.abs(exact) * 2.0 ** -8 + 1e-30
    assert np.all(np.abs(ref - exact) <= bound * 1.01)
    assert abs(np.std(exact) - 0.125) < 0.01  # 64 products of N(0,1/64) terms


def test_workload_fp32_pair_small(oracle):
    wl = W.single_fp32_pair(1 << 16)
    a, res, _ = oracle.run_workload(wl)
    r = res[0]
    ref, cand = _view(a, wl.pairs[0].ref_offset, "f32", 1 << 16), _view(a, wl.pairs[0].cand_offset, "f32", 1 << 16)
    changed = ref.view(np.uint32) != cand.view(np.uint32)
    # every change is a mismatch: +-1e-3 >> 1e-5 + 1e-5 |y| for |y| < 1
    assert r["mismatches"] == changed.sum() and r["nan_disagree"] == 3
    assert r["first_mismatch"] == int(np.argmax(changed))


def test_workload_ladder_closed_form(oracle):
    wl = W.progressive_ladder((10, 12, 14, 16, 18), deviate_stage=3, special_rate=1e-3)
    _, res, ff = oracle.run_workload(wl)
    assert ff == 3
    assert [r["state"] for r in res] == [1, 1, 1, 1, 2]
    assert [r["mismatches"] for r in res[:4]] == [0, 0, 0, 1]
    wl2 = W.progressive_ladder((10, 12, 14), deviate_stage=None, special_rate=1e-3)
    _, res2, ff2 = oracle.run_workload(wl2)
    assert ff2 == -1 and all(r["pass"] for r in res2)


def test_workload_segmented_small(oracle):
    wl = W.segmented_cases(n_cases=256, max_n=4096)
    _, res, _ = oracle.run_workload(wl)
    for s, r in zip(wl.gen_calls[0], res):
        hit = s.pcount.kind != "none"
        assert r["mismatches"] == (1 if hit else 0)


def test_workload_perm_small(oracle):
    wl = W.int64_permutation_pair(n=1 << 16)
    _, res, _ = oracle.run_workload(wl)
    r = res[0]
    assert 0 < r["mismatches"] <= 34 and r["mismatches"] % 2 == 0


@pytest.mark.parametrize("dtype", ["i32", "i64", "f32", "bf16"])
def test_from_arena_copies_the_source_and_applies_specials(oracle, dtype):
    # base values read from an existing array; specials (zero, duplicates of
    # the source) and an exact-count edit on top; a chunked run matches
    n = 5001
    sz = W.DTYPE_BYTES[dtype]
    rng = np.random.default_rng(3)
    src_off, ref_off, cand_off = 0, 32768 * sz // 4 * 4, 65536 * sz // 4 * 4
    size = cand_off + n * sz + 256
    arena = np.zeros(size, np.uint8)
    src = rng.integers(1, 1 << (8 * min(sz, 4)), n, dtype=np.uint64).astype({2: np.uint16, 4: np.uint32,
                                                                            8: np.uint64}[sz])
    if dtype in ("f32", "bf16"):  # finite, nonzero floats
        f = rng.uniform(1.0, 2.0, n).astype(np.float32)
        src = f.view(np.uint32) if dtype == "f32" else (f.view(np.uint32) >> 16).astype(np.uint16)
    arena[src_off: src_off + n * sz] = src.view(np.uint8)
    pc = W.Perturb("count_add", stream=2, count=3, value=1.0, ivalue=5)
    spec = W.GenSpec(dtype, "from_arena", n, seed=9, stream=1, ref_offset=ref_off, cand_offset=cand_off,
                     a_offset=src_off, specials=("zero", "dup"), special_rate=0.05, pcount=pc)
    assert oracle.check_spec(spec, size) == 0
    whole = arena.copy()
    oracle.generate([spec], whole)
    ut = {2: np.uint16, 4: np.uint32, 8: np.uint64}[sz]  # compare bit patterns
    src = src.view(ut)
    ref = _view(whole, ref_off, dtype, n).view(ut)
    cand = _view(whole, cand_off, dtype, n).view(ut)
    keep = ref == src
    special = ~keep
    assert 0.03 * n < special.sum() < 0.07 * n
    srcset = set(src.tolist())
    assert all(v == 0 or v in srcset for v in ref[special].tolist())  # zero or a duplicate
    assert 1 <= np.count_nonzero(cand != ref) <= 3
    assert np.array_equal(_view(whole, src_off, dtype, n).view(ut), src)  # the source is untouched
    # chunks of the same logical array give the same bytes
    chunked = arena.copy()
    cuts = [0, 1000, 2048, n]
    parts = [spec.replace(n=c1 - c0, elem_offset=c0, logical_n=n, ref_offset=ref_off + c0 * sz,
                          cand_offset=cand_off + c0 * sz) for c0, c1 in zip(cuts[:-1], cuts[1:])]
    oracle.generate(parts, chunked)
    assert np.array_equal(chunked, whole)
