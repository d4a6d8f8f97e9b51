"""Seeded random differential tests of synthesis: tables of random valid specs
-- every dtype and distribution, special values in both modes, element-wise and
exact-count perturbations, chunks of longer logical arrays, ragged sizes,
arena-source twins and dot-like values on generated factors -- synthesized on
the GPU (syn_generate and a plan) and by the oracle, output by output, with
the same value bounds as the hand-written parity tests (bit-exact unless a
value passes through the Box-Muller transform)."""
import numpy as np
import pytest

import paper_2609_00058_gb300 as sv
import workloads as W
from gpu_util import device
from test_gpu_generate import check_spec_outputs, gen_both

pytestmark = pytest.mark.gpu

FLOAT_DISTS = ("uniform", "normal", "raw_bits", "constant", "from_arena", "dotlike")
INT_DISTS = ("int_range", "permutation", "raw_bits", "constant", "from_arena")
SPECIALS_F = ("nan", "pinf", "ninf", "denorm", "zero", "dup")
SPECIALS_I = ("zero", "imin", "imax", "dup")
INT_RANGE = {"i32": (-(1 << 31), (1 << 31) - 1), "u32": (0, (1 << 32) - 1), "i64": (-(1 << 63), (1 << 63) - 1)}


@pytest.fixture(scope="module")
def dev():
    return device()


def random_table(rng, n_specs):
    """Two generator calls: the sources and factors first, then the specs."""
    ar = W.Arena()
    first, second = [], []
    for i in range(n_specs):
        dt = str(rng.choice(["f32", "f16", "bf16", "i32", "u32", "i64"]))
        fl = dt in W.FLOAT_DTYPES
        dist = str(rng.choice(FLOAT_DISTS if fl else INT_DISTS))
        sz = W.DTYPE_BYTES[dt]
        kw = dict(seed=int(rng.integers(0, 1 << 62)), stream=int(rng.integers(0, 1 << 20)))
        if dist == "dotlike":
            rows, cols, k = int(rng.integers(1, 70)), 4 * int(rng.integers(1, 70)), int(rng.integers(1, 70))
            n, eo, ln = rows * cols, 0, 0
            ao, bo = ar.take(4 * rows * k), ar.take(4 * k * cols)
            first.append(W.GenSpec("f32", "uniform", rows * k, seed=kw["seed"], stream=1, ref_offset=ao, p0=-1, p1=1))
            first.append(W.GenSpec("f32", "uniform", k * cols, seed=kw["seed"], stream=2, ref_offset=bo, p0=-1, p1=1))
            kw.update(rows=rows, cols=cols, dot_k=k, a_offset=ao, b_offset=bo)
        else:
            n = int(rng.choice([1, 3, 4, 7, 100, 1000, 4099, 20000]))
            eo, ln = 0, 0
            if rng.random() < 0.25:  # a chunk of a longer logical array
                eo = 4 * int(rng.integers(0, 500))
                ln = eo + n + int(rng.integers(0, 50))
        N = ln or eo + n
        if dist == "from_arena":  # the source: a generated array of the whole logical length
            src = ar.take(N * sz)
            first.append(W.GenSpec(dt, "uniform" if fl else "int_range", N, seed=kw["seed"], stream=3, ref_offset=src,
                                   p0=-50.0, p1=50.0, i0=0 if dt == "u32" else -1000, i1=1000))
            kw.update(a_offset=src)
        if dist == "uniform":
            a, b = sorted(rng.uniform(-1e3, 1e3, 2))
            kw.update(p0=float(a), p1=float(b))
        elif dist == "normal":
            kw.update(p0=float(rng.choice([0.0, 5.0, -2.5])), p1=float(rng.choice([1.0, 10.0, 0.25])))
        elif dist == "int_range":
            lo, hi = INT_RANGE[dt]
            a, b = sorted(int(x) for x in rng.integers(max(lo, -1000), 1000, 2))
            if rng.random() < 0.3:
                a, b = lo, hi
            kw.update(i0=max(lo, a), i1=min(hi, b))
        elif dist == "constant":
            kw.update(p0=float(rng.uniform(-10, 10)), i0=int(rng.integers(-100, 100)) if dt != "u32" else 7)
        kinds = SPECIALS_F if fl else SPECIALS_I
        if rng.random() < 0.6:
            pick = tuple(k for k in kinds if rng.random() < 0.5) or (kinds[0],)
            kw.update(specials=pick, special_rate=float(rng.choice([1e-3, 0.05, 0.3])),
                      special_exact=bool(rng.random() < 0.35))
        ref = ar.take(n * sz)
        cand = ar.take(n * sz) if rng.random() < 0.75 else None
        if cand is not None:
            r = rng.random()
            if r < 0.3:
                kw.update(pelem=W.Perturb("rate_add_pm", stream=5, rate=0.02, value=0.5, ivalue=3))
            elif r < 0.55 and fl:
                kw.update(pelem=W.Perturb("rel_noise", stream=6, value=2.0 ** -9))
            r = rng.random()
            if r < 0.2:
                kw.update(pcount=W.Perturb("count_set", stream=7, count=int(rng.integers(1, N + 1)) if N < 8 else 3,
                                           value=7.0, ivalue=7))
            elif r < 0.4:
                kw.update(pcount=W.Perturb("count_add", stream=8, count=min(N, 5), value=1.0, ivalue=1))
            elif r < 0.55 and N >= 2:
                kw.update(pcount=W.Perturb("swap_pairs", stream=9, count=max(1, min(N // 2, 4))))
        second.append(W.GenSpec(dt, dist, n, ref_offset=ref, cand_offset=cand, elem_offset=eo, logical_n=ln, **kw))
    return [first, second], ar.size


@pytest.mark.parametrize("seed", range(24))
def test_random_tables_match_the_oracle(dev, seed):
    import torch
    rng = np.random.default_rng(1000 + seed)
    calls, size = random_table(rng, 24)
    g, h = gen_both(dev, calls, size)
    for spec in calls[0] + calls[1]:
        check_spec_outputs(g, h, spec)
    # the same table through a plan writes the same bytes
    a = torch.zeros(size, dtype=torch.uint8, device=dev)
    for call in calls:
        sv.GeneratePlan(call, size, device=dev)(a)
    torch.cuda.synchronize()
    assert np.array_equal(a.cpu().numpy(), g)


def random_pairs(rng, n_pairs):
    """A table of pairs of random dtypes, sizes (empty, ragged, below and above
    the small-segment limit), tolerances and NaN rules over one arena of
    planted near and far mismatches and non-finite patterns."""
    ar = W.Arena()
    pairs, chunks = [], []
    for i in range(n_pairs):
        dt = str(rng.choice(["f32", "f16", "bf16", "i32", "u32", "i64"]))
        n = int(rng.choice([0, 1, 5, 8, 64, 1000, 4096, 16383, 20000, 70001]))
        c, r = W.random_pair_arrays(dt, max(n, 1), seed=int(rng.integers(0, 1 << 30)),
                                    mismatch_frac=float(rng.choice([0.0, 1e-3, 0.05])))
        sz = W.DTYPE_BYTES[dt]
        co, ro = ar.take(n * sz), ar.take(n * sz)
        chunks += [(co, c[:n * sz]), (ro, r[:n * sz])]
        atol, rtol = (float(rng.choice([0.0, 1e-6, 1e-3, 0.5])), float(rng.choice([0.0, 1e-5, 1e-2])))
        pairs.append(W.Pair(dt, n, co, ro, atol=atol, rtol=rtol, equal_nan=bool(rng.random() < 0.8)))
    buf = np.zeros(ar.size, np.uint8)
    for off, data in chunks:
        buf[off: off + data.size] = data
    return pairs, buf


@pytest.mark.parametrize("seed", range(12))
def test_random_pair_tables_match_the_oracle(dev, seed):
    import oracle
    import torch
    from gpu_util import assert_results_match
    rng = np.random.default_rng(5000 + seed)
    pairs, buf = random_pairs(rng, int(rng.choice([3, 40, 300])))
    a = torch.from_numpy(buf).to(dev)
    want = oracle.compare(pairs, buf, buf)
    got = sv.decode_results(sv.compare(pairs, a, a), len(pairs))
    assert_results_match(got, want, "seed %d" % seed)
    plan = sv.ComparePlan(pairs, buf.size, buf.size, device=dev)
    got_plan = sv.decode_results(plan(a, a), len(pairs))
    assert_results_match(got_plan, want, "plan, seed %d" % seed)


@pytest.mark.parametrize("seed", range(12))
def test_random_tile_geometries_match_the_oracle(dev, seed):
    """Shaped outputs of random rows, columns, padded pitches and tile sizes --
    side-by-side tile groups (with their staging ring), warp and CTA tiles,
    ragged edges -- against the oracle's tile compare."""
    import oracle
    from gpu_util import assert_results_match, to_dev
    from test_gpu_tiles import make_pair
    rng = np.random.default_rng(9000 + seed)
    dtype = str(rng.choice(["f32", "f16", "bf16", "i32", "i64", "u32"]))
    sz = W.DTYPE_BYTES[dtype]
    align = 16 // sz
    rows = int(rng.choice([1, 3, 17, 130, 2000, 9000]))
    cols = int(rng.choice([1, 3, 8, 40, 64, 100, 256, 520]))
    cp = -(-(cols + int(rng.integers(0, 20))) // align) * align
    rp = -(-(cols + int(rng.integers(0, 20))) // align) * align
    tr = int(rng.choice([1, 2, 3, 4, 5, 7, 8, 16, 33, 128]))
    tc = int(rng.choice([cols, 8, 16, 32, 64, 128]))
    if tc < cols:
        tc = -(-tc // align) * align
    x, y = make_pair(dtype, rows, cols, cp, rp, seed=9000 + seed)
    t = W.Tiles(dtype, rows, cols, 0, 0, cand_pitch=cp, ref_pitch=rp, tile_rows=tr, tile_cols=tc,
                atol=1e-3, rtol=1e-3)
    want = oracle.compare_tiles(t, x, y)
    got = sv.decode_results(sv.compare_tiles(t, to_dev(x, dev), to_dev(y, dev)), len(want))
    assert_results_match(got, want, "%s rows %d cols %d pitches %d/%d tile %dx%d" % (dtype, rows, cols, cp, rp, tr, tc))


@pytest.mark.parametrize("seed", range(12))
def test_random_ladders_match_the_oracle(dev, seed):
    """Progressive ladders of 1 to 12 stages of mixed dtypes and sizes (stage
    groups form and break on dtype changes and size limits), failing at a
    random stage or not at all: every stage's result, the skipped ones and the
    first failed index equal the oracle's."""
    import oracle
    import torch
    from gpu_util import assert_results_match
    rng = np.random.default_rng(13000 + seed)
    ar = W.Arena()
    stages, chunks = [], []
    n_st = int(rng.integers(1, 13))
    fail_at = int(rng.integers(0, n_st + 1))  # n_st: every stage passes
    for i in range(n_st):
        dt = str(rng.choice(["f32", "f32", "bf16", "i32", "i64"]))
        n = int(rng.choice([1, 100, 4096, 50000, 1 << 20]))
        c, r = W.random_pair_arrays(dt, n, seed=int(rng.integers(0, 1 << 30)), mismatch_frac=0.0,
                                    nonfinite_frac=0.0)
        if i == fail_at:
            k = int(rng.integers(0, n))
            sz = W.DTYPE_BYTES[dt]
            c = c.copy()
            c[k * sz] ^= 0x01
            c[k * sz + sz - 1] ^= 0x10
        sz = W.DTYPE_BYTES[dt]
        co, ro = ar.take(n * sz), ar.take(n * sz)
        chunks += [(co, c), (ro, r)]
        stages.append(W.Pair(dt, n, co, ro, atol=1e-6, rtol=1e-6))
    buf = np.zeros(ar.size, np.uint8)
    for off, data in chunks:
        buf[off: off + data.size] = data
    want, want_ff = oracle.progressive(stages, buf, buf)
    a = torch.from_numpy(buf).to(dev)
    res, ff = sv.progressive(stages, a, a)
    torch.cuda.synchronize()
    assert int(ff.item()) == want_ff
    assert_results_match(sv.decode_results(res, n_st), want, "seed %d" % seed)
