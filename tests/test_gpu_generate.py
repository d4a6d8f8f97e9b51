"""GPU parity of syn_generate (test-data synthesis, CUDA-Harness Sec. 4.2.1)
against the CPU oracle.

Bar: every stream that involves no transcendental function (uniform, integer
range, permutation, raw bits, constants, special-value selection and kinds,
+-delta perturbations, exact-count edits, swaps, dot-like sums on the same
factors) is bit-exact.  Box-Muller normals are computed in fp32 on the GPU:
N(0,1) samples are within 4 ulp of the oracle's fp64-computed, fp32-rounded
values; affine and 16-bit outputs inherit that bound (sigma * 4 ulp(z) plus
one rounding of the output type).
"""
import numpy as np
import pytest

import oracle
import paper_2609_00058_gb300 as sv
import workloads as W
from gpu_util import device, ordered_16, ordered_f32, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    return device()


def gen_both(dev, calls, size):
    import torch
    a = torch.zeros(size, dtype=torch.uint8, device=dev)
    h = np.zeros(size, dtype=np.uint8)
    for call in calls:
        sv.generate(call, a)
        oracle.generate(call, h)
    torch.cuda.synchronize()
    return a.cpu().numpy(), h


def _view(buf, off, dtype, n):
    t = {"f32": np.uint32, "f16": np.uint16, "bf16": np.uint16, "i32": np.uint32, "u32": np.uint32,
         "i64": np.uint64}[dtype]
    return buf[off: off + n * W.DTYPE_BYTES[dtype]].view(t)


def _uses_transcendentals(spec):
    return spec.dist == "normal" or spec.pelem.kind == "rel_noise"


def check_spec_outputs(g, h, spec, zbound_ulp=4):
    ref_h = _view(h, spec.ref_offset, spec.dtype, spec.n) if spec.ref_offset is not None else None
    for role, off in ((0, spec.ref_offset), (1, spec.cand_offset)):
        if off is None:
            continue
        gv, hv = _view(g, off, spec.dtype, spec.n), _view(h, off, spec.dtype, spec.n)
        if not _uses_transcendentals(spec):
            assert np.array_equal(gv, hv), "bit mismatch in %s/%s at %s" % (
                spec.dtype, spec.dist, np.nonzero(gv != hv)[0][:8])
            continue
        if spec.dtype == "f32":
            gf, hf = gv.view(np.float32), hv.view(np.float32)
            fin = np.isfinite(hf)
            assert np.array_equal(np.isfinite(gf), fin)
            assert np.array_equal(gv[~fin], hv[~fin])  # specials are bit-exact
            if role == 0 and spec.dist == "normal" and spec.p0 == 0.0 and spec.p1 == 1.0:
                d = np.abs(ordered_f32(gv[fin]) - ordered_f32(hv[fin]))
                assert d.max(initial=0) <= zbound_ulp
                continue
            # value bound: the clean value's z carries <= 4 ulp (scaled by
            # sigma), every later fp32 rounding adds <= 1 ulp of its result,
            # and the noise term c|x|z adds c|x| * 4 ulp(z) with |z| < 5.8
            x = hf[fin].astype(np.float64)
            xr = ref_h.view(np.float32)[fin].astype(np.float64) if ref_h is not None else x
            # a candidate value an exact-count edit made finite over a
            # non-finite reference carries no noise of the reference's
            xr = np.where(np.isfinite(xr), xr, x)
            sp = lambda v: np.spacing(np.abs(v).astype(np.float32)).astype(np.float64)
            err = np.zeros_like(x)
            if spec.dist == "normal":
                zr = (xr - spec.p0) / spec.p1
                err += abs(spec.p1) * zbound_ulp * sp(zr)
            err += sp(xr) + sp(x)
            if role == 1 and spec.pelem.kind == "rel_noise":
                err += abs(spec.pelem.value) * np.abs(xr) * zbound_ulp * np.spacing(np.float32(5.8)) + 2 * sp(x)
            if role == 1 and spec.pelem.kind == "rate_add_pm":
                err += 2 * sp(x) + sp(abs(spec.pelem.value))
            g64 = gf[fin].astype(np.float64)
            assert np.all((g64 == x) | (np.abs(g64 - x) <= err * 1.0001))
        else:
            fin_mask = 0x7C00 if spec.dtype == "f16" else 0x7F80
            fin = (hv & fin_mask) != fin_mask
            assert np.array_equal((gv & fin_mask) != fin_mask, fin)
            assert np.array_equal(gv[~fin], hv[~fin])
            d = np.abs(ordered_16(gv[fin], spec.dtype) - ordered_16(hv[fin], spec.dtype))
            assert d.max(initial=0) <= 1


ALL_SPECS = [
    dict(dtype="f32", dist="uniform", p0=-1.0, p1=1.0),
    dict(dtype="f16", dist="uniform", p0=-100.0, p1=100.0),
    dict(dtype="bf16", dist="uniform", p0=-100.0, p1=100.0, specials=("nan", "pinf", "denorm", "dup"),
         special_rate=0.01),
    dict(dtype="f32", dist="normal", p0=0.0, p1=1.0),
    dict(dtype="f32", dist="normal", p0=5.0, p1=10.0, specials=("nan", "pinf", "ninf", "denorm", "zero", "dup"),
         special_rate=0.05),
    dict(dtype="bf16", dist="normal", p0=0.0, p1=1.0, specials=("nan", "denorm"), special_rate=0.02),
    dict(dtype="f16", dist="normal", p0=0.0, p1=3.0),
    dict(dtype="i32", dist="int_range", i0=-100, i1=100, specials=("zero", "imin", "imax", "dup"), special_rate=0.03),
    dict(dtype="u32", dist="int_range", i0=0, i1=2**32 - 1),
    dict(dtype="u32", dist="int_range", i0=7, i1=70000),
    dict(dtype="i64", dist="int_range", i0=-(2**62), i1=2**62),
    dict(dtype="i64", dist="int_range", i0=-(2**63), i1=2**63 - 1),
    dict(dtype="i64", dist="permutation", specials=("dup", "zero", "imin", "imax"), special_rate=0.01),
    dict(dtype="i32", dist="permutation"),
    dict(dtype="u32", dist="permutation", logical_n=(1 << 33) // 3),
    dict(dtype="u32", dist="raw_bits"),
    dict(dtype="bf16", dist="raw_bits"),
    dict(dtype="f16", dist="raw_bits"),
    dict(dtype="i64", dist="raw_bits"),
    dict(dtype="f32", dist="constant", p0=2.5),
    dict(dtype="bf16", dist="constant", p0=float("nan")),
    dict(dtype="i64", dist="constant", i0=-7),
    # exact-count special values: round(rate * N), one per stratum
    dict(dtype="f32", dist="normal", p0=5.0, p1=10.0, specials=("nan", "pinf", "ninf", "denorm", "zero", "dup"),
         special_rate=0.01, special_exact=True),
    dict(dtype="bf16", dist="uniform", p0=-100.0, p1=100.0, specials=("nan", "denorm", "dup"), special_rate=3e-3,
         special_exact=True),
    dict(dtype="i64", dist="permutation", specials=("dup", "zero", "imin", "imax"), special_rate=0.01,
         special_exact=True),
    dict(dtype="i32", dist="int_range", i0=-100, i1=100, specials=("zero", "imin", "imax"), special_rate=1.0,
         special_exact=True),  # every element special: every edit lands on a special
]
PERTS = [
    (W.Perturb(), W.Perturb()),
    (W.Perturb("rate_add_pm", stream=3, rate=0.05, value=0.25, ivalue=3), W.Perturb()),
    (W.Perturb(), W.Perturb("count_set", stream=4, count=7, value=float("nan"), ivalue=-1)),
    (W.Perturb("rate_add_pm", stream=3, rate=0.02, value=1e-3, ivalue=1), W.Perturb("swap_pairs", stream=5, count=5)),
    (W.Perturb(), W.Perturb("count_add", stream=6, count=3, value=1e-2, ivalue=2)),
    (W.Perturb("rel_noise", stream=8, value=2.0 ** -9), W.Perturb("count_add", stream=6, count=2, value=1.0)),
]


@pytest.mark.parametrize("ki", range(len(ALL_SPECS)))
@pytest.mark.parametrize("pi", range(len(PERTS)))
def test_spec_matches_oracle(dev, ki, pi):
    kw = dict(ALL_SPECS[ki])
    pelem, pcount = PERTS[pi]
    if kw["dtype"] not in W.FLOAT_DTYPES and pelem.kind == "rel_noise":
        pytest.skip("rel_noise is float-only")
    n = 3 * 8192 + 13  # several tiles and a ragged last quantum
    sz = W.DTYPE_BYTES[kw["dtype"]]
    ln = kw.pop("logical_n", 0)
    spec = W.GenSpec(n=n, seed=4321, stream=9, ref_offset=0, cand_offset=(n * sz + 255) // 256 * 256,
                     logical_n=ln, pelem=pelem, pcount=pcount, **kw)
    g, h = gen_both(dev, [[spec]], 2 * spec.cand_offset)
    check_spec_outputs(g, h, spec)


def test_normal_unit_within_4_ulp_large_sample(dev):
    n = 1 << 22
    spec = W.GenSpec("f32", "normal", n, seed=7, stream=3, ref_offset=0, p0=0.0, p1=1.0)
    g, h = gen_both(dev, [[spec]], 4 * n)
    d = np.abs(ordered_f32(g.view(np.uint32)) - ordered_f32(h.view(np.uint32)))
    assert d.max() <= 4
    # and most are exact
    assert (d == 0).mean() > 0.5


def test_chunks_equal_whole_on_gpu(dev):
    n = 50000
    base = dict(dtype="f32", dist="uniform", seed=3, stream=1, p0=-2.0, p1=3.0, specials=("nan", "dup"),
                special_rate=0.01, pelem=W.Perturb("rate_add_pm", stream=2, rate=0.01, value=0.5),
                pcount=W.Perturb("swap_pairs", stream=3, count=9))
    whole = W.GenSpec(n=n, ref_offset=0, cand_offset=4 * n, **base)
    cuts = [0, 8192, 8196, 30000, n]
    chunks = [W.GenSpec(n=c1 - c0, ref_offset=4 * c0, cand_offset=4 * n + 4 * c0, elem_offset=c0, logical_n=n,
                        **base) for c0, c1 in zip(cuts[:-1], cuts[1:])]
    import torch
    a = torch.zeros(8 * n, dtype=torch.uint8, device=dev)
    b = torch.zeros(8 * n, dtype=torch.uint8, device=dev)
    sv.generate([whole], a)
    sv.generate(chunks, b)
    assert torch.equal(a, b)
    h = np.zeros(8 * n, np.uint8)
    oracle.generate([whole], h)
    assert np.array_equal(a.cpu().numpy(), h)


@pytest.mark.parametrize("case", [
    # few strata per CTA: the generating CTAs apply the edits (up to ~20 in one CTA here)
    dict(dtype="f32", dist="uniform", n=1 << 20, p0=-1.0, p1=1.0, pcount=W.Perturb("count_set", stream=2, count=2000,
                                                                              value=float("inf"))),
    dict(dtype="i64", dist="permutation", n=1 << 20, pcount=W.Perturb("swap_pairs", stream=2, count=700)),
    dict(dtype="f16", dist="uniform", n=300001, p0=-4.0, p1=4.0, pcount=W.Perturb("count_add", stream=2, count=90,
                                                                               value=0.125)),
    dict(dtype="bf16", dist="raw_bits", n=77777, pcount=W.Perturb("swap_pairs", stream=2, count=11)),
    # dense strata: the fixup kernel applies them
    dict(dtype="f32", dist="uniform", n=1000, p0=-1.0, p1=1.0, pcount=W.Perturb("count_set", stream=2, count=500,
                                                                             value=-3.0)),
    dict(dtype="i64", dist="permutation", n=4096, pcount=W.Perturb("swap_pairs", stream=2, count=1000)),
    dict(dtype="bf16", dist="normal", n=20000, p0=0.0, p1=1.0, pcount=W.Perturb("count_add", stream=2, count=300,
                                                                              value=0.5)),
    dict(dtype="i32", dist="int_range", n=5000, i0=-9, i1=9, pcount=W.Perturb("count_add", stream=2, count=5000,
                                                                            ivalue=1)),
])
def test_exact_count_edits_sparse_and_dense(dev, case):
    kw = dict(case)
    n = kw.pop("n")
    sz = W.DTYPE_BYTES[kw["dtype"]]
    spec = W.GenSpec(n=n, seed=11, stream=4, ref_offset=0, cand_offset=(n * sz + 255) // 256 * 256, **kw)
    g, h = gen_both(dev, [[spec]], 2 * spec.cand_offset)
    check_spec_outputs(g, h, spec)
    ref = _view(g, 0, spec.dtype, n)
    cand = _view(g, spec.cand_offset, spec.dtype, n)
    if spec.pcount.kind == "swap_pairs":
        assert np.count_nonzero(ref != cand) <= 2 * spec.pcount.count
    else:
        assert np.count_nonzero(ref != cand) <= spec.pcount.count


@pytest.mark.parametrize("kw", [
    dict(dtype="f32", dist="uniform", p0=-3.0, p1=7.0, specials=("nan", "dup", "denorm"), special_rate=0.01,
         pelem=W.Perturb("rate_add_pm", stream=5, rate=0.01, value=0.5)),
    dict(dtype="bf16", dist="normal", p0=5.0, p1=10.0, pelem=W.Perturb("rel_noise", stream=6, value=2.0 ** -9)),
    dict(dtype="i64", dist="permutation", specials=("dup", "imin"), special_rate=0.01,
         pcount=W.Perturb("swap_pairs", stream=7, count=3)),
    dict(dtype="i64", dist="int_range", i0=-(2 ** 40), i1=2 ** 40, pcount=W.Perturb("count_add", stream=8, count=5,
                                                                                  ivalue=-1)),
    dict(dtype="u32", dist="raw_bits", pcount=W.Perturb("count_set", stream=9, count=2, ivalue=7)),
])
def test_chunk_at_the_top_of_the_largest_logical_range(dev, kw):
    # a chunk ending at logical index 2^40: 64-bit counters, permutation
    # constants beyond 32 bits and strata of about 2^38 elements
    ln = 1 << 40
    n = 20001
    eo = ln - n - 3  # the quantum-aligned start (multiple of 4) of a ragged chunk
    eo -= eo % 4
    sz = W.DTYPE_BYTES[kw["dtype"]]
    spec = W.GenSpec(n=n, seed=77, stream=1, ref_offset=0, cand_offset=(n * sz + 255) // 256 * 256,
                     elem_offset=eo, logical_n=ln, **kw)
    g, h = gen_both(dev, [[spec]], 2 * spec.cand_offset)
    check_spec_outputs(g, h, spec)


@pytest.mark.parametrize("n_specs", [1, 8, 9, 40])
def test_many_specs_one_call(dev, n_specs):
    # inline (<= 8) and uploaded tables, mixed kinds grouped per launch
    kinds = [dict(dtype="f32", dist="uniform", p0=-1.0, p1=1.0),
             dict(dtype="i32", dist="int_range", i0=-5, i1=5),
             dict(dtype="bf16", dist="raw_bits"),
             dict(dtype="i64", dist="permutation"),
             dict(dtype="u32", dist="constant", i0=9)]
    ar = W.Arena()
    specs = []
    for i in range(n_specs):
        kw = kinds[i % len(kinds)]
        n = [1, 3, 4, 5, 100, 8192, 8193, 20000][i % 8]
        sz = W.DTYPE_BYTES[kw["dtype"]]
        specs.append(W.GenSpec(n=n, seed=i, stream=i, ref_offset=ar.take(n * sz), cand_offset=ar.take(n * sz),
                               specials=("zero",) if kw["dtype"] != "f32" else ("nan",), special_rate=0.1,
                               pcount=W.Perturb("count_set", stream=1, count=1, value=7.0, ivalue=7), **kw))
    g, h = gen_both(dev, [specs], ar.size)
    assert np.array_equal(g, h)


def test_dotlike_bit_exact_on_oracle_factors(dev):
    # the factors come from the oracle; the GPU's tiled FMA chains must equal
    # the oracle's sequential ones bit for bit
    rows, cols, k = 200, 520, 64
    wl = W.dotlike_bf16_pair(rows=rows, cols=cols, k=k)
    h = np.zeros(wl.arena_bytes, np.uint8)
    oracle.generate(wl.gen_calls[0], h)  # A and B
    import torch
    a = to_dev(h, dev)
    d = wl.gen_calls[1][0]
    sv.generate([d], a)
    oracle.generate([d], h)
    g = a.cpu().numpy()
    n = rows * cols
    assert np.array_equal(_view(g, d.ref_offset, "bf16", n), _view(h, d.ref_offset, "bf16", n))
    gc, hc = _view(g, d.cand_offset, "bf16", n), _view(h, d.cand_offset, "bf16", n)
    assert np.abs(ordered_16(gc, "bf16") - ordered_16(hc, "bf16")).max() <= 1


def test_dotlike_f32_and_odd_shapes(dev):
    for rows, cols, k in ((1, 4, 1), (65, 132, 33), (3, 256, 100)):
        ar = W.Arena()
        ao, bo = ar.take(4 * rows * k), ar.take(4 * k * cols)
        ro = ar.take(4 * rows * cols)
        fa = W.GenSpec("f32", "uniform", rows * k, seed=1, stream=0, ref_offset=ao, p0=-1, p1=1)
        fb = W.GenSpec("f32", "uniform", k * cols, seed=1, stream=1, ref_offset=bo, p0=-1, p1=1)
        d = W.GenSpec("f32", "dotlike", rows * cols, seed=1, stream=2, ref_offset=ro, rows=rows, cols=cols, dot_k=k,
                      a_offset=ao, b_offset=bo, specials=("nan", "dup"), special_rate=0.01)
        g, h = gen_both(dev, [[fa, fb], [d]], ar.size)
        assert np.array_equal(g, h), (rows, cols, k)


def test_dotlike_many_tiles_per_cta(dev):
    # more 64 x 128 tiles than resident CTAs, ragged in rows and columns, with
    # K a multiple of 4 (16-byte factor rows) and not (4-byte factor copies)
    for dtype, rows, cols, k in (("f16", 1100, 4100, 37), ("bf16", 1031, 4108, 68)):
        ar = W.Arena()
        ao, bo = ar.take(4 * rows * k), ar.take(4 * k * cols)
        ro = ar.take(2 * rows * cols)
        fa = W.GenSpec("f32", "uniform", rows * k, seed=5, stream=0, ref_offset=ao, p0=-1, p1=1)
        fb = W.GenSpec("f32", "uniform", k * cols, seed=5, stream=1, ref_offset=bo, p0=-1, p1=1)
        d = W.GenSpec(dtype, "dotlike", rows * cols, seed=5, stream=2, ref_offset=ro, rows=rows, cols=cols, dot_k=k,
                      a_offset=ao, b_offset=bo, specials=("pinf", "zero"), special_rate=1e-3)
        g, h = gen_both(dev, [[fa, fb], [d]], ar.size)
        assert np.array_equal(g, h), (dtype, rows, cols, k)


def test_dotlike_chunked(dev):
    rows, cols, k = 40, 64, 16
    ar = W.Arena()
    ao, bo = ar.take(4 * rows * k), ar.take(4 * k * cols)
    ro = ar.take(2 * rows * cols)
    fac = [W.GenSpec("f32", "uniform", rows * k, seed=2, ref_offset=ao, p0=-1, p1=1),
           W.GenSpec("f32", "uniform", k * cols, seed=2, stream=1, ref_offset=bo, p0=-1, p1=1)]
    whole = W.GenSpec("bf16", "dotlike", rows * cols, seed=2, stream=2, ref_offset=ro, rows=rows, cols=cols,
                      dot_k=k, a_offset=ao, b_offset=bo)
    g1, h1 = gen_both(dev, [fac, [whole]], ar.size)
    part = whole.replace(n=1000, elem_offset=704, logical_n=rows * cols, ref_offset=ro + 1408)
    g2, _ = gen_both(dev, [fac, [part]], ar.size)
    assert np.array_equal(g2[ro + 1408: ro + 1408 + 2000], g1[ro + 1408: ro + 1408 + 2000])
    assert np.array_equal(g1, h1)


@pytest.mark.parametrize("dtype,rows,cols,k", [
    ("bf16", 1031, 4108, 68),  # two k chunks per tile (64 + 4), ragged rows and columns
    ("f16", 1100, 4100, 37),   # K % 4 != 0: 4-byte factor copies; many tiles per CTA
    ("f32", 130, 260, 16),     # a chunk shorter than 64: the held tile's noise runs without FMAs beside it
    ("bf16", 300, 1032, 64),   # the bench shape's K: one 64-deep chunk per tile
])
def test_dotlike_noisy_twin_shapes(dev, dtype, rows, cols, k):
    """The relative-noise twin, which the kernel makes while it multiplies the
    next tile: the reference equals the oracle's bit for bit, the twin is
    within the Box-Muller bound of the oracle's, and it is bit-identical to
    the twin made afterwards from the stored reference (from_arena); a chunk
    that starts and ends inside rows writes the same bytes as the whole."""
    import torch
    sz = W.DTYPE_BYTES[dtype]
    n = rows * cols
    ar = W.Arena()
    ao, bo = ar.take(4 * rows * k), ar.take(4 * k * cols)
    ro, co, to = ar.take(sz * n), ar.take(sz * n), ar.take(sz * n)
    fa = W.GenSpec("f32", "uniform", rows * k, seed=7, stream=0, ref_offset=ao, p0=-1, p1=1)
    fb = W.GenSpec("f32", "uniform", k * cols, seed=7, stream=1, ref_offset=bo, p0=-1, p1=1)
    noise = W.Perturb("rel_noise", stream=3, value=2.0 ** -9)
    d = W.GenSpec(dtype, "dotlike", n, seed=7, stream=2, ref_offset=ro, cand_offset=co, rows=rows, cols=cols,
                  dot_k=k, a_offset=ao, b_offset=bo, specials=("nan", "pinf", "zero"), special_rate=1e-3,
                  pelem=noise)
    g, h = gen_both(dev, [[fa, fb], [d]], ar.size)
    assert np.array_equal(_view(g, ro, dtype, n), _view(h, ro, dtype, n))
    check_spec_outputs(g, h, d)
    a = to_dev(g, dev)
    twin = W.GenSpec(dtype, "from_arena", n, seed=7, stream=2, ref_offset=None, cand_offset=to, a_offset=ro,
                     pelem=noise)
    sv.generate([twin], a)
    out = a.cpu().numpy()
    assert np.array_equal(out[co: co + sz * n], out[to: to + sz * n])
    off = (3 * cols + 8) // 8 * 8  # inside row 3; 16-byte output offsets for every type
    m = n - off - 7
    part = d.replace(n=m, elem_offset=off, logical_n=n, ref_offset=ro + off * sz, cand_offset=co + off * sz)
    b = torch.zeros(ar.size, dtype=torch.uint8, device=dev)
    sv.generate([fa, fb], b)
    sv.generate([part], b)
    got = b.cpu().numpy()
    for base in (ro, co):
        lo_b, hi_b = base + off * sz, base + (off + m) * sz
        assert np.array_equal(got[lo_b: hi_b], g[lo_b: hi_b])
        assert not got[base: lo_b].any() and not got[hi_b: base + sz * n].any()


def test_zero_length_and_single_element(dev):
    specs = [W.GenSpec("f32", "uniform", 0, ref_offset=0, p0=0, p1=1),
             W.GenSpec("i64", "permutation", 1, ref_offset=256, cand_offset=512),
             W.GenSpec("bf16", "normal", 1, ref_offset=768, p0=0, p1=1, specials=("nan",), special_rate=1.0)]
    g, h = gen_both(dev, [specs], 1024)
    assert np.array_equal(g, h)


@pytest.mark.parametrize("dtype", ["f32", "f16", "bf16", "i32", "u32", "i64"])
def test_from_arena_matches_oracle(dev, dtype):
    # base values read from an existing array of N = 3 * 8192 + 13 elements
    # (its last quantum is ragged: the kernel must not read past it), with
    # specials, an element-wise and an exact-count perturbation; then a chunk
    # that ends at the array's end
    import torch
    n = 3 * 8192 + 13
    sz = W.DTYPE_BYTES[dtype]
    ar = W.Arena()
    src_off, ref_off, cand_off = ar.take(n * sz), ar.take(n * sz), ar.take(n * sz)
    h = np.zeros(ar.size, np.uint8)
    rng = np.random.default_rng(17)
    if dtype in W.FLOAT_DTYPES:
        f = rng.normal(0.0, 3.0, n).astype(np.float32)
        bits = f.view(np.uint32) if dtype == "f32" else (
            oracle.f32_to_bf16(f) if dtype == "bf16" else oracle.f32_to_f16(f))
        specials, pelem = ("nan", "pinf", "denorm", "dup"), W.Perturb("rel_noise", stream=3, value=2.0 ** -9)
        pcount = W.Perturb("count_add", stream=4, count=5, value=0.5)
    else:
        bits = rng.integers(0, 1 << 63, n, dtype=np.uint64).astype({4: np.uint32, 8: np.uint64}[sz])
        specials, pelem = ("zero", "imin", "dup"), W.Perturb("rate_add_pm", stream=3, rate=0.01, ivalue=7)
        pcount = W.Perturb("swap_pairs", stream=4, count=5)
    h[src_off: src_off + n * sz] = np.ascontiguousarray(bits).view(np.uint8)
    spec = W.GenSpec(dtype, "from_arena", n, seed=31, stream=2, ref_offset=ref_off, cand_offset=cand_off,
                     a_offset=src_off, specials=specials, special_rate=0.01, pelem=pelem, pcount=pcount)
    for specs in ([spec], [spec.replace(n=n - 8192, elem_offset=8192, logical_n=n, ref_offset=ref_off + 8192 * sz,
                                        cand_offset=cand_off + 8192 * sz)]):
        want = h.copy()
        oracle.generate(specs, want)
        a = torch.from_numpy(h.copy()).to(dev)
        sv.generate(specs, a)
        got = a.cpu().numpy()
        s0 = specs[0]
        if dtype in W.FLOAT_DTYPES:  # the noise runs Box-Muller: compare as the other parity tests do
            check_spec_outputs(got, want, s0)
            assert np.array_equal(got[:ref_off], want[:ref_off])  # the source is untouched
        else:
            assert np.array_equal(got, want), dtype


def test_candidate_pass_from_the_reference_equals_the_fused_twin(dev):
    # the dot-like kernel writes the reference and its noisy twin together; the
    # same twin made afterwards from the reference array (SV_FROM_ARENA with
    # the same noise) is bit-identical
    import torch
    rows, cols, k = 200, 520, 64
    wl = W.dotlike_bf16_pair(rows=rows, cols=cols, k=k)
    n = rows * cols
    extra = (2 * n + 255) // 256 * 256
    a = torch.zeros(wl.arena_bytes + extra, dtype=torch.uint8, device=dev)
    for call in wl.gen_calls:
        sv.generate(call, a)
    d = wl.gen_calls[1][0]
    twin = W.GenSpec("bf16", "from_arena", n, seed=d.seed, stream=d.stream, ref_offset=None,
                     cand_offset=wl.arena_bytes, a_offset=d.ref_offset, pelem=d.pelem)
    sv.generate([twin], a)
    h = a.cpu().numpy()
    assert np.array_equal(h[d.cand_offset: d.cand_offset + 2 * n], h[wl.arena_bytes: wl.arena_bytes + 2 * n])


# ---------------------------------------------------------------------------
# exact-count special values (one per stratum; SV_SP_EXACT)
# ---------------------------------------------------------------------------
def test_exact_specials_at_a_ladder_stage(dev):
    """A 2^22 fp32 N(0,1) stage with 1e-3 exact specials (4194 of them, over
    every CTA of the grid) and one +1e-2 edit: the specials land exactly on
    the oracle's indices, with its kinds, and nowhere else."""
    n = 1 << 22
    spec = W.GenSpec("f32", "normal", n, seed=7, stream=3, ref_offset=0, cand_offset=4 * n, p0=0.0, p1=1.0,
                     specials=("nan", "pinf", "ninf", "denorm"), special_rate=1e-3, special_exact=True,
                     pcount=W.Perturb("count_add", stream=103, count=1, value=1e-2))
    import torch
    a = torch.zeros(8 * n, dtype=torch.uint8, device=dev)
    sv.generate([spec], a)
    h = np.zeros(8 * n, np.uint8)
    oracle.generate([spec], h, threads=0)
    g = a.cpu().numpy()
    check_spec_outputs(g, h, spec)
    k = oracle.special_count(1e-3, n)
    idx = [oracle.special_index(n, k, 7, 3, s) for s in range(k)]
    gv = _view(g, 0, "f32", n)
    special = ~np.isfinite(gv.view(np.float32)) | ((gv & 0x7F800000) == 0)
    assert np.nonzero(special)[0].tolist() == idx
    assert np.array_equal(gv[idx], _view(h, 0, "f32", n)[idx])


def test_exact_specials_chunked_and_with_swaps(dev):
    n = 70_000
    base = dict(dtype="f32", dist="uniform", seed=3, stream=1, p0=-2.0, p1=3.0, specials=("nan", "dup", "zero"),
                special_rate=4e-3, special_exact=True,
                pelem=W.Perturb("rate_add_pm", stream=2, rate=0.01, value=0.5),
                pcount=W.Perturb("swap_pairs", stream=3, count=9))
    whole = W.GenSpec(n=n, ref_offset=0, cand_offset=4 * n, **base)
    cuts = [0, 8192, 8196, 40000, n]
    chunks = [W.GenSpec(n=c1 - c0, ref_offset=4 * c0, cand_offset=4 * n + 4 * c0, elem_offset=c0, logical_n=n,
                        **base) for c0, c1 in zip(cuts[:-1], cuts[1:])]
    import torch
    a = torch.zeros(8 * n, dtype=torch.uint8, device=dev)
    b = torch.zeros(8 * n, dtype=torch.uint8, device=dev)
    sv.generate([whole], a)
    sv.generate(chunks, b)
    assert torch.equal(a, b)
    h = np.zeros(8 * n, np.uint8)
    oracle.generate([whole], h)
    assert np.array_equal(a.cpu().numpy(), h)


@pytest.mark.parametrize("rate", [0.01, 1.0])
def test_exact_specials_on_dotlike_values(dev, rate):
    """Dot-like values take their exact specials from the fixup kernel; at
    rate 1 every element is special, so every edit lands on one."""
    rows, cols, k = 65, 132, 33
    ar = W.Arena()
    ao, bo = ar.take(4 * rows * k), ar.take(4 * k * cols)
    ro, co = ar.take(2 * rows * cols), ar.take(2 * rows * cols)
    fa = W.GenSpec("f32", "uniform", rows * k, seed=1, stream=0, ref_offset=ao, p0=-1, p1=1)
    fb = W.GenSpec("f32", "uniform", k * cols, seed=1, stream=1, ref_offset=bo, p0=-1, p1=1)
    d = W.GenSpec("bf16", "dotlike", rows * cols, seed=1, stream=2, ref_offset=ro, cand_offset=co, rows=rows,
                  cols=cols, dot_k=k, a_offset=ao, b_offset=bo, specials=("nan", "zero", "dup"), special_rate=rate,
                  special_exact=True, pelem=W.Perturb("rate_add_pm", stream=5, rate=0.05, value=0.25),
                  pcount=W.Perturb("count_add", stream=6, count=7, value=1.0))
    g, h = gen_both(dev, [[fa, fb], [d]], ar.size)
    assert np.array_equal(g, h)



@pytest.mark.parametrize("n_specs", [3, 40])
def test_generate_plan_equals_syn_generate(dev, n_specs):
    """A plan (table validated, grouped and staged once) writes the bytes of
    syn_generate, call after call."""
    import torch
    kinds = [dict(dtype="f32", dist="normal", p0=5.0, p1=10.0, specials=("nan", "pinf"), special_rate=1e-3,
                  special_exact=True),
             dict(dtype="i32", dist="int_range", i0=-5, i1=5),
             dict(dtype="bf16", dist="uniform", p0=-100.0, p1=100.0, specials=("denorm",), special_rate=0.01),
             dict(dtype="i64", dist="permutation", pcount=W.Perturb("swap_pairs", stream=4, count=3))]
    ar = W.Arena()
    specs = []
    for i in range(n_specs):
        kw = kinds[i % len(kinds)]
        n = [7, 100, 8192, 20001, 65536][i % 5]
        sz = W.DTYPE_BYTES[kw["dtype"]]
        specs.append(W.GenSpec(n=n, seed=i, stream=i, ref_offset=ar.take(n * sz), cand_offset=ar.take(n * sz),
                               **kw))
    a = torch.zeros(ar.size, dtype=torch.uint8, device=dev)
    sv.generate(specs, a)
    plan = sv.GeneratePlan(specs, ar.size, device=dev)
    for _ in range(2):
        b = torch.zeros(ar.size, dtype=torch.uint8, device=dev)
        plan(b)
        assert torch.equal(a, b)



@pytest.mark.parametrize("n_specs", [40, 300])
def test_plan_mixed_kinds(dev, n_specs):
    """A plan over many specs of every size class writes the bytes of
    syn_generate: arena-source twins, exact-count specials, fused and fixup
    edits, element-wise perturbations."""
    import torch
    ar = W.Arena()
    src_n = 70000
    src = ar.take(2 * src_n)
    kinds = [dict(dtype="f32", dist="normal", p0=0.0, p1=1.0, specials=("nan", "ninf"), special_rate=1e-3,
                  special_exact=True),
             dict(dtype="f16", dist="from_arena", a_offset=src, pelem=W.Perturb("rel_noise", stream=3, value=2.0 ** -9)),
             dict(dtype="i32", dist="int_range", i0=-9, i1=9, pcount=W.Perturb("count_add", stream=5, count=2, ivalue=1)),
             dict(dtype="bf16", dist="uniform", p0=-3.0, p1=3.0, pelem=W.Perturb("rate_add_pm", stream=6, rate=0.01,
                                                                                  value=0.5)),
             dict(dtype="i64", dist="permutation", pcount=W.Perturb("swap_pairs", stream=4, count=3))]
    specs = []
    for i in range(n_specs):
        kw = kinds[i % len(kinds)]
        n = [1, 7, 100, 8192, 20001, 65536][i % 6]
        if "pcount" in kw:
            n = max(n, 16)  # room for the edits' strata
        sz = W.DTYPE_BYTES[kw["dtype"]]
        specs.append(W.GenSpec(n=n, seed=i, stream=i, ref_offset=ar.take(n * sz), cand_offset=ar.take(n * sz), **kw))
    g = torch.Generator(device=dev)
    g.manual_seed(n_specs)
    base = torch.zeros(ar.size, dtype=torch.uint8, device=dev)
    base[src: src + 2 * src_n] = (torch.randn(src_n, device=dev, generator=g) * 4).half().view(torch.uint8)
    a = base.clone()
    sv.generate(specs, a)
    plan = sv.GeneratePlan(specs, ar.size, device=dev)
    for _ in range(2):
        b = base.clone()
        plan(b)
        assert torch.equal(a, b)
