"""Host validation under random and extreme tables (hypothesis, no GPU): every
check returns a status without crashing, and whatever it accepts stays inside
the caller's buffers by exact (Python integer) arithmetic -- the property the
kernels' 64-bit address arithmetic relies on.  Field values mix small aligned
numbers with the edges of their types (0, 2^31, 2^32, 2^40, 2^63, 2^64 - 1,
NaN, infinities) so that products and sums that could wrap are exercised;
specs start valid and have up to two fields moved to such edges (about 40%
of them stay accepted, so both sides of every rule get examples)."""
import ctypes as C

import pytest

hypothesis = pytest.importorskip("hypothesis")
from hypothesis import HealthCheck, given, settings
from hypothesis import strategies as st

import paper_2609_00058_gb300 as sv

EB = {0: 4, 1: 2, 2: 2, 3: 4, 4: 8, 5: 4}
NO_OUTPUT = (1 << 64) - 1
EDGES = [0, 1, 3, 4, 15, 16, 17, 64, 4096, (1 << 31) - 1, 1 << 31, 1 << 32, (1 << 40) - 4, 1 << 40,
         (1 << 40) + 16, 1 << 62, 1 << 63, (1 << 64) - 16, (1 << 64) - 1]
u64 = st.one_of(st.sampled_from(EDGES), st.integers(0, (1 << 64) - 1), st.integers(0, 1 << 16).map(lambda x: 16 * x),
                st.integers(0, 1 << 12))
small = st.one_of(st.integers(0, 64), st.sampled_from([0, 1, 4, 5, 128, 1 << 20, (1 << 20) + 1, 1 << 32]))
dbl = st.one_of(st.sampled_from([0.0, 1e-4, 0.5, 1.0, -1.0, 1e300]), st.floats(allow_nan=True, allow_infinity=True))
buf = st.sampled_from([0, 16, 4096, 1 << 20, 1 << 32, 1 << 40, 1 << 62, (1 << 64) - 1])
SETTINGS = settings(max_examples=2500, deadline=None, suppress_health_check=[HealthCheck.too_slow])


def perturb(kind_range):
    return st.builds(lambda k, s, r, c, v, iv: sv.sv_perturb(k, s, r, c, v, iv), kind_range,
                     st.integers(0, (1 << 32) - 1), dbl, st.one_of(small, u64), dbl,
                     st.integers(-(1 << 63), (1 << 63) - 1))


FLOAT_DISTS, INT_DISTS = (0, 1, 4, 5, 6, 7), (2, 3, 5, 6, 7)
FIELDS = ("dtype", "dist", "n", "special_mask", "special_rate", "ref_offset", "cand_offset", "elem_offset", "logical_n",
          "p0", "p1", "i0", "i1", "rows", "cols", "dot_k", "a_offset", "b_offset")


@st.composite
def specs(draw):
    """A spec that the rules accept, then 0 to 2 of its fields set to edge values:
    the accepted and the just-rejected neighbourhoods both get examples."""
    dt = draw(st.integers(0, 5))
    fl = dt <= 2
    di = draw(st.sampled_from(FLOAT_DISTS if fl else INT_DISTS))
    eb = EB[dt]
    s = sv.syn_spec()
    s.dtype, s.dist, s.seed, s.stream = dt, di, draw(st.integers(0, (1 << 64) - 1)), draw(st.integers(0, 1000))
    if di == 4:  # dot-like: rows x cols outputs from rows x K and K x cols factors
        s.rows, s.cols, s.dot_k = draw(st.integers(1, 64)), 4 * draw(st.integers(1, 64)), draw(st.integers(1, 130))
        n = s.rows * s.cols
        s.a_offset, s.b_offset = 1 << 30, (1 << 30) + 16 * draw(st.integers(1 << 12, 1 << 14))
    else:
        n = draw(st.one_of(st.integers(0, 1 << 16), st.sampled_from([1 << 20, 1 << 30, (1 << 40) - 4])))
    s.elem_offset = 4 * draw(st.integers(0, 64))
    s.n = n
    s.logical_n = draw(st.sampled_from([0, s.elem_offset + n, s.elem_offset + n + 4]))
    if di == 4:
        s.elem_offset, s.logical_n = 0, 0
    s.ref_offset = 16 * draw(st.integers(0, 1 << 20))
    s.cand_offset = draw(st.sampled_from([NO_OUTPUT, s.ref_offset + ((n * eb + 15) // 16) * 16]))
    if di == 7:  # the source lies past both outputs
        s.a_offset = ((s.ref_offset + 2 * n * eb + 31) // 16) * 16
    s.p0, s.p1 = sorted(draw(st.lists(st.floats(-1e6, 1e6), min_size=2, max_size=2)))
    lo_i, hi_i = {3: (-(1 << 31), (1 << 31) - 1), 5: (0, (1 << 32) - 1), 4: (-(1 << 63), (1 << 63) - 1)}.get(dt, (0, 0))
    s.i0, s.i1 = sorted(draw(st.lists(st.integers(lo_i, hi_i), min_size=2, max_size=2)))
    s.special_mask = draw(st.sampled_from([0, 0x1, 0x9F, 0x8000009F] if fl else [0, 0x10, 0xF0, 0x800000F0]))
    s.special_rate = draw(st.sampled_from([0.0, 1e-4, 0.5, 1.0]))
    pe = draw(st.sampled_from([0, 1, 5] if fl else [0, 1]))
    s.pelem = sv.sv_perturb(pe, 3, draw(st.sampled_from([0.0, 1e-3, 1.0])), 0, 2.0 ** -9, 1)
    pk = draw(st.sampled_from([0, 2, 3, 4]))
    s.pcount = sv.sv_perturb(pk, 4, 0.0, draw(st.integers(1, 8)), 1.0, 1)
    for _ in range(draw(st.integers(0, 2))):  # mutations towards the edges
        f = draw(st.sampled_from(FIELDS))
        if f in ("special_rate", "p0", "p1"):
            setattr(s, f, draw(dbl))
        elif f in ("i0", "i1"):
            setattr(s, f, draw(st.integers(-(1 << 63), (1 << 63) - 1)))
        elif f in ("dtype", "dist"):
            setattr(s, f, draw(st.integers(0, 9)))
        elif f == "special_mask":
            setattr(s, f, draw(st.integers(0, (1 << 32) - 1)))
        else:
            setattr(s, f, draw(u64))
    return s


@SETTINGS
@given(specs(), st.sampled_from([1 << 40, 1 << 62, (1 << 64) - 1, 1 << 31]))
def test_accepted_specs_stay_in_the_arena(s, arena):
    rc = sv.lib().sv_check_specs(C.byref(s), 1, arena)
    assert rc in (0, -1, -2, -3, -4, -5, -6, -7, -8, -9), rc
    if rc != 0:
        return
    assert s.dtype <= 5 and s.dist <= 7
    eb = EB[s.dtype]
    N = s.logical_n or s.elem_offset + s.n
    assert s.elem_offset % 4 == 0 and s.elem_offset + s.n <= N <= 1 << 40
    assert s.ref_offset != NO_OUTPUT or s.cand_offset != NO_OUTPUT
    for off in (s.ref_offset, s.cand_offset):
        if off != NO_OUTPUT:
            assert off % 16 == 0 and off + s.n * eb <= arena
    if s.dist == 4:  # dot-like factors
        assert s.rows * s.cols == N and s.cols % 4 == 0 and 0 < s.dot_k <= 1 << 20
        assert s.a_offset % 16 == 0 and s.a_offset + 4 * s.rows * s.dot_k <= arena
        assert s.b_offset % 16 == 0 and s.b_offset + 4 * s.dot_k * s.cols <= arena
    if s.dist == 7:  # arena source: the whole logical array
        assert s.a_offset % 16 == 0 and s.a_offset + N * eb <= arena
    if s.pcount.kind:
        strata = 2 * s.pcount.count if s.pcount.kind == 3 else s.pcount.count
        assert 0 < s.pcount.count <= 1 << 20 and strata <= N


pairs = st.builds(lambda dt, fl, n, co, ro, a, r: sv.vc_pair(dt, fl, n, co, ro, a, r),
                  st.integers(0, 7), st.sampled_from([0, 1, 2, 3]), st.one_of(small, u64), u64, u64, dbl, dbl)


@SETTINGS
@given(pairs, buf, buf)
def test_accepted_pairs_stay_in_their_buffers(p, cb, rb):
    rc = sv.lib().sv_check_pairs(C.byref(p), 1, cb, rb)
    if rc != 0:
        return
    assert p.dtype <= 5 and p.flags in (0, 1)
    eb = EB[p.dtype]
    assert p.cand_offset % 16 == 0 and p.cand_offset + p.n * eb <= cb
    assert p.ref_offset % 16 == 0 and p.ref_offset + p.n * eb <= rb
    if p.dtype in (0, 1, 2):
        assert p.atol >= 0 and p.rtol >= 0


tiles = st.builds(lambda dt, fl, rows, cols, co, ro, cp, rp, tr, tc, a, r:
                  sv.vc_tiles(dt, fl, rows, cols, co, ro, cp, rp, tr, tc, a, r),
                  st.integers(0, 7), st.sampled_from([0, 1, 2]), st.one_of(small, u64), st.one_of(small, u64), u64, u64,
                  st.one_of(small, u64), st.one_of(small, u64), st.one_of(small, u64), st.one_of(small, u64), dbl, dbl)


@SETTINGS
@given(tiles, buf, buf)
def test_accepted_tiles_stay_in_their_buffers(t, cb, rb):
    n = C.c_uint64(12345)
    rc = sv.lib().sv_check_tiles(C.byref(t), cb, rb, C.byref(n))
    if rc != 0:
        return
    assert t.dtype <= 5 and t.tile_rows > 0 and t.tile_cols > 0
    if t.rows == 0 or t.cols == 0:
        assert n.value == 0
        return
    eb = EB[t.dtype]
    for off, pitch, size in ((t.cand_offset, t.cand_pitch, cb), (t.ref_offset, t.ref_pitch, rb)):
        assert pitch >= t.cols and off % 16 == 0
        assert off + ((t.rows - 1) * pitch + t.cols) * eb <= size
        if t.rows > 1:
            assert pitch * eb % 16 == 0
    tiles_n = -(-t.rows // t.tile_rows) * -(-t.cols // t.tile_cols)
    assert n.value == tiles_n <= (1 << 31) - 1
