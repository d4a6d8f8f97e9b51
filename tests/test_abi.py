"""Host-side checks of the C ABI (no GPU needed, no compute call).

The library loads without a device (static CUDA runtime), exports every
function include/synverify.h declares, its structs have the header's layout,
and every validation error is reported before anything touches CUDA.
"""
import ctypes as C
import os
import re

import pytest

import paper_2609_00058_gb300 as sv
import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADERS = [os.path.join(ROOT, "include", f) for f in sorted(os.listdir(os.path.join(ROOT, "include")))
           if f.endswith(".h")]


@pytest.fixture(scope="module")
def lib():
    from paper_2609_00058_gb300 import build
    build.build()
    return sv.lib()


def declared_functions():
    text = "".join(open(h).read() for h in HEADERS)
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    names = re.findall(r"^[A-Za-z_][\w \t\*]*?\b([a-z_][a-z0-9_]*)\s*\([^;{]*\)\s*;", text, flags=re.M)
    return sorted(set(names))


def test_header_declares_the_three_entry_points():
    names = declared_functions()
    for n in ("syn_generate", "verify_compare", "verify_progressive"):
        assert n in names


def test_every_declared_function_is_exported(lib):
    names = declared_functions()
    assert len(names) >= 10
    for n in names:
        assert hasattr(lib, n), n
    assert {e[0] for e in sv.EXPORTS} == set(names)


def test_struct_layouts():
    assert C.sizeof(sv.syn_spec) == 224
    assert C.sizeof(sv.vc_pair) == 48
    assert C.sizeof(sv.vc_result) == 80
    assert C.sizeof(sv.sv_perturb) == 40


def test_abi_version_and_strerror(lib):
    assert lib.sv_abi_version() == 1
    for code in (0, -1, -2, -3, -4, -5):
        assert lib.sv_strerror(code)
    assert b"unknown" in lib.sv_strerror(-99)


def _spec(**kw):
    base = dict(dtype="f32", dist="uniform", n=1024, seed=1, ref_offset=0, p0=-1.0, p1=1.0)
    base.update(kw)
    return W.GenSpec(**base)


BAD_SPECS = [
    (dict(dtype="i32", dist="uniform"), -1),                      # float dist on an integer type
    (dict(dtype="f32", dist="int_range"), -1),                    # integer dist on a float type
    (dict(ref_offset=None), -1),                                   # no output at all
    (dict(ref_offset=8), -2),                                      # misaligned output
    (dict(elem_offset=2, logical_n=4096), -2),                     # elem_offset not a multiple of 4
    (dict(ref_offset=4096 * 4), -3),                               # output beyond the arena
    (dict(n=4096 * 4 + 1), -3),                                    # too many elements for the arena
    (dict(specials=("imin",), special_rate=0.1), -1),              # integer special on a float type
    (dict(specials=("nan",), special_rate=1.5), -1),               # rate above 1
    (dict(specials=("nan",), special_rate=float("nan")), -1),      # NaN rate
    (dict(p0=1.0, p1=-1.0), -1),                                   # empty uniform range
    (dict(p0=float("-inf"), p1=1.0), -1),                          # infinite uniform bound
    (dict(dist="normal", p0=0.0, p1=float("nan")), -1),            # non-finite normal scale
    (dict(logical_n=100), -1),                                     # n beyond the logical length
    (dict(logical_n=1 << 41), -3),                                 # logical length beyond the limit
    (dict(pelem=W.Perturb("count_set", count=1)), -1),             # count kind in the element-wise slot
    (dict(pcount=W.Perturb("rate_add_pm", rate=0.1)), -1),         # element-wise kind in the count slot
    (dict(pcount=W.Perturb("count_set", count=0)), -1),            # empty count
    (dict(pcount=W.Perturb("swap_pairs", count=600)), -1),         # more strata than elements
    (dict(dtype="i32", dist="int_range", i0=5, i1=4), -1),         # empty integer range
    (dict(dtype="i32", dist="int_range", i0=0, i1=1 << 31), -1),   # beyond int32
    (dict(dtype="u32", dist="int_range", i0=-1, i1=3), -1),        # negative unsigned
    (dict(dtype="i64", dist="int_range", pelem=W.Perturb("rel_noise", value=0.1)), -1),  # noise on ints
    (dict(dtype="bf16", dist="dotlike", rows=4, cols=6, dot_k=8, n=24), -1),   # cols % 4
    (dict(dtype="bf16", dist="dotlike", rows=4, cols=8, dot_k=8, n=24), -1),   # rows*cols != n
    (dict(dtype="bf16", dist="dotlike", rows=4, cols=8, dot_k=8, n=32, a_offset=8), -2),
    (dict(dtype="bf16", dist="dotlike", rows=4, cols=8, dot_k=8, n=32, b_offset=16256), -3),
    (dict(dtype="i32", dist="from_arena", n=256, a_offset=8192 + 8), -2),       # misaligned source
    (dict(dtype="i32", dist="from_arena", n=256, a_offset=16384 - 512), -3),    # source past the arena
    (dict(dtype="i32", dist="from_arena", n=256, a_offset=512), -1),            # source overlaps the output
    (dict(dtype="i32", dist="from_arena", n=256, a_offset=8192, logical_n=4096), -3),  # source of N elements
]


@pytest.mark.parametrize("kw,code", BAD_SPECS)
def test_invalid_specs_rejected_before_any_launch(lib, kw, code):
    s = _spec(**kw)
    assert sv.check_specs([s], 4096 * 4) == code
    tab = sv.SpecTable([s])
    # the entry point returns the same code without touching the (absent) GPU
    assert lib.syn_generate(tab.arr, 1, 0x1000, 4096 * 4, None, 0, None) == code


def test_valid_specs_accepted(lib):
    ok = [_spec(), _spec(dtype="bf16", dist="normal", p0=5.0, p1=10.0, specials=("nan", "dup"), special_rate=0.1),
          _spec(dtype="i64", dist="permutation", n=512, specials=("imin", "imax"), special_rate=0.01,
                pcount=W.Perturb("swap_pairs", count=17)),
          _spec(dtype="bf16", dist="dotlike", rows=4, cols=8, dot_k=8, n=32, a_offset=256, b_offset=512),
          _spec(dtype="i64", dist="from_arena", n=256, a_offset=8192, specials=("dup",), special_rate=0.1,
                pcount=W.Perturb("count_add", count=3, ivalue=1))]
    for s in ok:
        assert sv.check_specs([s], 4096 * 4) == 0


def _pair(**kw):
    base = dict(dtype="f32", n=1024, cand_offset=0, ref_offset=0, atol=1e-5, rtol=1e-5)
    base.update(kw)
    return W.Pair(**base)


BAD_PAIRS = [
    (dict(atol=-1.0), -1),
    (dict(rtol=float("nan")), -1),
    (dict(cand_offset=4), -2),
    (dict(ref_offset=8), -2),
    (dict(n=1025), -3),
    (dict(dtype="i64", n=600), -3),
    (dict(cand_offset=4096), -3),
]


@pytest.mark.parametrize("kw,code", BAD_PAIRS)
def test_invalid_pairs_rejected_before_any_launch(lib, kw, code):
    p = _pair(**kw)
    assert sv.check_pairs([p], 4096, 4096) == code
    tab = sv.PairTable([p])
    assert lib.verify_compare(tab.arr, 1, 0x1000, 4096, 0x2000, 4096, 0x3000, 0x4000, 1 << 20, None) == code
    ptab = sv.PairTable([p], progressive=True)
    assert lib.verify_progressive(ptab.arr, 1, 0x1000, 4096, 0x2000, 4096, 0x3000, 0x5000, 0x4000, 1 << 20,
                                  None) == code


def test_integer_pairs_ignore_tolerances(lib):
    assert sv.check_pairs([_pair(dtype="i32", atol=-1.0)], 4096, 4096) == 0


def test_workspace_sizes(lib):
    small = sv.SpecTable([_spec()] * 3)
    assert small.ws_bytes == 0  # inline table
    big = sv.SpecTable([_spec()] * 9)
    assert big.ws_bytes >= 9 * 240 and big.ws_bytes % 256 == 0
    pt = sv.PairTable([_pair()] * 3)
    assert pt.ws_bytes >= 64 * 4 and pt.ws_bytes % 256 == 0
    # partial slots: min(tiles, 4096) + pairs per dtype group
    huge = sv.PairTable([_pair(n=1 << 30)])
    assert huge.ws_bytes == ((4096 + 1) * 64 + 255) // 256 * 256
    mixed = sv.PairTable([_pair(n=4096), _pair(dtype="bf16", n=8192), _pair(dtype="i64", n=2048)] * 4)
    assert mixed.ws_bytes >= 12 * 80 + 24 * 64
    lad = sv.PairTable([_pair(n=1 << e) for e in (10, 20, 27)], progressive=True)
    assert lad.ws_bytes == ((4096 + 1) * 64 + 255) // 256 * 256


def test_workspace_too_small_rejected(lib):
    tab = sv.PairTable([_pair()])
    assert lib.verify_compare(tab.arr, 1, 0x1000, 4096, 0x2000, 4096, 0x3000, 0x4000, 64, None) == -4
    assert lib.verify_compare(tab.arr, 1, 0x1000, 4096, 0x2000, 4096, 0x3000, 0x4010, 1 << 20, None) == -4
    big = sv.SpecTable([_spec()] * 9)
    assert lib.syn_generate(big.arr, 9, 0x1000, 4096 * 4, None, 0, None) == -4


def test_zero_entries_is_a_no_op(lib):
    assert lib.syn_generate(None, 0, None, 0, None, 0, None) == 0
    assert lib.verify_compare(None, 0, None, 0, None, 0, None, None, 0, None) == 0


def test_binding_fails_loudly_without_library(monkeypatch, tmp_path):
    monkeypatch.setattr(sv, "_lib", None)
    monkeypatch.setattr(sv, "LIB_PATH", str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError, match="not built"):
        sv.lib()


def test_box_muller_entry_validates_before_any_launch():
    lib = sv.lib()
    assert lib.syn_box_muller(None, 0, None, None) == 0            # no-op
    assert lib.syn_box_muller(None, 4, 0x1000, None) == -1         # null words
    assert lib.syn_box_muller(0x1004, 4, 0x2000, None) == -2       # 4-byte aligned words
    assert lib.syn_box_muller(0x1000, 4, 0x2004, None) == -2       # 4-byte aligned output
    assert lib.syn_box_muller(0x1000, (1 << 39) + 1, 0x2000, None) == -3


def test_failure_hook_arguments():
    lib = sv.lib()
    assert lib.sv_debug_fail_launches(-1) == -1
    assert lib.sv_debug_fail_launches(0) == 0


def _tiles(**kw):
    base = dict(dtype="f32", rows=10, cols=16, cand_offset=0, ref_offset=0, tile_rows=4, tile_cols=8)
    base.update(kw)
    return W.Tiles(**base)


BAD_TILES = [
    (dict(dtype="f32", atol=-1.0), -1),
    (dict(tile_rows=0), -1),
    (dict(cand_pitch=15), -1),                         # pitch below cols
    (dict(cand_offset=8), -2),
    (dict(cand_pitch=17), -2),                         # pitch * 4 bytes not a multiple of 16
    (dict(tile_cols=6), -2),                           # tile width not whole vectors
    (dict(rows=10, ref_pitch=1 << 20), -3),            # the reference beyond its buffer
    (dict(rows=1 << 20, cols=1 << 16, tile_rows=1, tile_cols=4), -3),  # beyond the buffers, and 2^34 tiles
]


@pytest.mark.parametrize("kw,rc", BAD_TILES)
def test_tile_validation(lib, kw, rc):
    t = _tiles(**kw)
    n = C.c_uint64(7)
    got = lib.sv_check_tiles(C.byref(sv.to_c_tiles(t)), 1 << 20 if rc != -3 else 4096, 4096 * 16, C.byref(n))
    assert got == rc and n.value == 0


def test_tile_counts(lib):
    assert sv.tile_count(_tiles()) == 3 * 2
    assert sv.tile_count(_tiles(rows=0)) == 0
    assert sv.tile_count(_tiles(tile_rows=1, tile_cols=16)) == 10
    assert sv.tile_count(_tiles(rows=1, cols=3, tile_cols=3)) == 1  # one row, narrower than a vector: no pitch rule
    assert sv.tile_count(_tiles(rows=1 << 16, cols=1 << 16, tile_rows=1, tile_cols=4, cand_pitch=0, ref_pitch=0),
                         1 << 34, 1 << 34) == 1 << 30
    with pytest.raises(sv.SynVerifyError):
        sv.tile_count(_tiles(tile_cols=6))


def test_compare_plan_refusals_before_any_copy(lib):
    plan = C.c_void_p(123)
    good = sv.PairTable([W.Pair("f32", 64, 0, 0, 1e-5, 1e-5)])
    bad = sv.PairTable([W.Pair("f32", 64, 8, 0, 1e-5, 1e-5)])  # misaligned offset
    assert lib.sv_compare_plan_create(bad.arr, 1, 4096, 4096, None, 0, None, C.byref(plan)) == -2
    assert plan.value is None
    many = sv.PairTable([W.Pair("f32", 64, 256 * i, 0, 1e-5, 1e-5) for i in range(9)])  # needs a table
    assert lib.sv_compare_plan_create(many.arr, 9, 1 << 20, 4096, None, 0, None, C.byref(plan)) == -4
    assert lib.sv_compare_plan_create(good.arr, 1, 4096, 4096, None, 0, None, None) == -1
    assert lib.verify_compare_planned(None, None, None, None, None) == -1
    lib.sv_compare_plan_destroy(None)  # nothing to free


def test_misaligned_base_pointers_rejected_before_any_launch(lib):
    """Element buffers must start on 16 bytes and results on 8 (the kernels
    move 128-bit vectors and 64-bit fields); a misaligned base -- a byte view
    with an odd storage offset, say -- is refused with SV_EALIGN and nothing
    is enqueued (these calls would otherwise launch)."""
    tab = sv.PairTable([_pair()])
    ws, wsb = 0x100000, 1 << 20
    for cand, ref, res in ((0x1008, 0x2000, 0x3000), (0x1000, 0x2004, 0x3000), (0x1000, 0x2000, 0x3004)):
        assert lib.verify_compare(tab.arr, 1, cand, 4096, ref, 4096, res, ws, wsb, None) == -2
        assert lib.verify_compare_noalloc(tab.arr, 1, cand, 4096, ref, 4096, res, None) == -2
    stages = sv.PairTable([_pair()], progressive=True)
    assert lib.verify_progressive(stages.arr, 1, 0x1008, 4096, 0x2000, 4096, 0x3000, 0x5000, ws, wsb, None) == -2
    assert lib.verify_progressive(stages.arr, 1, 0x1000, 4096, 0x2000, 4096, 0x3000, 0x5002, ws, wsb, None) == -2
    spec = sv.SpecTable([_spec()])
    assert lib.syn_generate(spec.arr, 1, 0x1008, 4096 * 4, None, 0, None) == -2
    # a plan checks the buffers it is handed at every call
    plan = C.c_void_p()
    assert lib.sv_compare_plan_create(tab.arr, 1, 4096, 4096, ws, wsb, None, C.byref(plan)) == 0
    try:
        assert lib.verify_compare_planned(plan, 0x1000, 0x2008, 0x3000, None) == -2
        assert lib.verify_compare_planned(plan, 0x1000, 0x2000, 0x3001, None) == -2
    finally:
        lib.sv_compare_plan_destroy(plan)


def test_noalloc_slot_limit_boundary(lib):
    """verify_compare_noalloc counts min(tiles, 4096) + pairs partial slots
    per dtype against SV_NOALLOC_SLOTS = 4104.  A call landing exactly on
    the limit passes the slot check (it then stops at the misaligned result
    pointer, SV_EALIGN, before any launch); one slot more is SV_ERANGE."""
    big, n = 1 << 40, 1 << 22  # 2^22 fp32 elements: 16 MiB, 1024 tiles of 16 KiB per pair
    f32 = [W.Pair("f32", n, i << 24, i << 24) for i in range(8)]
    bf16 = W.Pair("bf16", 16, 8 << 24, 8 << 24)  # one tile
    # 8 f32 pairs: 8192 tiles -> 4096 + 8 = 4104 slots, exactly the limit
    at_limit = sv.PairTable(f32)
    assert lib.verify_compare_noalloc(at_limit.arr, 8, 0x1000, big, 0x1000, big, 0x2001, None) == -2
    # 7 f32 pairs (4096 + 7) and one bf16 pair (1 + 1): 4105 slots, one too many
    over = sv.PairTable(f32[:7] + [bf16])
    assert lib.verify_compare_noalloc(over.arr, 8, 0x1000, big, 0x1000, big, 0x2001, None) == -3
    # 6 f32 pairs (4096 + 6) and one bf16 pair (1 + 1): 4104 slots again
    fits = sv.PairTable(f32[:6] + [bf16])
    assert lib.verify_compare_noalloc(fits.arr, 7, 0x1000, big, 0x1000, big, 0x2001, None) == -2


def test_binding_refuses_host_and_strided_tensors_before_any_launch():
    """A CPU tensor's data_ptr() is a host address and a strided view is not
    the dense memory the library reads: every binding call refuses both with
    ValueError before it reaches the library."""
    torch = pytest.importorskip("torch")
    host = torch.zeros(4096, dtype=torch.uint8)
    pairs = [_pair()]
    with pytest.raises(ValueError, match="CUDA"):
        sv.compare(pairs, host, host)
    with pytest.raises(ValueError, match="CUDA"):
        sv.progressive(pairs, host, host)
    with pytest.raises(ValueError, match="CUDA"):
        sv.generate([_spec()], torch.zeros(4096 * 4, dtype=torch.uint8))
    with pytest.raises(ValueError, match="CUDA"):
        sv.compare_tiles(_tiles(), host, host)
    with pytest.raises(ValueError, match="CUDA"):
        sv.box_muller(torch.zeros(8, dtype=torch.int32))
    with pytest.raises(ValueError, match="CUDA"):
        sv.convert(host, "u8", "f32")
    strided = torch.zeros(8192, dtype=torch.uint8)[::2]
    with pytest.raises(ValueError):
        sv.compare(pairs, strided, strided)


def test_exact_specials_validation(lib):
    n = 1 << 22
    # 2^22 * 0.5 = 2^21 exact specials: beyond SV_MAX_COUNT (2^20) -> SV_ERANGE
    too_many = sv.SpecTable([W.GenSpec("f32", "uniform", n, ref_offset=0, p0=0, p1=1, specials=("nan",),
                                       special_rate=0.5, special_exact=True)])
    assert lib.sv_check_specs(too_many.arr, 1, 4 * n) == -3
    ok = sv.SpecTable([W.GenSpec("f32", "uniform", n, ref_offset=0, p0=0, p1=1, specials=("nan",),
                                 special_rate=0.25, special_exact=True)])
    assert lib.sv_check_specs(ok.arr, 1, 4 * n) == 0


def test_generate_plan_refusals_before_any_copy(lib):
    plan = C.c_void_p(123)
    bad = sv.SpecTable([_spec(ref_offset=8)])  # misaligned output
    assert lib.sv_generate_plan_create(bad.arr, 1, 4096 * 4, None, 0, None, C.byref(plan)) == -2
    assert plan.value is None
    many = sv.SpecTable([_spec(ref_offset=4096 * i) for i in range(9)])  # needs a table in the workspace
    assert lib.sv_generate_plan_create(many.arr, 9, 4096 * 4 * 9, None, 0, None, C.byref(plan)) == -4
    good = sv.SpecTable([_spec()])
    assert lib.sv_generate_plan_create(good.arr, 1, 4096 * 4, None, 0, None, None) == -1
    assert lib.syn_generate_planned(None, 0x1000, None) == -1
    # a plan of <= 8 specs needs no workspace and no copy; its calls check the arena
    assert lib.sv_generate_plan_create(good.arr, 1, 4096 * 4, None, 0, None, C.byref(plan)) == 0
    try:
        assert lib.syn_generate_planned(plan, None, None) == -1
        assert lib.syn_generate_planned(plan, 0x1008, None) == -2
    finally:
        lib.sv_generate_plan_destroy(plan)
    lib.sv_generate_plan_destroy(None)
