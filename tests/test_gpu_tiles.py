"""Parity of verify_compare_tiles (shaped outputs compared tile by tile) with
the oracle's or_compare_tiles, through the C ABI on the GPU: every dtype,
dense and padded pitches (different per operand), tiles that divide the
output and ragged ones, tiles narrower than a 16-byte vector, one row per
tile, one tile for everything; planted mismatches, NaN, infinities and
denormals; and the dot-like workload's 32768 x 32768 bf16 output in
128 x 128 tiles, checked on sampled tile rows the oracle computes."""
import numpy as np
import pytest

import oracle
import paper_2609_00058_gb300 as sv
import workloads as W
from gpu_util import assert_results_match, device, to_dev

pytestmark = pytest.mark.gpu
NP = {"f32": np.float32, "f16": np.float16, "i32": np.int32, "i64": np.int64, "u32": np.uint32}


@pytest.fixture(scope="module")
def dev():
    return device()


def make_pair(dtype, rows, cols, cpitch, rpitch, seed):
    """Reference and candidate of a rows x cols output in buffers with the given
    pitches; padding holds garbage that differs between the two."""
    rng = np.random.default_rng(seed)
    if dtype == "bf16":
        vals = rng.normal(5, 10, size=(rows, cols)).astype(np.float32)
        yv = (vals.view(np.uint32) >> 16).astype(np.uint16)
        xv = yv.copy()
        flat = xv.reshape(-1)
        k = rng.choice(flat.size, max(1, flat.size // 500), replace=False)
        flat[k] ^= rng.integers(1, 1 << 8, size=k.size, dtype=np.uint16)
        flat[rng.choice(flat.size, 3)] = 0x7FC0
        store = np.uint16
    elif dtype in ("f32", "f16"):
        yv = rng.normal(5, 10, size=(rows, cols)).astype(NP[dtype])
        xv = (yv + rng.normal(0, 1e-3, size=yv.shape).astype(NP[dtype])).astype(NP[dtype])
        flat, yflat = xv.reshape(-1), yv.reshape(-1)
        flat[rng.choice(flat.size, max(1, flat.size // 300), replace=False)] += 1
        flat[rng.choice(flat.size, 2)] = np.nan
        yflat[rng.choice(flat.size, 2)] = np.inf
        flat[rng.choice(flat.size, 2)] = np.finfo(NP[dtype]).tiny / 4
        store = NP[dtype]
    else:
        info = np.iinfo(NP[dtype])
        yv = rng.integers(max(info.min, -1000), min(info.max, 1000), size=(rows, cols), dtype=NP[dtype])
        xv = yv.copy()
        flat = xv.reshape(-1)
        flat[rng.choice(flat.size, max(1, flat.size // 400), replace=False)] = info.max
        store = NP[dtype]
    x = np.full((rows, cpitch), 0x55, dtype=np.uint8 if store is None else store)
    y = np.full((rows, rpitch), 0x33, dtype=x.dtype)
    x[:, :cols] = xv.view(x.dtype)
    y[:, :cols] = yv.view(y.dtype)
    return np.ascontiguousarray(x).view(np.uint8).reshape(-1), np.ascontiguousarray(y).view(np.uint8).reshape(-1)


CASES = [  # rows, cols, cand pitch, ref pitch, tile rows, tile cols
    (64, 256, 256, 256, 16, 64),
    (37, 100, 104, 112, 8, 32),      # ragged in both directions, padded pitches
    (5, 1000, 1000, 1024, 1, 1000),  # one row per tile
    (33, 36, 36, 40, 33, 36),        # one tile
    (50, 24, 24, 24, 7, 8),          # tiles of two 16-byte vectors
    (9, 3, 4, 8, 2, 3),              # rows narrower than a vector: ragged ends only
    (300, 513, 520, 520, 128, 128),
    (10000, 64, 64, 72, 1, 64),      # enough tiles for one warp per tile
    (12000, 37, 40, 48, 1, 37),      # one warp per tile, a ragged end in every row
    # enough tiles for warp teams, tiles narrower than the output: groups of
    # side-by-side tiles (their width in vectors divides 32) plus the ragged
    # last tile column one by one; 7 and 5 rows per tile, padded pitches
    (16000, 520, 528, 536, 7, 64),
    (20000, 100, 104, 112, 5, 32),   # (16-bit types: no whole group fits in a row)
]


@pytest.mark.parametrize("dtype", ["f32", "f16", "bf16", "i32", "i64", "u32"])
@pytest.mark.parametrize("case", CASES)
def test_tiles_match_oracle(dev, dtype, case):
    rows, cols, cp, rp, tr, tc = case
    sz = W.DTYPE_BYTES[dtype]
    align = 16 // sz  # pitches and tile widths in whole 16-byte vectors (the ABI's alignment rule)
    cp, rp = -(-cp // align) * align, -(-rp // align) * align
    if tc < cols:
        tc = -(-tc // align) * align
    x, y = make_pair(dtype, rows, cols, cp, rp, seed=rows * 7 + cols)
    t = W.Tiles(dtype, rows, cols, 0, 0, cand_pitch=cp, ref_pitch=rp, tile_rows=tr, tile_cols=tc,
                atol=1e-3, rtol=1e-3)
    want = oracle.compare_tiles(t, x, y)
    res = sv.compare_tiles(t, to_dev(x, dev), to_dev(y, dev))
    got = sv.decode_results(res, len(want))
    assert_results_match(got, want, "%s %r" % (dtype, case))
    assert any(not w["pass"] for w in want)


def test_offsets_and_shared_buffer(dev):
    """Both operands in one arena at 16-byte aligned offsets, a sub-matrix view."""
    rows, cols = 40, 64
    x, y = make_pair("f32", rows, 96, 96, 96, seed=5)
    arena = np.zeros(4096 + x.size + y.size + 64, np.uint8)
    arena[4096:4096 + x.size], arena[4096 + x.size + 48: 4096 + x.size + 48 + y.size] = x, y
    t = W.Tiles("f32", rows, cols, 4096 + 16 * 4, 4096 + x.size + 48 + 16 * 4, cand_pitch=96, ref_pitch=96,
                tile_rows=16, tile_cols=16, atol=1e-4, rtol=1e-4)  # columns 16..79 of each operand
    want = oracle.compare_tiles(t, arena, arena)
    a = to_dev(arena, dev)
    assert_results_match(sv.decode_results(sv.compare_tiles(t, a, a), len(want)), want, "sub-matrix")


def test_dotlike_output_per_tile(dev):
    """The dot-like workload's bf16 32768 x 32768 reference and its noisy twin,
    compared in 128 x 128 tiles (65536 results); sampled tile rows are
    recomputed by the oracle from the same bytes."""
    import torch
    wl = W.FULL_SIZE["dotlike_bf16"]()
    arena = torch.zeros(wl.arena_bytes, dtype=torch.uint8, device=dev)
    for call in wl.gen_calls:
        sv.generate(call, arena)
    pr = wl.pairs[0]
    side = 1 << 15
    t = W.Tiles("bf16", side, side, pr.cand_offset, pr.ref_offset, tile_rows=128, tile_cols=128,
                atol=pr.atol, rtol=pr.rtol)
    res = sv.compare_tiles(t, arena, arena)
    got = sv.decode_results(res, 256 * 256)
    whole = sv.decode_results(sv.compare([pr], arena, arena), 1)[0]
    assert sum(g["mismatches"] for g in got) == whole["mismatches"]
    assert sum(g["n_finite"] for g in got) == whole["n_finite"] == side * side
    firsts = [g["first_mismatch"] for g in got if g["first_mismatch"] >= 0]
    assert (min(firsts) if firsts else -1) == whole["first_mismatch"]
    for ti in (0, 97, 255):  # one tile row each: rows [128 ti, 128 ti + 128)
        rows0 = 128 * ti * side * 2
        c = arena[pr.cand_offset + rows0: pr.cand_offset + rows0 + 128 * side * 2].cpu().numpy()
        r = arena[pr.ref_offset + rows0: pr.ref_offset + rows0 + 128 * side * 2].cpu().numpy()
        sub = W.Tiles("bf16", 128, side, 0, 0, tile_rows=128, tile_cols=128, atol=pr.atol, rtol=pr.rtol)
        want = oracle.compare_tiles(sub, c, r)
        for w in want:  # the oracle's indices are relative to the sampled rows
            if w["first_mismatch"] >= 0:
                w["first_mismatch"] += 128 * ti * side
        assert_results_match(got[256 * ti: 256 * ti + 256], want, "tile row %d" % ti)


def test_manifest_plan_end_to_end(dev):
    """A manifest entry's plan on the GPU: inputs synthesized with the
    broad-range preset, a reference output (a copy of input a, as an identity
    kernel would write it) and a candidate with two planted errors, compared
    per 32 x 64 tile; the failing tiles are the ones holding the errors, and
    every tile's verdict equals the oracle's on the same bytes."""
    import json

    import torch

    from paper_2609_00058_gb300 import manifest as M
    entry = M.load(json.dumps({
        "kernel": "identity", "atol": 1e-5, "rtol": 1e-5,
        "inputs": [{"name": "a", "shape": [256, 384], "dtype": "f32"}],
        "outputs": [{"name": "c", "shape": [256, 384], "dtype": "f32", "tile": [32, 64]}]}))[0]
    p = M.plan(entry, seed=4)
    arena = torch.zeros(p.arena_bytes, dtype=torch.uint8, device=dev)
    M.synthesize(p, arena)
    a = arena[p.inputs["a"]: p.inputs["a"] + 4 * 256 * 384].view(torch.float32)
    assert abs(a.mean().item() - 5.0) < 0.2 and abs(a.std().item() - 10.0) < 0.2  # N(5, 10)
    n = 256 * 384
    sv.generate([sv.GenSpec("f32", "from_arena", n, seed=4, stream=9, ref_offset=p.ref_outputs["c"],
                            cand_offset=p.cand_outputs["c"], a_offset=p.inputs["a"],
                            pcount=sv.Perturb("count_add", stream=3, count=2, value=1.0))], arena)
    got = M.verify(p, arena)["c"]
    t = p.tiles["c"]
    bad = M.failing_tiles(got, t)
    assert len(bad) in (1, 2) and sum(r["mismatches"] for r in got) == 2
    for (ti, tj) in bad:
        f = got[ti * 6 + tj]["first_mismatch"]
        assert (f // 384 // 32, f % 384 // 64) == (ti, tj)
    want = oracle.compare_tiles(t, arena.cpu().numpy(), arena.cpu().numpy())
    assert_results_match(got, want, "manifest plan")


def test_medium_output_per_tile(dev):
    """An 8192 x 8192 bf16 output (2 x 128 MiB, beyond L2) in 64 x 64 tiles
    (16384 verdicts, one warp per tile), with relative noise on the candidate;
    sampled tile rows are recomputed by the oracle from the same bytes."""
    import torch
    side = 8192
    g = torch.Generator(device=dev)
    g.manual_seed(8192)
    ref = torch.randn(side * side, dtype=torch.float32, device=dev, generator=g) * 10 + 5
    cand = ref * (1 + torch.randn(side * side, dtype=torch.float32, device=dev, generator=g) * 2 ** -9)
    ref16, cand16 = ref.to(torch.bfloat16), cand.to(torch.bfloat16)
    cand16[123456] = float("nan")
    cand16[side * 4000 + 77] += 3.0
    arena = torch.cat([cand16.view(torch.uint8), ref16.view(torch.uint8)])
    t = W.Tiles("bf16", side, side, 0, 2 * side * side, tile_rows=64, tile_cols=64, atol=1e-2, rtol=1e-2)
    got = sv.decode_results(sv.compare_tiles(t, arena, arena), 128 * 128)
    for ti in (0, 62, 127):
        lo, hi = 64 * ti * side * 2, 64 * (ti + 1) * side * 2
        c = arena[lo:hi].cpu().numpy()
        r = arena[2 * side * side + lo: 2 * side * side + hi].cpu().numpy()
        want = oracle.compare_tiles(W.Tiles("bf16", 64, side, 0, 0, tile_rows=64, tile_cols=64, atol=1e-2,
                                            rtol=1e-2), c, r)
        for w in want:
            if w["first_mismatch"] >= 0:
                w["first_mismatch"] += 64 * ti * side
        assert_results_match(got[128 * ti: 128 * ti + 128], want, "tile row %d" % ti)
    # the planted +3 is a mismatch of its tile (a natural one may come first)
    assert sum(r["mismatches"] for r in got) >= 2
    assert 0 <= got[62 * 128 + 1]["first_mismatch"] <= side * 4000 + 77
