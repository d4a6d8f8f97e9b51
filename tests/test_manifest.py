"""Manifest entries (Sec. 4.1.1) turned into a verification plan: parsing,
the broad-range input preset of Sec. 4.2.1, the arena layout, the specs and
tile descriptions passing the library's own validation (host only)."""
import json

import pytest

import paper_2609_00058_gb300 as sv
from paper_2609_00058_gb300 import manifest as M

ENTRY = {
    "kernel": "scaled_residual", "description": "c = a * s + b, row-wise scale s",
    "atol": 1e-4, "rtol": 1e-4,
    "inputs": [{"name": "a", "shape": [96, 128], "dtype": "f32"},
               {"name": "s", "shape": [96], "dtype": "bf16"},
               {"name": "idx", "shape": [96], "dtype": "i32"},
               {"name": "mask", "shape": [96], "dtype": "u32"},
               {"name": "b", "shape": [96, 128], "dtype": "f32", "dist": "uniform", "params": [-1, 1]}],
    "outputs": [{"name": "c", "shape": [96, 128], "dtype": "f32", "tile": [32, 64]},
                {"name": "stats", "shape": [2, 3, 8], "dtype": "i64"}],
}


def test_load_text_and_file(tmp_path):
    e = M.load(json.dumps(ENTRY))
    p = tmp_path / "m.json"
    p.write_text(json.dumps([ENTRY, dict(ENTRY, kernel="other")]))
    both = M.load(str(p))
    assert len(e) == 1 and [x.kernel for x in both] == ["scaled_residual", "other"]
    assert e[0].outputs[0].tile == (32, 64) and e[0].atol == 1e-4
    with pytest.raises(ValueError):
        M.load(json.dumps(dict(ENTRY, inputs=[{"name": "x", "shape": [4], "dtype": "f64"}])))


def test_broad_range_preset():
    e = M.load(json.dumps(ENTRY))[0]
    by = {t.name: M.preset(t) for t in e.inputs}
    assert by["a"] == ("normal", (5.0, 10.0)) and by["s"] == ("normal", (5.0, 10.0))
    assert by["idx"] == ("int_range", (-1000, 1000)) and by["mask"] == ("int_range", (0, 1000))
    assert by["b"] == ("uniform", (-1, 1))


def test_plan_layout_specs_and_tiles():
    e = M.load(json.dumps(ENTRY))[0]
    p = M.plan(e, seed=11)
    spans = [(p.inputs[t.name], t.nbytes) for t in e.inputs]
    spans += [(p.ref_outputs[t.name], t.nbytes) for t in e.outputs]
    spans += [(p.cand_outputs[t.name], t.nbytes) for t in e.outputs]
    spans.sort()
    assert all(off % 256 == 0 for off, _ in spans)
    assert all(a + n <= b for (a, n), (b, _) in zip(spans[:-1], spans[1:]))
    assert spans[-1][0] + spans[-1][1] <= p.arena_bytes
    assert sv.check_specs(p.specs, p.arena_bytes) == 0
    assert [s.stream for s in p.specs] == list(range(5)) and {s.seed for s in p.specs} == {11}
    a = p.specs[0]
    assert (a.dist, a.p0, a.p1, a.n) == ("normal", 5.0, 10.0, 96 * 128)
    c, st = p.tiles["c"], p.tiles["stats"]
    assert (c.rows, c.cols, c.tile_rows, c.tile_cols) == (96, 128, 32, 64)
    assert sv.tile_count(c, p.arena_bytes, p.arena_bytes) == 3 * 2
    assert (st.rows, st.cols, st.tile_rows, st.tile_cols) == (6, 8, 1, 8)  # 2 x 3 x 8: six rows of 8
    assert sv.tile_count(st, p.arena_bytes, p.arena_bytes) == 6
    assert c.cand_offset == p.cand_outputs["c"] and c.ref_offset == p.ref_outputs["c"]
    assert p.calling_convention().startswith("scaled_residual(a: f32 [96, 128], s: bf16 [96]")


def test_invalid_tile_shape_is_refused():
    bad = dict(ENTRY, outputs=[{"name": "c", "shape": [96, 128], "dtype": "f32", "tile": [32, 6]}])
    with pytest.raises(sv.SynVerifyError):
        M.plan(M.load(json.dumps(bad))[0])
