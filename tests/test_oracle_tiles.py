"""Pins of the oracle's tile-by-tile compare of shaped outputs
(or_compare_tiles), independent of its code:
- the tiles partition the output: their counts add up to the whole array's
  verdict from or_compare (pinned in test_oracle_compare.py);
- a single planted mismatch at every position of a small output is found by
  exactly the tile that contains it, at index row * cols + col (brute force);
- bytes in the pitch padding never count, whatever they hold;
- one tile per row equals or_compare run on each row as its own segment;
- ragged edge tiles have the area that the geometry gives.
"""
import numpy as np
import pytest

import oracle
import workloads as W

F32 = 4


def dense(rows, cols, pitch, seed, dtype=np.float32):
    rng = np.random.default_rng(seed)
    a = np.full((rows, pitch), np.nan, dtype=dtype)
    a[:, :cols] = rng.normal(5, 10, size=(rows, cols)).astype(dtype)
    return a


def as_bytes(a):
    return np.ascontiguousarray(a).view(np.uint8).reshape(-1)


def test_tiles_partition_the_whole_compare():
    rows, cols = 37, 53
    y = dense(rows, cols, cols, 1)
    x = y.copy()
    rng = np.random.default_rng(2)
    x.reshape(-1)[rng.choice(rows * cols, 40, replace=False)] += 1.0
    x[3, 4], x[10, 10], y[20, 7] = np.nan, np.inf, np.nan
    whole = oracle.compare([W.Pair("f32", rows * cols, 0, 0, 1e-5, 1e-5)], as_bytes(x), as_bytes(y))[0]
    for tr, tc in ((1, cols), (5, 7), (rows, cols), (8, 53), (37, 1)):
        t = W.Tiles("f32", rows, cols, 0, 0, tile_rows=tr, tile_cols=tc, atol=1e-5, rtol=1e-5)
        res = oracle.compare_tiles(t, as_bytes(x), as_bytes(y))
        assert len(res) == -(-rows // tr) * -(-cols // tc)
        for k in ("mismatches", "nan_disagree", "inf_disagree", "n_finite"):
            assert sum(r[k] for r in res) == whole[k], (tr, tc, k)
        assert min(r["first_mismatch"] for r in res if r["first_mismatch"] >= 0) == whole["first_mismatch"]
        assert max(r["max_abs"] for r in res) == whole["max_abs"]
        assert max(r["max_rel"] for r in res) == whole["max_rel"]
        ssq = sum(r["rms"] ** 2 * r["n_finite"] for r in res)
        assert np.sqrt(ssq / whole["n_finite"]) == pytest.approx(whole["rms"], rel=1e-12)


@pytest.mark.parametrize("pitch", [11, 16])
def test_every_single_mismatch_lands_in_its_tile(pitch):
    rows, cols, tr, tc = 7, 11, 3, 4
    y = dense(rows, cols, pitch, 3)
    t = W.Tiles("f32", rows, cols, 0, 0, cand_pitch=pitch, ref_pitch=pitch, tile_rows=tr, tile_cols=tc)
    ntc = -(-cols // tc)
    for r in range(rows):
        for c in range(cols):
            x = y.copy()
            x[r, c] += 1.0
            res = oracle.compare_tiles(t, as_bytes(x), as_bytes(y))
            hit = (r // tr) * ntc + c // tc
            assert [q["mismatches"] for q in res] == [1 if i == hit else 0 for i in range(len(res))]
            assert res[hit]["first_mismatch"] == r * cols + c
            assert all(q["first_mismatch"] == -1 for i, q in enumerate(res) if i != hit)


def test_pitch_padding_never_counts():
    rows, cols, pitch = 9, 10, 24
    y = dense(rows, cols, pitch, 4)
    x = y.copy()
    x[:, cols:] = 7.0       # the candidate's padding holds other values (the reference's is NaN)
    t = W.Tiles("f32", rows, cols, 0, 0, cand_pitch=pitch, ref_pitch=pitch, tile_rows=4, tile_cols=3)
    res = oracle.compare_tiles(t, as_bytes(x), as_bytes(y))
    assert all(r["pass"] and r["mismatches"] == 0 for r in res)
    assert sum(r["n_finite"] for r in res) == rows * cols
    # different pitches per operand: the same values, laid out differently
    xd = np.ascontiguousarray(y[:, :cols])
    t2 = W.Tiles("f32", rows, cols, 0, 0, cand_pitch=cols, ref_pitch=pitch, tile_rows=2, tile_cols=5)
    assert all(r["pass"] for r in oracle.compare_tiles(t2, as_bytes(xd), as_bytes(y)))


def test_row_tiles_equal_per_row_segments():
    rows, cols = 12, 33
    y = dense(rows, cols, cols, 5)
    x = y + np.random.default_rng(6).normal(0, 1e-4, size=y.shape).astype(np.float32)
    t = W.Tiles("f32", rows, cols, 0, 0, tile_rows=1, tile_cols=cols, atol=1e-4, rtol=1e-4)
    res = oracle.compare_tiles(t, as_bytes(x), as_bytes(y))
    pairs = [W.Pair("f32", cols, r * cols * F32, r * cols * F32, 1e-4, 1e-4) for r in range(rows)]
    want = oracle.compare(pairs, as_bytes(x), as_bytes(y))
    for r, (g, w) in enumerate(zip(res, want)):
        for k in ("mismatches", "n_finite", "max_abs", "max_rel", "rms", "pass"):
            assert g[k] == w[k]
        assert g["first_mismatch"] == (-1 if w["first_mismatch"] < 0 else r * cols + w["first_mismatch"])


def test_ragged_edges_and_integers():
    rows, cols = 10, 13
    y = np.arange(rows * cols, dtype=np.int64).reshape(rows, cols) - 60
    x = y.copy()
    x[9, 12] = np.iinfo(np.int64).min
    t = W.Tiles("i64", rows, cols, 0, 0, tile_rows=4, tile_cols=5)
    res = oracle.compare_tiles(t, as_bytes(x), as_bytes(y))
    assert [r["n_finite"] for r in res] == [20, 20, 12, 20, 20, 12, 10, 10, 6]
    assert res[-1]["mismatches"] == 1 and res[-1]["first_mismatch"] == 9 * cols + 12
    assert res[-1]["max_abs_u64"] == 69 + 2 ** 63  # |y - INT64_MIN| with y = 9 * 13 + 12 - 60 = 69
