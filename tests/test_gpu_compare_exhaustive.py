"""Brute force over 16-bit encodings: the GPU compare (Eq. 1) against the
oracle on ALL 2^32 (candidate, reference) pairs of fp16 and of bf16
encodings, for three tolerance sets.

Layout: 65,536 segments of 65,536 elements.  Segment s pairs candidate
encoding i with reference encoding (i + s) mod 2^16 for every i, so the
segments together hold every pair exactly once.  The candidate operand is
one array of all encodings (every segment starts at offset 0); the reference
operand is eight copies of the encodings, two periods long, copy k rotated by
k, so segment s reads copy s mod 8 from element s - s mod 8 (a 16-byte
aligned offset).  Every statistic of every segment must match the oracle's
on the same bytes (its multi-threaded driver: one job per segment)."""
import numpy as np
import pytest

import oracle
import workloads as W
import paper_2609_00058_gb300 as sv
from gpu_util import assert_results_match, device, to_dev

pytestmark = pytest.mark.gpu
N = 1 << 16
COPY = 2 * N  # elements of one rotated reference copy


@pytest.fixture(scope="module")
def dev():
    return device()


def layout(dtype, atol, rtol):
    cand = np.arange(N, dtype=np.uint32).astype(np.uint16)
    j = np.arange(COPY, dtype=np.uint32)
    ref = np.concatenate([((j + k) % N).astype(np.uint16) for k in range(8)])
    pairs = []
    for s in range(N):
        k, m = s % 8, s - s % 8
        pairs.append(W.Pair(dtype, N, 0, 2 * (k * COPY + m), atol, rtol))
    return pairs, cand.view(np.uint8), ref.view(np.uint8)


def test_layout_covers_every_pair_once():
    _, c8, r8 = layout("f16", 0.0, 0.0)
    c, r = c8.view(np.uint16), r8.view(np.uint16)
    for s in (0, 1, 7, 8, 9, 4095, 65535):
        k, m = s % 8, s - s % 8
        y = r[k * COPY + m: k * COPY + m + N].astype(np.int64)
        assert np.array_equal(y, (np.arange(N) + s) % N)
        assert np.array_equal(c.astype(np.int64), np.arange(N))


@pytest.mark.parametrize("dtype", ["f16", "bf16"])
@pytest.mark.parametrize("atol,rtol", [(1e-3, 1e-3), (0.0, 0.0), (1e-2, 0.0)])
def test_all_encoding_pairs(dev, dtype, atol, rtol):
    pairs, c8, r8 = layout(dtype, atol, rtol)
    want = oracle.compare(pairs, c8, r8, threads=0)
    got = sv.decode_results(sv.compare(pairs, to_dev(c8, dev), to_dev(r8, dev)), len(pairs))
    assert_results_match(got, want, "%s atol=%g rtol=%g" % (dtype, atol, rtol))
    assert sum(w["nan_disagree"] for w in want) > 0 and sum(w["inf_disagree"] for w in want) > 0
    assert sum(w["mismatches"] for w in want) > 0 and sum(w["n_finite"] for w in want) > (1 << 31)
