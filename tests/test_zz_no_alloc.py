"""verify_compare_noalloc through the C ABI, against verify_compare and the
CPU oracle.

The allocation-free entry point serves callers that cannot allocate device
memory (their process's GPU memory belongs to another component, or their
path must not pay for an allocation): they pass only inputs and outputs and
the library uses a fixed scratch array in its own device memory.  Its
verdicts must equal those of verify_compare (which takes a caller
workspace) and those of the CPU oracle on the same bytes, within the
tolerance the other parity tests use: every integer field and the max
statistics exactly, RMS within 1e-6 relative.  Two calls in
a row check that the shared scratch left by one call does not leak into the
next.  This file is collected last so that a run stopping at the first
failure has already run every other test; it also passes alone in a fresh
process (the first call on the device performs the scratch-address lookup).
"""
import ctypes as C

import numpy as np
import pytest

import paper_2609_00058_gb300 as sv
import workloads as W
from gpu_util import assert_results_match, device, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    return device()


def _case(seed, specs):
    ar = W.Arena()
    placed = [(dt, n, ar.take(max(n, 1) * W.DTYPE_BYTES[dt])) for dt, n in specs]
    cand = np.zeros(ar.size, np.uint8)
    ref = np.zeros(ar.size, np.uint8)
    pairs = []
    for i, (dt, n, off) in enumerate(placed):
        if n:
            c, r = W.random_pair_arrays(dt, n, seed=seed + i, mismatch_frac=3e-3, nonfinite_frac=1e-3)
            cand[off:off + c.size] = c
            ref[off:off + r.size] = r
        pairs.append(W.Pair(dt, n, off, off, 1e-3, 1e-3))
    return pairs, cand, ref


def _noalloc(pairs, dcand, dref, results, stream):
    tab = sv.PairTable(pairs)
    return sv.lib().verify_compare_noalloc(tab.arr, tab.n, dcand.data_ptr(), dcand.numel(), dref.data_ptr(),
                                           dref.numel(), results.data_ptr(), stream)


def test_noalloc_matches_workspace_compare_on_two_calls(dev, oracle):
    import torch
    stream = torch.cuda.current_stream().cuda_stream
    cases = [
        _case(100, [("f32", 300007), ("bf16", 65537), ("i64", 4099), ("f16", 7), ("u32", 1), ("f32", 0)]),
        _case(200, [("f32", 1 << 22), ("i32", 5000), ("bf16", 3), ("f16", 20000), ("i64", 1 << 16),
                    ("u32", 12345), ("f32", 17), ("bf16", 1 << 18)]),
    ]
    for pairs, cand, ref in cases:  # two calls in a row, different shapes
        dc, dr = to_dev(cand, dev), to_dev(ref, dev)
        want = sv.decode_results(sv.compare(pairs, dc, dr), len(pairs))
        results = torch.full((len(pairs) * sv.RESULT_BYTES,), 0xAB, dtype=torch.uint8, device=dev)
        assert _noalloc(pairs, dc, dr, results, stream) == 0
        got = sv.decode_results(results, len(pairs))
        assert_results_match(got, want, "noalloc vs verify_compare")
        assert_results_match(got, oracle.compare(pairs, cand, ref), "noalloc vs oracle")
    # and the same call twice on the same buffers
    pairs, cand, ref = cases[0]
    dc, dr = to_dev(cand, dev), to_dev(ref, dev)
    first = torch.empty(len(pairs) * sv.RESULT_BYTES, dtype=torch.uint8, device=dev)
    second = torch.empty_like(first)
    assert _noalloc(pairs, dc, dr, first, stream) == 0
    assert _noalloc(pairs, dc, dr, second, stream) == 0
    assert sv.decode_results(first, len(pairs)) == sv.decode_results(second, len(pairs))


def test_noalloc_rejects_calls_beyond_its_scratch(dev):
    lib = sv.lib()
    big = 1 << 34  # sizes are validated before any pointer is used
    nine = sv.PairTable([W.Pair("f32", 16, 0, 0)] * 9)
    assert lib.verify_compare_noalloc(nine.arr, 9, 0x1000, big, 0x1000, big, 0x2000, None) == -3
    # one large pair of any size fits (4096 + 1 slots) ...
    one = sv.PairTable([W.Pair("f32", 1 << 30, 0, 0)])
    assert lib.sv_check_pairs(one.arr, 1, big, big) == 0
    # ... two large pairs of different dtypes do not (8194 slots > 4104)
    two = sv.PairTable([W.Pair("f32", 1 << 30, 0, 0), W.Pair("bf16", 1 << 30, 0, 0)])
    assert lib.verify_compare_noalloc(two.arr, 2, 0x1000, big, 0x1000, big, 0x2000, None) == -3
    assert b"size beyond" in lib.sv_strerror(-3)
    assert C.sizeof(sv.vc_result) == 80
