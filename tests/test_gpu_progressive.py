"""GPU parity of verify_progressive (progressive multi-stage validation,
CUDA-Harness Sec. 4.2.2, fail-fast order) against the CPU oracle."""
import numpy as np
import pytest

import oracle
import paper_2609_00058_gb300 as sv
import workloads as W
from gpu_util import assert_results_match, device, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    return device()


@pytest.mark.parametrize("deviate", [None, 0, 2, 4])
def test_ladder_on_oracle_bytes(dev, deviate):
    wl = W.progressive_ladder((10, 12, 14, 16, 18), deviate_stage=deviate, special_rate=1e-3)
    h = np.zeros(wl.arena_bytes, np.uint8)
    for call in wl.gen_calls:
        oracle.generate(call, h)
    want, want_ff = oracle.progressive(wl.pairs, h, h)
    a = to_dev(h, dev)
    res, ff = sv.progressive(wl.pairs, a, a)
    got = sv.decode_results(res, len(wl.pairs))
    assert int(ff.item()) == want_ff == (-1 if deviate is None else deviate)
    assert_results_match(got, want, "ladder")


def test_ladder_generated_on_gpu_has_closed_form_verdict(dev):
    # the GPU's own synthesis feeding its own ladder: stage 3 fails at the
    # index the oracle's stratum map names, later stages are skipped
    import torch
    wl = W.progressive_ladder((10, 14, 18, 20, 22), deviate_stage=3, special_rate=1e-4)
    a = torch.zeros(wl.arena_bytes, dtype=torch.uint8, device=dev)
    sv.generate(wl.gen_calls[0], a)
    res, ff = sv.progressive(wl.pairs, a, a)
    got = sv.decode_results(res, len(wl.pairs))
    assert int(ff.item()) == 3
    assert [g["state"] for g in got] == [1, 1, 1, 1, 2]
    assert [g["mismatches"] for g in got[:4]] == [0, 0, 0, 1]
    n3 = 1 << 20
    spec3 = wl.gen_calls[0][3]
    assert got[3]["first_mismatch"] == oracle.stratum_index(n3, 1, spec3.seed, spec3.pcount.stream, 0)


def test_mixed_dtype_stages_and_repeat(dev):
    # the flag is re-armed by every call
    n = 5000
    c16, r16 = W.random_pair_arrays("f16", n, seed=1, mismatch_frac=0.0, nonfinite_frac=0.0)
    ci, ri = W.random_pair_arrays("i64", n, seed=2, mismatch_frac=1e-3)
    cand = np.concatenate([c16, np.zeros(16, np.uint8), ci])
    ref = np.concatenate([r16, np.zeros(16, np.uint8), ri])
    stages = [W.Pair("f16", n, 0, 0, 1e-3, 1e-3), W.Pair("i64", n, 10016, 10016)]
    want, want_ff = oracle.progressive(stages, cand, ref)
    dc, dr = to_dev(cand, dev), to_dev(ref, dev)
    for _ in range(2):
        res, ff = sv.progressive(stages, dc, dr)
        assert want_ff == 1
        assert int(ff.item()) == want_ff
        assert_results_match(sv.decode_results(res, 2), want)
    res, ff = sv.progressive(stages[:1], dc, dr)
    assert int(ff.item()) == -1


def test_empty_ladder_and_empty_stage(dev):
    import torch
    a = torch.zeros(256, dtype=torch.uint8, device=dev)
    _, ff = sv.progressive([], a, a)
    assert int(ff.item()) == -1
    res, ff = sv.progressive([W.Pair("f32", 0, 0, 0)], a, a)
    g = sv.decode_results(res, 1)[0]
    assert int(ff.item()) == -1 and g["pass"] == 1 and g["state"] == 1 and g["first_mismatch"] == -1


def test_library_counts_its_own_launches(dev):
    # one generator launch for a one-kind batch (its sparse exact-count edit is
    # applied in the generating CTAs), then one compare and one ordered
    # combine per stage group of the ladder (five small fp32 stages: one group)
    import torch
    wl = W.progressive_ladder((10, 12, 14, 16, 18), deviate_stage=2, special_rate=1e-3)
    a = torch.zeros(wl.arena_bytes, dtype=torch.uint8, device=dev)
    lib = sv.lib()
    n0 = lib.sv_kernel_launches()
    sv.generate(wl.gen_calls[0], a)
    n1 = lib.sv_kernel_launches()
    res, ff = sv.progressive(wl.pairs, a, a)
    n2 = lib.sv_kernel_launches()
    assert (n1 - n0, n2 - n1) == (1, 2)
    assert int(ff.item()) == 2
    # two pairs of different dtypes: a compare per dtype and one combine
    pairs = [W.Pair("f32", 1000, 0, 0), W.Pair("i32", 1000, 4096, 4096)]
    n3 = lib.sv_kernel_launches()
    sv.compare(pairs, a, a)
    assert lib.sv_kernel_launches() - n3 == 3
