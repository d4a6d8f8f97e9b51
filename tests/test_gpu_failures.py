"""Failure handling without a GPU fault: the library's test hook makes the next
launches fail with an invalid launch configuration (nothing runs, the context
stays usable), so each entry point's error path is exercised: it returns
SV_ECUDA, the binding raises, and the next call works and is correct.
"""
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


@pytest.fixture(autouse=True)
def no_pending_failures():
    yield
    sv.lib().sv_debug_fail_launches(0)


def _expect_ecuda(fn):
    with pytest.raises(sv.SynVerifyError) as e:
        fn()
    assert e.value.status == -5


def test_generate_fails_loudly_then_recovers(dev):
    import torch
    spec = W.GenSpec("f32", "normal", 10007, seed=2, stream=1, ref_offset=0, cand_offset=40192, p0=5.0, p1=10.0,
                     specials=("nan",), special_rate=0.01, pcount=W.Perturb("count_add", stream=2, count=3, value=1.0))
    a = torch.zeros(2 * 40192, dtype=torch.uint8, device=dev)
    assert sv.lib().sv_debug_fail_launches(1) == 0
    _expect_ecuda(lambda: sv.generate([spec], a))
    torch.cuda.synchronize()  # nothing ran, nothing is pending
    sv.generate([spec], a)
    h = np.zeros(a.numel(), np.uint8)
    oracle.generate([spec], h)
    g = a.cpu().numpy()
    gf, hf = g[:40028].view(np.float32), h[:40028].view(np.float32)
    assert np.array_equal(np.isnan(gf), np.isnan(hf))


def test_compare_and_progressive_fail_loudly_then_recover(dev):
    pairs = [W.Pair("f32", 5000, 0, 0, 1e-5, 1e-5), W.Pair("i32", 3000, 20480, 20480)]
    cand, ref = W.random_pair_arrays("f32", 5000, seed=3, mismatch_frac=1e-2)
    c = np.zeros(40960, np.uint8)
    r = np.zeros(40960, np.uint8)
    c[:cand.size], r[:ref.size] = cand, ref
    ci, ri = W.random_pair_arrays("i32", 3000, seed=4, mismatch_frac=1e-2)
    c[20480:20480 + ci.size], r[20480:20480 + ri.size] = ci, ri
    dc, dr = to_dev(c, dev), to_dev(r, dev)
    want = oracle.compare(pairs, c, r)
    for n_fail in (1, 2, 3):  # pending failures: the call's first launch fails, the rest are cancelled
        sv.lib().sv_debug_fail_launches(n_fail)
        _expect_ecuda(lambda: sv.compare(pairs, dc, dr))
        sv.lib().sv_debug_fail_launches(0)
        assert_results_match(sv.decode_results(sv.compare(pairs, dc, dr), 2), want, "after a failed call")
    stages = [W.Pair("f32", 1000, 0, 0, 1e-5, 1e-5), W.Pair("f32", 5000, 0, 0, 1e-5, 1e-5)]
    want_s, want_ff = oracle.progressive(stages, c, r)
    sv.lib().sv_debug_fail_launches(1)
    _expect_ecuda(lambda: sv.progressive(stages, dc, dr))
    res, ff = sv.progressive(stages, dc, dr)
    assert int(ff.item()) == want_ff
    assert_results_match(sv.decode_results(res, 2), want_s, "progressive after a failed call")


def test_box_muller_entry_fails_loudly(dev):
    import torch
    w = torch.arange(64, dtype=torch.int32, device=dev)
    sv.lib().sv_debug_fail_launches(1)
    _expect_ecuda(lambda: sv.box_muller(w))
    z = sv.box_muller(w).cpu().numpy()
    assert np.abs(z - oracle.box_muller(np.arange(64, dtype=np.uint32))).max() < 1e-5  # within a few ulp
