"""Helpers shared by the GPU parity tests (no method arithmetic here)."""
import numpy as np
import pytest

FIELDS_EXACT = ("mismatches", "nan_disagree", "inf_disagree", "n_finite", "first_mismatch", "max_abs_u64",
                "max_abs", "pass", "state")
RMS_RTOL = 1e-6  # RMS error: within 1e-6 relative of the oracle's fp64 value


def device():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    return torch.device("cuda:0")


def to_dev(arr, dev):
    import torch
    return torch.from_numpy(np.ascontiguousarray(arr).view(np.uint8).copy()).to(dev)


def assert_results_match(got, want, ctx="", max_rel_exact=True):
    assert len(got) == len(want)
    for i, (g, w) in enumerate(zip(got, want)):
        for k in FIELDS_EXACT:
            assert g[k] == w[k], "%s pair %d field %s: gpu %r oracle %r" % (ctx, i, k, g[k], w[k])
        if max_rel_exact:
            assert g["max_rel"] == w["max_rel"], "%s pair %d max_rel %r vs %r" % (ctx, i, g["max_rel"], w["max_rel"])
        else:
            assert g["max_rel"] == pytest.approx(w["max_rel"], rel=1e-6)
        if np.isfinite(w["rms"]):
            assert g["rms"] == pytest.approx(w["rms"], rel=RMS_RTOL, abs=0.0), "%s pair %d rms" % (ctx, i)
        else:
            assert g["rms"] == w["rms"] or (np.isnan(g["rms"]) and np.isnan(w["rms"]))


def ordered_f32(bits):
    """fp32 bit patterns -> integers in value order (ulp distance = difference)."""
    b = np.asarray(bits, dtype=np.uint32).astype(np.int64)
    return np.where(b >= 0x80000000, 0x80000000 - b, b)


def ordered_16(bits, dtype):
    b = np.asarray(bits, dtype=np.uint16).astype(np.int64)
    return np.where(b >= 0x8000, 0x8000 - b, b)
