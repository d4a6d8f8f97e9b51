"""The Box-Muller polynomial coefficients and constant splits in the kernel
header are the ones fit_box_muller.py derives (Lawson minimax fits of the
sin, cos and ln corrections), and the fits are as accurate as stated."""
import importlib.util
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2609_00058_gb300", "csrc")


def _fit_module():
    spec = importlib.util.spec_from_file_location("fit_box_muller", os.path.join(CSRC, "fit_box_muller.py"))
    m = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(m)
    return m


@pytest.fixture(scope="module")
def k():
    return _fit_module().coefficients()


def test_header_constants_come_from_the_fit(k):
    src = open(os.path.join(CSRC, "sv_device.cuh")).read()
    got = {name: float(v) for name, v in re.findall(r"constexpr float kBm(\w+) = ([-+0-9.e]+)f;", src)}
    want = {}
    for name in ("T", "P", "R"):
        for i, v in enumerate(k[name]):
            want["%s%d" % (name, i)] = v
    for name in ("LN2_HI", "LN2_LO", "PI_HI", "PI_LO"):
        want[name.replace("_", "")] = k[name]
    assert set(got) == set(want)
    for name, v in want.items():
        assert np.float32(got[name]) == np.float32(v), name
    # the approximation errors are far below an fp32 ulp (2^-24 relative)
    assert max(k["errors"]) < 2 ** -24 / 10


def test_constant_splits_are_exact_where_it_matters(k):
    # e * LN2_HI is exact for |e| <= 25 (the exponents of u1 in [2^-24, 1])
    hi = np.float32(k["LN2_HI"])
    for e in range(-25, 26):
        assert float(np.float32(e) * hi) == e * float(hi)
    assert abs(float(hi) + float(np.float32(k["LN2_LO"])) - np.log(2.0)) < 1e-13
    assert abs(float(np.float32(k["PI_HI"])) + float(np.float32(k["PI_LO"])) - np.pi) < 1e-14
