"""Brute force over 16-bit encodings: the GPU compare against the oracle on
every fp16 / bf16 candidate encoding paired with every 64th reference
encoding, and every reference encoding paired with every 64th candidate
encoding (2 x 67,108,864 pairs per case), for three tolerance sets.  One
segment per fixed operand value, so each of its 65,536 elements meets every
encoding of the other side; all statistics of every segment must match."""
import numpy as np
import pytest

import oracle
import workloads as W
import paper_2609_00058_gb300 as sv
from gpu_util import assert_results_match, device, to_dev

pytestmark = pytest.mark.gpu
ALL = np.arange(1 << 16, dtype=np.uint32).astype(np.uint16)
STRIDE = 64


@pytest.fixture(scope="module")
def dev():
    return device()


@pytest.mark.parametrize("dtype", ["f16", "bf16"])
@pytest.mark.parametrize("atol,rtol", [(1e-3, 1e-3), (0.0, 0.0), (1e-2, 0.0)])
@pytest.mark.parametrize("sweep", ["candidate", "reference"])
def test_all_encodings(dev, dtype, atol, rtol, sweep):
    fixed = ALL[7::STRIDE]  # 1024 values of the other side, a spread over every exponent and sign
    every = np.tile(ALL, fixed.size)
    const = np.repeat(fixed, ALL.size)
    cand, ref = (every, const) if sweep == "candidate" else (const, every)
    seg = ALL.size * 2
    pairs = [W.Pair(dtype, ALL.size, i * seg, i * seg, atol, rtol) for i in range(fixed.size)]
    c8, r8 = cand.view(np.uint8), ref.view(np.uint8)
    want = oracle.compare(pairs, c8, r8)
    got = sv.decode_results(sv.compare(pairs, to_dev(c8, dev), to_dev(r8, dev)), len(pairs))
    assert_results_match(got, want, "%s %s atol=%g rtol=%g" % (dtype, sweep, atol, rtol))
    assert sum(w["nan_disagree"] for w in want) > 0 and sum(w["inf_disagree"] for w in want) > 0
