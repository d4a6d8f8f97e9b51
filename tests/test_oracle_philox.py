"""Pins of the oracle's Philox-4x32-10 against an independent implementation.

The counter-based generator is Philox-4x32-10 (Salmon et al., SC'11).  The
oracle's implementation is checked against PyTorch's own Philox engine
(ATen/core/PhiloxRNGEngine.h, compiled here from its source and run), whose
state maps onto ours as: key = seed (lo, hi); counter = (offset lo, offset hi,
subsequence lo, subsequence hi).  Our draw for (seed, stream, purpose, block)
is counter (block lo, block hi, stream, purpose), i.e. offset = block and
subsequence = stream | purpose << 32.
"""
import os
import subprocess
import tempfile

import numpy as np
import pytest

PROBE = r"""
#include <ATen/core/PhiloxRNGEngine.h>
#include <cstdio>
int main() {
  unsigned long long seed, sub, off;
  while (std::scanf("%llu %llu %llu", &seed, &sub, &off) == 3) {
    at::philox_engine e(seed, sub, off);
    unsigned a = e(), b = e(), c = e(), d = e();
    std::printf("%u %u %u %u\n", a, b, c, d);
  }
  return 0;
}
"""


def _torch_include_dirs():
    import torch
    base = os.path.join(os.path.dirname(torch.__file__), "include")
    hdr = os.path.join(base, "ATen", "core", "PhiloxRNGEngine.h")
    if not os.path.exists(hdr):
        pytest.skip("PyTorch Philox engine header not available")
    return [base, os.path.join(base, "torch", "csrc", "api", "include")]


@pytest.fixture(scope="module")
def torch_philox():
    incs = _torch_include_dirs()
    d = tempfile.mkdtemp(prefix="philox_probe_")
    src, exe = os.path.join(d, "p.cpp"), os.path.join(d, "p")
    with open(src, "w") as f:
        f.write(PROBE)
    subprocess.check_call(["g++", "-O1", "-std=c++17", *["-I" + i for i in incs], src, "-o", exe])

    def run(triples):
        inp = "".join("%d %d %d\n" % t for t in triples)
        out = subprocess.run([exe], input=inp, capture_output=True, text=True, check=True).stdout
        return [list(map(int, line.split())) for line in out.strip().splitlines()]
    return run


def _cases():
    rng = np.random.default_rng(20260101)
    cases = [(0, 0, 0, 0), (2**64 - 1, 2**32 - 1, 2**32 - 1, 2**64 - 1), (1, 0, 0, 1), (7, 3, 0, 0),
             (7, 3, 1, 5), (5, 0, 6, 2), (0x0123456789ABCDEF, 17, 2, 2**40 + 3)]
    for _ in range(200):
        cases.append((int(rng.integers(0, 2**63)) * 2 + int(rng.integers(0, 2)),
                      int(rng.integers(0, 2**32)), int(rng.integers(0, 8)), int(rng.integers(0, 2**62))))
    return cases


def test_philox_matches_pytorch_engine(oracle, torch_philox):
    cases = _cases()
    triples = [(seed, stream | (purpose << 32), block) for seed, stream, purpose, block in cases]
    ref = torch_philox(triples)
    names = {v: k for k, v in oracle.PURPOSES.items()}
    for (seed, stream, purpose, block), want in zip(cases, ref):
        ctr = [block & 0xFFFFFFFF, block >> 32, stream, purpose]
        key = [seed & 0xFFFFFFFF, seed >> 32]
        assert oracle.philox(ctr, key) == want, (seed, stream, purpose, block)
        if purpose in names:
            assert oracle.draw(seed, stream, names[purpose], block) == want


def test_philox_raw_counter_key_layout(oracle, torch_philox):
    # the raw entry point: counter words and key words in their natural order
    ctr, key = [0x11111111, 0x22222222, 0x33333333, 0x44444444], [0xA5A5A5A5, 0x5A5A5A5A]
    seed = key[0] | (key[1] << 32)
    sub = ctr[2] | (ctr[3] << 32)
    off = ctr[0] | (ctr[1] << 32)
    assert oracle.philox(ctr, key) == torch_philox([(seed, sub, off)])[0]


def test_philox_distinct_purposes_decorrelate(oracle):
    # different purpose words give different blocks (no accidental aliasing)
    blocks = {tuple(oracle.draw(9, 0, p, 0)) for p in oracle.PURPOSES}
    assert len(blocks) == len(oracle.PURPOSES)


def test_philox_word_bits_unbiased(oracle):
    # each output bit of 4096 consecutive blocks is set about half the time
    w = np.array([oracle.draw(3, 1, "value", b) for b in range(4096)], dtype=np.uint64).ravel()
    bits = ((w[:, None] >> np.arange(32, dtype=np.uint64)) & 1).mean(axis=0)
    # 16384 words: sd of a bit frequency = 0.5/128 ~ 0.0039; allow 5 sd
    assert np.all(np.abs(bits - 0.5) < 0.02)
