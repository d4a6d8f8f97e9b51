"""Guard bytes: every byte a call may not write keeps its canary value.

Output arrays of many kinds and ragged sizes sit in an arena between gaps
filled with a canary pattern; after syn_generate the gaps, and after the
compare calls the results buffer's spare records and the workspace's tail,
must be unchanged.  A kernel that wrote past a segment, a quantum or a
partial record would show here even where the written values look right.
"""
import numpy as np
import pytest

import paper_2609_00058_gb300 as sv
import workloads as W
from gpu_util import device

pytestmark = pytest.mark.gpu
CANARY = 0xA5


@pytest.fixture(scope="module")
def dev():
    return device()


KINDS = [
    dict(dtype="f32", dist="uniform", p0=-1.0, p1=1.0, specials=("nan", "dup"), special_rate=0.02),
    dict(dtype="bf16", dist="normal", p0=5.0, p1=10.0, pelem=W.Perturb("rel_noise", stream=3, value=2.0 ** -9)),
    dict(dtype="f16", dist="uniform", p0=-8.0, p1=8.0, pcount=W.Perturb("count_set", stream=4, count=2, value=0.0)),
    dict(dtype="i32", dist="int_range", i0=-50, i1=50, pelem=W.Perturb("rate_add_pm", stream=3, rate=0.05, ivalue=1)),
    dict(dtype="u32", dist="raw_bits"),
    dict(dtype="i64", dist="permutation", specials=("imax",), special_rate=0.01,
         pcount=W.Perturb("swap_pairs", stream=4, count=3)),
    dict(dtype="i64", dist="constant", i0=-3),
]
SIZES = [1, 2, 3, 5, 7, 13, 255, 1001, 8191, 8193, 40001]


def _layout(seed):
    rng = np.random.default_rng(seed)
    off, specs, outs = 256, [], []
    for i, n in enumerate(SIZES * 2):
        kw = dict(KINDS[(i + seed) % len(KINDS)])
        if n < 8:  # too few elements for the exact-count strata
            kw.pop("pcount", None)
        sz = W.DTYPE_BYTES[kw["dtype"]]
        ref = off
        off = (off + n * sz + 256 + int(rng.integers(0, 4)) * 16 + 15) // 16 * 16
        cand = off
        off = (off + n * sz + 256 + 15) // 16 * 16
        specs.append(W.GenSpec(n=n, seed=seed + i, stream=i, ref_offset=ref, cand_offset=cand, **kw))
        outs += [(ref, n * sz), (cand, n * sz)]
    return specs, outs, off + 256


@pytest.mark.parametrize("seed", [1, 2])
def test_generate_writes_nothing_outside_its_outputs(dev, seed):
    import torch
    specs, outs, size = _layout(seed)
    assert sv.check_specs(specs, size) == 0
    a = torch.full((size,), CANARY, dtype=torch.uint8, device=dev)
    sv.generate(specs, a)
    h = a.cpu().numpy()
    mask = np.ones(size, bool)
    for off, nb in outs:
        mask[off: off + nb] = False
    assert np.all(h[mask] == CANARY)


def test_compare_writes_nothing_outside_results_and_workspace(dev):
    import torch
    specs, outs, size = _layout(3)
    a = torch.zeros(size, dtype=torch.uint8, device=dev)
    sv.generate(specs, a)
    pairs = [W.Pair(s.dtype, s.n, s.cand_offset, s.ref_offset, 1e-3, 1e-3) for s in specs]
    tab = sv.PairTable(pairs)
    spare = 4 * sv.RESULT_BYTES
    results = torch.full((len(pairs) * sv.RESULT_BYTES + spare,), CANARY, dtype=torch.uint8, device=dev)
    ws = torch.full((tab.ws_bytes + 4096,), CANARY, dtype=torch.uint8, device=dev)
    sv.compare(tab, a, a, results=results, workspace=ws[: tab.ws_bytes])
    assert np.all(results[len(pairs) * sv.RESULT_BYTES:].cpu().numpy() == CANARY)
    assert np.all(ws[tab.ws_bytes:].cpu().numpy() == CANARY)
    got = sv.decode_results(results, len(pairs))
    assert all(g["state"] == sv.STAGE_RUN for g in got)
    # the twins differ from the clean outputs only where a perturbation applies
    for s, g in zip(specs, got):
        if s.pelem.kind == "none" and s.pcount.kind == "none":
            assert g["mismatches"] == 0, s
