"""Parity at the five workloads' full sizes, through the same calls bench.py
times (syn_generate on the workload's spec tables, then verify_compare or
verify_progressive on the arena).

Where the oracle can follow the whole workload in seconds (the fp32 pair, the
segmented cases, the stages the ladder actually verifies) it does, and the
GPU must match it as in the small-size tests.  Otherwise the oracle computes
sampled elements one by one (synthesis), the compare runs on neutral seeded
arrays of the full size that both sides read (verification), and properties
that hold at any size are checked on the GPU's own output.
"""
import numpy as np
import pytest

import oracle
import paper_2609_00058_gb300 as sv
import workloads as W
from gpu_util import assert_results_match, device, ordered_16, ordered_f32, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    return device()


def gpu_run(wl, dev):
    import torch
    arena = torch.zeros(wl.arena_bytes, dtype=torch.uint8, device=dev)
    for call in wl.gen_calls:
        sv.generate(sv.SpecTable(call), arena)
    if wl.progressive:
        res, ff = sv.progressive(sv.PairTable(wl.pairs, progressive=True), arena, arena)
        out = sv.decode_results(res, len(wl.pairs)), int(ff.item())
    else:
        out = sv.decode_results(sv.compare(sv.PairTable(wl.pairs), arena, arena), len(wl.pairs)), None
    torch.cuda.synchronize()
    return arena, out


def _u(dtype):
    return {2: np.uint16, 4: np.uint32, 8: np.uint64}[W.DTYPE_BYTES[dtype]]


def oracle_verdicts_on(arena_dev, wl):
    """The oracle's verdicts on the GPU's own synthesized bytes (the arena
    copied to the host), through its multi-threaded driver on every core."""
    h = arena_dev.cpu().numpy()
    if wl.progressive:
        return oracle.progressive(wl.pairs, h, h, threads=0)
    return oracle.compare(wl.pairs, h, h, threads=0), None


def sample_indices(n, k, seed):
    rng = np.random.default_rng(seed)
    idx = set(rng.integers(0, n, size=k).tolist())
    idx.update({0, 1, 2, 3, n - 1, n - 2, max(0, n - 5)})
    return sorted(i for i in idx if 0 <= i < n)


def gather(arena_dev, off, dtype, idx):
    """Elements idx of the array at byte offset off, gathered on the device."""
    import torch
    sz = W.DTYPE_BYTES[dtype]
    tt = {2: torch.int16, 4: torch.int32, 8: torch.int64}[sz]
    n = max(idx) + 1
    v = arena_dev[off: off + n * sz].view(tt)
    g = v[torch.as_tensor(idx, device=arena_dev.device)].cpu().numpy()
    return g.view(_u(dtype))


def check_sampled(arena_dev, spec, host_arena, idx, exact):
    """GPU values at sampled indices against the oracle's per-index values."""
    for role, off in ((0, spec.ref_offset), (1, spec.cand_offset)):
        if off is None:
            continue
        g = gather(arena_dev, off, spec.dtype, idx)
        want = np.array([oracle.value_at(spec, host_arena, spec.elem_offset + i, role) for i in idx], dtype=np.uint64)
        if exact:
            assert np.array_equal(g.astype(np.uint64), want), (spec.dist, role)
        elif spec.dtype == "f32":
            w32 = want.astype(np.uint32)
            fin = np.isfinite(w32.view(np.float32))
            assert np.array_equal(g[~fin], w32[~fin])
            assert np.abs(ordered_f32(g[fin]) - ordered_f32(w32[fin])).max(initial=0) <= 4
        else:
            w16 = want.astype(np.uint16)
            assert np.abs(ordered_16(g, spec.dtype) - ordered_16(w16, spec.dtype)).max(initial=0) <= 1


def test_fp32_pair_full(dev):
    wl = W.single_fp32_pair()
    arena, (got, _) = gpu_run(wl, dev)
    h, want, _ = oracle.run_workload(wl)
    assert np.array_equal(arena.cpu().numpy(), h)  # uniform, +-delta, NaN edits: all bit-exact
    assert_results_match(got, want, "fp32 pair")
    # the GPU compare on the oracle's bytes too
    d = to_dev(h, dev)
    assert_results_match(sv.decode_results(sv.compare(wl.pairs, d, d), 1), want)


def test_ladder_full(dev):
    wl = W.progressive_ladder()
    arena, (got, ff) = gpu_run(wl, dev)
    # closed form of the verdict: stage 3 fails at the one edited element, 4-5 skipped
    assert ff == 3
    assert [g["state"] for g in got] == [1, 1, 1, 1, 2, 2]
    assert [g["mismatches"] for g in got[:4]] == [0, 0, 0, 1]
    s3 = wl.gen_calls[0][3]
    assert got[3]["first_mismatch"] == oracle.stratum_index(s3.n, 1, s3.seed, s3.pcount.stream, 0)
    # the oracle's verdicts on the GPU's own bytes
    want_g, want_gff = oracle_verdicts_on(arena, wl)
    assert want_gff == 3
    assert_results_match(got, want_g, "ladder, GPU bytes")
    # sampled synthesis of every stage, including the 2^25 and 2^27 ones
    h0 = np.zeros(16, np.uint8)
    for k, s in enumerate(wl.gen_calls[0]):
        idx = sample_indices(s.n, 3000, 100 + k)
        if s.pcount.kind != "none":
            idx = sorted(set(idx) | {oracle.stratum_index(s.n, 1, s.seed, s.pcount.stream, 0)})
        check_sampled(arena, s, h0, idx, exact=False)
    # the verified stages on the oracle's own bytes (stages 4-5 stay zero: skipped)
    h = np.zeros(wl.arena_bytes, np.uint8)
    oracle.generate(wl.gen_calls[0][:4], h)
    want, want_ff = oracle.progressive(wl.pairs, h, h)
    d = to_dev(h, dev)
    res, gff = sv.progressive(sv.PairTable(wl.pairs, progressive=True), d, d)
    assert int(gff.item()) == want_ff == 3
    assert_results_match(sv.decode_results(res, len(wl.pairs)), want, "ladder")


def test_segmented_full(dev):
    wl = W.segmented_cases()
    arena, (got, _) = gpu_run(wl, dev)
    h, want, _ = oracle.run_workload(wl)
    assert np.array_equal(arena.cpu().numpy(), h)
    assert_results_match(got, want, "segmented")
    hits = sum(1 for s in wl.gen_calls[0] if s.pcount.kind != "none")
    assert sum(1 for g in got if not g["pass"]) == hits


def test_dotlike_full(dev):
    import torch
    wl = W.dotlike_bf16_pair()
    arena, (got, _) = gpu_run(wl, dev)
    # the verdict on the synthesized 2^30 pair equals the oracle's on the same bytes
    assert_results_match(got, oracle_verdicts_on(arena, wl)[0], "dot-like, GPU bytes")
    fa, fb = wl.gen_calls[0]
    d = wl.gen_calls[1][0]
    # the oracle's own factors (2M normals each), uploaded in place of the
    # GPU's: the GPU's dot-like values on them must equal the oracle's bit for bit
    hfac = np.zeros(fb.ref_offset + 4 * fb.n, np.uint8)
    oracle.generate([fa, fb], hfac)
    check_sampled(arena, fa, hfac, sample_indices(fa.n, 4000, 7), exact=False)  # GPU factors: <= 4 ulp
    arena[: hfac.size].copy_(torch.from_numpy(hfac).to(dev))
    sv.generate([d], arena)
    idx = sample_indices(d.n, 4000, 8)
    want = np.array([oracle.value_at(d, hfac, i, 0) for i in idx], dtype=np.uint16)
    assert np.array_equal(gather(arena, d.ref_offset, "bf16", idx), want)
    wantc = np.array([oracle.value_at(d, hfac, i, 1) for i in idx], dtype=np.uint16)
    gc = gather(arena, d.cand_offset, "bf16", idx)
    assert np.abs(ordered_16(gc, "bf16") - ordered_16(wantc, "bf16")).max() <= 1
    # verdict properties: noise of 2^-9 |ref| never exceeds 1e-2 + 1e-2 |ref|
    # except in the far tail; the stats are those of the two arrays
    assert got[0]["n_finite"] == d.n and got[0]["max_rel"] < 2 ** -9 * 6 + 2 ** -7
    # the compare on a full-size neutral bf16 pair that both sides read
    n = d.n
    cand, ref = W.random_bits_pair("bf16", n, seed=44, n_changes=5000)
    pairs = [W.Pair("bf16", n, 0, 0, 1e-2, 1e-2)]
    gres = sv.decode_results(sv.compare(pairs, to_dev(cand, dev), to_dev(ref, dev)), 1)
    assert_results_match(gres, oracle.compare(pairs, cand, ref), "bf16 2^30")


def test_perm_full(dev):
    import torch
    wl = W.int64_permutation_pair()
    arena, (got, _) = gpu_run(wl, dev)
    # the verdict on the synthesized 2^28 pair equals the oracle's on the same bytes
    want_g = oracle_verdicts_on(arena, wl)[0]
    assert_results_match(got, want_g, "permutation, GPU bytes")
    assert want_g[0]["mismatches"] <= 34
    s = wl.gen_calls[0][0]
    idx = sample_indices(s.n, 20000, 9)
    strata = [oracle.stratum_index(s.n, 34, s.seed, s.pcount.stream, k) for k in range(34)]
    check_sampled(arena, s, np.zeros(16, np.uint8), sorted(set(idx) | set(strata)), exact=True)
    # the verdict equals the count of positions where the two GPU arrays differ
    r = arena[s.ref_offset: s.ref_offset + 8 * s.n].view(torch.int64)
    c = arena[s.cand_offset: s.cand_offset + 8 * s.n].view(torch.int64)
    diff = torch.nonzero(r != c).flatten().cpu().numpy()
    assert got[0]["mismatches"] == diff.size <= 34
    assert got[0]["first_mismatch"] == (int(diff[0]) if diff.size else -1)
    assert set(diff.tolist()) <= set(strata)
    # the compare on a full-size neutral int64 pair that both sides read
    n = s.n
    rng = np.random.default_rng(55)
    ref = rng.permutation(n).astype(np.int64)
    cand = ref.copy()
    sw = rng.choice(n, size=34, replace=False)
    cand[sw[0::2]], cand[sw[1::2]] = ref[sw[1::2]], ref[sw[0::2]]
    pairs = [W.Pair("i64", n, 0, 0)]
    gres = sv.decode_results(sv.compare(pairs, to_dev(cand.view(np.uint8), dev), to_dev(ref.view(np.uint8), dev)), 1)
    want = oracle.compare(pairs, cand.view(np.uint8), ref.view(np.uint8))
    assert_results_match(gres, want, "int64 2^28")
    assert want[0]["mismatches"] == 34
