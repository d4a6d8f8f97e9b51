"""Capture into CUDA graphs: a generator plan followed by a compare plan
(many segments, chained launches) and a progressive ladder, captured once
and replayed, write exactly what the direct calls write."""
import pytest

import paper_2609_00058_gb300 as sv
import workloads as W
from gpu_util import device

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    return device()


def _capture(step, dev):
    import torch
    s = torch.cuda.Stream(dev)
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):  # warm-up outside the capture (first-use allocations, caches)
        step()
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        step()
    return g


def test_plans_replay_in_a_graph(dev):
    import torch
    wl = W.segmented_cases(n_cases=300, max_n=20000, seed=9)
    arena = torch.zeros(wl.arena_bytes, dtype=torch.uint8, device=dev)
    gens = [sv.GeneratePlan(sv.SpecTable(c), wl.arena_bytes, device=dev) for c in wl.gen_calls]
    plan = sv.ComparePlan(sv.PairTable(wl.pairs), wl.arena_bytes, wl.arena_bytes, device=dev)
    res = torch.empty(len(wl.pairs) * sv.RESULT_BYTES, dtype=torch.uint8, device=dev)

    def step():
        for g in gens:
            g(arena)
        plan(arena, arena, results=res)

    step()
    torch.cuda.synchronize()
    want_arena, want_res = arena.clone(), res.clone()
    g = _capture(step, dev)
    for _ in range(2):
        arena.zero_()
        res.zero_()
        g.replay()
        torch.cuda.synchronize()
        assert torch.equal(arena, want_arena) and torch.equal(res, want_res)


def test_progressive_replays_in_a_graph(dev):
    import torch
    wl = W.progressive_ladder((10, 14, 18, 20), deviate_stage=2, special_rate=1e-3)
    arena = torch.zeros(wl.arena_bytes, dtype=torch.uint8, device=dev)
    for c in wl.gen_calls:
        sv.generate(c, arena)
    pt = sv.PairTable(wl.pairs, progressive=True)
    res = torch.empty(len(wl.pairs) * sv.RESULT_BYTES, dtype=torch.uint8, device=dev)
    ff = torch.empty(1, dtype=torch.int32, device=dev)
    ws = torch.empty(pt.ws_bytes + 256, dtype=torch.uint8, device=dev)

    def step():
        sv.progressive(pt, arena, arena, results=res, first_failed=ff, workspace=ws)

    step()
    torch.cuda.synchronize()
    want_res, want_ff = res.clone(), int(ff.item())
    assert want_ff == 2
    g = _capture(step, dev)
    res.zero_()
    ff.fill_(-7)
    g.replay()
    torch.cuda.synchronize()
    assert torch.equal(res, want_res) and int(ff.item()) == want_ff
