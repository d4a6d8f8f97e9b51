"""One candidate round end to end: compilation tool (Eq. 2), synthesized stage
inputs, reference and candidate runs, fail-fast validation (Sec. 4.2.2 with
Eq. 1), latency performance (Eq. 3) and reward (Eq. 4).

CPU: the reward's three cases, the compilation tool on sources that do and do
not compile, and the stage inputs passing the library's own validation.
GPU: full rounds for a correct candidate (V = 1, r = P > 0), a candidate with
a planted fault beyond 2^20 elements (stages 0-2 pass, stage 3 fails, later
stages are skipped, r = 0) and one that does not compile (r = -1).
"""
import ctypes as C
import os

import numpy as np
import pytest

import paper_2609_00058_gb300 as sv
from paper_2609_00058_gb300 import candidate_round as cr

HERE = os.path.dirname(os.path.abspath(__file__))
CAND = os.path.join(HERE, "candidates")
TASK = cr.Task("vecAddInplace")


def src(name):
    return os.path.join(CAND, name + ".cu")


def test_reward_follows_eq4():
    assert cr.reward(0, 0, 0.0) == -1.0
    assert cr.reward(0, 1, 5.0) == -1.0  # nothing counts without compilation
    assert cr.reward(1, 0, 5.0) == 0.0
    assert cr.reward(1, 1, 2.5) == 2.5


def test_compilation_tool(tmp_path):
    bad = cr.compile_kernel(src("vec_add_inplace_broken"), str(tmp_path))
    assert not bad.ok and bad.path is None and "scale_factor" in bad.log
    good = cr.compile_kernel(src("vec_add_inplace"), str(tmp_path))
    assert good.ok and os.path.exists(good.path)
    assert hasattr(C.CDLL(good.path), cr.LAUNCH_SYMBOL)


def test_stage_inputs_are_valid_specs():
    layout, nbytes = cr.stage_layout(TASK)
    assert [row[0] % 256 for row in layout] == [0] * len(TASK.stages)
    specs = cr.input_specs(TASK, layout)
    assert len(specs) == 2 * len(TASK.stages)
    assert sv.check_specs(specs, nbytes) == 0
    # the four arrays of a stage do not overlap and fit the arena
    for n, row in zip(TASK.stages, layout):
        assert all(b - a >= 4 * n for a, b in zip(row[:-1], row[1:]))
    assert layout[-1][3] + 4 * TASK.stages[-1] <= nbytes


def test_broken_candidate_scores_minus_one(tmp_path):
    r = cr.run_round(TASK, src("vec_add_inplace_broken"), src("vec_add_reference"), str(tmp_path))
    assert (r.C, r.V, r.r) == (0, 0, -1.0)
    assert "scale_factor" in r.compile_log


def assert_oracle_verdicts(r, progressive=True):
    """The round's per-stage verdicts against the oracle on the bytes the
    round verified (Eq. 1 per stage; Sec. 4.2.2 fail-fast for the ladder)."""
    import oracle
    from gpu_util import assert_results_match
    pairs, h = r.snapshot
    if progressive:
        want, ff = oracle.progressive(pairs, h, h)
        assert ff == r.first_failed
    else:
        want = oracle.compare(pairs, h, h)
    assert_results_match(r.stages[:len(want)], want, "candidate round")
    return want


@pytest.mark.gpu
def test_correct_candidate_round(tmp_path):
    from gpu_util import device
    device()
    r = cr.run_round(TASK, src("vec_add_inplace"), src("vec_add_reference"), str(tmp_path), snapshot=True)
    assert (r.C, r.V, r.first_failed) == (1, 1, -1)
    assert_oracle_verdicts(r)
    assert r.latency_ms > 0 and r.P == pytest.approx(1.0 / r.latency_ms) and r.r == r.P
    assert all(s["state"] == sv.STAGE_RUN and s["pass"] and s["mismatches"] == 0 for s in r.stages)
    # the synthesized a carries NaN/Inf at the specials rate: both sides agree on them
    assert sum(s["nan_disagree"] + s["inf_disagree"] for s in r.stages) == 0
    assert r.stages[-1]["n_finite"] < TASK.stages[-1]


@pytest.mark.gpu
def test_faulty_candidate_fails_at_the_first_large_stage(tmp_path):
    from gpu_util import device
    device()
    r = cr.run_round(TASK, src("vec_add_inplace_faulty"), src("vec_add_reference"), str(tmp_path), snapshot=True)
    assert (r.C, r.V, r.r, r.first_failed) == (1, 0, 0.0, 3)
    assert [s["state"] for s in r.stages] == [sv.STAGE_RUN] * 4
    assert [s["pass"] for s in r.stages] == [True, True, True, False]
    # every statistic of every stage equals the oracle's on the same bytes
    want = assert_oracle_verdicts(r)
    assert want[3]["first_mismatch"] >= 1 << 20


@pytest.mark.gpu
def test_fault_found_at_the_right_stage_on_other_ladders(tmp_path):
    from gpu_util import device
    device()
    task = cr.Task("vecAddInplace", stages=(1000, (1 << 20) - 1, (1 << 20) + 1, 1 << 21), seed=9)
    r = cr.run_round(task, src("vec_add_inplace_faulty"), src("vec_add_reference"), str(tmp_path), snapshot=True)
    assert r.first_failed == 2
    assert [s["state"] for s in r.stages] == [sv.STAGE_RUN] * 3 + [sv.STAGE_SKIPPED]
    assert_oracle_verdicts(r)
    assert r.stages[2]["mismatches"] == 1 and r.stages[2]["first_mismatch"] == 1 << 20


# ---------------------------------------------------------------------------
# self-contained programs exchanging tensor files (the scaffold's process boundary)
# ---------------------------------------------------------------------------
def test_broken_program_scores_minus_one(tmp_path):
    r = cr.run_program_round(TASK, src("vec_add_inplace_broken"), src("vec_add_reference"), str(tmp_path))
    assert (r.C, r.V, r.r) == (0, 0, -1.0)


@pytest.mark.gpu
def test_correct_program_round(tmp_path):
    from gpu_util import device
    device()
    r = cr.run_program_round(TASK, src("vec_add_inplace"), src("vec_add_reference"), str(tmp_path), snapshot=True)
    assert (r.C, r.V, r.first_failed) == (1, 1, -1)
    assert_oracle_verdicts(r, progressive=False)
    assert r.latency_ms > 0 and r.r == r.P == pytest.approx(1.0 / r.latency_ms)
    assert len(r.stages) == len(TASK.stages) and all(s["pass"] and s["mismatches"] == 0 for s in r.stages)
    # the files the programs exchanged are tensor files of the stage sizes
    import tensor_files as TF
    name, shape, data = TF.parse(os.path.join(str(tmp_path), "files", "cand_3.svt"))
    assert (name, shape) == ("f32", (TASK.stages[3],))


@pytest.mark.gpu
def test_faulty_program_stops_at_the_failing_stage(tmp_path):
    """Fail-fast across processes: stage 3 fails, and no later stage is run."""
    from gpu_util import device
    device()
    task = cr.Task("vecAddInplace", stages=(1000, 1 << 16, 1 << 21, 1 << 22), seed=3)
    r = cr.run_program_round(task, src("vec_add_inplace_faulty"), src("vec_add_reference"), str(tmp_path),
                             snapshot=True)
    assert (r.C, r.V, r.r, r.first_failed) == (1, 0, 0.0, 2)
    assert_oracle_verdicts(r, progressive=False)
    assert [s["pass"] for s in r.stages] == [True, True, False]
    assert r.stages[2]["first_mismatch"] >= 1 << 20
    assert not os.path.exists(os.path.join(str(tmp_path), "files", "a_3.svt"))
