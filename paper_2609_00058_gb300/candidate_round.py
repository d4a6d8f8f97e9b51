"""One candidate round of the harness, end to end (CUDA-Harness Sec. 4.2.2 and
Sec. 4.3.2): the compilation tool C (Eq. 2), synthesis of the test inputs of
every stage (syn_generate), the trusted reference and the candidate run on
them, functional validation V by the fail-fast stage ladder
(verify_progressive, Eq. 1 per element), the latency performance P (Eq. 3)
and the reward r = -1 + C + C * V * P (Eq. 4).

A task here is an in-place binary fp32 vector operation, a <- f(a, b), the
shape of the paper's running example (vecAddInplace).  A candidate is a CUDA
source defining

    extern "C" int candidate_launch(float* a, const float* b, long long n, void* stream);

which enqueues the operation on `stream` and returns 0 (or a CUDA error
code).  The reference is a source with the same export that the caller
trusts.  Two ways to run them:
- run_round: both compiled by nvcc into shared libraries (the compilation
  parameters phi of Eq. 2 are the nvcc flags), loaded with ctypes and run on
  device buffers that syn_generate filled;
- run_program_round: both compiled into self-contained programs behind the
  scaffold's main() (scaffold/vec_inplace_main.h, Sec. 4.1.2), which read
  their inputs from tensor files named on the command line and write their
  outputs to files that are loaded back dtype-correctly (sv_read_tensor).
The paper leaves the unit of the latency open: P is reported in 1/ms.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
from dataclasses import dataclass, field
from typing import List, Optional, Sequence

from . import GenSpec, Pair, SynVerifyError, compare, decode_results, generate, progressive, read_tensor, write_tensor
from .build import ARCH, nvcc

DEFAULT_FLAGS = (*ARCH, "-O3", "-shared", "-Xcompiler", "-fPIC")
PROGRAM_FLAGS = (*ARCH, "-O3")
LAUNCH_SYMBOL = "candidate_launch"
SCAFFOLD_DIR = os.path.join(os.path.dirname(os.path.abspath(__file__)), "scaffold")
VEC_INPLACE_MAIN = "vec_inplace_main.h"


@dataclass
class Task:
    """An in-place fp32 vector operation checked on size-ascending stages."""
    name: str
    stages: Sequence[int] = (1 << 10, 1 << 14, 1 << 18, 1 << 22)
    seed: int = 1
    # inputs: a ~ N(mu, sigma) with special values (the paper's broad-range
    # example is N(5, 10)), b ~ U[lo, hi)
    a_normal: tuple = (5.0, 10.0)
    a_specials: tuple = ("nan", "pinf", "ninf", "denorm")
    a_special_rate: float = 1e-4
    b_uniform: tuple = (-100.0, 100.0)
    atol: float = 1e-5
    rtol: float = 1e-5


@dataclass
class Compiled:
    ok: bool  # C of Eq. 2
    path: Optional[str]
    log: str
    calling_convention: Optional[str] = None  # emitted at compile time (#pragma message)


@dataclass
class RoundResult:
    C: int
    V: int
    P: float  # 1 / latency, latency in ms; 0 unless C and V
    r: float
    latency_ms: Optional[float]
    first_failed: int  # index of the first failing stage, -1 if none (or not run)
    stages: List[dict] = field(default_factory=list)
    compile_log: str = ""
    # with snapshot=True: (the compare pairs of the stages that ran, the
    # arena's bytes on the host as they were verified), so the verdicts can
    # be re-derived from the same data
    snapshot: Optional[tuple] = None


def reward(c: int, v: int, p: float) -> float:
    """Eq. 4: -1 for a kernel that does not compile, 0 for one that compiles but
    fails validation, and its performance P otherwise."""
    return -1.0 + c + c * v * p


def compile_kernel(src: str, out_dir: str, flags: Sequence[str] = DEFAULT_FLAGS) -> Compiled:
    """The compilation tool of Eq. 2: 1 iff `src` compiles under `flags` into a
    shared library that exports the launcher."""
    os.makedirs(out_dir, exist_ok=True)
    out = os.path.join(out_dir, os.path.splitext(os.path.basename(src))[0] + ".so")
    p = subprocess.run([nvcc(), *flags, "-o", out, src], capture_output=True, text=True)
    log = (p.stdout + p.stderr).strip()
    if p.returncode != 0 or not os.path.exists(out):
        return Compiled(False, None, log)
    return Compiled(True, out, log)


def _calling_convention(log: str) -> Optional[str]:
    for line in log.splitlines():
        k = line.find("Calling convention:")
        if k >= 0:
            return line[k + len("Calling convention:"):].strip().strip("\"'\u2018\u2019")
    return None


def compile_program(src: str, out_dir: str, main_header: str = VEC_INPLACE_MAIN,
                    flags: Sequence[str] = PROGRAM_FLAGS) -> Compiled:
    """The compilation tool of Eq. 2 for a self-contained program: the
    candidate's source compiled behind the scaffold's main() (which reads the
    test inputs, calls the launcher and writes the outputs, Sec. 4.1.2).  The
    calling convention the scaffold emits at compile time is returned."""
    os.makedirs(out_dir, exist_ok=True)
    out = os.path.join(out_dir, os.path.splitext(os.path.basename(src))[0])
    p = subprocess.run([nvcc(), *flags, "-I" + SCAFFOLD_DIR, "-include", main_header, "-o", out, src],
                       capture_output=True, text=True)
    log = (p.stdout + p.stderr).strip()
    if p.returncode != 0 or not os.path.exists(out):
        return Compiled(False, None, log, _calling_convention(log))
    return Compiled(True, out, log, _calling_convention(log))


def _launcher(path: str):
    lib = C.CDLL(path)
    f = getattr(lib, LAUNCH_SYMBOL)
    f.argtypes = [C.c_void_p, C.c_void_p, C.c_longlong, C.c_void_p]
    f.restype = C.c_int
    f._keep = lib  # the library stays loaded while the launcher is in use
    return f


def stage_layout(task: Task):
    """Byte offsets of every stage's four arrays in one arena: the input a, the
    input b, the reference's output and the candidate's output (256-aligned)."""
    off, out = 0, []
    for n in task.stages:
        row = []
        for _ in range(4):
            row.append(off)
            off += (4 * n + 255) // 256 * 256
        out.append(tuple(row))
    return out, off


def input_specs(task: Task, layout) -> List[GenSpec]:
    specs = []
    for s, (n, (a_off, b_off, _, _)) in enumerate(zip(task.stages, layout)):
        specs.append(GenSpec("f32", "normal", n, seed=task.seed, stream=2 * s, ref_offset=a_off,
                             p0=task.a_normal[0], p1=task.a_normal[1], specials=tuple(task.a_specials),
                             special_rate=task.a_special_rate))
        specs.append(GenSpec("f32", "uniform", n, seed=task.seed, stream=2 * s + 1, ref_offset=b_off,
                             p0=task.b_uniform[0], p1=task.b_uniform[1]))
    return specs


def run_round(task: Task, candidate_src: str, reference_src: str, work_dir: str, runs: int = 20,
              flags: Sequence[str] = DEFAULT_FLAGS, device=None, snapshot: bool = False) -> RoundResult:
    """Compile, synthesize, run, validate, time and score one candidate
    (snapshot: also return the verified bytes, copied before the timing runs)."""
    import torch
    cand = compile_kernel(candidate_src, os.path.join(work_dir, "candidate"), flags)
    if not cand.ok:
        return RoundResult(0, 0, 0.0, reward(0, 0, 0.0), None, -1, [], cand.log)
    ref = compile_kernel(reference_src, os.path.join(work_dir, "reference"), flags)
    if not ref.ok:
        raise RuntimeError("the reference does not compile:\n" + ref.log)
    run_cand, run_ref = _launcher(cand.path), _launcher(ref.path)

    dev = torch.device(device or "cuda")
    stream = torch.cuda.current_stream(dev)
    layout, nbytes = stage_layout(task)
    arena = torch.zeros(nbytes, dtype=torch.uint8, device=dev)
    generate(input_specs(task, layout), arena, stream=stream)

    def f32(off, n):
        return arena[off: off + 4 * n].view(torch.float32)

    def launch(fn, out_off, b_off, n):
        rc = fn(arena.data_ptr() + out_off, arena.data_ptr() + b_off, n, stream.cuda_stream)
        if rc != 0:
            raise RuntimeError("launcher returned %d" % rc)

    # every stage: out = a, then the operation in place, for the reference and the candidate
    for n, (a_off, b_off, r_off, c_off) in zip(task.stages, layout):
        f32(r_off, n).copy_(f32(a_off, n))
        f32(c_off, n).copy_(f32(a_off, n))
        launch(run_ref, r_off, b_off, n)
        launch(run_cand, c_off, b_off, n)
    pairs = [Pair("f32", n, c_off, r_off, task.atol, task.rtol)
             for n, (_, _, r_off, c_off) in zip(task.stages, layout)]
    res, ff = progressive(pairs, arena, arena, stream=stream)
    stages = decode_results(res, len(pairs))
    first_failed = int(ff.item())
    snap = (pairs, arena.cpu().numpy()) if snapshot else None
    v = int(first_failed < 0)
    if not v:
        return RoundResult(1, 0, 0.0, reward(1, 0, 0.0), None, first_failed, stages, cand.log, snap)

    # P of Eq. 3 on the largest stage: mean latency of `runs` launches (CUDA
    # events on the launching stream, after warm-up), reusing the candidate's
    # output buffer of that stage now that its verdict is in
    n = task.stages[-1]
    a_off, b_off, _, c_off = layout[-1]
    for _ in range(3):
        launch(run_cand, c_off, b_off, n)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    stream.synchronize()
    e0.record(stream)
    for _ in range(runs):
        launch(run_cand, c_off, b_off, n)
    e1.record(stream)
    e1.synchronize()
    latency = e0.elapsed_time(e1) / runs
    p = 1.0 / latency
    return RoundResult(1, 1, p, reward(1, 1, p), latency, -1, stages, cand.log, snap)


def run_program_round(task: Task, candidate_src: str, reference_src: str, work_dir: str, runs: int = 20,
                      timeout: float = 120.0, device=None, snapshot: bool = False) -> RoundResult:
    """One round with self-contained programs exchanging tensor files (the
    scaffold's process boundary, Sec. 4.1.2): the stage inputs are synthesized
    on the GPU and written to files; stage by stage, the reference and the
    candidate program read them, run and write their outputs; the outputs are
    loaded back dtype-correctly (a file that is not float32 of the stage's
    size fails the stage) and compared with Eq. 1; the first failing stage
    ends the round (later stages are not run at all).  P is the candidate
    program's mean latency over `runs` launches on the largest stage.
    snapshot: also return the loaded outputs as they were compared."""
    import torch
    cand = compile_program(candidate_src, os.path.join(work_dir, "candidate"))
    if not cand.ok:
        return RoundResult(0, 0, 0.0, reward(0, 0, 0.0), None, -1, [], cand.log)
    ref = compile_program(reference_src, os.path.join(work_dir, "reference"))
    if not ref.ok:
        raise RuntimeError("the reference does not compile:\n" + ref.log)
    dev = torch.device(device or "cuda")
    layout, nbytes = stage_layout(task)
    arena = torch.zeros(nbytes, dtype=torch.uint8, device=dev)
    generate(input_specs(task, layout), arena)
    files = os.path.join(work_dir, "files")
    os.makedirs(files, exist_ok=True)

    def path(kind, s):
        return os.path.join(files, "%s_%d.svt" % (kind, s))

    def run(prog, s, out, extra=()):
        return subprocess.run([prog, path("a", s), path("b", s), out, *extra], capture_output=True, text=True,
                              timeout=timeout)

    stages: List[dict] = []
    compared: List[Pair] = []
    first_failed = -1
    for s, (n, (a_off, b_off, r_off, c_off)) in enumerate(zip(task.stages, layout)):
        write_tensor(path("a", s), arena[a_off: a_off + 4 * n], dtype="f32", shape=(n,))
        write_tensor(path("b", s), arena[b_off: b_off + 4 * n], dtype="f32", shape=(n,))
        rr = run(ref.path, s, path("ref", s))
        if rr.returncode != 0:
            raise RuntimeError("the reference program failed:\n" + rr.stderr)
        read_tensor(path("ref", s), file_dtype="f32", n=n, strict=True, out=arena[r_off: r_off + 4 * n])
        cr = run(cand.path, s, path("cand", s))
        ok = cr.returncode == 0
        if ok:
            try:  # the output must be float32 with the stage's element count
                read_tensor(path("cand", s), file_dtype="f32", n=n, strict=True, out=arena[c_off: c_off + 4 * n])
            except SynVerifyError:
                ok = False
        if ok:
            pair = Pair("f32", n, c_off, r_off, task.atol, task.rtol)
            compared.append(pair)
            res = decode_results(compare([pair], arena, arena), 1)[0]
        else:
            res = {"state": 1, "pass": 0, "mismatches": n, "first_mismatch": 0, "max_abs": float("nan"),
                   "program_error": (cr.stderr or "").strip()[-500:]}
        stages.append(res)
        if not res["pass"]:
            first_failed = s
            break
    snap = (compared, arena.cpu().numpy()) if snapshot else None
    if first_failed >= 0:
        return RoundResult(1, 0, 0.0, reward(1, 0, 0.0), None, first_failed, stages, cand.log, snap)
    last = len(task.stages) - 1
    cr = run(cand.path, last, path("cand_t", last), (str(runs),))
    latency = None
    for line in cr.stdout.splitlines():
        if line.startswith("latency_ms "):
            latency = float(line.split()[1])
    if cr.returncode != 0 or latency is None or latency <= 0:
        return RoundResult(1, 0, 0.0, reward(1, 0, 0.0), None, last, stages, cand.log, snap)
    p = 1.0 / latency
    return RoundResult(1, 1, p, reward(1, 1, p), latency, -1, stages, cand.log, snap)


def main(argv=None) -> int:
    """python -m paper_2609_00058_gb300.candidate_round CANDIDATE.cu REFERENCE.cu [--work DIR]:
    one round of the in-place vector task, printed as one JSON line."""
    import argparse
    import json
    import tempfile
    ap = argparse.ArgumentParser()
    ap.add_argument("candidate")
    ap.add_argument("reference")
    ap.add_argument("--work", default=None)
    ap.add_argument("--runs", type=int, default=20)
    ap.add_argument("--programs", action="store_true",
                    help="run self-contained programs that exchange tensor files instead of shared libraries")
    a = ap.parse_args(argv)
    work = a.work or tempfile.mkdtemp(prefix="candidate_round_")
    rnd = run_program_round if a.programs else run_round
    r = rnd(Task("vecAddInplace"), a.candidate, a.reference, work, runs=a.runs)
    print(json.dumps({"C": r.C, "V": r.V, "P_per_ms": r.P, "r": r.r, "latency_ms": r.latency_ms,
                      "first_failed_stage": r.first_failed,
                      "stages": [{k: s[k] for k in ("state", "pass", "mismatches", "first_mismatch", "max_abs")}
                                 for s in r.stages]}))
    return 0


if __name__ == "__main__":
    raise SystemExit(main())
