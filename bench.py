"""Benchmark of the synthesis + verification path on GB300.

One step = the whole path over one batch of one workload: syn_generate of
every reference and candidate array (test-data synthesis, CUDA-Harness Sec.
4.2.1), then the compare of every pair (Eq. 1) -- verify_progressive for the
ladder (fail-fast, Sec. 4.2.2), a compare plan otherwise.

Workloads (workloads.py): perm_i64 (int64 permutation n = 2^28, 17 swapped
pairs; the default and headline: 4.29 GB synthesized and 4.29 GB verified
per step), dotlike_bf16 (bf16 32768^2, K = 64), ladder (n = 2^10 .. 2^27
fp32 N(0,1), exit at stage 3), segmented (4096 mixed-dtype cases) and
fp32_pair (n = 2^20).  By default every workload is measured and the JSON
line carries one object per workload under "workloads"; the top-level
fields are the headline workload's.

Prints ONE JSON line (rank 0).  `value` is synthesized + verified bytes per
second with every buffer resident in HBM; `e2e` is the same metric through
the public API with the synthesized test data delivered to pinned host
memory and the verdicts read back every step.  `roofline` is the headline
workload's dominant kernel against the measured HBM copy bandwidth; the
dot-like workload also reports its dot products' FMAs against a measured
fp32 FMA rate (bench_alu_peak.cu).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                  [--workload perm_i64|dotlike_bf16|ladder|segmented|fp32_pair|tensor_io]
                  [--only-headline] [--no-cpu-baseline] [--oracle-threads T]

--workload tensor_io measures the test-data I/O path instead (sv_read_tensor
of a 1 GiB uint8 tensor file into fp32, the conversion kernel alone, the
pinned copy rate and sv_write_tensor) and prints its own JSON line.

Under torchrun (N > 1) every rank runs an independent replica on its own
GPU (the path needs no exchange at this size); the time is the max over ranks.
"""
import argparse
import ctypes
import hashlib
import json
import os
import statistics
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import workloads as W  # noqa: E402

METRIC = "verified GB/s and synthesized GB/s on 1 GB300, as % of HBM peak"
L2_BYTES = 129 * 1000 * 1000  # GB300 L2 (bytes, nominal 129 MB)
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
# DRAM bytes per step of each workload's generator and compare kernels
# (dram__bytes_read.sum + dram__bytes_write.sum), keyed by (workload, role,
# hash of the sources of that role's kernels): a figure taken on other
# sources is not reported (null)
NCU_TRAFFIC = {
    # one single-pass launch list per workload (python bench.py --workload W
    # --only-headline --steps 2 --warmup 1 --no-cpu-baseline): the step's own
    # launches of each role, summed over its 7 steps and divided by 7
    ("perm_i64", "generate", "1c4f4b4c9fb23b7d"): 4234255799,  # gen_kernel<i64, permutation>, edits fused
    ("perm_i64", "verify", "792e3c49e8acd81c"): 4295342738,    # cmp_kernel<i64> + combine_kernel
    ("ladder", "generate", "1c4f4b4c9fb23b7d"): 1316475611,    # gen_kernel<f32, normal>, one launch
    ("ladder", "verify", "792e3c49e8acd81c"): 36022930,        # 3 stage groups: cmp_kernel + combine_stages_kernel
    ("dotlike_bf16", "generate", "1c4f4b4c9fb23b7d"): 4442408814,  # factors gen_kernel + dot_kernel<bf16>
    ("dotlike_bf16", "verify", "792e3c49e8acd81c"): 4298158373,    # cmp_kernel<bf16> + combine_kernel
    # the two small workloads' outputs stay in L2 through the step (DRAM
    # counts only what the caches write back meanwhile)
    ("segmented", "generate", "1c4f4b4c9fb23b7d"): 5694427,
    ("segmented", "verify", "792e3c49e8acd81c"): 146442240,
    ("fp32_pair", "generate", "1c4f4b4c9fb23b7d"): 90514,
    ("fp32_pair", "verify", "792e3c49e8acd81c"): 8452718,
}
ROLE_SOURCES = {"generate": ("generate.cu", "sv_device.cuh", "sv_kernels.h"),
                "verify": ("compare.cu", "sv_device.cuh", "sv_kernels.h")}


def log(*a):
    print(*a, file=sys.stderr, flush=True)


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return FALLBACK_PEAKS, "fallback"


def alu_peaks():
    """Hardware issue rates (fp32 FMA, 32-bit IMAD, 32x32->64 IMAD per second
    and per SM-cycle) measured now on this GPU by bench_alu_peak.cu, a plain
    loop of independent chains of each instruction (built on demand)."""
    import subprocess
    src = os.path.join(ROOT, "bench_alu_peak.cu")
    exe = os.path.join(ROOT, "_build", "bench_alu_peak")
    try:
        if not os.path.exists(exe) or os.path.getmtime(exe) < os.path.getmtime(src):
            from paper_2609_00058_gb300 import build as b
            os.makedirs(os.path.dirname(exe), exist_ok=True)
            subprocess.run([b.nvcc(), *b.ARCH, "-O3", "-std=c++17", "-o", exe, src], check=True,
                           capture_output=True, timeout=300)
        out = subprocess.run([exe], check=True, capture_output=True, text=True, timeout=120).stdout
        return json.loads(out.strip().splitlines()[-1])
    except Exception as e:  # the dot-like ALU fraction is then left out
        log("alu probe unavailable:", e)
        return None


def source_hash(role):
    """Hash of the kernel sources of one role ("generate" or "verify")."""
    h = hashlib.sha256()
    d = os.path.join(ROOT, "paper_2609_00058_gb300", "csrc")
    for f in ROLE_SOURCES[role]:
        with open(os.path.join(d, f), "rb") as fh:
            h.update(f.encode() + fh.read())
    return h.hexdigest()[:16]


# ---------------------------------------------------------------------------
# clocks sampled during the timed region (NVML through ctypes; read-only)
# ---------------------------------------------------------------------------
REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown", 0x40: "hw_thermal_slowdown",
           0x80: "hw_power_brake_slowdown", 0x2: "applications_clocks_setting", 0x10: "sync_boost"}


class ClockSampler:
    def __init__(self, torch_device):
        self.samples, self.ok, self.max_mhz = [], False, None
        try:
            self.nv = ctypes.CDLL("libnvidia-ml.so.1")
            if self.nv.nvmlInit_v2() != 0:
                return
            self.h = ctypes.c_void_p()
            bus = None
            try:
                import torch
                pr = torch.cuda.get_device_properties(torch_device)
                bus = "%08x:%02x:%02x.0" % (pr.pci_domain_id, pr.pci_bus_id, pr.pci_device_id)
            except Exception:
                bus = None
            rc = self.nv.nvmlDeviceGetHandleByPciBusId_v2(bus.encode(), ctypes.byref(self.h)) if bus else 1
            if rc != 0 and self.nv.nvmlDeviceGetHandleByIndex_v2(0, ctypes.byref(self.h)) != 0:
                return
            m = ctypes.c_uint()
            if self.nv.nvmlDeviceGetMaxClockInfo(self.h, 1, ctypes.byref(m)) == 0:
                self.max_mhz = m.value
            self.ok = True
        except OSError:
            pass

    def _loop(self):
        mhz, rs = ctypes.c_uint(), ctypes.c_ulonglong()
        while not self.stop_ev.is_set():
            if self.nv.nvmlDeviceGetClockInfo(self.h, 1, ctypes.byref(mhz)) == 0 and \
                    self.nv.nvmlDeviceGetCurrentClocksEventReasons(self.h, ctypes.byref(rs)) == 0:
                self.samples.append((time.perf_counter(), mhz.value, rs.value))
            time.sleep(0.002)

    def start(self):
        if not self.ok:
            return
        self.stop_ev = threading.Event()
        self.th = threading.Thread(target=self._loop, daemon=True)
        self.th.start()

    def stop(self, t0, t1):
        if not self.ok:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvml unavailable"]}
        self.stop_ev.set()
        self.th.join()
        inside = [s for s in self.samples if t0 <= s[0] <= t1] or \
            sorted(self.samples, key=lambda s: min(abs(s[0] - t0), abs(s[0] - t1)))[:3]
        bits = 0
        for s in inside:
            bits |= s[2]
        return {"sm_mhz": statistics.median(s[1] for s in inside) if inside else None,
                "sm_max_mhz": self.max_mhz, "samples": len(inside),
                "reasons": [v for k, v in sorted(REASONS.items()) if bits & k]}


# ---------------------------------------------------------------------------
# the CPU oracle on a bounded sample (baseline / reference arm)
# ---------------------------------------------------------------------------
def oracle_sample(workload):
    if workload == "ladder":
        return W.progressive_ladder((10, 14, 18, 22)), "ladder stages n=2^10,2^14,2^18,2^22 (same seeds)"
    if workload == "fp32_pair":
        return W.single_fp32_pair(1 << 20), "the whole fp32 pair n=2^20"
    if workload == "segmented":
        return W.segmented_cases(1024), "the first 1024 of the 4096 cases"
    if workload == "dotlike_bf16":
        return W.dotlike_bf16_pair(rows=256, cols=32768), "256 of the 32768 rows"
    return W.int64_permutation_pair(1 << 22), "n=2^22 of the 2^28 permutation"


def run_oracle_once(wl, threads=1):
    """One step of the oracle on host memory: generate every call, then
    verify; returns (seconds, synthesized + verified bytes)."""
    import oracle
    arena = np.zeros(wl.arena_bytes, np.uint8)
    t0 = time.perf_counter()
    for call in wl.gen_calls:
        oracle.generate(call, arena, threads=threads)
    if wl.progressive:
        _, ff = oracle.progressive(wl.pairs, arena, arena, threads=threads)
        stages = len(wl.pairs) if ff < 0 else ff + 1
    else:
        oracle.compare(wl.pairs, arena, arena, threads=threads)
        stages = None
    dt = time.perf_counter() - t0
    return dt, wl.synth_bytes() + wl.verify_bytes(stages)


CPU_BASELINE_SECONDS = 8.0  # per leg of the headline workload's baseline
CPU_SUB_SECONDS = 2.0       # per leg of every other workload's baseline


def oracle_rate(wl, threads, seconds):
    """GB/s of the oracle on `wl`, repeating it until `seconds` are timed."""
    tot, nbytes, reps = 0.0, 0, 0
    while reps == 0 or tot < seconds:
        dt, nb = run_oracle_once(wl, threads)
        tot, nbytes, reps = tot + dt, nbytes + nb, reps + 1
    return nbytes / tot / 1e9, reps, tot


def cpu_baseline(workload, seconds=CPU_BASELINE_SECONDS, threads=0):
    """The oracle as it stands on a bounded sample of the workload, timed two
    ways: single-threaded (the plain oracle) and on every host core (its
    multi-threaded driver, same bytes and verdicts).  The top-level value is
    the all-cores figure."""
    import oracle
    oracle.build()
    wl, sample = oracle_sample(workload)
    cores = threads if threads > 0 else oracle.threads_default()
    v1, r1, t1 = oracle_rate(wl, 1, seconds)
    vt, rt, tt = oracle_rate(wl, cores, seconds)
    single = {"value": v1, "unit": "GB/s", "cores": 1,
              "sample": "%d x (%s), generate + verify, single-threaded C oracle, %.1f s" % (r1, sample, t1)}
    threaded = {"value": vt, "unit": "GB/s", "cores": cores,
                "sample": "%d x (%s), generate + verify, C oracle on %d threads, %.1f s" % (rt, sample, cores, tt)}
    return {"value": vt, "unit": "GB/s", "cores": cores, "kind": "oracle", "sample": threaded["sample"],
            "single": single, "threaded": threaded}


def reference_arm(args, rank, world):
    """The oracle arm: the CPU oracle on all host cores (its multi-threaded
    driver), one bounded sample of the workload per step."""
    if rank != 0:
        return
    import oracle
    oracle.build()
    if args.workload == "tensor_io":
        return io_reference_arm(args)
    cores = args.oracle_threads if args.oracle_threads > 0 else oracle.threads_default()
    wl, sample = oracle_sample(args.workload)
    for _ in range(args.warmup):
        run_oracle_once(wl, cores)
    times, nbytes = [], 0
    for _ in range(args.steps):
        dt, nbytes = run_oracle_once(wl, cores)
        times.append(dt)
    tot = sum(times)
    value = nbytes * args.steps / tot / 1e9
    what = "%s, C oracle on %d threads" % (sample, cores)
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * tot / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": workload_dtype(args.workload),
            "data": "synthetic (seeded counter-based specs)",
            "config": {"workload": full_workload(args.workload).name, "sample": sample},
            "cpu_baseline": {"value": value, "unit": "GB/s", "cores": cores, "kind": "oracle", "sample": what},
            "e2e": {"value": value, "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def io_reference_arm(args):
    """The oracle's load of test data: a 16 MiB uint8 file read by numpy and
    converted to fp32 by the oracle, per step."""
    import shutil
    import tempfile

    import oracle
    host = np.random.default_rng(0).integers(0, 256, size=16 << 20, dtype=np.uint8)
    tmp = tempfile.mkdtemp(prefix="svio_")
    try:
        p = os.path.join(tmp, "s.bin")
        host.tofile(p)
        for _ in range(args.warmup):
            oracle.convert(np.fromfile(p, np.uint8), "u8", "f32")
        t0 = time.perf_counter()
        for _ in range(args.steps):
            oracle.convert(np.fromfile(p, np.uint8), "u8", "f32")
        tot = time.perf_counter() - t0
    finally:
        shutil.rmtree(tmp, ignore_errors=True)
    value = host.size * args.steps / tot / 1e9
    sample = "16 MiB uint8 file read by numpy, converted to fp32 by the oracle (single thread)"
    print(json.dumps({"impl": "reference", "metric": IO_METRIC, "value": value, "unit": "GB/s", "n_gpus": args.gpus,
                      "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * tot / args.steps,
                      "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "u8->f32",
                      "data": "synthetic (uniform random bytes)",
                      "config": {"workload": "1 GiB uint8 tensor file loaded as fp32", "sample": sample},
                      "cpu_baseline": {"value": value, "unit": "GB/s", "cores": 1, "kind": "oracle",
                                       "sample": sample},
                      "e2e": {"value": value, "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}),
          flush=True)


# ---------------------------------------------------------------------------
# the GPU arm
# ---------------------------------------------------------------------------
SMALL = {  # the same kernels on cases of a few GB at most (for ncu captures): --small
    "dotlike_bf16": lambda: W.dotlike_bf16_pair(rows=8192),
    "perm_i64": lambda: W.int64_permutation_pair(1 << 26),
    "ladder": lambda: W.progressive_ladder(W.LADDER_EXPONENTS[:-1]),
}
_small = False


def full_workload(name):
    if _small and name in SMALL:
        return SMALL[name]()
    return W.FULL_SIZE[name]()


def workload_dtype(name):
    """The element type the workload's arithmetic runs on."""
    return {"ladder": "f32", "fp32_pair": "f32", "segmented": "mixed f32/f16/bf16/i32", "dotlike_bf16": "bf16",
            "perm_i64": "int64"}[name]


WORKLOAD_ORDER = ("perm_i64", "dotlike_bf16", "ladder", "segmented", "fp32_pair")
HEADLINE = "perm_i64"  # the largest single-GPU workload: 4.29 GB synthesized + 4.29 GB verified per step


def timed_events(stream, fn, reps):
    """Mean ms of fn() over reps calls, CUDA events on `stream` (after 3 warm-up calls)."""
    import torch
    for _ in range(3):
        fn()
    c0, c1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    c0.record(stream)
    for _ in range(reps):
        fn()
    c1.record(stream)
    torch.cuda.synchronize()
    return c0.elapsed_time(c1) / reps


def measure_workload(name, args, dev, world, steps, warmup, alu):
    """Time one workload's step (syn_generate, then the compare) with its
    inputs resident in HBM, then the same step end to end through the
    binding with the arena delivered to pinned host memory.  Returns the
    workload's object of the JSON line (rank 0's view; times are max over
    ranks)."""
    import torch

    import paper_2609_00058_gb300 as sv

    wl = full_workload(name)
    arena = torch.zeros(wl.arena_bytes, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)
    spec_tabs = [sv.SpecTable(c) for c in wl.gen_calls]
    pair_tab = sv.PairTable(wl.pairs, progressive=wl.progressive)
    ws_bytes = max([t.ws_bytes for t in spec_tabs] + [pair_tab.ws_bytes, 256])
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=dev)
    n_pairs = len(wl.pairs)
    results = torch.empty(n_pairs * sv.RESULT_BYTES, dtype=torch.uint8, device=dev)
    ff = torch.empty(1, dtype=torch.int32, device=dev)

    # every generator call goes through a plan built once before the steps
    # (the spec table validated, grouped, scheduled and staged), as the
    # stages of a round are synthesized again for every candidate
    gen_plans = [sv.GeneratePlan(t, wl.arena_bytes, device=dev) for t in spec_tabs]

    def do_generate():
        for pl in gen_plans:
            pl(arena)

    # a compare workload verifies through a plan built once (the pair table
    # grouped and staged before the steps, as for every candidate of a round)
    plan = None if wl.progressive else sv.ComparePlan(pair_tab, wl.arena_bytes, wl.arena_bytes, device=dev)

    def do_verify():
        if wl.progressive:
            sv.progressive(pair_tab, arena, arena, results=results, first_failed=ff, workspace=ws)
        else:
            plan(arena, arena, results=results)

    # one untimed pass to learn how many stages the ladder runs
    do_generate()
    do_verify()
    torch.cuda.synchronize()
    stages_run = None
    if wl.progressive:
        f = int(ff.item())
        stages_run = n_pairs if f < 0 else f + 1
    synth_b, verify_b = wl.synth_bytes(), wl.verify_bytes(stages_run)
    step_bytes = synth_b + verify_b

    for _ in range(warmup):
        do_generate()
        do_verify()
    torch.cuda.synchronize()
    barrier(world)

    # a working set that fits twice in L2 is evicted before every timed step
    # by writing a buffer of twice the L2 size (outside the step's events)
    flush = None
    if wl.arena_bytes <= 2 * L2_BYTES:
        flush = torch.empty(2 * L2_BYTES, dtype=torch.uint8, device=dev)
    sampler = ClockSampler(dev)
    sampler.start()
    time.sleep(0.05)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(steps)]
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier(world)
    torch.cuda.synchronize()
    launches0 = sv.lib().sv_kernel_launches()
    t_host0 = time.perf_counter()
    start.record(stream)
    for k in range(steps):
        if flush is not None:
            flush.fill_(k & 0xFF)
        ev[k][0].record(stream)
        do_generate()
        ev[k][1].record(stream)
        do_verify()
        ev[k][2].record(stream)
    end.record(stream)
    torch.cuda.synchronize()
    t_host1 = time.perf_counter()
    launches = sv.lib().sv_kernel_launches() - launches0
    barrier(world)
    clocks = sampler.stop(t_host0, t_host1)
    gen_each = [e[0].elapsed_time(e[1]) for e in ev]
    ver_each = [e[1].elapsed_time(e[2]) for e in ev]
    step_each = [g + v for g, v in zip(gen_each, ver_each)]
    gen_ms = max_over_ranks(sum(gen_each) / steps, world)
    ver_ms = max_over_ranks(sum(ver_each) / steps, world)
    # the job's time: start to end, or the sum of the steps when flushes sit between them
    total_ms = sum(step_each) if flush is not None else start.elapsed_time(end)
    total_ms = max_over_ranks(total_ms, world)

    peaks, peak_kind = load_peaks()
    hbm = float(peaks["hbm_gbs"])
    reps = max(5, min(steps, 20))
    extra = {}
    if name == "dotlike_bf16":
        # the candidate pass alone: the noisy twin of the existing reference
        # array (SV_FROM_ARENA + relative noise), the part of its synthesis
        # that is not the dot product
        d = wl.gen_calls[1][0]
        cp = sv.SpecTable([W.GenSpec(d.dtype, "from_arena", d.n, seed=d.seed, stream=d.stream, ref_offset=None,
                                     cand_offset=d.cand_offset, a_offset=d.ref_offset, pelem=d.pelem)])
        cp_ms = timed_events(stream, lambda: sv.generate(cp, arena, workspace=ws), reps)
        cp_bytes = 2 * d.n * W.DTYPE_BYTES[d.dtype]  # reference read + candidate written
        extra["candidate_pass"] = {"what": "candidate pass alone: reference read, noisy twin written", "ms": cp_ms,
                                   "bytes": cp_bytes, "gbs": cp_bytes / (cp_ms * 1e-3) / 1e9,
                                   "frac_of_hbm": cp_bytes / (cp_ms * 1e-3) / 1e9 / hbm}
        # the dot products alone (factors in L2 or HBM, outputs written, no noise)
        dot_only = sv.SpecTable([d.replace(cand_offset=None, pelem=W.Perturb())])
        do_ms = timed_events(stream, lambda: sv.generate(dot_only, arena, workspace=ws), reps)
        fmas = d.n * d.dot_k
        extra["dot_only"] = {"what": "dot products alone: reference written, no candidate", "ms": do_ms,
                             "fma_per_s": fmas / (do_ms * 1e-3)}
        # the output compared per 128 x 128 tile (shaped outputs): the same
        # bytes as the verify step, 65536 verdicts instead of one
        pr = wl.pairs[0]
        tt = sv.Tiles(pr.dtype, d.rows, d.cols, pr.cand_offset, pr.ref_offset, tile_rows=128, tile_cols=128,
                      atol=pr.atol, rtol=pr.rtol)
        n_t = sv.tile_count(tt, wl.arena_bytes, wl.arena_bytes)
        tres = torch.empty(n_t * sv.RESULT_BYTES, dtype=torch.uint8, device=dev)
        tp_ms = timed_events(stream, lambda: sv.compare_tiles(tt, arena, arena, results=tres), reps)
        tp_bytes = 2 * pr.n * W.DTYPE_BYTES[pr.dtype]
        extra["tile_verify"] = {"what": "verify_compare_tiles, %d x %d output in 128 x 128 tiles (%d verdicts)"
                                        % (d.rows, d.cols, n_t), "ms": tp_ms, "bytes": tp_bytes,
                                "gbs": tp_bytes / (tp_ms * 1e-3) / 1e9,
                                "frac_of_hbm": tp_bytes / (tp_ms * 1e-3) / 1e9 / hbm}
        if alu:
            # the dot products' fp32 FMAs (K per output) against the measured
            # FMA issue rate; the noise's Philox and Box-Muller work is not counted
            peak = 2 * alu["ffma_per_s"] / 1e12
            ach = 2 * fmas / (gen_ms * 1e-3) / 1e12
            extra["alu"] = {"bound": "alu", "kernel": "dot_kernel<bf16> (syn_generate of the pair)",
                            "achieved": ach, "peak": peak, "unit": "TFLOP/s", "frac": ach / peak,
                            "dot_only_frac": 2 * fmas / (do_ms * 1e-3) / 1e12 / peak,
                            "work": "%d outputs x K=%d fp32 FMAs (2 flops each); noise not counted" % (d.n, d.dot_k),
                            "peak_kind": "measured fp32 FMA issue rate (bench_alu_peak.cu): %.1f FMA per SM-cycle "
                                         "at %.0f MHz" % (alu["ffma_per_sm_cycle"], alu["ffma_mhz"])}
        del tres

    # end to end: synthesized data delivered to pinned host buffers, verdicts read back
    host = torch.empty(wl.arena_bytes, dtype=torch.uint8, pin_memory=True)
    host_res = torch.empty(results.numel(), dtype=torch.uint8, pin_memory=True)
    host_ff = torch.empty(1, dtype=torch.int32, pin_memory=True)
    d2h = wl.arena_bytes + host_res.numel() + (4 if wl.progressive else 0)
    # host-to-device bytes per step: the tables that ride in kernel parameters
    # (up to 8 entries); a plan's larger table stays on the device
    h2d = sum(t.n * ctypes.sizeof(sv.syn_spec) for t in spec_tabs if t.n <= sv.INLINE_ENTRIES) + \
        (pair_tab.n * ctypes.sizeof(sv.vc_pair) if wl.progressive else 0)

    # the whole arena (every output array and the few alignment gaps between
    # them) goes to pinned host memory in pieces of at most 64 MiB spread over
    # four copy streams (several copy engines at once); the verify runs beside
    # them on the compute stream, as both only read the arena
    copy_streams = [torch.cuda.Stream(dev) for _ in range(4)]
    pieces = [[] for _ in copy_streams]
    for k, o in enumerate(range(0, wl.arena_bytes, 64 << 20)):
        pieces[k % len(pieces)].append((o, min(64 << 20, wl.arena_bytes - o)))

    def e2e_step():
        do_generate()
        generated = torch.cuda.Event()
        generated.record(stream)
        for cs, ps in zip(copy_streams, pieces):
            cs.wait_event(generated)
            with torch.cuda.stream(cs):
                for off, nb in ps:
                    host[off:off + nb].copy_(arena[off:off + nb], non_blocking=True)
        do_verify()
        host_res.copy_(results, non_blocking=True)
        if wl.progressive:
            host_ff.copy_(ff, non_blocking=True)
        for cs in copy_streams:
            cs.synchronize()
        stream.synchronize()

    e2e_steps = max(1, min(steps, 20))
    for _ in range(min(warmup, 3)):
        e2e_step()
    barrier(world)
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        e2e_step()
    e2e_s = max_over_ranks(time.perf_counter() - t0, world)
    l2_note = ("L2 flushed before every timed step (%d MiB written, outside the step's events)"
               % (2 * L2_BYTES >> 20)) if flush is not None else \
        ("working set %.2f GB > 2 x 129 MB L2 per step (no flush)" % (wl.arena_bytes / 1e9))
    del host, host_res, host_ff, arena, ws, results, flush, plan, gen_plans
    torch.cuda.synchronize()
    torch.cuda.empty_cache()

    gen_gbs = synth_b / (gen_ms * 1e-3) / 1e9
    ver_gbs = verify_b / (ver_ms * 1e-3) / 1e9
    gen_kernel = {"perm_i64": "gen_kernel<i64, permutation>", "ladder": "gen_kernel<f32, normal>",
                  "dotlike_bf16": "dot_kernel<bf16>", "fp32_pair": "gen_kernel<f32, uniform>",
                  "segmented": "gen_kernel<f32|f16|bf16 uniform, i32 int_range>"}[name]
    cmp_kernel = "cmp_kernel<%s> + combine" % ("mixed" if name == "segmented" else wl.pairs[0].dtype)
    out = {
        "workload": wl.name,
        "steps": steps, "warmup": warmup,
        "synth_bytes_per_step": synth_b, "verified_bytes_per_step": verify_b, "stages_run": stages_run,
        "l2": l2_note,
        "generate_call": "syn_generate_planned (plan built once, before the steps)",
        "verify": "verify_progressive" if wl.progressive else
                  "verify_compare_planned (plan built once, before the steps)",
        "value": job_throughput(step_bytes, steps, world, total_ms * 1e-3),
        "ms_per_step": total_ms / steps,
        "step_ms_median": statistics.median(step_each), "step_ms_best": min(step_each),
        "gen_ms": gen_ms, "verify_ms": ver_ms,
        "synth_gbs": gen_gbs, "verify_gbs": ver_gbs,
        "synth_frac_of_hbm": gen_gbs / hbm, "verify_frac_of_hbm": ver_gbs / hbm,
        "generate": {"kernel": gen_kernel, "ms": gen_ms, "bytes": synth_b, "gbs": gen_gbs, "frac_of_hbm": gen_gbs / hbm,
                     "traffic": NCU_TRAFFIC.get((name, "generate", source_hash("generate")))},
        "compare": {"kernel": cmp_kernel, "ms": ver_ms, "bytes": verify_b, "gbs": ver_gbs,
                    "frac_of_hbm": ver_gbs / hbm, "traffic": NCU_TRAFFIC.get((name, "verify", source_hash("verify")))},
        **extra,
        "e2e": {"value": job_throughput(step_bytes, e2e_steps, world, e2e_s), "unit": "GB/s",
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "steps": e2e_steps},
        "clocks": clocks,
        "gpu_launches": launches,
        "hbm_peak": {"value": hbm, "unit": "GB/s", "kind": "%s (hbm_gbs)" % peak_kind},
    }
    return out


def roofline_of(sub):
    """The dominant kernel of a workload's step against its bound: the
    generator or the compare (whichever takes longer per step) against the
    measured HBM copy bandwidth; the dot-like generator against the
    measured fp32 FMA rate."""
    dom = "generate" if sub["gen_ms"] >= sub["verify_ms"] else "compare"
    if dom == "generate" and "alu" in sub:
        r = dict(sub["alu"])
        r["traffic"] = sub["generate"]["traffic"]
        r["hbm_frac"] = sub["generate"]["frac_of_hbm"]
        return r
    k = sub[dom]
    other = sub["compare" if dom == "generate" else "generate"]
    return {"bound": "hbm", "kernel": k["kernel"], "achieved": k["gbs"], "peak": sub["hbm_peak"]["value"],
            "unit": "GB/s", "frac": k["frac_of_hbm"], "traffic": k["traffic"],
            "peak_kind": sub["hbm_peak"]["kind"],
            "other_kernel": {"kernel": other["kernel"], "frac": other["frac_of_hbm"]}}


def ours_arm(args, rank, world):
    import torch

    import paper_2609_00058_gb300 as sv

    dev = torch.device("cuda", int(os.environ.get("LOCAL_RANK", 0)))
    torch.cuda.set_device(dev)
    sv.lib()
    headline = args.workload
    names = [headline] + ([] if args.only_headline else [w for w in WORKLOAD_ORDER if w != headline])
    alu = alu_peaks() if "dotlike_bf16" in names and rank == 0 else None
    subs = {}
    for name in names:
        steps = args.steps if name == headline else min(args.steps, 20)
        warmup = args.warmup if name == headline else max(3, min(args.warmup, 5))
        log("measuring", name)
        subs[name] = measure_workload(name, args, dev, world, steps, warmup, alu)
    if rank != 0:
        return
    if not args.no_cpu_baseline:
        for name in names:
            subs[name]["cpu_baseline"] = cpu_baseline(
                name, CPU_BASELINE_SECONDS if name == headline else CPU_SUB_SECONDS, args.oracle_threads)
    h = subs[headline]
    reasons = sorted({r for s in subs.values() for r in (s["clocks"].get("reasons") or [])})
    line = {
        "metric": METRIC,
        "value": h["value"],
        "unit": "GB/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": h["ms_per_step"],
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": workload_dtype(headline),
        "data": "synthetic (seeded counter-based specs)",
        "config": {"workload": h["workload"], "synth_bytes_per_step": h["synth_bytes_per_step"],
                   "verified_bytes_per_step": h["verified_bytes_per_step"], "stages_run": h["stages_run"],
                   "l2": h["l2"], "generate": h["generate_call"], "verify": h["verify"],
                   "parallelism": "replicas" if world > 1 else "single GPU"},
        "synth_gbs": h["synth_gbs"], "verify_gbs": h["verify_gbs"],
        "synth_frac_of_hbm": h["synth_frac_of_hbm"], "verify_frac_of_hbm": h["verify_frac_of_hbm"],
        "gen_ms": h["gen_ms"], "verify_ms": h["verify_ms"],
        "roofline": roofline_of(h),
        "e2e": h["e2e"],
        "clocks": dict(h["clocks"], reasons_any_workload=reasons),
        "gpu_launches": h["gpu_launches"],
        "workloads": {n: dict(s, roofline=roofline_of(s)) for n, s in subs.items()},
    }
    if "cpu_baseline" in h:
        line["cpu_baseline"] = h["cpu_baseline"]
    if alu:
        line["alu_peaks"] = alu
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------------------
# the test-data I/O path (include/sv_io.h)
# ---------------------------------------------------------------------------
IO_METRIC = "test-data load GB/s (file bytes into HBM, values converted) on 1 GB300"
IO_FILE_ELEMS = 1 << 30  # uint8 elements of the timed file (1 GiB), loaded as fp32 (4 GiB)
IO_CONVERSIONS = [("u8", "f32"), ("f32", "bf16"), ("i32", "f32"), ("f64", "f32"), ("f32", "f64"), ("i64", "f32"),
                  ("f64", "bf16"), ("i32", "f64"), ("u16", "f16")]


def io_arm(args, rank, world):
    """One step = sv_read_tensor of a 1 GiB uint8 tensor file (page cache warm)
    into an fp32 buffer: host threads read the file into pinned chunks, the
    chunks cross to the GPU and the GPU converts each one.  Also measured: the
    conversion kernel alone (device to device, HBM roofline), the pinned
    host-to-device copy rate (the link's ceiling for the file path) and
    sv_write_tensor of the same bytes."""
    import shutil
    import tempfile

    import torch

    import oracle
    import paper_2609_00058_gb300 as sv

    dev = torch.device("cuda", int(os.environ.get("LOCAL_RANK", 0)))
    torch.cuda.set_device(dev)
    stream = torch.cuda.current_stream(dev)
    n = IO_FILE_ELEMS
    src = torch.randint(0, 256, (n,), dtype=torch.uint8, device=dev)
    out = torch.empty(4 * n, dtype=torch.uint8, device=dev)
    ws = torch.empty(sv.lib().sv_io_workspace_bytes(sv.IO_DTYPES["u8"], sv.IO_DTYPES["f32"], n),
                     dtype=torch.uint8, device=dev)
    tmp = tempfile.mkdtemp(prefix="svio_")
    path = os.path.join(tmp, "input.svt")
    try:
        t0 = time.perf_counter()
        sv.write_tensor(path, src, dtype="u8", shape=(n,))
        write_s = time.perf_counter() - t0
        for _ in range(max(args.warmup, 3)):
            sv.read_tensor(path, dtype="f32", out=out, workspace=ws)
        torch.cuda.synchronize()
        barrier(world)
        sampler = ClockSampler(dev)
        sampler.start()
        time.sleep(0.05)
        launches0 = sv.lib().sv_kernel_launches()
        times = []
        t_host0 = time.perf_counter()
        for _ in range(args.steps):
            t0 = time.perf_counter()
            sv.read_tensor(path, dtype="f32", out=out, workspace=ws)  # returns with the data in place
            times.append(time.perf_counter() - t0)
        t_host1 = time.perf_counter()
        launches = sv.lib().sv_kernel_launches() - launches0
        clocks = sampler.stop(t_host0, t_host1)
        total_s = max_over_ranks(sum(times), world)
        ok = bool(torch.equal(out.view(torch.float32)[:: 1 << 16], src[:: 1 << 16].float()))
        t0 = time.perf_counter()
        for _ in range(3):
            sv.write_tensor(path, src, dtype="u8", shape=(n,))
        write_s = min(write_s, (time.perf_counter() - t0) / 3)
    finally:
        shutil.rmtree(tmp, ignore_errors=True)

    # the conversion kernel alone, inputs resident (larger than L2)
    peaks, peak_kind = load_peaks()
    hbm = float(peaks["hbm_gbs"])
    conv = {}
    lost = torch.zeros(1, dtype=torch.int64, device=dev)
    for s_t, d_t in IO_CONVERSIONS:
        m = (1 << 30) // sv.IO_DTYPE_BYTES[s_t]  # 1 GiB of source
        a = torch.randint(0, 256, (m * sv.IO_DTYPE_BYTES[s_t],), dtype=torch.uint8, device=dev)
        if s_t in ("f32", "f64"):  # finite float test values rather than random encodings
            a = (torch.randn(m, device=dev, dtype=torch.float64 if s_t == "f64" else torch.float32)
                 * 100).view(torch.uint8)
        elif s_t in ("i32", "i64"):  # integers of every magnitude
            a = torch.randint(-2 ** 31, 2 ** 31, (m,), device=dev, dtype=torch.int64)
            a = (a if s_t == "i64" else a.to(torch.int32)).view(torch.uint8)
        b = torch.empty(m * sv.IO_DTYPE_BYTES[d_t], dtype=torch.uint8, device=dev)
        for _ in range(3):
            sv.convert(a, s_t, d_t, n=m, out=b, lost=lost)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        reps = max(5, min(args.steps, 20))
        torch.cuda.synchronize()
        e0.record(stream)
        for _ in range(reps):
            sv.convert(a, s_t, d_t, n=m, out=b, lost=lost)
        e1.record(stream)
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / reps
        nbytes = m * (sv.IO_DTYPE_BYTES[s_t] + sv.IO_DTYPE_BYTES[d_t])
        conv["%s->%s" % (s_t, d_t)] = {"ms": ms, "bytes": nbytes, "gbs": nbytes / (ms * 1e-3) / 1e9,
                                       "frac_of_hbm": nbytes / (ms * 1e-3) / 1e9 / hbm}
        del a, b
    # the link: pinned host -> device copy of 1 GiB
    pinned = torch.empty(1 << 30, dtype=torch.uint8, pin_memory=True)
    for _ in range(2):
        out[: 1 << 30].copy_(pinned, non_blocking=True)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(5):
        out[: 1 << 30].copy_(pinned, non_blocking=True)
    torch.cuda.synchronize()
    link_gbs = 5 * (1 << 30) / (time.perf_counter() - t0) / 1e9
    if rank != 0:
        return
    value = world * n * args.steps / total_s / 1e9
    main_conv = conv["u8->f32"]
    line = {
        "metric": IO_METRIC, "value": value, "unit": "GB/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": 1e3 * total_s / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "u8->f32", "data": "synthetic (uniform random bytes)",
        "config": {"workload": "1 GiB uint8 tensor file loaded as fp32 (sv_read_tensor, page cache warm)",
                   "file_bytes": n + 128, "loaded_bytes": 4 * n, "chunk_bytes": 32 << 20,
                   "host_threads": os.cpu_count(), "l2": "1 GiB source, 4 GiB destination: larger than L2",
                   "values_checked": ok, "parallelism": "replicas" if world > 1 else "single GPU"},
        "roofline": {"bound": "hbm", "kernel": "cvt_kernel<u8, f32> (sv_convert, device to device)",
                     "achieved": main_conv["gbs"], "peak": hbm, "unit": "GB/s", "frac": main_conv["frac_of_hbm"],
                     "peak_kind": "%s (%s)" % (peak_kind, "hbm_gbs"), "traffic": None},
        "convert": conv,
        "link_h2d_gbs": link_gbs, "file_path_frac_of_link": value / world / link_gbs,
        "write_gbs": n / write_s / 1e9,
        "e2e": {"value": value, "unit": "GB/s", "h2d_bytes_per_step": n, "d2h_bytes_per_step": 0,
                "what": "the public call itself: file on the host, result in HBM"},
        "clocks": clocks, "gpu_launches": launches,
    }
    if not args.no_cpu_baseline:  # the oracle's conversion after a numpy read of the same bytes
        host = np.random.default_rng(0).integers(0, 256, size=16 << 20, dtype=np.uint8)
        tmp = tempfile.mkdtemp(prefix="svio_")
        try:
            p = os.path.join(tmp, "s.bin")
            host.tofile(p)
            tot, reps = 0.0, 0
            while reps == 0 or tot < CPU_BASELINE_SECONDS:
                t0 = time.perf_counter()
                oracle.convert(np.fromfile(p, np.uint8), "u8", "f32")
                tot += time.perf_counter() - t0
                reps += 1
        finally:
            shutil.rmtree(tmp, ignore_errors=True)
        line["cpu_baseline"] = {"value": reps * host.size / tot / 1e9, "unit": "GB/s", "cores": 1, "kind": "oracle",
                                "sample": "%d x (16 MiB uint8 file read by numpy, converted to fp32 by the oracle), "
                                          "%.1f s" % (reps, tot)}
    print(json.dumps(line), flush=True)


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x, world):
    """The largest of the ranks' x (the slowest rank's time): one all-reduce on
    the process group's device (CUDA for NCCL, host memory for gloo)."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(bytes_per_rank_step, steps, world, slowest_s):
    """Whole-job GB/s of N independent replicas: every rank processes the same
    bytes per step, and the job takes as long as its slowest rank."""
    return world * bytes_per_rank_step * steps / slowest_s / 1e9


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default=HEADLINE, choices=sorted(W.FULL_SIZE) + ["tensor_io"])
    ap.add_argument("--only-headline", action="store_true", help="measure the --workload alone")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--oracle-threads", type=int, default=0, help="oracle threads (0: every host core)")
    ap.add_argument("--small", action="store_true",
                    help="smaller cases of the large workloads (profiling; not the configured sizes)")
    args = ap.parse_args()
    global _small
    _small = args.small
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if world > 1:
        import torch
        import torch.distributed as dist
        backend = "gloo" if args.impl == "reference" else "nccl"
        if backend == "nccl":
            torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", 0)))
        dist.init_process_group(backend)
    if args.impl == "reference":
        reference_arm(args, rank, world)
    else:
        from __graft_entry__ import build
        if rank == 0:
            build()
        barrier(world)
        build()
        (io_arm if args.workload == "tensor_io" else ours_arm)(args, rank, world)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
