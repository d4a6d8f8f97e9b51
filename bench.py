"""Benchmark of the synthesis + verification path on GB300.

One step = the whole path over one batch: syn_generate of every stage's
reference and candidate (test-data synthesis, CUDA-Harness Sec. 4.2.1) and
verify_progressive over the stages (Eq. 1 and the fail-fast ladder,
Sec. 4.2.2).  Default workload: the six-stage ladder n = 2^10 .. 2^27 fp32
N(0,1) with 0.01% NaN/+-Inf/denormal injected, the candidate deviating at
stage 4 (1.38 GB synthesized per step, 35.8 MB verified before the exit).

Prints ONE JSON line (rank 0).  `value` is synthesized + verified bytes per
second with every buffer resident in HBM; `e2e` is the same metric through
the public API with the synthesized test data delivered to pinned host
memory and the verdicts read back every step.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                  [--workload ladder|fp32_pair|segmented|dotlike_bf16|perm_i64|tensor_io]

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
# dram bytes per launch of the dominant kernel from one ncu capture, keyed by
# a hash of the generator's sources they were taken on (None once they change)
NCU_TRAFFIC = {
    # gen_kernel<f32, normal>, median of the 7 launches of one single-pass ncu launch
    # list of the ladder step: 122,880 B read + 1,312,933,120 B written; no
    # fixup launch (the one exact-count edit is applied by the generating CTA)
    ("ladder", "c7ab7035e73bbe0a"): 1313085696,
    # gen_kernel<i64, permutation>, median of 7 launches of the permutation step:
    # 2,013,440 B read + 4,231,760,384 B written; the 34 swap edits are fused
    ("perm_i64", "c7ab7035e73bbe0a"): 4233829888,
}


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
    """Philox blocks, Box-Muller pairs and fp32 FMAs per SM per cycle of the
    library's own device code, measured now on this GPU by
    paper_2609_00058_gb300/probes/alu_peak.cu (built on demand)."""
    import subprocess
    src = os.path.join(ROOT, "paper_2609_00058_gb300", "probes", "alu_peak.cu")
    exe = os.path.join(ROOT, "paper_2609_00058_gb300", "_build", "alu_peak")
    try:
        deps = [src] + [os.path.join(ROOT, "paper_2609_00058_gb300", "csrc", f) for f in ("sv_device.cuh", "sv_kernels.h")]
        if not os.path.exists(exe) or os.path.getmtime(exe) < max(os.path.getmtime(d) for d in deps):
            from paper_2609_00058_gb300 import build as b
            subprocess.run([b.nvcc(), *b.ARCH, "-O3", "-std=c++17", "--fmad=false", "-o", exe, src], check=True,
                           capture_output=True, timeout=300)
        out = subprocess.run([exe], check=True, capture_output=True, text=True, timeout=120).stdout
        return json.loads(out.strip().splitlines()[-1])
    except Exception as e:  # the roofline falls back to HBM alone
        log("alu probe unavailable:", e)
        return None


def alu_floor_s(wl, peaks):
    """Seconds the generator needs at the measured ALU rates: per 4-element
    quantum, its Philox blocks (value, special selection, element-wise
    perturbation) and Box-Muller pairs (normal values, noise); for dot-like
    values also the K fp32 FMAs of every output."""
    cycles = 0.0
    for call in wl.gen_calls:
        for s in call:
            quanta = (s.n + 3) // 4
            if s.dist == "dotlike":  # K fp32 FMAs per output, then the same per-quantum noise
                cycles += 4 * quanta * s.dot_k / peaks["ffma_per_sm_cycle"]
                blocks = 1 if s.pelem.kind in ("rate_add_pm", "rel_noise") and s.cand_offset is not None else 0
                pairs = 2 if s.pelem.kind == "rel_noise" else 0
                cycles += quanta * (blocks / peaks["philox_blocks_per_sm_cycle"] +
                                    pairs / peaks["box_muller_pairs_per_sm_cycle"])
                continue
            blocks = {"uniform": 1, "normal": 1, "int_range": 2 if s.dtype == "i64" else 1,
                      "raw_bits": 2 if s.dtype == "i64" else 1}.get(s.dist, 0)
            blocks += 1 if s.specials and s.special_rate > 0 else 0
            blocks += 1 if s.pelem.kind in ("rate_add_pm", "rel_noise") and s.cand_offset is not None else 0
            pairs = (2 if s.dist == "normal" else 0) + (2 if s.pelem.kind == "rel_noise" else 0)
            cycles += quanta * (blocks / peaks["philox_blocks_per_sm_cycle"] +
                                pairs / peaks["box_muller_pairs_per_sm_cycle"])
    return cycles / (peaks["sms"] * peaks["clock_mhz"] * 1e6)


def source_hash():
    """Hash of the generator's kernel sources (the roofline's kernel)."""
    h = hashlib.sha256()
    d = os.path.join(ROOT, "paper_2609_00058_gb300", "csrc")
    for f in ("generate.cu", "sv_device.cuh", "sv_kernels.h"):
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


def run_oracle_once(wl):
    import oracle
    arena = np.zeros(wl.arena_bytes, np.uint8)
    t0 = time.perf_counter()
    for call in wl.gen_calls:
        oracle.generate(call, arena)
    if wl.progressive:
        _, ff = oracle.progressive(wl.pairs, arena, arena)
        stages = len(wl.pairs) if ff < 0 else ff + 1
    else:
        oracle.compare(wl.pairs, arena, arena)
        stages = None
    dt = time.perf_counter() - t0
    return dt, wl.synth_bytes() + wl.verify_bytes(stages)


CPU_BASELINE_SECONDS = 10.0  # the sample is repeated until this much CPU work is timed


def cpu_baseline(workload):
    wl, sample = oracle_sample(workload)
    import oracle
    oracle.build()
    tot, nbytes, reps = 0.0, 0, 0
    while reps == 0 or tot < CPU_BASELINE_SECONDS:
        dt, nb = run_oracle_once(wl)
        tot, nbytes, reps = tot + dt, nbytes + nb, reps + 1
    return {"value": nbytes / tot / 1e9, "unit": "GB/s", "cores": 1, "kind": "oracle",
            "sample": "%d x (%s), generate + verify, single-threaded C oracle, %.1f s" % (reps, sample, tot)}


def reference_arm(args, rank, world):
    if rank != 0:
        return
    import oracle
    oracle.build()
    if args.workload == "tensor_io":
        return io_reference_arm(args)
    wl, sample = oracle_sample(args.workload)
    for _ in range(args.warmup):
        run_oracle_once(wl)
    times, nbytes = [], 0
    for _ in range(args.steps):
        dt, nbytes = run_oracle_once(wl)
        times.append(dt)
    tot = sum(times)
    value = nbytes * args.steps / tot / 1e9
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * tot / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": workload_dtype(args.workload),
            "data": "synthetic (seeded counter-based specs)",
            "config": {"workload": full_workload(args.workload).name, "sample": sample},
            "cpu_baseline": {"value": value, "unit": "GB/s", "cores": 1, "kind": "oracle", "sample": sample},
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
def full_workload(name):
    return W.FULL_SIZE[name]()


def workload_dtype(name):
    """The element type the workload's arithmetic runs on."""
    return {"ladder": "f32", "fp32_pair": "f32", "segmented": "mixed f32/f16/bf16/i32", "dotlike_bf16": "bf16",
            "perm_i64": "int64"}[name]


def ours_arm(args, rank, world):
    import torch

    import paper_2609_00058_gb300 as sv

    dev = torch.device("cuda", int(os.environ.get("LOCAL_RANK", 0)))
    torch.cuda.set_device(dev)
    sv.lib()
    wl = full_workload(args.workload)
    arena = torch.zeros(wl.arena_bytes, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)
    spec_tabs = [sv.SpecTable(c) for c in wl.gen_calls]
    pair_tab = sv.PairTable(wl.pairs, progressive=wl.progressive)
    ws_bytes = max([t.ws_bytes for t in spec_tabs] + [pair_tab.ws_bytes, 256])
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=dev)
    n_pairs = len(wl.pairs)
    results = torch.empty(n_pairs * sv.RESULT_BYTES, dtype=torch.uint8, device=dev)
    ff = torch.empty(1, dtype=torch.int32, device=dev)
    synth_calls = [(t, c) for t, c in zip(spec_tabs, wl.gen_calls)]

    def do_generate():
        for t, _ in synth_calls:
            sv.generate(t, arena, workspace=ws)

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

    for _ in range(args.warmup):
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
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier(world)
    torch.cuda.synchronize()
    launches0 = sv.lib().sv_kernel_launches()
    t_host0 = time.perf_counter()
    start.record(stream)
    for k in range(args.steps):
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
    gen_ms = sum(gen_each) / args.steps
    ver_ms = sum(ver_each) / args.steps
    # the job's time: start to end, or the sum of the steps when flushes sit between them
    total_ms = sum(step_each) if flush is not None else start.elapsed_time(end)
    total_ms = max_over_ranks(total_ms, world)

    # the dot-like workload's candidate pass alone: the noisy twin of the
    # existing reference array (SV_FROM_ARENA + relative noise), the part of
    # its synthesis that is not the dot product
    cand_pass = None
    if args.workload == "dotlike_bf16":
        d = wl.gen_calls[1][0]
        cp = sv.SpecTable([W.GenSpec(d.dtype, "from_arena", d.n, seed=d.seed, stream=d.stream, ref_offset=None,
                                     cand_offset=d.cand_offset, a_offset=d.ref_offset, pelem=d.pelem)])
        for _ in range(3):
            sv.generate(cp, arena, workspace=ws)
        c0, c1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        c0.record(stream)
        for _ in range(args.steps):
            sv.generate(cp, arena, workspace=ws)
        c1.record(stream)
        torch.cuda.synchronize()
        cp_ms = c0.elapsed_time(c1) / args.steps
        cp_bytes = 2 * d.n * W.DTYPE_BYTES[d.dtype]  # reference read + candidate written
        cand_pass = {"what": "candidate pass alone: reference read, noisy twin written", "ms": cp_ms,
                     "bytes": cp_bytes, "gbs": cp_bytes / (cp_ms * 1e-3) / 1e9}

    # the dot-like output compared per 128 x 128 tile (shaped outputs): the
    # same bytes as the verify step, 65536 verdicts instead of one
    tile_pass = None
    if args.workload == "dotlike_bf16":
        pr = wl.pairs[0]
        side = int(round(pr.n ** 0.5))
        tt = sv.Tiles(pr.dtype, side, side, pr.cand_offset, pr.ref_offset, tile_rows=128, tile_cols=128,
                      atol=pr.atol, rtol=pr.rtol)
        n_t = sv.tile_count(tt, wl.arena_bytes, wl.arena_bytes)
        tres = torch.empty(n_t * sv.RESULT_BYTES, dtype=torch.uint8, device=dev)
        for _ in range(3):
            sv.compare_tiles(tt, arena, arena, results=tres)
        c0, c1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        c0.record(stream)
        for _ in range(args.steps):
            sv.compare_tiles(tt, arena, arena, results=tres)
        c1.record(stream)
        torch.cuda.synchronize()
        tp_ms = c0.elapsed_time(c1) / args.steps
        tp_bytes = 2 * pr.n * W.DTYPE_BYTES[pr.dtype]
        tile_pass = {"what": "verify_compare_tiles, %d x %d output in 128 x 128 tiles (%d verdicts)" % (side, side, n_t),
                     "ms": tp_ms, "bytes": tp_bytes, "gbs": tp_bytes / (tp_ms * 1e-3) / 1e9}

    # end to end: synthesized data delivered to pinned host buffers, verdicts read back
    host = torch.empty(wl.arena_bytes, dtype=torch.uint8, pin_memory=True)
    host_res = torch.empty(results.numel(), dtype=torch.uint8, pin_memory=True)
    host_ff = torch.empty(1, dtype=torch.int32, pin_memory=True)
    # the whole arena (every output array and the few alignment gaps between
    # them) goes back, in large pieces rather than one copy per array
    out_ranges = [(0, wl.arena_bytes)]
    d2h = wl.arena_bytes + host_res.numel() + (4 if wl.progressive else 0)
    h2d = sum(C.n * ctypes.sizeof(sv.syn_spec) for C in spec_tabs) + \
        (pair_tab.n * ctypes.sizeof(sv.vc_pair) if wl.progressive else 0)  # a plan's table stays on the device

    # the arena goes to pinned host memory in pieces of at most 64 MiB spread
    # over four copy streams (several copy engines at once); the verify runs
    # beside them on the compute stream, as both only read the arena
    copy_streams = [torch.cuda.Stream(dev) for _ in range(4)]
    pieces = [[] for _ in copy_streams]
    k = 0
    for off, nb in out_ranges:
        for o in range(off, off + nb, 64 << 20):
            pieces[k % len(pieces)].append((o, min(64 << 20, off + nb - o)))
            k += 1

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

    e2e_steps = max(1, min(args.steps, 20))
    for _ in range(min(args.warmup, 3)):
        e2e_step()
    barrier(world)
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        e2e_step()
    e2e_s = max_over_ranks(time.perf_counter() - t0, world)

    if rank != 0:
        return
    peaks, peak_kind = load_peaks()
    hbm = float(peaks["hbm_gbs"])
    gen_bytes_launch = synth_b  # algorithmic bytes: every output element written once
    achieved = gen_bytes_launch / (gen_ms * 1e-3) / 1e9
    src = source_hash()
    traffic = NCU_TRAFFIC.get((args.workload, src))
    alu = alu_peaks()
    alu_s = alu_floor_s(wl, alu) if alu else None
    hbm_s = gen_bytes_launch / (hbm * 1e9)
    if alu_s is not None and alu_s > hbm_s:
        # the ALU floor is above the HBM floor: report against the output rate
        # the measured Philox / Box-Muller throughput allows
        alu_gbs = gen_bytes_launch / alu_s / 1e9
        roofline = {"bound": "alu", "kernel": "syn_generate (gen_kernel + exact-count fixup)",
                    "achieved": achieved, "peak": alu_gbs, "unit": "GB/s", "frac": achieved / alu_gbs,
                    "peak_kind": "measured ALU rates (Philox %.3f blocks, Box-Muller %.3f pairs, %.1f fp32 FMAs "
                                 "per SM-cycle, %d SMs at %d MHz) as output GB/s" % (
                                     alu["philox_blocks_per_sm_cycle"], alu["box_muller_pairs_per_sm_cycle"],
                                     alu["ffma_per_sm_cycle"], alu["sms"], alu["clock_mhz"]),
                    "hbm_peak": hbm, "hbm_frac": achieved / hbm, "traffic": traffic}
    else:
        roofline = {"bound": "hbm", "kernel": "syn_generate (gen_kernel + exact-count fixup)",
                    "achieved": achieved, "peak": hbm, "unit": "GB/s", "frac": achieved / hbm,
                    "peak_kind": "%s (%s)" % (peak_kind, "hbm_gbs"), "traffic": traffic}
    line = {
        "metric": METRIC,
        "value": job_throughput(step_bytes, args.steps, world, total_ms * 1e-3),
        "unit": "GB/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": total_ms / args.steps,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": workload_dtype(args.workload),
        "data": "synthetic (seeded counter-based specs)",
        "config": {"workload": wl.name, "synth_bytes_per_step": synth_b, "verified_bytes_per_step": verify_b,
                   "stages_run": stages_run,
                   "l2": ("L2 flushed before every timed step (%d MiB written, outside the step's events)"
                          % (2 * L2_BYTES >> 20)) if flush is not None else
                         ("working set %.2f GB > 2 x 129 MB L2 per step (no flush)" % (wl.arena_bytes / 1e9)),
                   "verify": "verify_progressive" if wl.progressive else
                             "verify_compare_planned (plan built once, before the steps)",
                   "parallelism": "replicas" if world > 1 else "single GPU"},
        "synth_gbs": synth_b / (gen_ms * 1e-3) / 1e9,
        "verify_gbs": verify_b / (ver_ms * 1e-3) / 1e9,
        "synth_frac_of_hbm": synth_b / (gen_ms * 1e-3) / 1e9 / hbm,
        "verify_frac_of_hbm": verify_b / (ver_ms * 1e-3) / 1e9 / hbm,
        "gen_ms": gen_ms,
        "verify_ms": ver_ms,
        "step_ms_median": statistics.median(step_each),
        "step_ms_best": min(step_each),
        "roofline": roofline,
        **({"candidate_pass": dict(cand_pass, frac_of_hbm=cand_pass["gbs"] / hbm)} if cand_pass else {}),
        **({"tile_verify": dict(tile_pass, frac_of_hbm=tile_pass["gbs"] / hbm)} if tile_pass else {}),
        "e2e": {"value": job_throughput(step_bytes, e2e_steps, world, e2e_s), "unit": "GB/s",
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "steps": e2e_steps},
        "clocks": clocks,
        "gpu_launches": launches,
    }
    if not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(args.workload)
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
    ap.add_argument("--workload", default="ladder", choices=sorted(W.FULL_SIZE) + ["tensor_io"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    args = ap.parse_args()
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
