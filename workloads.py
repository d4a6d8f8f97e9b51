"""Seeded synthetic workloads for the synthesis + verification path.

This module only DESCRIBES inputs: generator spec tables, compare-pair tables,
arena layouts, and seeded numpy arrays used as compare inputs.  It holds none
of the method's arithmetic (no Philox, no value maps, no Eq. 1), so both the
CUDA library's binding and the CPU oracle's wrapper can consume the same
descriptions while sharing no code with each other.

Names are strings; each side maps them onto its own enumerations:
  dtypes        f32 f16 bf16 i32 i64 u32
  dists         uniform normal int_range permutation dotlike raw_bits constant from_arena
  special kinds nan pinf ninf denorm zero imin imax dup
  perturbations none rate_add_pm rel_noise count_set count_add swap_pairs

The five workloads follow the paper's synthesis-based verification setting
(CUDA-Harness Sec. 4.2): broad-range inputs (Sec. 4.2.1), Eq. 1 tolerances,
and a size-ascending progressive ladder (Sec. 4.2.2).
"""
from __future__ import annotations

import dataclasses
import math
from dataclasses import dataclass, field
from typing import List, Optional, Sequence, Tuple

import numpy as np

DTYPE_BYTES = {"f32": 4, "f16": 2, "bf16": 2, "i32": 4, "i64": 8, "u32": 4}
FLOAT_DTYPES = ("f32", "f16", "bf16")
INT_DTYPES = ("i32", "i64", "u32")
ALIGN = 256  # arena offsets are aligned well beyond the 16-byte requirement


@dataclass
class Perturb:
    kind: str = "none"
    stream: int = 0
    rate: float = 0.0
    count: int = 0
    value: float = 0.0
    ivalue: int = 0


@dataclass
class GenSpec:
    dtype: str
    dist: str
    n: int
    seed: int = 0
    stream: int = 0
    ref_offset: Optional[int] = None
    cand_offset: Optional[int] = None
    elem_offset: int = 0
    logical_n: int = 0
    p0: float = 0.0
    p1: float = 0.0
    i0: int = 0
    i1: int = 0
    specials: Tuple[str, ...] = ()
    special_rate: float = 0.0
    special_exact: bool = False  # exactly round(rate * N) specials, one per stratum
    rows: int = 0
    cols: int = 0
    dot_k: int = 0
    a_offset: int = 0
    b_offset: int = 0
    pelem: Perturb = field(default_factory=Perturb)
    pcount: Perturb = field(default_factory=Perturb)

    def replace(self, **kw) -> "GenSpec":
        return dataclasses.replace(self, **kw)


@dataclass
class Pair:
    dtype: str
    n: int
    cand_offset: int
    ref_offset: int
    atol: float = 0.0
    rtol: float = 0.0
    equal_nan: bool = True


@dataclass
class Tiles:
    """A 2-D output (rows x cols elements, row-major) compared tile by tile;
    each operand has its own row pitch (elements between row starts).  Zero
    pitches and a zero tile_cols mean cols."""
    dtype: str
    rows: int
    cols: int
    cand_offset: int
    ref_offset: int
    cand_pitch: int = 0
    ref_pitch: int = 0
    tile_rows: int = 1
    tile_cols: int = 0
    atol: float = 0.0
    rtol: float = 0.0
    equal_nan: bool = True

    def __post_init__(self):
        self.cand_pitch = self.cand_pitch or self.cols
        self.ref_pitch = self.ref_pitch or self.cols
        self.tile_cols = self.tile_cols or self.cols


class Arena:
    """Bump allocator for byte offsets inside one arena."""

    def __init__(self) -> None:
        self.size = 0

    def take(self, nbytes: int) -> int:
        off = self.size
        self.size = off + ((nbytes + ALIGN - 1) // ALIGN) * ALIGN
        return off


@dataclass
class Workload:
    """One verification job: generator calls (run in order), then compare pairs."""

    name: str
    gen_calls: List[List[GenSpec]]
    pairs: List[Pair]
    arena_bytes: int
    progressive: bool = False

    def synth_bytes(self) -> int:
        """Bytes the generator writes (every output of every spec)."""
        tot = 0
        for call in self.gen_calls:
            for s in call:
                outs = (s.ref_offset is not None) + (s.cand_offset is not None)
                tot += outs * s.n * DTYPE_BYTES[s.dtype]
        return tot

    def verify_bytes(self, stages_run: Optional[int] = None) -> int:
        """Candidate + reference bytes read by the compare (first stages_run pairs)."""
        ps = self.pairs if stages_run is None else self.pairs[:stages_run]
        return sum(2 * p.n * DTYPE_BYTES[p.dtype] for p in ps)


# ---------------------------------------------------------------------------
# the five workloads
# ---------------------------------------------------------------------------

def single_fp32_pair(n: int = 1 << 20) -> Workload:
    """fp32 pair: reference ~U[-1,1) (seed 1); candidate = reference with
    0.1% Bernoulli-selected elements moved by +-1e-3 and 3 elements set to
    NaN; atol = rtol = 1e-5."""
    ar = Arena()
    ref, cand = ar.take(4 * n), ar.take(4 * n)
    spec = GenSpec("f32", "uniform", n, seed=1, stream=0, ref_offset=ref, cand_offset=cand,
                   p0=-1.0, p1=1.0,
                   pelem=Perturb("rate_add_pm", stream=1, rate=1e-3, value=1e-3),
                   pcount=Perturb("count_set", stream=2, count=3, value=float("nan")))
    pair = Pair("f32", n, cand, ref, atol=1e-5, rtol=1e-5)
    return Workload("single fp32 pair n=%d" % n, [[spec]], [pair], ar.size)


LADDER_EXPONENTS = (10, 14, 18, 22, 25, 27)


def progressive_ladder(exponents: Sequence[int] = LADDER_EXPONENTS, deviate_stage: Optional[int] = 3,
                       special_rate: float = 1e-4) -> Workload:
    """Size-ascending ladder of fp32 N(0,1) stages (seed 7, stream = stage),
    0.01% injected NaN/+Inf/-Inf/denormal (exactly round(1e-4 N) of them per
    stage, one per stratum); the candidate equals the reference
    except for one element moved by +1e-2 at stage `deviate_stage` (0-based),
    so validation stops there.  atol = rtol = 1e-5."""
    ar = Arena()
    specs, pairs = [], []
    for s, e in enumerate(exponents):
        n = 1 << e
        ref, cand = ar.take(4 * n), ar.take(4 * n)
        pc = Perturb("count_add", stream=100 + s, count=1, value=1e-2) if s == deviate_stage else Perturb()
        specs.append(GenSpec("f32", "normal", n, seed=7, stream=s, ref_offset=ref, cand_offset=cand,
                             p0=0.0, p1=1.0, specials=("nan", "pinf", "ninf", "denorm"),
                             special_rate=special_rate, special_exact=True, pcount=pc))
        pairs.append(Pair("f32", n, cand, ref, atol=1e-5, rtol=1e-5))
    name = "progressive ladder n=2^{%s} fp32 N(0,1)" % ",".join(str(e) for e in exponents)
    return Workload(name, [specs], pairs, ar.size, progressive=True)


def segmented_cases(n_cases: int = 4096, max_n: int = 65536, seed: int = 3) -> Workload:
    """Many small cases: sizes log-uniform in [1, max_n], dtypes cycling
    f32/f16/bf16/i32, values U[-100,100) (ints: [-100,100]); atol = rtol =
    1e-3 for floats, exact for int32; 5% of cases carry one +1 mismatch.
    Sizes and the 5% selection are drawn with numpy's PCG64 (seed `seed`)."""
    rng = np.random.default_rng(seed)
    u = rng.random(n_cases)
    sizes = np.clip(np.floor(np.exp(u * math.log(max_n + 1))), 1, max_n).astype(np.int64)
    hit = rng.random(n_cases) < 0.05
    dts = ("f32", "f16", "bf16", "i32")
    ar = Arena()
    specs, pairs = [], []
    for i in range(n_cases):
        dt, n = dts[i % 4], int(sizes[i])
        nb = n * DTYPE_BYTES[dt]
        ref, cand = ar.take(nb), ar.take(nb)
        pc = Perturb("count_add", stream=10000 + i, count=1, value=1.0, ivalue=1) if hit[i] else Perturb()
        if dt == "i32":
            s = GenSpec(dt, "int_range", n, seed=seed, stream=i, ref_offset=ref, cand_offset=cand,
                        i0=-100, i1=100, pcount=pc)
            pairs.append(Pair(dt, n, cand, ref))
        else:
            s = GenSpec(dt, "uniform", n, seed=seed, stream=i, ref_offset=ref, cand_offset=cand,
                        p0=-100.0, p1=100.0, pcount=pc)
            pairs.append(Pair(dt, n, cand, ref, atol=1e-3, rtol=1e-3))
        specs.append(s)
    return Workload("%d segmented cases, log-uniform sizes in [1,%d]" % (n_cases, max_n), [specs], pairs, ar.size)


def dotlike_bf16_pair(rows: int = 32768, cols: int = 32768, k: int = 64, seed: int = 4) -> Workload:
    """bf16 pair of GEMM-shaped values: ref[i,j] = sum_k A[i,k] B[k,j] in fp32
    (k in order, fused multiply-add) rounded to bf16, A and B ~ N(0,1)/8;
    candidate = reference + N(0, (2^-9 |ref|)^2) noise; atol = rtol = 1e-2.
    First call generates A and B (fp32), the second the pair."""
    ar = Arena()
    a_off, b_off = ar.take(4 * rows * k), ar.take(4 * k * cols)
    n = rows * cols
    ref, cand = ar.take(2 * n), ar.take(2 * n)
    fa = GenSpec("f32", "normal", rows * k, seed=seed, stream=0, ref_offset=a_off, p0=0.0, p1=0.125)
    fb = GenSpec("f32", "normal", k * cols, seed=seed, stream=1, ref_offset=b_off, p0=0.0, p1=0.125)
    d = GenSpec("bf16", "dotlike", n, seed=seed, stream=2, ref_offset=ref, cand_offset=cand,
                rows=rows, cols=cols, dot_k=k, a_offset=a_off, b_offset=b_off,
                pelem=Perturb("rel_noise", stream=3, value=2.0 ** -9))
    pair = Pair("bf16", n, cand, ref, atol=1e-2, rtol=1e-2)
    return Workload("bf16 pair %dx%d dot-like K=%d" % (rows, cols, k), [[fa, fb], [d]], [pair], ar.size)


def int64_permutation_pair(n: int = 1 << 28, seed: int = 5, swaps: int = 17) -> Workload:
    """int64 pair for index outputs: reference = seeded permutation of [0, n)
    with 0.01% duplicates / 0 / INT64_MIN / INT64_MAX injected; candidate =
    reference with `swaps` seeded pairs of elements exchanged; exact compare."""
    ar = Arena()
    ref, cand = ar.take(8 * n), ar.take(8 * n)
    spec = GenSpec("i64", "permutation", n, seed=seed, stream=0, ref_offset=ref, cand_offset=cand,
                   specials=("dup", "zero", "imin", "imax"), special_rate=1e-4,
                   pcount=Perturb("swap_pairs", stream=1, count=swaps))
    pair = Pair("i64", n, cand, ref)
    return Workload("int64 permutation pair n=%d, %d swaps" % (n, swaps), [[spec]], [pair], ar.size)


FULL_SIZE = {
    "fp32_pair": single_fp32_pair,
    "ladder": progressive_ladder,
    "segmented": segmented_cases,
    "dotlike_bf16": dotlike_bf16_pair,
    "perm_i64": int64_permutation_pair,
}


# ---------------------------------------------------------------------------
# seeded compare inputs (numpy PCG64), for parity of the compare alone
# ---------------------------------------------------------------------------

def _f32_to_bf16_truncate(x: np.ndarray) -> np.ndarray:
    """bf16 bit patterns by dropping the low 16 bits (input synthesis only)."""
    return (np.ascontiguousarray(x, dtype=np.float32).view(np.uint32) >> 16).astype(np.uint16)


def random_pair_arrays(dtype: str, n: int, seed: int, scale: float = 10.0, mismatch_frac: float = 1e-3,
                       nonfinite_frac: float = 1e-3) -> Tuple[np.ndarray, np.ndarray]:
    """(cand_bytes, ref_bytes) uint8 arrays of one pair: ref ~ N(0, scale^2)
    (ints: uniform in +-2^30 / +-2^62), cand = ref with a fraction of elements
    nudged by a few ulps, some moved far, and NaN/Inf/denormal/zero patterns
    planted on either side."""
    rng = np.random.default_rng(seed)
    if dtype in FLOAT_DTYPES:
        ref = (rng.standard_normal(n) * scale).astype(np.float32)
        if dtype == "f32":
            rb = ref.view(np.uint32).copy()
        elif dtype == "f16":
            rb = ref.astype(np.float16).view(np.uint16).copy()
        else:
            rb = _f32_to_bf16_truncate(ref)
        cb = rb.copy()
        m = rng.random(n)
        # small nudges of the bit pattern (a few ulps either way)
        near = m < mismatch_frac * 4
        step = rng.integers(-3, 4, size=n).astype(np.int64)
        cb[near] = (cb[near].astype(np.int64) + step[near]).astype(cb.dtype)
        # far moves: flip a high mantissa bit
        far = m > 1 - mismatch_frac
        hb = 1 << (22 if dtype == "f32" else (9 if dtype == "f16" else 6))
        cb[far] ^= cb.dtype.type(hb)
        # non-finite and tiny patterns on either side
        pats = {"f32": [0x7FC00000, 0x7F800000, 0xFF800000, 0x00000001, 0x80000000, 0x00000000],
                "f16": [0x7E00, 0x7C00, 0xFC00, 0x0001, 0x8000, 0x0000],
                "bf16": [0x7FC0, 0x7F80, 0xFF80, 0x0001, 0x8000, 0x0000]}[dtype]
        for arr in (cb, rb):
            sel = np.nonzero(rng.random(n) < nonfinite_frac)[0]
            arr[sel] = np.array(pats, dtype=np.uint64)[rng.integers(0, len(pats), size=sel.size)].astype(arr.dtype)
        return cb.view(np.uint8), rb.view(np.uint8)
    if dtype == "i64":
        ref = rng.integers(-(1 << 62), 1 << 62, size=n, dtype=np.int64)
        lim = np.array([np.iinfo(np.int64).min, np.iinfo(np.int64).max, 0], dtype=np.int64)
    elif dtype == "i32":
        ref = rng.integers(-(1 << 30), 1 << 30, size=n, dtype=np.int64).astype(np.int32)
        lim = np.array([np.iinfo(np.int32).min, np.iinfo(np.int32).max, 0], dtype=np.int32)
    else:
        ref = rng.integers(0, 1 << 32, size=n, dtype=np.int64).astype(np.uint32)
        lim = np.array([0, np.iinfo(np.uint32).max, 1], dtype=np.uint32)
    cand = ref.copy()
    sel = np.nonzero(rng.random(n) < mismatch_frac)[0]
    cand[sel] = cand[sel] + ref.dtype.type(1)
    for arr in (cand, ref):
        s2 = np.nonzero(rng.random(n) < nonfinite_frac)[0]
        arr[s2] = lim[rng.integers(0, lim.size, size=s2.size)]
    return cand.view(np.uint8), ref.view(np.uint8)


def random_bits_pair(dtype: str, n: int, seed: int, n_changes: int) -> Tuple[np.ndarray, np.ndarray]:
    """(cand_bytes, ref_bytes): ref = uniformly random bit patterns of the
    dtype (every class of value: normals, denormals, zeros, infinities,
    NaNs), cand = ref with `n_changes` random elements given new random bits
    and as many nudged by one unit in the last place.  Cheap at any size."""
    rng = np.random.default_rng(seed)
    t = {2: np.uint16, 4: np.uint32, 8: np.uint64}[DTYPE_BYTES[dtype]]
    ref = rng.integers(0, np.iinfo(t).max, size=n, dtype=t, endpoint=True)
    cand = ref.copy()
    idx = rng.integers(0, n, size=n_changes)
    cand[idx] = rng.integers(0, np.iinfo(t).max, size=n_changes, dtype=t, endpoint=True)
    idx2 = rng.integers(0, n, size=n_changes)
    cand[idx2] = cand[idx2] + t(1)
    return cand.view(np.uint8), ref.view(np.uint8)
