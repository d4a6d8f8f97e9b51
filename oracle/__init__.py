"""ctypes wrapper of the CPU oracle (oracle.c).

TEST INFRASTRUCTURE ONLY: imported by tests/, by the package's smoke check
and by bench.py's CPU-baseline / reference arm.  The product path never
imports it.  Specs and pairs are the neutral descriptions of `workloads.py`
(any object with the same attribute names works); names are mapped onto the
oracle's own enumerations here.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
from typing import List, Sequence, Tuple

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "oracle.c")
SRCS = [SRC, os.path.join(HERE, "convert.c"), os.path.join(HERE, "threads.c")]
HDR = os.path.join(HERE, "oracle.h")
LIB = os.path.join(HERE, "_build", "liboracle.so")
CFLAGS = ["-O2", "-std=c11", "-Wall", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared", "-pthread"]

DTYPES = {"f32": 0, "f16": 1, "bf16": 2, "i32": 3, "i64": 4, "u32": 5}
DTYPE_BYTES = {"f32": 4, "f16": 2, "bf16": 2, "i32": 4, "i64": 8, "u32": 4}
DISTS = {"uniform": 0, "normal": 1, "int_range": 2, "permutation": 3, "dotlike": 4, "raw_bits": 5,
         "constant": 6, "from_arena": 7}
SPECIALS = {"nan": 1, "pinf": 2, "ninf": 4, "denorm": 8, "zero": 16, "imin": 32, "imax": 64, "dup": 128}
SPECIAL_EXACT = 1 << 31
PERTS = {"none": 0, "rate_add_pm": 1, "rel_noise": 2, "count_set": 3, "count_add": 4, "swap_pairs": 5}
PURPOSES = {"value": 0, "special_sel": 1, "special_kind": 2, "pert_sel": 3, "pert_val": 4, "index": 5,
            "perm": 6, "noise": 7}
# element types of test-data files: the six array types and six more
IO_DTYPES = dict(DTYPES, u8=6, i8=7, i16=8, u16=9, u64=10, f64=11)
IO_DTYPE_BYTES = dict(DTYPE_BYTES, u8=1, i8=1, i16=2, u16=2, u64=8, f64=8)
ABSENT = (1 << 64) - 1
STAGE_RUN, STAGE_SKIPPED = 1, 2


def build(force: bool = False) -> str:
    """Compile liboracle.so with gcc (seconds)."""
    os.makedirs(os.path.dirname(LIB), exist_ok=True)
    newest = max(os.path.getmtime(f) for f in SRCS + [HDR])
    if force or not os.path.exists(LIB) or os.path.getmtime(LIB) < newest:
        tmp = LIB + ".%d.tmp" % os.getpid()
        subprocess.check_call(["gcc", *CFLAGS, "-o", tmp, *SRCS, "-lm", "-lpthread"])
        os.replace(tmp, LIB)
    return LIB


class Perturb(C.Structure):
    _fields_ = [("kind", C.c_uint32), ("stream", C.c_uint32), ("rate", C.c_double), ("count", C.c_uint64),
                ("value", C.c_double), ("ivalue", C.c_int64)]


class Spec(C.Structure):
    _fields_ = [("dtype", C.c_uint32), ("dist", C.c_uint32), ("n", C.c_uint64), ("seed", C.c_uint64),
                ("stream", C.c_uint32), ("special_mask", C.c_uint32), ("special_rate", C.c_double),
                ("ref_offset", C.c_uint64), ("cand_offset", C.c_uint64), ("elem_offset", C.c_uint64),
                ("logical_n", C.c_uint64), ("p0", C.c_double), ("p1", C.c_double), ("i0", C.c_int64),
                ("i1", C.c_int64), ("rows", C.c_uint64), ("cols", C.c_uint64), ("dot_k", C.c_uint64),
                ("a_offset", C.c_uint64), ("b_offset", C.c_uint64), ("pelem", Perturb), ("pcount", Perturb)]


class PairC(C.Structure):
    _fields_ = [("dtype", C.c_uint32), ("flags", C.c_uint32), ("n", C.c_uint64), ("cand_offset", C.c_uint64),
                ("ref_offset", C.c_uint64), ("atol", C.c_double), ("rtol", C.c_double)]


class TilesC(C.Structure):
    _fields_ = [("dtype", C.c_uint32), ("flags", C.c_uint32), ("rows", C.c_uint64), ("cols", C.c_uint64),
                ("cand_offset", C.c_uint64), ("ref_offset", C.c_uint64), ("cand_pitch", C.c_uint64),
                ("ref_pitch", C.c_uint64), ("tile_rows", C.c_uint64), ("tile_cols", C.c_uint64),
                ("atol", C.c_double), ("rtol", C.c_double)]


class Result(C.Structure):
    _fields_ = [("mismatches", C.c_uint64), ("nan_disagree", C.c_uint64), ("inf_disagree", C.c_uint64),
                ("n_finite", C.c_uint64), ("first_mismatch", C.c_int64), ("max_abs_u64", C.c_uint64),
                ("max_abs", C.c_double), ("max_rel", C.c_double), ("rms", C.c_double), ("pass_", C.c_uint32),
                ("state", C.c_uint32)]


_lib = None


def lib() -> C.CDLL:
    global _lib
    if _lib is None:
        L = C.CDLL(build())
        u32p, u16p, f32p, u64p = (C.POINTER(C.c_uint32), C.POINTER(C.c_uint16), C.POINTER(C.c_float),
                                  C.POINTER(C.c_uint64))
        L.or_philox4x32_10.argtypes = [u32p, u32p, u32p]
        L.or_draw.argtypes = [C.c_uint64, C.c_uint32, C.c_uint32, C.c_uint64, u32p]
        L.or_f32_to_bf16.argtypes = [C.c_float]
        L.or_f32_to_bf16.restype = C.c_uint16
        L.or_f32_to_f16.argtypes = [C.c_float]
        L.or_f32_to_f16.restype = C.c_uint16
        L.or_bf16_to_f32.argtypes = [C.c_uint16]
        L.or_bf16_to_f32.restype = C.c_float
        L.or_f16_to_f32.argtypes = [C.c_uint16]
        L.or_f16_to_f32.restype = C.c_float
        L.or_uniform_map.argtypes = [C.c_float, C.c_float, C.c_uint32]
        L.or_uniform_map.restype = C.c_float
        L.or_box_muller.argtypes = [C.c_uint32, C.c_uint32, f32p, f32p]
        L.or_int_range_map32.argtypes = [C.c_int64, C.c_uint64, C.c_uint32]
        L.or_int_range_map32.restype = C.c_int64
        L.or_perm_value.argtypes = [C.c_uint64, C.c_uint64, C.c_uint32, C.c_uint64]
        L.or_perm_value.restype = C.c_uint64
        L.or_stratum_index.argtypes = [C.c_uint64, C.c_uint64, C.c_uint64, C.c_uint32, C.c_uint64]
        L.or_stratum_index.restype = C.c_uint64
        L.or_special_count.argtypes = [C.c_double, C.c_uint64]
        L.or_special_count.restype = C.c_uint64
        L.or_special_index.argtypes = [C.c_uint64, C.c_uint64, C.c_uint64, C.c_uint32, C.c_uint64]
        L.or_special_index.restype = C.c_uint64
        L.or_stratum_of.argtypes = [C.c_uint64, C.c_uint64, C.c_uint64]
        L.or_stratum_of.restype = C.c_uint64
        L.or_map_uniform.argtypes = [C.c_float, C.c_float, u32p, C.c_uint64, f32p]
        L.or_map_box_muller.argtypes = [u32p, C.c_uint64, f32p]
        L.or_map_f32_to_bf16.argtypes = [f32p, C.c_uint64, u16p]
        L.or_map_f32_to_f16.argtypes = [f32p, C.c_uint64, u16p]
        L.or_int_range_histogram.argtypes = [C.c_uint64, u64p]
        L.or_map_perm.argtypes = [C.c_uint64, C.c_uint64, C.c_uint32, C.c_uint64, C.c_uint64, u64p]
        L.or_check_spec.argtypes = [C.POINTER(Spec), C.c_uint64]
        L.or_check_spec.restype = C.c_int
        L.or_value_at.argtypes = [C.POINTER(Spec), C.c_void_p, C.c_uint64, C.c_int]
        L.or_value_at.restype = C.c_uint64
        L.or_generate.argtypes = [C.POINTER(Spec), C.c_int, C.c_void_p, C.c_uint64]
        L.or_generate.restype = C.c_int
        L.or_compare.argtypes = [C.POINTER(PairC), C.c_int, C.c_void_p, C.c_uint64, C.c_void_p, C.c_uint64,
                                 C.POINTER(Result)]
        L.or_compare.restype = C.c_int
        L.or_progressive.argtypes = [C.POINTER(PairC), C.c_int, C.c_void_p, C.c_uint64, C.c_void_p,
                                     C.c_uint64, C.POINTER(Result), C.POINTER(C.c_int32)]
        L.or_progressive.restype = C.c_int
        L.or_compare_sums.argtypes = [C.POINTER(PairC), C.c_int, C.c_void_p, C.c_uint64, C.c_void_p,
                                      C.c_uint64, C.POINTER(Result), C.POINTER(C.c_double)]
        L.or_compare_sums.restype = C.c_int
        L.or_check_pair.argtypes = [C.POINTER(PairC), C.c_uint64, C.c_uint64]
        L.or_check_pair.restype = C.c_int
        L.or_threads_default.argtypes = []
        L.or_threads_default.restype = C.c_int
        L.or_generate_mt.argtypes = [C.POINTER(Spec), C.c_int, C.c_void_p, C.c_uint64, C.c_int]
        L.or_generate_mt.restype = C.c_int
        L.or_compare_mt.argtypes = [C.POINTER(PairC), C.c_int, C.c_void_p, C.c_uint64, C.c_void_p, C.c_uint64,
                                    C.POINTER(Result), C.c_int]
        L.or_compare_mt.restype = C.c_int
        L.or_progressive_mt.argtypes = [C.POINTER(PairC), C.c_int, C.c_void_p, C.c_uint64, C.c_void_p,
                                        C.c_uint64, C.POINTER(Result), C.POINTER(C.c_int32), C.c_int]
        L.or_progressive_mt.restype = C.c_int
        L.or_compare_tiles.argtypes = [C.POINTER(TilesC), C.c_void_p, C.c_uint64, C.c_void_p, C.c_uint64,
                                       C.POINTER(Result)]
        L.or_compare_tiles.restype = C.c_int
        L.or_dtype_bytes.argtypes = [C.c_int]
        L.or_dtype_bytes.restype = C.c_int
        L.or_convert.argtypes = [C.c_int, C.c_void_p, C.c_uint64, C.c_int, C.c_void_p, u64p]
        L.or_convert.restype = C.c_int
        _lib = L
    return _lib


def _ptr(a: np.ndarray, ct):
    return a.ctypes.data_as(C.POINTER(ct))


# ---------------------------------------------------------------------------
# primitives
# ---------------------------------------------------------------------------

def philox(ctr: Sequence[int], key: Sequence[int]) -> List[int]:
    c = (C.c_uint32 * 4)(*[x & 0xFFFFFFFF for x in ctr])
    k = (C.c_uint32 * 2)(*[x & 0xFFFFFFFF for x in key])
    o = (C.c_uint32 * 4)()
    lib().or_philox4x32_10(c, k, o)
    return list(o)


def draw(seed: int, stream: int, purpose: str, block: int) -> List[int]:
    o = (C.c_uint32 * 4)()
    lib().or_draw(seed, stream, PURPOSES[purpose], block, o)
    return list(o)


def f32_to_bf16(x: np.ndarray) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float32)
    out = np.empty(x.shape, dtype=np.uint16)
    lib().or_map_f32_to_bf16(_ptr(x, C.c_float), x.size, _ptr(out, C.c_uint16))
    return out


def f32_to_f16(x: np.ndarray) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float32)
    out = np.empty(x.shape, dtype=np.uint16)
    lib().or_map_f32_to_f16(_ptr(x, C.c_float), x.size, _ptr(out, C.c_uint16))
    return out


def bf16_to_f32(h: int) -> float:
    return lib().or_bf16_to_f32(h)


def f16_to_f32(h: int) -> float:
    return lib().or_f16_to_f32(h)


def uniform_map(a: float, b: float, words: np.ndarray) -> np.ndarray:
    w = np.ascontiguousarray(words, dtype=np.uint32)
    out = np.empty(w.shape, dtype=np.float32)
    lib().or_map_uniform(a, b, _ptr(w, C.c_uint32), w.size, _ptr(out, C.c_float))
    return out


def box_muller(words: np.ndarray) -> np.ndarray:
    """words: uint32 array of even length (pairs); returns z0,z1 per pair."""
    w = np.ascontiguousarray(words, dtype=np.uint32)
    out = np.empty(w.shape, dtype=np.float32)
    lib().or_map_box_muller(_ptr(w, C.c_uint32), w.size // 2, _ptr(out, C.c_float))
    return out


def int_range_map32(lo: int, r: int, w: int) -> int:
    return lib().or_int_range_map32(lo, r, w)


def int_range_histogram(r: int) -> np.ndarray:
    counts = np.zeros(r, dtype=np.uint64)
    lib().or_int_range_histogram(r, _ptr(counts, C.c_uint64))
    return counts


def perm_value(N: int, seed: int, stream: int, g: int) -> int:
    return lib().or_perm_value(N, seed, stream, g)


def perm_values(N: int, seed: int, stream: int, g0: int, n: int) -> np.ndarray:
    out = np.empty(n, dtype=np.uint64)
    lib().or_map_perm(N, seed, stream, g0, n, _ptr(out, C.c_uint64))
    return out


def stratum_index(N: int, k: int, seed: int, stream: int, s: int) -> int:
    return lib().or_stratum_index(N, k, seed, stream, s)


def special_count(rate: float, N: int) -> int:
    return lib().or_special_count(rate, N)


def special_index(N: int, k: int, seed: int, stream: int, s: int) -> int:
    return lib().or_special_index(N, k, seed, stream, s)


def stratum_of(g: int, k: int, N: int) -> int:
    return lib().or_stratum_of(g, k, N)


# ---------------------------------------------------------------------------
# marshalling of the neutral descriptions
# ---------------------------------------------------------------------------

def _perturb(p) -> Perturb:
    return Perturb(PERTS[p.kind], p.stream, p.rate, p.count, p.value, p.ivalue)


def to_spec(s) -> Spec:
    mask = SPECIAL_EXACT if getattr(s, "special_exact", False) else 0
    for k in s.specials:
        mask |= SPECIALS[k]
    return Spec(DTYPES[s.dtype], DISTS[s.dist], s.n, s.seed, s.stream, mask, s.special_rate,
                ABSENT if s.ref_offset is None else s.ref_offset,
                ABSENT if s.cand_offset is None else s.cand_offset,
                s.elem_offset, s.logical_n, s.p0, s.p1, s.i0, s.i1, s.rows, s.cols, s.dot_k,
                s.a_offset, s.b_offset, _perturb(s.pelem), _perturb(s.pcount))


def to_pair(p) -> PairC:
    return PairC(DTYPES[p.dtype], 1 if p.equal_nan else 0, p.n, p.cand_offset, p.ref_offset, p.atol, p.rtol)


def result_dict(r: Result) -> dict:
    return {"mismatches": r.mismatches, "nan_disagree": r.nan_disagree, "inf_disagree": r.inf_disagree,
            "n_finite": r.n_finite, "first_mismatch": r.first_mismatch, "max_abs_u64": r.max_abs_u64,
            "max_abs": r.max_abs, "max_rel": r.max_rel, "rms": r.rms, "pass": r.pass_, "state": r.state}


def check_spec(spec, arena_bytes: int) -> int:
    s = to_spec(spec)
    return lib().or_check_spec(C.byref(s), arena_bytes)


def threads_default() -> int:
    """Online host cores (the thread count of threads=0)."""
    return lib().or_threads_default()


def generate(specs, arena: np.ndarray, threads: int = 1) -> None:
    """Run the specs into `arena` (uint8 numpy array, modified in place); the
    specs of one call are independent.  threads != 1: the multi-threaded
    driver (same bytes; 0 = every host core)."""
    assert arena.dtype == np.uint8 and arena.flags.c_contiguous
    arr = (Spec * max(len(specs), 1))(*[to_spec(s) for s in specs])
    if threads == 1:
        rc = lib().or_generate(arr, len(specs), arena.ctypes.data, arena.size)
    else:
        rc = lib().or_generate_mt(arr, len(specs), arena.ctypes.data, arena.size, threads)
    if rc != 0:
        raise ValueError("oracle: invalid generator spec")


def value_at(spec, arena: np.ndarray, g: int, role: int) -> int:
    s = to_spec(spec)
    return lib().or_value_at(C.byref(s), arena.ctypes.data, g, role)


def compare(pairs, cand: np.ndarray, ref: np.ndarray, threads: int = 1) -> List[dict]:
    """Eq. 1 verdicts per pair; threads != 1: the multi-threaded driver
    (integer fields identical, rms up to the order of its sum)."""
    arr = (PairC * max(len(pairs), 1))(*[to_pair(p) for p in pairs])
    out = (Result * max(len(pairs), 1))()
    if threads == 1:
        rc = lib().or_compare(arr, len(pairs), cand.ctypes.data, cand.nbytes, ref.ctypes.data, ref.nbytes, out)
    else:
        rc = lib().or_compare_mt(arr, len(pairs), cand.ctypes.data, cand.nbytes, ref.ctypes.data, ref.nbytes,
                                 out, threads)
    if rc != 0:
        raise ValueError("oracle: invalid compare pair")
    return [result_dict(r) for r in out][:len(pairs)]


def compare_sums(pairs, cand: np.ndarray, ref: np.ndarray) -> Tuple[List[dict], List[float]]:
    """compare() plus each pair's sum of squared differences (index order)."""
    arr = (PairC * max(len(pairs), 1))(*[to_pair(p) for p in pairs])
    out = (Result * max(len(pairs), 1))()
    sums = (C.c_double * max(len(pairs), 1))()
    rc = lib().or_compare_sums(arr, len(pairs), cand.ctypes.data, cand.nbytes, ref.ctypes.data, ref.nbytes, out,
                               sums)
    if rc != 0:
        raise ValueError("oracle: invalid compare pair")
    return [result_dict(r) for r in out][:len(pairs)], list(sums)[:len(pairs)]


def progressive(stages, cand: np.ndarray, ref: np.ndarray, threads: int = 1) -> Tuple[List[dict], int]:
    arr = (PairC * max(len(stages), 1))(*[to_pair(p) for p in stages])
    out = (Result * max(len(stages), 1))()
    ff = C.c_int32(0)
    if threads == 1:
        rc = lib().or_progressive(arr, len(stages), cand.ctypes.data, cand.nbytes, ref.ctypes.data, ref.nbytes,
                                  out, C.byref(ff))
    else:
        rc = lib().or_progressive_mt(arr, len(stages), cand.ctypes.data, cand.nbytes, ref.ctypes.data,
                                     ref.nbytes, out, C.byref(ff), threads)
    if rc != 0:
        raise ValueError("oracle: invalid stage")
    return [result_dict(r) for r in out][:len(stages)], ff.value


def run_workload(wl, arena: np.ndarray = None, threads: int = 1):
    """Generate every call of a workload, then verify; returns (arena, results, first_failed)."""
    if arena is None:
        arena = np.zeros(wl.arena_bytes, dtype=np.uint8)
    for call in wl.gen_calls:
        generate(call, arena, threads=threads)
    if wl.progressive:
        res, ff = progressive(wl.pairs, arena, arena, threads=threads)
        return arena, res, ff
    return arena, compare(wl.pairs, arena, arena, threads=threads), None


def convert(src: np.ndarray, src_dtype: str, dst_dtype: str) -> Tuple[np.ndarray, int]:
    """Dtype-correct value conversion of `src` (its bytes are read as
    `src_dtype` elements): returns (destination bytes as uint8, number of
    clamped / overflowed elements).  Raises ValueError for a refused pair
    (float to integer)."""
    raw = np.ascontiguousarray(src).view(np.uint8).reshape(-1)
    sb, db = IO_DTYPE_BYTES[src_dtype], IO_DTYPE_BYTES[dst_dtype]
    assert raw.size % sb == 0
    n = raw.size // sb
    out = np.zeros(n * db, np.uint8)
    bad = C.c_uint64(0)
    rc = lib().or_convert(IO_DTYPES[src_dtype], raw.ctypes.data, n, IO_DTYPES[dst_dtype], out.ctypes.data,
                          C.byref(bad))
    if rc != 0:
        raise ValueError("conversion %s -> %s refused" % (src_dtype, dst_dtype))
    return out, bad.value


def tile_grid(t) -> Tuple[int, int]:
    return (-(-t.rows // t.tile_rows), -(-t.cols // t.tile_cols))


def compare_tiles(t, cand: np.ndarray, ref: np.ndarray) -> List[dict]:
    """Tile-by-tile verdicts of a shaped output `t` (any object with the
    fields of workloads.Tiles), row-major over the tile grid."""
    tr, tc = tile_grid(t)
    n = tr * tc
    out = (Result * max(n, 1))()
    c = TilesC(DTYPES[t.dtype], 1 if t.equal_nan else 0, t.rows, t.cols, t.cand_offset, t.ref_offset,
               t.cand_pitch, t.ref_pitch, t.tile_rows, t.tile_cols, t.atol, t.rtol)
    rc = lib().or_compare_tiles(C.byref(c), cand.ctypes.data, cand.nbytes, ref.ctypes.data, ref.nbytes, out)
    if rc != 0:
        raise ValueError("invalid tiles")
    return [result_dict(out[i]) for i in range(n)]
