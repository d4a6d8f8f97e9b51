"""Python binding of libsynverify (include/synverify.h): argument marshalling only.

GB300 (sm_103a) implementation of the data-parallel path of Synthesis-Based
Verification (CUDA-Harness, Sec. 4.2):

  generate(specs, arena)            syn_generate: seeded test-data synthesis
  compare(pairs, cand, ref)         verify_compare: Eq. 1 per segment
  progressive(stages, cand, ref)    verify_progressive: fail-fast stage ladder

Device memory and streams come from PyTorch (tensors are passed by
data_ptr(); the current CUDA stream is used unless one is given).  Every step
of the path runs in the library's CUDA kernels; there is no CPU fallback: if
the compiled library is missing, importing works but every call raises.

Specs and pairs are any objects with the attribute names of `GenSpec`,
`Perturb` and `Pair` below (string-valued enums).
"""
from __future__ import annotations

import ctypes as C
import os
from dataclasses import dataclass, field
from typing import List, Optional, Sequence, Tuple

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "_build", "libsynverify.so")

DTYPES = {"f32": 0, "f16": 1, "bf16": 2, "i32": 3, "i64": 4, "u32": 5}
DTYPE_BYTES = {"f32": 4, "f16": 2, "bf16": 2, "i32": 4, "i64": 8, "u32": 4}
DISTS = {"uniform": 0, "normal": 1, "int_range": 2, "permutation": 3, "dotlike": 4, "raw_bits": 5,
         "constant": 6, "from_arena": 7}
SPECIALS = {"nan": 1, "pinf": 2, "ninf": 4, "denorm": 8, "zero": 16, "imin": 32, "imax": 64, "dup": 128}
SPECIAL_EXACT = 1 << 31
PERTS = {"none": 0, "rate_add_pm": 1, "rel_noise": 2, "count_set": 3, "count_add": 4, "swap_pairs": 5}
EQUAL_NAN = 1
STAGE_RUN, STAGE_SKIPPED = 1, 2
NO_OUTPUT = (1 << 64) - 1
INLINE_ENTRIES = 8
STATUS = {0: "SV_OK", -1: "SV_EINVAL", -2: "SV_EALIGN", -3: "SV_ERANGE", -4: "SV_EWORKSPACE", -5: "SV_ECUDA",
          -6: "SV_EIO", -7: "SV_EFORMAT", -8: "SV_ELOSSY"}
# element types of test-data files and buffers (include/sv_io.h)
IO_DTYPES = dict(DTYPES, u8=6, i8=7, i16=8, u16=9, u64=10, f64=11)
IO_DTYPE_BYTES = dict(DTYPE_BYTES, u8=1, i8=1, i16=2, u16=2, u64=8, f64=8)
IO_DTYPE_NAMES = {v: k for k, v in IO_DTYPES.items()}
IO_RAW, IO_STRICT = 1, 2
TENSOR_MAX_DIMS = 8


# ---------------------------------------------------------------------------
# public spec types (mirrors of the C structs with string enums)
# ---------------------------------------------------------------------------
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
    """A shaped output (rows x cols, row-major) compared tile by tile; zero
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


# ---------------------------------------------------------------------------
# C structs (layouts of synverify.h)
# ---------------------------------------------------------------------------
class sv_perturb(C.Structure):
    _fields_ = [("kind", C.c_uint32), ("stream", C.c_uint32), ("rate", C.c_double), ("count", C.c_uint64),
                ("value", C.c_double), ("ivalue", C.c_int64)]


class syn_spec(C.Structure):
    _fields_ = [("dtype", C.c_uint32), ("dist", C.c_uint32), ("n", C.c_uint64), ("seed", C.c_uint64),
                ("stream", C.c_uint32), ("special_mask", C.c_uint32), ("special_rate", C.c_double),
                ("ref_offset", C.c_uint64), ("cand_offset", C.c_uint64), ("elem_offset", C.c_uint64),
                ("logical_n", C.c_uint64), ("p0", C.c_double), ("p1", C.c_double), ("i0", C.c_int64),
                ("i1", C.c_int64), ("rows", C.c_uint64), ("cols", C.c_uint64), ("dot_k", C.c_uint64),
                ("a_offset", C.c_uint64), ("b_offset", C.c_uint64), ("pelem", sv_perturb), ("pcount", sv_perturb)]


class vc_pair(C.Structure):
    _fields_ = [("dtype", C.c_uint32), ("flags", C.c_uint32), ("n", C.c_uint64), ("cand_offset", C.c_uint64),
                ("ref_offset", C.c_uint64), ("atol", C.c_double), ("rtol", C.c_double)]


class vc_result(C.Structure):
    _fields_ = [("mismatches", C.c_uint64), ("nan_disagree", C.c_uint64), ("inf_disagree", C.c_uint64),
                ("n_finite", C.c_uint64), ("first_mismatch", C.c_int64), ("max_abs_u64", C.c_uint64),
                ("max_abs", C.c_double), ("max_rel", C.c_double), ("rms", C.c_double), ("pass_", C.c_uint32),
                ("state", C.c_uint32)]


class vc_tiles(C.Structure):
    _fields_ = [("dtype", C.c_uint32), ("flags", C.c_uint32), ("rows", C.c_uint64), ("cols", C.c_uint64),
                ("cand_offset", C.c_uint64), ("ref_offset", C.c_uint64), ("cand_pitch", C.c_uint64),
                ("ref_pitch", C.c_uint64), ("tile_rows", C.c_uint64), ("tile_cols", C.c_uint64),
                ("atol", C.c_double), ("rtol", C.c_double)]


class sv_tensor_header(C.Structure):
    _fields_ = [("magic", C.c_uint32), ("header_bytes", C.c_uint32), ("dtype", C.c_uint32), ("ndim", C.c_uint32),
                ("shape", C.c_uint64 * TENSOR_MAX_DIMS), ("n", C.c_uint64), ("data_bytes", C.c_uint64),
                ("reserved", C.c_uint64 * 4)]


assert C.sizeof(syn_spec) == 224 and C.sizeof(vc_pair) == 48 and C.sizeof(vc_result) == 80
assert C.sizeof(sv_tensor_header) == 128 and C.sizeof(vc_tiles) == 88
RESULT_BYTES = C.sizeof(vc_result)

# every function the header declares: (name, restype, argtypes)
_VP, _SZ = C.c_void_p, C.c_size_t
EXPORTS = [
    ("sv_generate_workspace_bytes", _SZ, [C.POINTER(syn_spec), C.c_int]),
    ("sv_compare_workspace_bytes", _SZ, [C.POINTER(vc_pair), C.c_int]),
    ("sv_progressive_workspace_bytes", _SZ, [C.POINTER(vc_pair), C.c_int]),
    ("sv_check_specs", C.c_int, [C.POINTER(syn_spec), C.c_int, _SZ]),
    ("sv_check_pairs", C.c_int, [C.POINTER(vc_pair), C.c_int, _SZ, _SZ]),
    ("syn_generate", C.c_int, [C.POINTER(syn_spec), C.c_int, _VP, _SZ, _VP, _SZ, _VP]),
    ("verify_compare", C.c_int, [C.POINTER(vc_pair), C.c_int, _VP, _SZ, _VP, _SZ, _VP, _VP, _SZ, _VP]),
    ("verify_progressive", C.c_int, [C.POINTER(vc_pair), C.c_int, _VP, _SZ, _VP, _SZ, _VP, _VP, _VP, _SZ, _VP]),
    ("verify_compare_noalloc", C.c_int, [C.POINTER(vc_pair), C.c_int, _VP, _SZ, _VP, _SZ, _VP, _VP]),
    ("sv_strerror", C.c_char_p, [C.c_int]),
    ("sv_abi_version", C.c_int, []),
    ("sv_kernel_launches", C.c_uint64, []),
    ("syn_box_muller", C.c_int, [C.c_void_p, C.c_size_t, C.c_void_p, C.c_void_p]),
    ("sv_debug_fail_launches", C.c_int, [C.c_int]),
    ("sv_compare_plan_create", C.c_int, [C.POINTER(vc_pair), C.c_int, _SZ, _SZ, _VP, _SZ, _VP,
                                         C.POINTER(C.c_void_p)]),
    ("verify_compare_planned", C.c_int, [_VP, _VP, _VP, _VP, _VP]),
    ("sv_compare_plan_destroy", None, [_VP]),
    ("sv_generate_plan_create", C.c_int, [C.POINTER(syn_spec), C.c_int, _SZ, _VP, _SZ, _VP, C.POINTER(C.c_void_p)]),
    ("syn_generate_planned", C.c_int, [_VP, _VP, _VP]),
    ("sv_generate_plan_destroy", None, [_VP]),
    ("sv_check_tiles", C.c_int, [C.POINTER(vc_tiles), _SZ, _SZ, C.POINTER(C.c_uint64)]),
    ("verify_compare_tiles", C.c_int, [C.POINTER(vc_tiles), _VP, _SZ, _VP, _SZ, _VP, _VP]),
    # include/sv_io.h
    ("sv_dtype_bytes", C.c_int, [C.c_int]),
    ("sv_tensor_probe", C.c_int, [C.c_char_p, C.POINTER(sv_tensor_header)]),
    ("sv_io_workspace_bytes", _SZ, [C.c_int, C.c_int, C.c_uint64]),
    ("sv_read_tensor", C.c_int, [C.c_char_p, C.c_uint32, C.c_int, C.c_uint64, C.c_int, _VP, _SZ, _VP, _SZ, _VP,
                                 C.POINTER(sv_tensor_header), C.POINTER(C.c_uint64)]),
    ("sv_write_tensor", C.c_int, [C.c_char_p, C.c_uint32, C.c_int, C.POINTER(C.c_uint64), C.c_int, _VP, _SZ, _VP]),
    ("sv_convert", C.c_int, [C.c_int, _VP, C.c_uint64, C.c_int, _VP, _VP, _VP]),
    ("sv_debug_io_chunk_bytes", C.c_int, [_SZ]),
]

_lib = None


def lib() -> C.CDLL:
    """The loaded library; raises if it has not been built (no fallback)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError("libsynverify.so is not built (%s); run __graft_entry__.build() or "
                               "python -m paper_2609_00058_gb300.build" % LIB_PATH)
        L = C.CDLL(LIB_PATH)
        for name, res, args in EXPORTS:
            f = getattr(L, name)
            f.restype, f.argtypes = res, args
        _lib = L
    return _lib


class SynVerifyError(RuntimeError):
    def __init__(self, status: int, where: str):
        msg = lib().sv_strerror(status).decode()
        super().__init__("%s failed: %s (%s)" % (where, STATUS.get(status, status), msg))
        self.status = status


def _ok(status: int, where: str) -> None:
    if status != 0:
        raise SynVerifyError(status, where)


# ---------------------------------------------------------------------------
# marshalling
# ---------------------------------------------------------------------------
def _perturb(p) -> sv_perturb:
    return sv_perturb(PERTS[p.kind], p.stream, p.rate, p.count, p.value, p.ivalue)


def to_c_spec(s) -> syn_spec:
    mask = SPECIAL_EXACT if getattr(s, "special_exact", False) else 0
    for k in s.specials:
        mask |= SPECIALS[k]
    return syn_spec(DTYPES[s.dtype], DISTS[s.dist], s.n, s.seed, s.stream, mask, s.special_rate,
                    NO_OUTPUT if s.ref_offset is None else s.ref_offset,
                    NO_OUTPUT if s.cand_offset is None else s.cand_offset,
                    s.elem_offset, s.logical_n, s.p0, s.p1, s.i0, s.i1, s.rows, s.cols, s.dot_k,
                    s.a_offset, s.b_offset, _perturb(s.pelem), _perturb(s.pcount))


def to_c_pair(p) -> vc_pair:
    return vc_pair(DTYPES[p.dtype], EQUAL_NAN if p.equal_nan else 0, p.n, p.cand_offset, p.ref_offset,
                   p.atol, p.rtol)


def _host_array(ctype, items):
    """A ctypes array of `items` in ordinary host memory (the library reads it
    during the call and stages its own device table from pinned buffers)."""
    n = max(len(items), 1)
    return (ctype * n)(*items), None


class SpecTable:
    """A prepared host table of generator specs (reusable across calls)."""

    def __init__(self, specs: Sequence):
        self.n = len(specs)
        self.arr, self._keep = _host_array(syn_spec, [to_c_spec(s) for s in specs])
        self.ws_bytes = lib().sv_generate_workspace_bytes(self.arr, self.n)


class PairTable:
    """A prepared host table of compare pairs / ladder stages."""

    def __init__(self, pairs: Sequence, progressive: bool = False):
        self.n = len(pairs)
        self.arr, self._keep = _host_array(vc_pair, [to_c_pair(p) for p in pairs])
        f = lib().sv_progressive_workspace_bytes if progressive else lib().sv_compare_workspace_bytes
        self.ws_bytes = f(self.arr, self.n)


def _stream_ptr(stream) -> int:
    import torch
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _workspace(nbytes: int, device, workspace):
    import torch
    if nbytes == 0:
        return None, 0
    if workspace is not None:
        _dense_cuda(workspace, "workspace")
        return workspace.data_ptr(), workspace.numel() * workspace.element_size()
    ws = torch.empty(nbytes + 256, dtype=torch.uint8, device=device)
    base = ws.data_ptr()
    off = (-base) % 256
    return base + off, nbytes, ws  # keep the tensor alive


def _nbytes(t) -> int:
    return t.numel() * t.element_size()


# ---------------------------------------------------------------------------
# entry points
# ---------------------------------------------------------------------------
def generate(specs, arena, workspace=None, stream=None) -> None:
    """syn_generate into `arena` (a CUDA tensor; offsets are bytes into it)."""
    _dense_cuda(arena, "arena")
    tab = specs if isinstance(specs, SpecTable) else SpecTable(specs)
    ws = _workspace(tab.ws_bytes, arena.device, workspace)
    rc = lib().syn_generate(tab.arr, tab.n, arena.data_ptr(), _nbytes(arena), ws[0], ws[1] if ws[0] else 0,
                            _stream_ptr(stream))
    _ok(rc, "syn_generate")


def compare(pairs, cand, ref, results=None, workspace=None, stream=None):
    """verify_compare; returns the device results tensor (uint8, n x 80 bytes)."""
    import torch
    _dense_cuda(cand, "cand")
    _dense_cuda(ref, "ref")
    tab = pairs if isinstance(pairs, PairTable) else PairTable(pairs)
    if results is None:
        results = torch.empty(max(tab.n, 1) * RESULT_BYTES, dtype=torch.uint8, device=cand.device)
    _dense_cuda(results, "results")
    ws = _workspace(tab.ws_bytes, cand.device, workspace)
    rc = lib().verify_compare(tab.arr, tab.n, cand.data_ptr(), _nbytes(cand), ref.data_ptr(), _nbytes(ref),
                              results.data_ptr(), ws[0], ws[1] if ws[0] else 0, _stream_ptr(stream))
    _ok(rc, "verify_compare")
    return results


class GeneratePlan:
    """sv_generate_plan_create: a syn_generate whose spec table is validated,
    grouped, scheduled and staged once (in a workspace this object owns), for
    arenas of at least arena_bytes."""

    def __init__(self, specs, arena_bytes: int, device=None, stream=None):
        import torch
        self.tab = specs if isinstance(specs, SpecTable) else SpecTable(specs)
        self.arena_bytes = arena_bytes
        dev = torch.device(device) if device is not None else torch.device("cuda", torch.cuda.current_device())
        self._ws = _workspace(self.tab.ws_bytes, dev, None)
        self._h = C.c_void_p()
        rc = lib().sv_generate_plan_create(self.tab.arr, self.tab.n, arena_bytes, self._ws[0],
                                           self._ws[1] if self._ws[0] else 0, _stream_ptr(stream), C.byref(self._h))
        _ok(rc, "sv_generate_plan_create")
        self.n = self.tab.n
        self.device = dev

    def __call__(self, arena, stream=None) -> None:
        """syn_generate_planned into `arena`."""
        _dense_cuda(arena, "arena")
        if _nbytes(arena) < self.arena_bytes:
            raise ValueError("arena smaller than the plan was made for")
        _ok(lib().syn_generate_planned(self._h, arena.data_ptr(), _stream_ptr(stream)), "syn_generate_planned")

    def __del__(self):
        h = getattr(self, "_h", None)
        if h is not None and h.value and _lib is not None:
            _lib.sv_generate_plan_destroy(h)
            self._h = None


class ComparePlan:
    """sv_compare_plan_create: a verify_compare whose table is prepared once,
    in a workspace this object owns, for buffers of cand_bytes / ref_bytes."""

    def __init__(self, pairs, cand_bytes: int, ref_bytes: int, device=None, stream=None):
        import torch
        self.tab = pairs if isinstance(pairs, PairTable) else PairTable(pairs)
        self.cand_bytes, self.ref_bytes = cand_bytes, ref_bytes
        dev = torch.device(device) if device is not None else torch.device("cuda", torch.cuda.current_device())
        self._ws = _workspace(self.tab.ws_bytes, dev, None)
        self._h = C.c_void_p()
        rc = lib().sv_compare_plan_create(self.tab.arr, self.tab.n, cand_bytes, ref_bytes, self._ws[0],
                                          self._ws[1] if self._ws[0] else 0, _stream_ptr(stream), C.byref(self._h))
        _ok(rc, "sv_compare_plan_create")
        self.n = self.tab.n
        self.device = dev

    def __call__(self, cand, ref, results=None, stream=None):
        """verify_compare_planned; returns the device results tensor."""
        import torch
        _dense_cuda(cand, "cand")
        _dense_cuda(ref, "ref")
        if _nbytes(cand) < self.cand_bytes or _nbytes(ref) < self.ref_bytes:
            raise ValueError("buffers smaller than the plan was made for")
        if results is None:
            results = torch.empty(max(self.n, 1) * RESULT_BYTES, dtype=torch.uint8, device=cand.device)
        _dense_cuda(results, "results")
        _ok(lib().verify_compare_planned(self._h, cand.data_ptr(), ref.data_ptr(), results.data_ptr(),
                                         _stream_ptr(stream)), "verify_compare_planned")
        return results

    def __del__(self):
        h = getattr(self, "_h", None)
        if h is not None and h.value and _lib is not None:
            _lib.sv_compare_plan_destroy(h)
            self._h = None


def progressive(stages, cand, ref, results=None, first_failed=None, workspace=None, stream=None):
    """verify_progressive; returns (device results, device int32 first-failed index)."""
    import torch
    _dense_cuda(cand, "cand")
    _dense_cuda(ref, "ref")
    tab = stages if isinstance(stages, PairTable) else PairTable(stages, progressive=True)
    if results is None:
        results = torch.empty(max(tab.n, 1) * RESULT_BYTES, dtype=torch.uint8, device=cand.device)
    if first_failed is None:
        first_failed = torch.empty(1, dtype=torch.int32, device=cand.device)
    _dense_cuda(results, "results")
    _dense_cuda(first_failed, "first_failed")
    ws = _workspace(tab.ws_bytes, cand.device, workspace)
    rc = lib().verify_progressive(tab.arr, tab.n, cand.data_ptr(), _nbytes(cand), ref.data_ptr(), _nbytes(ref),
                                  results.data_ptr(), first_failed.data_ptr(), ws[0], ws[1] if ws[0] else 0,
                                  _stream_ptr(stream))
    _ok(rc, "verify_progressive")
    return results, first_failed


def to_c_tiles(t) -> vc_tiles:
    """A shaped output (any object with the fields of workloads.Tiles)."""
    return vc_tiles(DTYPES[t.dtype], EQUAL_NAN if t.equal_nan else 0, t.rows, t.cols, t.cand_offset, t.ref_offset,
                    t.cand_pitch or t.cols, t.ref_pitch or t.cols, t.tile_rows, t.tile_cols or t.cols, t.atol, t.rtol)


def tile_count(t, cand_bytes: int = 1 << 62, ref_bytes: int = 1 << 62) -> int:
    """sv_check_tiles: the number of tiles (raises on an invalid description)."""
    n = C.c_uint64(0)
    _ok(lib().sv_check_tiles(C.byref(to_c_tiles(t)), cand_bytes, ref_bytes, C.byref(n)), "sv_check_tiles")
    return n.value


def compare_tiles(tiles, cand, ref, results=None, stream=None):
    """verify_compare_tiles; returns the device results tensor (uint8, one
    80-byte vc_result per tile, row-major over the tile grid)."""
    import torch
    _dense_cuda(cand, "cand")
    _dense_cuda(ref, "ref")
    c = to_c_tiles(tiles)
    n = tile_count(tiles, _nbytes(cand), _nbytes(ref))
    if results is None:
        results = torch.empty(max(n, 1) * RESULT_BYTES, dtype=torch.uint8, device=cand.device)
    _dense_cuda(results, "results")
    _ok(lib().verify_compare_tiles(C.byref(c), cand.data_ptr(), _nbytes(cand), ref.data_ptr(), _nbytes(ref),
                                   results.data_ptr(), _stream_ptr(stream)), "verify_compare_tiles")
    return results


def box_muller(words, out=None, stream=None):
    """syn_box_muller: the generator's Box-Muller step on a CUDA uint32 tensor
    of word pairs; returns (or fills) a float32 tensor of the same length."""
    import torch
    _dense_cuda(words, "words")
    n_pairs = words.numel() // 2
    if out is None:
        out = torch.empty(2 * n_pairs, dtype=torch.float32, device=words.device)
    _dense_cuda(out, "out")
    _ok(lib().syn_box_muller(words.data_ptr(), n_pairs, out.data_ptr(), _stream_ptr(stream)), "syn_box_muller")
    return out


def decode_results(results, n: int) -> List[dict]:
    """Copy n vc_result records to the host as dicts."""
    raw = bytes(results[: n * RESULT_BYTES].cpu().numpy().tobytes()) if hasattr(results, "cpu") else bytes(results)
    out = []
    for i in range(n):
        r = vc_result.from_buffer_copy(raw, i * RESULT_BYTES)
        out.append({"mismatches": r.mismatches, "nan_disagree": r.nan_disagree, "inf_disagree": r.inf_disagree,
                    "n_finite": r.n_finite, "first_mismatch": r.first_mismatch, "max_abs_u64": r.max_abs_u64,
                    "max_abs": r.max_abs, "max_rel": r.max_rel, "rms": r.rms, "pass": r.pass_, "state": r.state})
    return out


def check_specs(specs, arena_bytes: int) -> int:
    tab = SpecTable(specs)
    return lib().sv_check_specs(tab.arr, tab.n, arena_bytes)


def check_pairs(pairs, cand_bytes: int, ref_bytes: int) -> int:
    tab = PairTable(pairs)
    return lib().sv_check_pairs(tab.arr, tab.n, cand_bytes, ref_bytes)


# ---------------------------------------------------------------------------
# test-data I/O (include/sv_io.h)
# ---------------------------------------------------------------------------
def _torch_dtype(name: str):
    import torch
    return {"f32": torch.float32, "f16": torch.float16, "bf16": torch.bfloat16, "f64": torch.float64,
            "i32": torch.int32, "i64": torch.int64, "i16": torch.int16, "i8": torch.int8, "u8": torch.uint8,
            "u16": torch.uint16, "u32": torch.uint32, "u64": torch.uint64}[name]


def _header_dict(h: sv_tensor_header) -> dict:
    return {"dtype": IO_DTYPE_NAMES.get(h.dtype, h.dtype), "ndim": h.ndim, "shape": tuple(h.shape[: h.ndim]),
            "n": h.n, "data_bytes": h.data_bytes}


def _path(path) -> bytes:
    return os.fsencode(os.fspath(path))


def _dense_cuda(t, what: str):
    """The library reads and writes n * size bytes from data_ptr(): only a
    dense CUDA tensor describes that memory."""
    if t.device.type != "cuda":
        raise ValueError("%s must be a CUDA tensor (got %s)" % (what, t.device))
    if not t.is_contiguous():
        raise ValueError("%s must be contiguous (a strided view would be read as dense memory)" % what)


def tensor_probe(path) -> dict:
    """sv_tensor_probe: the checked header of a tensor file."""
    h = sv_tensor_header()
    _ok(lib().sv_tensor_probe(_path(path), C.byref(h)), "sv_tensor_probe")
    return _header_dict(h)


def read_tensor(path, dtype: Optional[str] = None, out=None, *, file_dtype: Optional[str] = None,
                n: Optional[int] = None, raw: bool = False, strict: bool = False, lossy_ok: bool = False,
                device=None, workspace=None, stream=None):
    """sv_read_tensor: load a test-data file into device memory, converting
    values to `dtype` (default: the file's type).  Returns (tensor, header,
    lost): the tensor has the file's shape when `out` is not given, else it is
    `out` (a CUDA tensor whose bytes receive the data).  Raises on every error,
    and on lost values (clamped or overflowed) unless lossy_ok."""
    import torch
    flags = (IO_RAW if raw else 0) | (IO_STRICT if strict else 0)
    if raw:
        if file_dtype is None:
            raise ValueError("a headerless file needs file_dtype")
        shape, src = None, file_dtype
        if n is None:
            n_file = os.path.getsize(path) // IO_DTYPE_BYTES[file_dtype]
        else:
            n_file = n
    else:
        info = tensor_probe(path)
        shape, src, n_file = info["shape"], info["dtype"], info["n"]
    dst = dtype or src
    if out is not None:
        dev = out.device
    else:
        dev = torch.device(device) if device is not None else torch.device("cuda", torch.cuda.current_device())
    if out is None:
        buf = torch.empty(max(n_file, 1) * IO_DTYPE_BYTES[dst], dtype=torch.uint8, device=dev)
    else:
        _dense_cuda(out, "out")
        buf = out
    ws = _workspace(lib().sv_io_workspace_bytes(IO_DTYPES[src], IO_DTYPES[dst], n_file), dev, workspace)
    h = sv_tensor_header()
    lost = C.c_uint64(0)
    rc = lib().sv_read_tensor(_path(path), flags, -1 if file_dtype is None else IO_DTYPES[file_dtype],
                              n or 0, IO_DTYPES[dst], buf.data_ptr(), _nbytes(buf), ws[0], ws[1] if ws[0] else 0,
                              _stream_ptr(stream), C.byref(h), C.byref(lost))
    if rc != -8 or not lossy_ok:
        _ok(rc, "sv_read_tensor")
    hd = _header_dict(h)
    if out is None:
        t = buf[: hd["n"] * IO_DTYPE_BYTES[dst]].view(_torch_dtype(dst))
        out = t.reshape(hd["shape"]) if not raw else t
    return out, hd, lost.value


def write_tensor(path, src, dtype: Optional[str] = None, shape: Optional[Sequence[int]] = None, raw: bool = False,
                 stream=None) -> None:
    """sv_write_tensor: write a CUDA tensor's bytes to a tensor file (header
    with `dtype` and `shape`, default: the tensor's own)."""
    _dense_cuda(src, "src")
    if dtype is None:
        names = {_torch_dtype(k): k for k in IO_DTYPES}
        dtype = names[src.dtype]
    if shape is None:  # the tensor's own shape, or its bytes as a vector of `dtype`
        shape = tuple(src.shape) if src.dtype == _torch_dtype(dtype) else (_nbytes(src) // IO_DTYPE_BYTES[dtype],)
    arr = (C.c_uint64 * max(len(shape), 1))(*shape)
    rc = lib().sv_write_tensor(_path(path), IO_RAW if raw else 0, IO_DTYPES[dtype], arr, len(shape), src.data_ptr(),
                               _nbytes(src), _stream_ptr(stream))
    _ok(rc, "sv_write_tensor")


def convert(src, src_dtype: str, dst_dtype: str, n: Optional[int] = None, out=None, lost=None, stream=None):
    """sv_convert: device-to-device value conversion; returns (out, lost),
    `lost` a device uint64 counter (added to, not reset, when given)."""
    import torch
    _dense_cuda(src, "src")
    if out is not None:
        _dense_cuda(out, "out")
    if n is None:
        n = _nbytes(src) // IO_DTYPE_BYTES[src_dtype]
    if out is None:
        out = torch.empty(max(n, 1) * IO_DTYPE_BYTES[dst_dtype], dtype=torch.uint8, device=src.device)
    if lost is None:
        lost = torch.zeros(1, dtype=torch.int64, device=src.device)
    _ok(lib().sv_convert(IO_DTYPES[src_dtype], src.data_ptr(), n, IO_DTYPES[dst_dtype], out.data_ptr(),
                         lost.data_ptr(), _stream_ptr(stream)), "sv_convert")
    return out, lost
