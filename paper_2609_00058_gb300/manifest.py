"""Kernel implementation manifest entries (CUDA-Harness Sec. 4.1.1) turned into
a verification plan on the GPU: test-input synthesis specs and shaped-output
comparisons.

A manifest entry records, per kernel, its name, a functional description and
the shapes and element types of its test inputs and outputs.  From an entry,
`plan()` lays out one arena holding every input, the trusted reference's
outputs and the candidate's outputs (16-byte aligned, 256-byte spaced), and
derives:
- one syn_generate spec per input.  Unless the entry says otherwise, float
  inputs follow the broad-range rule of Sec. 4.2.1, N(5, 10), so that the
  relative term of Eq. 1 is not swamped by the absolute one; integer inputs
  are uniform over [-1000, 1000] (unsigned: [0, 1000]);
- one tile-by-tile comparison per output (verify_compare_tiles): the output
  viewed as rows x cols, with rows the product of every extent but the last,
  in tiles of the entry's tile shape (default: one row per tile), so a wrong
  result is located to the rows, or the blocks, that hold it.

Entries load from JSON:
  {"kernel": "...", "description": "...", "atol": 1e-5, "rtol": 1e-5,
   "inputs":  [{"name": "a", "shape": [1024, 512], "dtype": "f32",
                "dist": "normal", "params": [5.0, 10.0]}, ...],
   "outputs": [{"name": "c", "shape": [1024, 512], "dtype": "f32",
                "tile": [64, 128]}, ...]}
"dist"/"params" and "tile" are optional.  Names and values are marshalled
into the library's structures only; no step of synthesis or comparison runs
on the host.
"""
from __future__ import annotations

import json
import math
from dataclasses import dataclass, field
from typing import Dict, List, Optional, Sequence, Tuple

from . import DTYPE_BYTES, GenSpec, Tiles, compare_tiles, decode_results, generate, tile_count

BROAD_RANGE_NORMAL = (5.0, 10.0)  # Sec. 4.2.1: mean 5, standard deviation 10
INT_RANGE = (-1000, 1000)
ALIGN = 256
FLOATS = ("f32", "f16", "bf16")


@dataclass
class TensorDesc:
    name: str
    shape: Tuple[int, ...]
    dtype: str
    dist: Optional[str] = None           # syn_generate distribution; None: the preset
    params: Tuple[float, ...] = ()       # (p0, p1) for float dists, (i0, i1) for int_range
    tile: Optional[Tuple[int, int]] = None  # outputs: (tile_rows, tile_cols); None: one row per tile

    @property
    def n(self) -> int:
        return math.prod(self.shape) if self.shape else 1

    @property
    def nbytes(self) -> int:
        return self.n * DTYPE_BYTES[self.dtype]

    def matrix(self) -> Tuple[int, int]:
        """(rows, cols): every extent but the last as rows."""
        if not self.shape:
            return 1, 1
        return math.prod(self.shape[:-1]) if len(self.shape) > 1 else 1, self.shape[-1]


@dataclass
class ManifestEntry:
    kernel: str
    inputs: List[TensorDesc]
    outputs: List[TensorDesc]
    description: str = ""
    atol: float = 1e-5
    rtol: float = 1e-5


def _tensor(d: dict) -> TensorDesc:
    if d["dtype"] not in DTYPE_BYTES:
        raise ValueError("unknown dtype %r of %r" % (d["dtype"], d.get("name")))
    tile = tuple(d["tile"]) if d.get("tile") is not None else None
    return TensorDesc(d["name"], tuple(int(x) for x in d["shape"]), d["dtype"], d.get("dist"),
                      tuple(d.get("params", ())), tile)


def entry_from_dict(d: dict) -> ManifestEntry:
    return ManifestEntry(d["kernel"], [_tensor(x) for x in d.get("inputs", [])],
                         [_tensor(x) for x in d.get("outputs", [])], d.get("description", ""),
                         float(d.get("atol", 1e-5)), float(d.get("rtol", 1e-5)))


def load(path_or_text) -> List[ManifestEntry]:
    """Entries of a manifest: a JSON file path or text holding one entry or a list."""
    text = path_or_text
    if not str(path_or_text).lstrip().startswith(("{", "[")):
        with open(path_or_text) as f:
            text = f.read()
    data = json.loads(text)
    return [entry_from_dict(d) for d in (data if isinstance(data, list) else [data])]


def preset(t: TensorDesc) -> Tuple[str, Tuple]:
    """The distribution and parameters an input is synthesized from."""
    if t.dist is not None:
        return t.dist, t.params
    if t.dtype in FLOATS:
        return "normal", BROAD_RANGE_NORMAL
    return "int_range", (0, INT_RANGE[1]) if t.dtype == "u32" else INT_RANGE


@dataclass
class Plan:
    entry: ManifestEntry
    arena_bytes: int
    inputs: Dict[str, int] = field(default_factory=dict)       # name -> byte offset
    ref_outputs: Dict[str, int] = field(default_factory=dict)  # name -> byte offset of the reference's output
    cand_outputs: Dict[str, int] = field(default_factory=dict)
    specs: List[GenSpec] = field(default_factory=list)
    tiles: Dict[str, object] = field(default_factory=dict)     # name -> Tiles description

    def calling_convention(self) -> str:
        def one(t):
            return "%s: %s %s" % (t.name, t.dtype, list(t.shape))
        e = self.entry
        return "%s(%s) -> (%s)" % (e.kernel, ", ".join(one(t) for t in e.inputs),
                                   ", ".join(one(t) for t in e.outputs))


def plan(entry: ManifestEntry, seed: int = 1) -> Plan:
    """Arena layout, input specs and per-output tile descriptions of an entry.
    Input i is drawn from Philox stream i of `seed`."""
    off = 0

    def take(nbytes):
        nonlocal off
        at = off
        off += (nbytes + ALIGN - 1) // ALIGN * ALIGN
        return at

    p = Plan(entry, 0)
    for i, t in enumerate(entry.inputs):
        at = take(t.nbytes)
        p.inputs[t.name] = at
        dist, prm = preset(t)
        kw = dict(dtype=t.dtype, dist=dist, n=t.n, seed=seed, stream=i, ref_offset=at)
        if dist in ("uniform", "normal", "constant") and t.dtype in FLOATS:
            kw.update(p0=float(prm[0]), p1=float(prm[1]) if len(prm) > 1 else 0.0)
        elif dist == "int_range" or dist == "constant":
            kw.update(i0=int(prm[0]), i1=int(prm[1]) if len(prm) > 1 else 0)
        p.specs.append(GenSpec(**kw))
    for t in entry.outputs:
        p.ref_outputs[t.name] = take(t.nbytes)
        p.cand_outputs[t.name] = take(t.nbytes)
        rows, cols = t.matrix()
        tr, tc = t.tile if t.tile else (1, cols)
        p.tiles[t.name] = Tiles(t.dtype, rows, cols, p.cand_outputs[t.name], p.ref_outputs[t.name],
                                  tile_rows=tr, tile_cols=min(tc, cols), atol=entry.atol, rtol=entry.rtol)
    p.arena_bytes = max(off, ALIGN)
    for name, t in p.tiles.items():
        tile_count(t, p.arena_bytes, p.arena_bytes)  # validates the geometry (raises if the tiles are invalid)
    return p


def synthesize(p: Plan, arena, stream=None) -> None:
    """syn_generate of every input of the plan into `arena`."""
    if p.specs:
        generate(p.specs, arena, stream=stream)


def verify(p: Plan, arena, stream=None) -> Dict[str, List[dict]]:
    """Eq. 1 per tile of every output: candidate against reference."""
    out = {}
    for name, t in p.tiles.items():
        res = compare_tiles(t, arena, arena, stream=stream)
        out[name] = decode_results(res, tile_count(t, arena.numel(), arena.numel()))
    return out


def failing_tiles(results: Sequence[dict], tiles) -> List[Tuple[int, int]]:
    """(tile row, tile column) of every tile that failed, from per-tile results."""
    ntc = -(-tiles.cols // tiles.tile_cols)
    return [(i // ntc, i % ntc) for i, r in enumerate(results) if not r["pass"]]
