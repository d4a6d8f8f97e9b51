"""Tensor files written and parsed by the tests themselves, from the layout
that include/sv_io.h documents: a 128-byte little-endian header (magic
"SVT1", header size, element type, rank, eight extents, element count, data
bytes, four reserved words), then the elements."""
import struct

import numpy as np

DTYPES = {"f32": 0, "f16": 1, "bf16": 2, "i32": 3, "i64": 4, "u32": 5, "u8": 6, "i8": 7, "i16": 8, "u16": 9,
          "u64": 10, "f64": 11}
NAMES = {v: k for k, v in DTYPES.items()}
BYTES = {"f32": 4, "f16": 2, "bf16": 2, "i32": 4, "i64": 8, "u32": 4, "u8": 1, "i8": 1, "i16": 2, "u16": 2,
         "u64": 8, "f64": 8}
FMT = "<4sIII8QQQ4Q"
assert struct.calcsize(FMT) == 128


def header(dtype, shape, n=None, data_bytes=None, magic=b"SVT1", header_bytes=128, reserved=(0, 0, 0, 0)):
    shape = tuple(shape)
    if n is None:
        n = int(np.prod(shape, dtype=object)) if shape else 1
    if data_bytes is None:
        data_bytes = n * BYTES[dtype]
    ext = list(shape) + [0] * (8 - len(shape))
    return struct.pack(FMT, magic, header_bytes, DTYPES[dtype], len(shape), *ext, n, data_bytes, *reserved)


def write(path, raw_bytes, dtype, shape=None, headerless=False):
    raw_bytes = np.ascontiguousarray(raw_bytes).view(np.uint8).reshape(-1)
    if shape is None:
        shape = (raw_bytes.size // BYTES[dtype],)
    with open(path, "wb") as f:
        if not headerless:
            f.write(header(dtype, shape))
        f.write(raw_bytes.tobytes())


def parse(path):
    """(dtype name, shape, data bytes as uint8)"""
    blob = open(path, "rb").read()
    fields = struct.unpack(FMT, blob[:128])
    magic, hb, dt, ndim = fields[:4]
    ext = fields[4:12]
    n, nbytes = fields[12], fields[13]
    assert magic == b"SVT1" and hb == 128 and ndim <= 8
    assert len(blob) == 128 + nbytes
    return NAMES[dt], tuple(ext[:ndim]), np.frombuffer(blob[128:], np.uint8)
