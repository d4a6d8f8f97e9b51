"""Host-side checks of the test-data I/O entry points (include/sv_io.h), no
GPU: header parsing and every refusal that happens before a CUDA call (a bad
header, a type, count or size that differs from what the caller stated, a
refused conversion, bad arguments), plus empty tensors, which need no copy.
The device pointers passed here are never dereferenced: each case is
rejected (or complete) before anything touches CUDA."""
import ctypes as C
import os

import pytest

import paper_2609_00058_gb300 as sv
import tensor_files as TF

FAKE = 1 << 20  # an aligned address that is never used


@pytest.fixture(scope="module")
def lib():
    from paper_2609_00058_gb300 import build
    build.build()
    return sv.lib()


def read(lib, path, flags=0, file_dtype=-1, n=0, dst="f32", dst_bytes=1 << 30, ws=FAKE, ws_bytes=1 << 30, dptr=FAKE):
    h = sv.sv_tensor_header()
    lost = C.c_uint64(0)
    rc = lib.sv_read_tensor(os.fsencode(str(path)), flags, file_dtype, n, sv.IO_DTYPES[dst], dptr, dst_bytes, ws,
                            ws_bytes, None, C.byref(h), C.byref(lost))
    return rc, h


def test_dtype_bytes(lib):
    for k, v in sv.IO_DTYPES.items():
        assert lib.sv_dtype_bytes(v) == sv.IO_DTYPE_BYTES[k]
    assert lib.sv_dtype_bytes(12) == 0 and lib.sv_dtype_bytes(-1) == 0


def test_probe_reads_header(lib, tmp_path):
    p = tmp_path / "a.svt"
    import numpy as np
    TF.write(p, np.arange(24, dtype=np.int16), "i16", shape=(2, 3, 4))
    info = sv.tensor_probe(p)
    assert info == {"dtype": "i16", "ndim": 3, "shape": (2, 3, 4), "n": 24, "data_bytes": 48}
    TF.write(p, np.zeros(0, np.uint8), "u8", shape=())  # rank 0 holds one element: the size is wrong
    with pytest.raises(sv.SynVerifyError) as e:
        sv.tensor_probe(p)
    assert e.value.status == -7
    TF.write(p, np.zeros(1, np.uint8), "u8", shape=())
    assert sv.tensor_probe(p)["n"] == 1


BAD_HEADERS = [
    dict(magic=b"SVT2"),
    dict(header_bytes=64),
    dict(n=25),                      # not the product of the extents
    dict(data_bytes=50),             # not n * element size
    dict(reserved=(0, 0, 1, 0)),
]


@pytest.mark.parametrize("bad", BAD_HEADERS)
def test_probe_rejects_bad_headers(lib, tmp_path, bad):
    p = tmp_path / "b.svt"
    with open(p, "wb") as f:
        f.write(TF.header("i16", (2, 3, 4), **bad))
        f.write(bytes(48))
    assert lib.sv_tensor_probe(os.fsencode(str(p)), C.byref(sv.sv_tensor_header())) == -7


def test_probe_rejects_sizes_and_types(lib, tmp_path):
    p = tmp_path / "c.svt"
    with open(p, "wb") as f:  # one byte short
        f.write(TF.header("f32", (10,)))
        f.write(bytes(39))
    assert lib.sv_tensor_probe(os.fsencode(str(p)), C.byref(sv.sv_tensor_header())) == -7
    blob = bytearray(TF.header("f32", (10,)) + bytes(40))
    blob[8] = 12  # unknown element type
    p.write_bytes(bytes(blob))
    assert lib.sv_tensor_probe(os.fsencode(str(p)), C.byref(sv.sv_tensor_header())) == -7
    blob = bytearray(TF.header("f32", (10,)) + bytes(40))
    blob[12] = 9  # rank above 8
    p.write_bytes(bytes(blob))
    assert lib.sv_tensor_probe(os.fsencode(str(p)), C.byref(sv.sv_tensor_header())) == -7
    p.write_bytes(b"SVT1")  # shorter than a header
    assert lib.sv_tensor_probe(os.fsencode(str(p)), C.byref(sv.sv_tensor_header())) == -7
    assert lib.sv_tensor_probe(os.fsencode(str(tmp_path / "missing")), C.byref(sv.sv_tensor_header())) == -6
    assert lib.sv_tensor_probe(os.fsencode(str(tmp_path)), C.byref(sv.sv_tensor_header())) == -6  # a directory
    assert lib.sv_tensor_probe(None, C.byref(sv.sv_tensor_header())) == -1


def test_read_refusals_before_any_copy(lib, tmp_path):
    import numpy as np
    p = tmp_path / "d.svt"
    TF.write(p, np.arange(100, dtype=np.uint8), "u8")
    assert read(lib, p, file_dtype=sv.IO_DTYPES["f32"])[0] == -7     # the file is not what the caller says
    assert read(lib, p, n=99)[0] == -7                               # count differs
    assert read(lib, p, flags=sv.IO_STRICT, dst="f32")[0] == -7      # strict: no conversion allowed
    assert read(lib, p, flags=4)[0] == -1                            # unknown flag
    assert read(lib, p, dst="f32", dptr=FAKE + 8)[0] == -2           # misaligned destination
    assert read(lib, p, dst="f32", dst_bytes=399)[0] == -3           # destination too small
    assert read(lib, p, dst="f32", ws=0)[0] == -4                    # conversion without workspace
    assert read(lib, p, dst="f32", ws_bytes=16)[0] == -4
    assert read(lib, p, dst="f32", ws=FAKE + 128)[0] == -4           # workspace not 256-aligned
    assert read(lib, tmp_path / "nope.svt")[0] == -6
    f = tmp_path / "e.svt"
    TF.write(f, np.ones(10, np.float32), "f32")
    assert read(lib, f, dst="i32")[0] == -1                          # float -> integer refused
    assert read(lib, f, dst="u8")[0] == -1


def test_defect_raw_uint8_read_as_float(lib, tmp_path):
    """The loading defect of Sec. 5.2.3: n bytes of uint8 data read as n floats.
    Stating the type and count of a headerless file turns it into an error."""
    import numpy as np
    p = tmp_path / "img.bin"
    TF.write(p, np.arange(1000, dtype=np.uint16).astype(np.uint8), "u8", headerless=True)
    assert read(lib, p, flags=sv.IO_RAW, file_dtype=sv.IO_DTYPES["f32"], n=1000)[0] == -7
    # 1000 bytes do hold 250 floats: the format checks pass (and the small destination is refused next)
    assert read(lib, p, flags=sv.IO_RAW, file_dtype=sv.IO_DTYPES["f32"], n=250, dst_bytes=999)[0] == -3
    TF.write(p, np.zeros(1001, np.uint8), "u8", headerless=True)
    assert read(lib, p, flags=sv.IO_RAW, file_dtype=sv.IO_DTYPES["f32"])[0] == -7  # not a whole number of floats
    assert read(lib, p, flags=sv.IO_RAW)[0] == -1  # a raw file needs its type


def test_empty_tensors_need_no_device(lib, tmp_path):
    import numpy as np
    p = tmp_path / "z.svt"
    TF.write(p, np.zeros(0, np.float32), "f32", shape=(0, 7))
    rc, h = read(lib, p, dst="bf16", ws=0, ws_bytes=0, dptr=0)
    assert rc == 0 and h.n == 0 and h.ndim == 2 and h.shape[1] == 7
    q = tmp_path / "w.svt"
    shape = (C.c_uint64 * 2)(3, 0)
    assert lib.sv_write_tensor(os.fsencode(str(q)), 0, sv.IO_DTYPES["i64"], shape, 2, None, 0, None) == 0
    dt, shp, data = TF.parse(q)
    assert (dt, shp, data.size) == ("i64", (3, 0), 0)
    assert lib.sv_write_tensor(os.fsencode(str(q)), sv.IO_RAW, sv.IO_DTYPES["i64"], shape, 2, None, 0, None) == 0
    assert os.path.getsize(q) == 0


def test_write_refusals(lib, tmp_path):
    q = os.fsencode(str(tmp_path / "v.svt"))
    one = (C.c_uint64 * 1)(10)
    assert lib.sv_write_tensor(q, 0, 12, one, 1, FAKE, 1 << 20, None) == -1          # unknown type
    assert lib.sv_write_tensor(q, 0, 0, one, 9, FAKE, 1 << 20, None) == -1           # rank above 8
    assert lib.sv_write_tensor(q, 0, 0, None, 1, FAKE, 1 << 20, None) == -1          # no shape
    assert lib.sv_write_tensor(q, 2, 0, one, 1, FAKE, 1 << 20, None) == -1           # strict is a read flag
    assert lib.sv_write_tensor(q, 0, 0, one, 1, FAKE + 4, 1 << 20, None) == -2       # misaligned source
    assert lib.sv_write_tensor(q, 0, 0, one, 1, FAKE, 39, None) == -3                # source too small
    big = (C.c_uint64 * 2)(1 << 40, 1 << 40)
    assert lib.sv_write_tensor(q, 0, 0, big, 2, FAKE, 1 << 20, None) == -3           # count overflow
    assert lib.sv_write_tensor(os.fsencode(str(tmp_path / "no" / "dir.svt")), 0, 0, one, 1, FAKE, 1 << 20,
                               None) == -6


def test_convert_refusals_and_workspace_sizes(lib):
    assert lib.sv_convert(0, FAKE, 10, 3, FAKE, FAKE, None) == -1   # f32 -> i32 refused
    assert lib.sv_convert(12, FAKE, 10, 0, FAKE, FAKE, None) == -1
    assert lib.sv_convert(6, FAKE + 8, 10, 0, FAKE, FAKE, None) == -2
    assert lib.sv_convert(6, FAKE, 10, 0, FAKE, FAKE + 4, None) == -2
    assert lib.sv_convert(6, FAKE, 10, 0, FAKE, None, None) == -1  # conversion needs the lost counter
    assert lib.sv_convert(6, FAKE, (1 << 40) + 1, 0, FAKE, FAKE, None) == -3
    assert lib.sv_convert(6, 0, 0, 0, 0, 0, None) == 0              # nothing to do
    assert lib.sv_io_workspace_bytes(0, 0, 1 << 30) == 0
    assert lib.sv_io_workspace_bytes(6, 0, 100) == 256 + 2 * 256
    assert lib.sv_io_workspace_bytes(6, 0, 1 << 30) == 256 + 2 * (32 << 20)
    assert lib.sv_io_workspace_bytes(6, 12, 100) == 0


def test_chunk_hook_arguments(lib):
    assert lib.sv_debug_io_chunk_bytes(4095) == -1
    assert lib.sv_debug_io_chunk_bytes((32 << 20) + 4096) == -1
    assert lib.sv_debug_io_chunk_bytes(8192) == 0
    assert lib.sv_debug_io_chunk_bytes(0) == 0


def test_binding_refuses_host_and_strided_tensors(lib, tmp_path):
    """The binding passes data_ptr(): a host tensor or a strided view would be
    taken for dense device memory, so both are refused before any call."""
    torch = pytest.importorskip("torch")
    host = torch.zeros(64, dtype=torch.float32)
    with pytest.raises(ValueError, match="CUDA"):
        sv.write_tensor(tmp_path / "h.svt", host)
    with pytest.raises(ValueError, match="CUDA"):
        sv.convert(host, "f32", "f64")
    class FakeCuda:  # a strided view on a CUDA device, as far as the checks can tell
        device = torch.device("cuda", 0)

        def is_contiguous(self):
            return False
    with pytest.raises(ValueError, match="contiguous"):
        sv.write_tensor(tmp_path / "s.svt", FakeCuda(), dtype="f32", shape=(8,))
    with pytest.raises(ValueError, match="contiguous"):
        sv.convert(FakeCuda(), "f32", "f64", n=8)
