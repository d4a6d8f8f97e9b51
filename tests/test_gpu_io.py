"""Parity of the dtype-correct test-data I/O (include/sv_io.h) with the
oracle's value conversion (oracle/convert.c), through the C ABI on the GPU.

- sv_convert, every allowed pair of the 12 element types, random encodings
  (NaN payloads, infinities, subnormals, every integer range), sizes from one
  element to several vectors per thread with ragged tails: bytes identical
  to the oracle's, lost counts equal;
- sv_read_tensor from files the tests write themselves (tests/tensor_files.py),
  into every target type, across many pipeline chunks (small chunk hook) and
  at the default chunk size; headerless files; the loading defect of Sec. 5.2.3;
- sv_write_tensor read back by the tests' own parser.
"""
import numpy as np
import pytest

import oracle
import paper_2609_00058_gb300 as sv
import tensor_files as TF
from gpu_util import device

pytestmark = pytest.mark.gpu
FLOATS = ["f16", "bf16", "f32", "f64"]
INTS = ["u8", "i8", "i16", "u16", "i32", "u32", "i64", "u64"]
ALL = FLOATS + INTS
PAIRS = [(s, d) for s in ALL for d in ALL if s != d and not (s in FLOATS and d in INTS)]


@pytest.fixture(scope="module")
def dev():
    return device()


@pytest.fixture(autouse=True)
def default_chunks():
    yield
    sv.lib().sv_debug_io_chunk_bytes(0)
    sv.lib().sv_debug_fail_launches(0)


def source_bytes(dtype, n, seed):
    """Random encodings, plus integer values spread over every magnitude."""
    rng = np.random.default_rng(seed)
    nb = oracle.IO_DTYPE_BYTES[dtype]
    raw = rng.integers(0, 256, size=n * nb, dtype=np.uint8)
    if dtype in INTS and n >= 4:  # a quarter of the elements: small magnitudes, both signs
        k = n // 4
        mags = np.floor(np.exp2(rng.uniform(0, 8 * nb - 1, size=k))).astype(np.uint64)
        vals = mags.view(np.int64) * np.where(rng.integers(0, 2, size=k) == 1, -1, 1)
        raw[: k * nb] = vals.astype(TF_NP[dtype]).view(np.uint8)
    return raw


TF_NP = {"u8": np.uint8, "i8": np.int8, "i16": np.int16, "u16": np.uint16, "i32": np.int32, "u32": np.uint32,
         "i64": np.int64, "u64": np.uint64}


def as_bytes(t):
    import torch
    return t.reshape(-1).view(torch.uint8).cpu().numpy()


def to_dev(raw, dev):
    import torch
    t = torch.empty(max(raw.size, 16), dtype=torch.uint8, device=dev)
    t[: raw.size].copy_(torch.from_numpy(raw))
    return t


@pytest.mark.parametrize("s,d", PAIRS)
def test_convert_matches_oracle(dev, s, d):
    import torch
    for n in (1, 3, 16, 17, 1000, 4099, 70001):
        raw = source_bytes(s, n, seed=ALL.index(s) * 1000 + ALL.index(d) * 37 + n)
        want, want_lost = oracle.convert(raw, s, d)
        out, lost = sv.convert(to_dev(raw, dev), s, d, n=n)
        torch.cuda.synchronize()
        got = out[: want.size].cpu().numpy()
        assert np.array_equal(got, want), (s, d, n, np.flatnonzero(got != want)[:8])
        assert int(lost.item()) == want_lost, (s, d, n)


def test_convert_same_type_is_a_copy_and_refusals(dev):
    import torch
    raw = source_bytes("f32", 1001, 5)
    out, _ = sv.convert(to_dev(raw, dev), "f32", "f32", n=1001)
    torch.cuda.synchronize()
    assert np.array_equal(out[: raw.size].cpu().numpy(), raw)
    for s in FLOATS:
        for d in INTS:
            with pytest.raises(sv.SynVerifyError) as e:
                sv.convert(to_dev(raw, dev), s, d, n=16)
            assert e.value.status == -1


def test_convert_accumulates_lost(dev):
    import torch
    raw = np.array([300, -5, 7, 256], np.int32).view(np.uint8)
    lost = torch.full((1,), 10, dtype=torch.int64, device=dev)
    out, lost = sv.convert(to_dev(raw, dev), "i32", "u8", n=4, lost=lost)
    torch.cuda.synchronize()
    assert list(out[:4].cpu().numpy()) == [255, 0, 7, 255] and int(lost.item()) == 13


def test_convert_large(dev):
    """One launch over 2^25 + 3 elements, every vector and the ragged tail."""
    import torch
    n = (1 << 25) + 3
    raw = source_bytes("f64", n, 11)
    want, want_lost = oracle.convert(raw, "f64", "bf16")
    out, lost = sv.convert(to_dev(raw, dev), "f64", "bf16", n=n)
    torch.cuda.synchronize()
    assert np.array_equal(out[: want.size].cpu().numpy(), want) and int(lost.item()) == want_lost


# ---------------------------------------------------------------------------
# files
# ---------------------------------------------------------------------------
READ_PAIRS = [("u8", "f32"), ("i32", "f32"), ("u8", "u8"), ("f32", "bf16"), ("f64", "f32"), ("i64", "i32"),
              ("u16", "f16"), ("bf16", "f32"), ("f32", "f32"), ("i8", "i64"), ("u64", "f64")]


@pytest.mark.parametrize("chunk", [4096, 12288, 0])
@pytest.mark.parametrize("s,d", READ_PAIRS)
def test_read_tensor_matches_oracle(dev, tmp_path, s, d, chunk):
    assert sv.lib().sv_debug_io_chunk_bytes(chunk) == 0
    for n in (1, 5, 4096 + 17, 3 * 4096 // oracle.IO_DTYPE_BYTES[s] + 1, 50003):
        raw = source_bytes(s, n, seed=n)
        p = tmp_path / ("%s_%d.svt" % (s, n))
        TF.write(p, raw, s, shape=(n,))
        want, want_lost = oracle.convert(raw, s, d)
        t, hdr, lost = sv.read_tensor(p, dtype=d, lossy_ok=True, device=dev)
        assert hdr["dtype"] == s and hdr["n"] == n and hdr["shape"] == (n,)
        assert np.array_equal(as_bytes(t), want), (s, d, n, chunk)
        assert lost == want_lost


def test_read_shapes_and_into_arena(dev, tmp_path):
    import torch
    raw = np.arange(2 * 3 * 5, dtype=np.int16)
    p = tmp_path / "s.svt"
    TF.write(p, raw, "i16", shape=(2, 3, 5))
    t, hdr, _ = sv.read_tensor(p, device=dev)
    assert t.dtype == torch.int16 and tuple(t.shape) == (2, 3, 5)
    assert np.array_equal(t.cpu().numpy().reshape(-1), raw)
    arena = torch.zeros(4096, dtype=torch.uint8, device=dev)
    out, _, _ = sv.read_tensor(p, dtype="f32", out=arena[1024:1024 + 120], device=dev)
    assert np.array_equal(arena[1024:1144].cpu().numpy().view(np.float32), raw.astype(np.float32))
    assert not arena[:1024].any().item() and not arena[1144:].any().item()


def test_the_loading_defect(dev, tmp_path):
    """uint8 and int32 test data loaded for a float kernel arrive as their values,
    not as reinterpreted bytes (Sec. 5.2.3)."""
    img = np.random.default_rng(3).integers(0, 256, size=4096, dtype=np.uint8)
    p = tmp_path / "img.svt"
    TF.write(p, img, "u8")
    t, _, _ = sv.read_tensor(p, dtype="f32", device=dev)
    assert np.array_equal(t.cpu().numpy(), img.astype(np.float32))
    ints = np.random.default_rng(4).integers(-2 ** 31, 2 ** 31, size=4096, dtype=np.int64).astype(np.int32)
    q = tmp_path / "ints.svt"
    TF.write(q, ints, "i32")
    t, _, _ = sv.read_tensor(q, dtype="f32", device=dev)
    assert np.array_equal(t.cpu().numpy(), ints.astype(np.float32))  # one rounding to nearest even
    # the defect itself, for contrast: the same bytes taken as floats are not the data
    assert not np.array_equal(ints.view(np.float32), ints.astype(np.float32))
    # stated type and count of a headerless file: uint8 bytes cannot pass as floats
    r = tmp_path / "img.bin"
    TF.write(r, img, "u8", headerless=True)
    with pytest.raises(sv.SynVerifyError) as e:
        sv.read_tensor(r, raw=True, file_dtype="f32", n=4096, device=dev)
    assert e.value.status == -7
    t, hdr, _ = sv.read_tensor(r, raw=True, file_dtype="u8", n=4096, dtype="f32", device=dev)
    assert np.array_equal(t.cpu().numpy(), img.astype(np.float32)) and hdr["n"] == 4096
    with pytest.raises(sv.SynVerifyError) as e:  # the header says u8: the caller's f32 is wrong
        sv.read_tensor(p, file_dtype="f32", device=dev)
    assert e.value.status == -7
    with pytest.raises(sv.SynVerifyError) as e:
        sv.read_tensor(p, dtype="f32", strict=True, device=dev)
    assert e.value.status == -7


def test_lossy_loads_raise_unless_allowed(dev, tmp_path):
    vals = np.array([1, 255, 256, -1, 70000, 3], np.int32)
    p = tmp_path / "l.svt"
    TF.write(p, vals, "i32")
    with pytest.raises(sv.SynVerifyError) as e:
        sv.read_tensor(p, dtype="u8", device=dev)
    assert e.value.status == -8
    t, _, lost = sv.read_tensor(p, dtype="u8", lossy_ok=True, device=dev)
    assert list(t.cpu().numpy()) == [1, 255, 255, 0, 255, 3] and lost == 3
    t, _, lost = sv.read_tensor(p, dtype="f16", lossy_ok=True, device=dev)
    assert lost == 1 and np.isinf(t.cpu().numpy()[4])


@pytest.mark.parametrize("chunk", [4096, 0])
def test_write_tensor_round_trip(dev, tmp_path, chunk):
    import torch
    assert sv.lib().sv_debug_io_chunk_bytes(chunk) == 0
    for dt, n in (("f32", 1), ("bf16", 4097), ("i64", 3 * 512 + 1), ("u8", 100003), ("f64", 70000)):
        raw = source_bytes(dt, n, seed=n)
        src = to_dev(raw, dev)
        p = tmp_path / ("w_%s.svt" % dt)
        sv.write_tensor(p, src[: raw.size], dtype=dt, shape=(n,))
        name, shape, data = TF.parse(p)
        assert (name, shape) == (dt, (n,)) and np.array_equal(data, raw)
        q = tmp_path / ("w_%s.bin" % dt)
        sv.write_tensor(q, src[: raw.size], dtype=dt, raw=True)
        assert np.array_equal(np.fromfile(q, np.uint8), raw)
        back, hdr, _ = sv.read_tensor(p, device=dev)
        assert hdr["dtype"] == dt
        assert np.array_equal(as_bytes(back), raw)


def test_large_file_default_chunks(dev, tmp_path):
    """A 96 MiB uint8 file (three default chunks) loaded as fp32 (384 MiB)."""
    n = 96 << 20
    raw = np.random.default_rng(9).integers(0, 256, size=n, dtype=np.uint8)
    p = tmp_path / "big.svt"
    TF.write(p, raw, "u8")
    want, want_lost = oracle.convert(raw, "u8", "f32")
    t, hdr, lost = sv.read_tensor(p, dtype="f32", device=dev)
    assert hdr["n"] == n and lost == want_lost == 0
    assert np.array_equal(as_bytes(t), want)


def test_read_fails_loudly_then_recovers(dev, tmp_path):
    raw = source_bytes("i16", 10000, 1)
    p = tmp_path / "f.svt"
    TF.write(p, raw, "i16")
    sv.lib().sv_debug_fail_launches(1)
    with pytest.raises(sv.SynVerifyError) as e:
        sv.read_tensor(p, dtype="f32", device=dev)
    assert e.value.status == -5
    t, _, _ = sv.read_tensor(p, dtype="f32", device=dev)
    assert np.array_equal(t.cpu().numpy(), raw.view(np.int16).astype(np.float32))
