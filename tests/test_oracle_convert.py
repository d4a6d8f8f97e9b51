"""Pins of the oracle's dtype-correct value conversion (oracle/convert.c).

What fixes the expected values, independently of the oracle's code:
- numpy's own casts (float64/float32/int -> float32/float64/float16) and
  torch's float32 -> bfloat16, both round to nearest even;
- an exact nearest-value search with Python fractions that bisects over the
  ordered encodings of the target format (a different algorithm from the
  oracle's mantissa shifting), for every source type into every float type;
- exhaustive passes over all 2^16 half and bfloat16 encodings;
- integer clamping against Python integers;
- the refusal of float -> integer and the byte copy of same-type loads.
"""
from fractions import Fraction

import numpy as np
import pytest

import oracle

FLOATS = ["f16", "bf16", "f32", "f64"]
INTS = ["u8", "i8", "i16", "u16", "i32", "u32", "i64", "u64"]
ALL = FLOATS + INTS
NP = {"f16": np.float16, "f32": np.float32, "f64": np.float64, "u8": np.uint8, "i8": np.int8, "i16": np.int16,
      "u16": np.uint16, "i32": np.int32, "u32": np.uint32, "i64": np.int64, "u64": np.uint64}
UINT = {1: np.uint8, 2: np.uint16, 4: np.uint32, 8: np.uint64}
# precision (with the hidden bit), exponent bits, bias
FMT = {"f16": (11, 5, 15), "bf16": (8, 8, 127), "f32": (24, 8, 127), "f64": (53, 11, 1023)}


def random_bits(dtype, n, seed):
    rng = np.random.default_rng(seed)
    nb = oracle.IO_DTYPE_BYTES[dtype]
    return rng.integers(0, 256, size=n * nb, dtype=np.uint8)


def small_ints(dtype, n, seed):
    """Values of an integer type concentrated where float targets round."""
    rng = np.random.default_rng(seed)
    info = np.iinfo(NP[dtype])
    mags = np.exp2(rng.uniform(0, np.log2(float(info.max)), size=n)).astype(np.float64)
    v = np.floor(mags).astype(object)
    sign = rng.integers(0, 2, size=n) if info.min < 0 else np.zeros(n, int)
    out = [int(-x) if s else int(x) for x, s in zip(v, sign)]
    out = [min(max(x, int(info.min)), int(info.max)) for x in out]
    return np.array(out, dtype=NP[dtype]).view(np.uint8)


def cvt(raw, s, d):
    out, bad = oracle.convert(raw, s, d)
    return out, bad


def bits_of(out, d):
    return out.view(UINT[oracle.IO_DTYPE_BYTES[d]])


# ---------------------------------------------------------------------------
# exact decoding of an encoding (Python integers and fractions)
# ---------------------------------------------------------------------------
def float_value(bits, d):
    p, eb, bias = FMT[d]
    frac = bits & ((1 << (p - 1)) - 1)
    e = (bits >> (p - 1)) & ((1 << eb) - 1)
    neg = (bits >> (p - 1 + eb)) & 1
    if e == (1 << eb) - 1:
        return "nan" if frac else ("-inf" if neg else "inf")
    v = Fraction(frac, 1) * Fraction(2) ** (1 - bias - (p - 1)) if e == 0 else \
        Fraction(frac | (1 << (p - 1))) * Fraction(2) ** (e - bias - (p - 1))
    return -v if neg else v


def source_value(raw_elem, s):
    nb = oracle.IO_DTYPE_BYTES[s]
    if s in FLOATS:
        return float_value(int.from_bytes(raw_elem.tobytes(), "little"), s)
    return int(raw_elem.view(NP[s])[0])


def nearest(x, d):
    """Round the exact rational x to format d, to nearest with ties to even, by
    bisection over the ordered encodings of the positive finite values.
    Returns (bits, overflowed)."""
    p, eb, bias = FMT[d]
    sign = 1 << (p - 1 + eb)
    neg = x < 0
    a = -x if neg else x
    max_bits = (((1 << eb) - 2) << (p - 1)) | ((1 << (p - 1)) - 1)
    inf_bits = ((1 << eb) - 1) << (p - 1)
    lo, hi = 0, max_bits  # largest encoding with value <= a
    if float_value(max_bits, d) <= a:
        lo = max_bits
    else:
        while hi - lo > 1:
            mid = (lo + hi) // 2
            if float_value(mid, d) <= a:
                lo = mid
            else:
                hi = mid
    below = float_value(lo, d)
    if below == a:
        b = lo
    else:
        if lo == max_bits:
            up, upv = inf_bits, below + Fraction(2) ** ((1 << eb) - 2 - bias - (p - 1))
        else:
            up, upv = lo + 1, float_value(lo + 1, d)
        dl, du = a - below, upv - a
        b = lo if dl < du else up if du < dl else (lo if lo % 2 == 0 else up)
    over = b == inf_bits
    return (b | sign) if neg else b, over


# ---------------------------------------------------------------------------
def test_refuses_float_to_int():
    for s in FLOATS:
        for d in INTS:
            with pytest.raises(ValueError):
                cvt(random_bits(s, 4, 0), s, d)


@pytest.mark.parametrize("t", ALL)
def test_same_type_is_a_byte_copy(t):
    raw = random_bits(t, 1001, 1)
    out, bad = cvt(raw, t, t)
    assert bad == 0 and np.array_equal(out, raw)


@pytest.mark.parametrize("s", INTS)
@pytest.mark.parametrize("d", INTS)
def test_int_to_int_clamps(s, d):
    if s == d:
        return
    raw = np.concatenate([random_bits(s, 3000, 2), small_ints(s, 1000, 3)])
    out, bad = cvt(raw, s, d)
    src = raw.view(NP[s]).astype(object)
    info = np.iinfo(NP[d])
    want = [min(max(int(v), int(info.min)), int(info.max)) for v in src]
    assert [int(v) for v in out.view(NP[d])] == want
    assert bad == sum(1 for v in src if int(v) < info.min or int(v) > info.max)


def test_int_edges():
    i64 = np.array([np.iinfo(np.int64).min, -1, 0, np.iinfo(np.int64).max], np.int64).view(np.uint8)
    assert list(cvt(i64, "i64", "u64")[0].view(np.uint64)) == [0, 0, 0, 2 ** 63 - 1]
    assert list(cvt(i64, "i64", "i8")[0].view(np.int8)) == [-128, -1, 0, 127]
    u64 = np.array([2 ** 64 - 1, 2 ** 63, 2 ** 63 - 1], np.uint64).view(np.uint8)
    out, bad = cvt(u64, "u64", "i64")
    assert list(out.view(np.int64)) == [2 ** 63 - 1, 2 ** 63 - 1, 2 ** 63 - 1] and bad == 2


@pytest.mark.parametrize("s", ALL)
@pytest.mark.parametrize("d", ["f32", "f64", "f16"])
def test_matches_numpy_casts(s, d):
    """Non-NaN results equal numpy's cast; overflow counted where numpy gives
    inf from a finite value."""
    if s == "bf16":
        pytest.skip("numpy has no bfloat16")
    raw = random_bits(s, 20000, 4) if s in FLOATS else np.concatenate([random_bits(s, 10000, 5),
                                                                        small_ints(s, 10000, 6)])
    out, bad = cvt(raw, s, d)
    src = raw.view(NP[s])
    with np.errstate(over="ignore", invalid="ignore"):
        want = src.astype(NP[d])
    got = out.view(NP[d])
    nan = np.isnan(want)
    assert np.array_equal(np.isnan(got), nan)
    if s == d:
        assert np.array_equal(got.view(UINT[got.itemsize]), want.view(UINT[got.itemsize]))
        return
    assert np.array_equal(got[~nan].view(UINT[got.itemsize]), want[~nan].view(UINT[got.itemsize]))
    canon = {"f16": 0x7E00, "f32": 0x7FC00000, "f64": 0x7FF8000000000000}[d]
    assert np.all(got[nan].view(UINT[got.itemsize]) == canon)
    with np.errstate(invalid="ignore"):
        finite = np.isfinite(src.astype(np.float64)) if s in FLOATS else np.ones(src.size, bool)
    assert bad == int(np.sum(finite & np.isinf(want)))


@pytest.mark.parametrize("s", ["f32", "f16", "u8", "i8", "i16", "u16"])
def test_bf16_matches_torch(s):
    """torch's float32 -> bfloat16 rounds to nearest even; sources exact in
    float32 go through it with a single rounding."""
    torch = pytest.importorskip("torch")
    raw = random_bits(s, 20000, 7)
    out, _ = cvt(raw, s, "bf16")
    src = raw.view(NP[s]).astype(np.float32)
    want = torch.from_numpy(src).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = out.view(np.uint16)
    nan = np.isnan(src)
    assert np.array_equal(got[~nan], want[~nan])
    assert np.all(got[nan] == 0x7FC0)


@pytest.mark.parametrize("s", ALL)
@pytest.mark.parametrize("d", FLOATS)
def test_nearest_by_exact_search(s, d):
    """Every result is the nearest encoding (ties to even) of the exact source
    value, found by bisection over the target's encodings with fractions."""
    if s == d:
        return
    n = 150
    raw = random_bits(s, n, 8) if s in FLOATS else np.concatenate([random_bits(s, n // 2, 9),
                                                                    small_ints(s, n - n // 2, 10)])
    out, bad = cvt(raw, s, d)
    sb, db = oracle.IO_DTYPE_BYTES[s], oracle.IO_DTYPE_BYTES[d]
    n_over = 0
    for i in range(raw.size // sb):
        x = source_value(raw[i * sb:(i + 1) * sb], s)
        got = int.from_bytes(out[i * db:(i + 1) * db].tobytes(), "little")
        p, eb, bias = FMT[d]
        if x == "nan":
            assert got == (((1 << eb) - 1) << (p - 1)) | (1 << (p - 2))
            continue
        if x in ("inf", "-inf"):
            assert got == (((1 << eb) - 1) << (p - 1)) | ((1 << (p - 1 + eb)) if x == "-inf" else 0)
            continue
        if x == 0:
            neg_zero = s in FLOATS and (int.from_bytes(raw[i * sb:(i + 1) * sb].tobytes(), "little") >> (8 * sb - 1))
            assert got == ((1 << (p - 1 + eb)) if neg_zero else 0)
            continue
        want, over = nearest(Fraction(x), d)
        assert got == want, (s, d, x, hex(got), hex(want))
        n_over += over
    assert bad == n_over


def test_exhaustive_half_and_bfloat16_sources():
    torch = pytest.importorskip("torch")
    allb = np.arange(1 << 16, dtype=np.uint16)
    h = allb.view(np.float16)
    nan_h = np.isnan(h)
    for d in ("f32", "f64"):
        got = cvt(allb.view(np.uint8), "f16", d)[0].view(NP[d])
        assert np.array_equal(got[~nan_h], h[~nan_h].astype(NP[d]))
    got = cvt(allb.view(np.uint8), "f16", "bf16")[0].view(np.uint16)
    want = torch.from_numpy(h.copy()).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(got[~nan_h], want[~nan_h]) and np.all(got[nan_h] == 0x7FC0)
    b32 = (allb.astype(np.uint32) << 16).view(np.float32)  # bfloat16 widened exactly
    nan_b = np.isnan(b32)
    got = cvt(allb.view(np.uint8), "bf16", "f32")[0].view(np.float32)
    assert np.array_equal(got[~nan_b].view(np.uint32), b32[~nan_b].view(np.uint32))
    assert np.all(got[nan_b].view(np.uint32) == 0x7FC00000)
    got, bad = cvt(allb.view(np.uint8), "bf16", "f16")
    with np.errstate(over="ignore"):
        want = b32.astype(np.float16)  # exact widening then one rounding
    assert np.array_equal(got.view(np.uint16)[~nan_b], want.view(np.uint16)[~nan_b])
    assert bad == int(np.sum(np.isfinite(b32) & np.isinf(want)))


def test_closed_forms():
    f = np.array([65519.99, 65520.0, -65536.0, 2.0 ** -25, 2.0 ** -24 * 1.5, -0.0, 1e-300], np.float64)
    out, bad = cvt(f.view(np.uint8), "f64", "f16")
    h = out.view(np.float16)
    assert h[0] == 65504 and np.isinf(h[1]) and h[2] == -np.inf and bad == 2
    assert h[3] == 0 and h[4] == 2.0 ** -23  # tie to even at 2^-25; 1.5 * 2^-24 rounds up
    assert np.signbit(h[5]) and h[5] == 0 and h[6] == 0
    big = np.array([2 ** 63 - 1, -(2 ** 63), 2 ** 24 + 1, 2 ** 24 + 3], np.int64)
    got = cvt(big.view(np.uint8), "i64", "f32")[0].view(np.float32)
    assert list(got) == [2.0 ** 63, -(2.0 ** 63), 2.0 ** 24, 2.0 ** 24 + 4]
    nanp = np.array([0x7FF0000000000001, 0xFFF8000000000123], np.uint64).view(np.uint8)
    for d, canon in (("f32", 0x7FC00000), ("f16", 0x7E00), ("bf16", 0x7FC0)):
        assert set(bits_of(cvt(nanp, "f64", d)[0], d)) == {canon}
