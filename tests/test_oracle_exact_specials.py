"""Pins of the oracle's exact-count special values.

Reading (Sec. 4.2.1 asks for broad, special-laden inputs; the workload's
"0.01% injected" is read as a count): with the exact flag, a logical array of
N elements holds exactly round(rate * N) special values, one at an index
drawn uniformly in each of that many equal strata of [0, N) (SPECIAL_SEL
purpose of the spec's stream); each special's kind follows the same rule as
in the Bernoulli mode.  Every other element keeps its base value.
"""
import numpy as np
import pytest

import workloads as W

KINDS_F = ("nan", "pinf", "ninf", "denorm")


def _spec(n, rate, exact=True, **kw):
    base = dict(dtype="f32", dist="normal", n=n, seed=11, stream=3, ref_offset=0, p0=0.0, p1=1.0,
                specials=KINDS_F, special_rate=rate, special_exact=exact)
    base.update(kw)
    return W.GenSpec(**base)


def _gen(oracle, spec, nbytes=None):
    a = np.zeros(nbytes or spec.n * W.DTYPE_BYTES[spec.dtype] + 256, np.uint8)
    oracle.generate([spec], a)
    return a


def test_stratum_of_by_brute_force(oracle):
    for N in (1, 2, 5, 17, 100, 1000, 4099):
        for k in sorted({1, 2, 3, 7, min(N, 40), N}):
            if k > N:
                continue
            owner = np.empty(N, np.int64)
            for s in range(k):
                owner[s * N // k:(s + 1) * N // k] = s
            got = [oracle.stratum_of(g, k, N) for g in range(N)]
            assert got == owner.tolist(), (N, k)


def test_count_rounds_to_nearest_and_is_capped():
    import oracle
    oracle.build()
    assert oracle.special_count(1e-4, 1 << 27) == 13422      # 13421.77
    assert oracle.special_count(1e-4, 1 << 10) == 0          # 0.10
    assert oracle.special_count(0.5, 3) == 2                 # 1.5 rounds up
    assert oracle.special_count(1.0, 1000) == 1000
    assert oracle.special_count(0.0, 1000) == 0


@pytest.mark.parametrize("n,rate", [(1 << 16, 1e-3), (10_007, 3e-3), (4096, 0.25)])
def test_exact_count_one_per_stratum_rest_untouched(oracle, n, rate):
    spec = _spec(n, rate)
    got = _gen(oracle, spec)[:4 * n].view(np.uint32)
    clean = _gen(oracle, spec.replace(specials=(), special_rate=0.0))[:4 * n].view(np.uint32)
    k = oracle.special_count(rate, n)
    assert k == int(np.floor(rate * n + 0.5))
    want = [oracle.special_index(n, k, spec.seed, spec.stream, s) for s in range(k)]
    for s, g in enumerate(want):  # each index inside its own stratum
        assert s * n // k <= g < (s + 1) * n // k
    changed = np.nonzero(got != clean)[0]
    assert changed.tolist() == want  # exactly k elements, the drawn ones, and nothing else changed


def test_kinds_uniform_over_the_mask(oracle):
    n, rate = 1 << 20, 0.05
    got = _gen(oracle, _spec(n, rate))[:4 * n].view(np.uint32)
    clean = _gen(oracle, _spec(n, 0.0))[:4 * n].view(np.uint32)
    sp = got[got != clean]
    assert sp.size == oracle.special_count(rate, n)
    f = sp.view(np.float32)
    counts = np.array([np.isnan(f).sum(), (f == np.inf).sum(), (f == -np.inf).sum(),
                       ((sp & 0x7F800000) == 0).sum()])
    assert counts.sum() == sp.size
    expect = sp.size / 4
    chi2 = ((counts - expect) ** 2 / expect).sum()
    assert chi2 < 16.27  # 3 degrees of freedom, p = 0.001


def test_purpose_is_not_the_perturbation_index(oracle):
    """Specials draw on SPECIAL_SEL, exact-count edits on INDEX: with the same
    seed, stream and count the two sets of indices differ."""
    n, k = 1 << 16, 64
    a = [oracle.special_index(n, k, 5, 2, s) for s in range(k)]
    b = [oracle.stratum_index(n, k, 5, 2, s) for s in range(k)]
    assert a != b and sum(x == y for x, y in zip(a, b)) < 4


def test_rate_one_makes_every_element_special(oracle):
    n = 1000
    got = _gen(oracle, _spec(n, 1.0))[:4 * n].view(np.uint32)
    f = got.view(np.float32)
    assert (~np.isfinite(f) | ((got & 0x7F800000) == 0)).all()


def test_tiny_rate_is_the_clean_stream(oracle):
    n = 1 << 12
    assert np.array_equal(_gen(oracle, _spec(n, 1e-5)), _gen(oracle, _spec(n, 0.0)))


def test_chunks_give_the_bytes_of_the_whole(oracle):
    n, rate = 60_000, 2e-3
    whole = _gen(oracle, _spec(n, rate, pcount=W.Perturb("count_add", stream=9, count=5, value=1.0),
                               cand_offset=4 * n + 256), nbytes=8 * n + 512)
    parts = np.zeros_like(whole)
    for a, b in ((0, 20_000), (20_000, 44_000), (44_000, n)):
        s = _spec(b - a, rate, elem_offset=a, logical_n=n, ref_offset=4 * a, cand_offset=4 * n + 256 + 4 * a,
                  pcount=W.Perturb("count_add", stream=9, count=5, value=1.0))
        oracle.generate([s], parts)
    assert np.array_equal(whole, parts)


def test_integer_exact_specials(oracle):
    n, rate = 1 << 16, 1e-3
    spec = W.GenSpec("i64", "permutation", n, seed=5, stream=0, ref_offset=0,
                     specials=("dup", "zero", "imin", "imax"), special_rate=rate, special_exact=True)
    got = _gen(oracle, spec)[:8 * n].view(np.int64)
    clean = _gen(oracle, spec.replace(specials=(), special_rate=0.0))[:8 * n].view(np.int64)
    k = oracle.special_count(rate, n)
    idx = {oracle.special_index(n, k, 5, 0, s) for s in range(k)}
    changed = set(np.nonzero(got != clean)[0].tolist())
    assert changed <= idx and len(changed) >= k - 4  # a DUP or ZERO may equal the value it replaces
    assert set(got[sorted(idx)].tolist()) - set(clean.tolist()) <= {np.iinfo(np.int64).min,
                                                                     np.iinfo(np.int64).max}
