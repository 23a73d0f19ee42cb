"""Pins of the oracle's quantizers and random numbers against what the paper and mathematics fix.

Definition 1 (quantization mapping), Definition 3 (compressor), Example 1 (l_inf-scaled uniform
grid), Example 2 (nearest power of two), the bounds in the appendix proof sketches of Examples 1-2,
and the published known-answer vectors of Philox4x32-10.  CPU only.
"""
import itertools
import os
import subprocess
import sys

import numpy as np
import pytest

import oracle as O

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _q(kind, bits, d, group=0, segments=None, **kw):
    return O.Quantizer(kind, bits, O.group_offsets(d, group, segments), **kw)


# ------------------------------------------------------------------------------------- Philox

def test_philox_known_answers():
    """Philox4x32-10 reproduces the published known-answer vectors (tests/golden)."""
    path = os.path.join(ROOT, "tests", "golden", "philox4x32_10_kat.txt")
    rows = [l.split() for l in open(path) if l.strip() and not l.startswith("#")]
    assert len(rows) == 3
    for r in rows:
        vals = [int(x, 16) for x in r]
        out = O.philox4x32_10(vals[0:4], vals[4:6])
        assert [int(x) for x in out] == vals[6:10]


_TRITON_PROBE = r"""
import os, sys
os.environ["TRITON_INTERPRET"] = "1"
import torch, triton, triton.language as tl
@triton.jit
def k(out_ptr, seed, N: tl.constexpr):
    offs = tl.arange(0, N)
    a, b, c, d = tl.randint4x(seed, offs, 10)
    tl.store(out_ptr + offs * 4 + 0, a)
    tl.store(out_ptr + offs * 4 + 1, b)
    tl.store(out_ptr + offs * 4 + 2, c)
    tl.store(out_ptr + offs * 4 + 3, d)
out = torch.zeros(64 * 4, dtype=torch.int32)
k[(1,)](out, int(sys.argv[1]), N=64)
print(" ".join(str(x & 0xffffffff) for x in out.tolist()))
"""


def test_philox_matches_triton_library():
    """Triton's philox (counter = (offset, 0, 0, 0), key = (seed_lo, seed_hi), 10 rounds), run in
    its CPU interpreter, is an independent library implementation of the same generator."""
    pytest.importorskip("triton")
    seed = 0x1234ABCD
    r = subprocess.run([sys.executable, "-c", _TRITON_PROBE, str(seed)], capture_output=True, text=True,
                       timeout=300)
    if r.returncode != 0:
        pytest.skip("triton interpreter unavailable: " + r.stderr.strip().splitlines()[-1][:200])
    got = np.array([int(x) for x in r.stdout.split()], dtype=np.uint64).reshape(64, 4)
    for off in range(64):
        ref = O.philox4x32_10([off, 0, 0, 0], [seed & 0xFFFFFFFF, seed >> 32])
        assert [int(x) for x in ref] == [int(x) for x in got[off]]


def test_uniform_variate_mapping():
    """U_j comes from word j mod 4 of the block j/4; 24 bits; keyed by (seed, id, round)."""
    seed, qid, t = 0x0123456789ABCDEF, 3, 7
    for j in [0, 1, 2, 3, 4, 5, 1023, 2**32 + 6, 2**33 + 3]:
        blk = j >> 2
        w = O.philox4x32_10([blk & 0xFFFFFFFF, blk >> 32, qid, t], [seed & 0xFFFFFFFF, seed >> 32])
        assert O.uniform(seed, qid, t, j) == np.float32(int(w[j & 3]) >> 8) * np.float32(2.0**-24)
    # distinct streams for distinct (id, round)
    assert O.uniform(seed, 0, 0, 5) != O.uniform(seed, 1, 0, 5)
    assert O.uniform(seed, 0, 0, 5) != O.uniform(seed, 0, 1, 5)


# -------------------------------------------------------------------------- scaled sign (Def. 3)

@pytest.mark.parametrize("d,group", [(1, 0), (7, 0), (4096, 0), (10_000, 4096), (333, 100)])
def test_sign_closed_form_error(d, group):
    """||u - Q(u)||^2 = ||u||^2 - ||u||_1^2 / G per group (the scale is the mean |u|, which is the
    least-squares scale for the fixed sign pattern), hence Definition 3 with delta > 0 and
    ||Q(u)|| <= ||u|| (Cauchy-Schwarz)."""
    rng = np.random.default_rng(d + group)
    u = (rng.standard_normal(d) * rng.choice([1e-4, 1.0, 30.0], size=d)).astype(np.float32)
    q = _q(O.Q_SIGN_L1, 1, d, group)
    words, scales, dec = q.quantize(u)
    off = q.offsets
    for g in range(q.n_groups):
        a, b = off[g], off[g + 1]
        ug, dg = u[a:b].astype(np.float64), dec[a:b].astype(np.float64)
        G = b - a
        np.testing.assert_allclose(scales[g], np.abs(ug).sum() / G, rtol=2**-23)
        err2 = ((ug - dg) ** 2).sum()
        closed = (ug ** 2).sum() - np.abs(ug).sum() ** 2 / G
        assert abs(err2 - closed) <= 1e-5 * (ug ** 2).sum() + 1e-30
        nu, nerr = np.sqrt((ug ** 2).sum()), np.sqrt(err2)
        if G > 1:
            delta = 1 - np.sqrt(max(0.0, 1 - np.abs(ug).sum() ** 2 / (G * (ug ** 2).sum())))
            assert delta > 0 and nerr <= (1 - delta) * nu * (1 + 1e-6)
        assert np.sqrt((dg ** 2).sum()) <= nu * (1 + 1e-6)


def test_sign_of_zero_is_plus_one_and_bits():
    u = np.array([0.0, -0.0, 1.0, -1.0, 2.0, -3.0], dtype=np.float32)
    q = _q(O.Q_SIGN_L1, 1, 6, 0)
    words, scales, dec = q.quantize(u)
    s = np.float32(7.0 / 6.0)
    assert scales[0] == s
    np.testing.assert_array_equal(dec, np.array([s, s, s, -s, s, -s], np.float32))
    bits = np.unpackbits(words.view(np.uint8), bitorder="little")[:6]
    np.testing.assert_array_equal(bits, [1, 1, 1, 0, 1, 0])


def test_sign_all_patterns_brute_force():
    """Every sign pattern of a 10-vector: decoded values are s * sign(u) and the packed bit of
    coordinate j is bit j of the stream (least significant first)."""
    rng = np.random.default_rng(1)
    mags = rng.uniform(0.1, 2.0, size=10).astype(np.float32)
    q = _q(O.Q_SIGN_L1, 1, 10, 0)
    for pat in range(1 << 10):
        sgn = np.array([1 if (pat >> j) & 1 else -1 for j in range(10)], np.float32)
        u = mags * sgn
        words, scales, dec = q.quantize(u)
        assert int(words[0]) == pat
        np.testing.assert_array_equal(dec, scales[0] * sgn)


def test_sign_segments_use_true_lengths():
    segs = [3, 1, 64, 5]
    d = sum(segs)
    u = np.arange(1, d + 1, dtype=np.float32)
    q = _q(O.Q_SIGN_L1, 1, d, -1, segs)
    _, scales, _ = q.quantize(u)
    off = np.cumsum([0] + segs)
    for g in range(4):
        assert scales[g] == np.float32(u[off[g]:off[g + 1]].astype(np.float64).mean())


# ------------------------------------------------------------------ Example 1: uniform l_inf grid

def _grid_argmin(u, s, L):
    """Brute force: the point of s * {i/L : |i| <= L}^d nearest to u, by enumerating the grid."""
    d = len(u)
    best, best_err = None, np.inf
    for idx in itertools.product(range(-L, L + 1), repeat=d):
        p = s * np.array(idx, dtype=np.float64) / L
        err = np.sum((u.astype(np.float64) - p) ** 2)
        if err < best_err:
            best, best_err = np.array(idx), err
    return best


@pytest.mark.parametrize("bits,d", [(2, 3), (2, 5), (4, 3)])
def test_uniform_is_grid_argmin(bits, d):
    """Q(x) = Q1(||x||_inf) * argmin over M_2^d of ||x/Q1 - y|| (Example 1), checked by enumerating
    M_2^d, with M_2 = {i/(2^k - 1) : |i| <= 2^k - 1} and k = bits - 1."""
    L = 2 ** (bits - 1) - 1
    rng = np.random.default_rng(bits * 10 + d)
    q = _q(O.Q_UNIFORM_MAX, bits, d, 0)
    for _ in range(60):
        u = rng.standard_normal(d).astype(np.float32)
        words, scales, dec = q.quantize(u)
        s = float(np.max(np.abs(u)))
        assert scales[0] == np.float32(s)
        idx = _grid_argmin(u, s, L)
        np.testing.assert_allclose(dec, s * idx / L, rtol=2e-7, atol=0)
        # offset-binary code q + L in b bits, least significant first
        raw = np.array([(int(words[(j * bits) // 32]) >> ((j * bits) % 32)) & ((1 << bits) - 1)
                        for j in range(d)])
        np.testing.assert_array_equal(raw - L, idx)


@pytest.mark.parametrize("bits", [2, 4, 8])
def test_uniform_error_bounds(bits):
    """The Example 1 bound of the appendix, ||Q(x) - x|| <= sqrt((d-1)/(d-1+2^k)) ||x|| (+ the Q1
    rounding term), the tighter per-coordinate form |x_j - Q(x)_j| <= s/(2L), and Definition 1's
    ||Q(x)|| <= (2 - delta) ||x||.  The largest coordinate is exact."""
    k = bits - 1
    L = 2 ** k - 1
    rng = np.random.default_rng(bits)
    for d in [1, 2, 5, 64, 1000]:
        q = _q(O.Q_UNIFORM_MAX, bits, d, 0)
        for _ in range(20):
            x = (rng.standard_normal(d) * 10 ** rng.uniform(-6, 3)).astype(np.float32)
            _, scales, dec = q.quantize(x)
            x64, q64 = x.astype(np.float64), dec.astype(np.float64)
            s = float(scales[0])
            err = np.linalg.norm(x64 - q64)
            bound = np.sqrt((d - 1) / (d - 1 + 2 ** k)) * np.linalg.norm(x64)
            assert err <= bound * (1 + 1e-6) + 2.0 ** -126 * np.sqrt(d)
            assert np.all(np.abs(x64 - q64) <= s / (2 * L) * (1 + 1e-6))
            j = int(np.argmax(np.abs(x)))
            assert dec[j] == x[j]
            delta = 1 - bound / max(np.linalg.norm(x64), 1e-300)
            assert np.linalg.norm(q64) <= (2 - delta) * np.linalg.norm(x64) * (1 + 1e-6)


def test_uniform_tight_bound_attained():
    """The worst case of the grid: all but one coordinate just below a midpoint s/(2L); the
    error then equals sqrt((d-1)/(d-1+4L^2)) ||x|| (within float rounding)."""
    bits, d = 4, 9
    L = 7
    x = np.full(d, np.float32(0.5 / L * (1 - 1e-5)), np.float32)
    x[0] = 1.0
    q = _q(O.Q_UNIFORM_MAX, bits, d, 0)
    _, _, dec = q.quantize(x)
    err = np.linalg.norm(x.astype(np.float64) - dec)
    tight = np.sqrt((d - 1) / (d - 1 + 4 * L * L)) * np.linalg.norm(x.astype(np.float64))
    assert abs(err - tight) <= 1e-4 * tight


def test_uniform_zero_group_and_ties():
    q = _q(O.Q_UNIFORM_MAX, 4, 8, 4)
    x = np.array([0, 0, 0, 0, 7, 3.5, -0.5, 1.5], np.float32)  # block 2: s = 7, y = x (L = 7)
    words, scales, dec = q.quantize(x)
    assert scales[0] == 0 and np.all(dec[:4] == 0)          # Q = 0 when Q1(||x||_inf) = 0
    # ties of the nearest grid point go to the even index: 3.5 -> 4, -0.5 -> 0, 1.5 -> 2
    np.testing.assert_array_equal(dec[4:], np.array([7, 4, 0, 2], np.float32))


def test_uniform_stochastic_rounding_properties():
    """Stochastic grid rounding: q is floor(y) or ceil(y); over independent rounds its mean is
    y (unbiased up to 2^-24 of a step); the up-probability of a fixed y equals frac(y)."""
    d, bits = 4096, 4
    L = 7
    rng = np.random.default_rng(5)
    x = rng.standard_normal(d).astype(np.float32)
    x[0] = 4.0                        # s = 4 -> the grid step is 4/7
    q = _q(O.Q_UNIFORM_MAX, bits, d, 0, stochastic=True)
    y = (x / np.float32(4.0)) * np.float32(L)
    fl = np.floor(y.astype(np.float64))
    R = 400
    acc = np.zeros(d)
    for t in range(R):
        words, scales, dec = q.quantize(x, seed=99, qid=2, t=t)
        qi = np.rint(dec.astype(np.float64) / (4.0 / L)).astype(np.int64)
        assert np.all((qi == fl) | (qi == fl + 1))
        acc += dec
    mean_err = acc / R - x.astype(np.float64)
    step = 4.0 / L
    sigma = step * 0.5 / np.sqrt(R)  # the largest per-coordinate std of the mean
    assert np.abs(mean_err).max() < 5.5 * sigma
    assert abs(mean_err.mean()) < 5 * step * 0.5 / np.sqrt(R * d)
    # frequency of rounding up for one coordinate across many counters: frac(y)
    xs = np.full(4096, np.float32(0.3), np.float32)
    xs[0] = 1.0
    q1 = _q(O.Q_UNIFORM_MAX, 2, 4096, 0, stochastic=True)  # L = 1: y = x, up means 1
    ups = 0
    for t in range(25):
        _, _, dec = q1.quantize(xs, seed=7, qid=0, t=t)
        ups += int((dec[1:] == 1.0).sum())
    n = 25 * 4095
    p = 0.3
    assert abs(ups / n - p) < 5 * np.sqrt(p * (1 - p) / n)


# --------------------------------------------------------------------- Example 2: powers of two

def test_pow2_is_nearest_power_and_bounds():
    """Example 2 with the paper's k = -17, K = -11: Q(x) = sign(x) * argmin over {2^k..2^K} of
    | |x| - y | (enumerated), 4 bits (1 + ceil(log2(K - k + 1))), Q(0) = 0, and the appendix
    constants delta = 1/2, delta' = 2^k sqrt(d) when ||x||_inf <= 2^K + 2^(K-1)."""
    k, K, bits = -17, -11, 4
    M = np.array([2.0 ** j for j in range(k, K + 1)])
    rng = np.random.default_rng(3)
    d = 2000
    x = (np.sign(rng.standard_normal(d)) * 2.0 ** rng.uniform(k - 3, K + 0.5, d)).astype(np.float32)
    x[:3] = [0.0, 2.0 ** k, -(2.0 ** K + 2.0 ** (K - 1))]
    q = O.Quantizer(O.Q_POW2, bits, O.group_offsets(d, 0), pow2_k=k, pow2_K=K)
    words, _, dec = q.quantize(x)
    assert dec[0] == 0.0
    for j in range(1, d):
        a = abs(float(x[j]))
        dist = np.abs(M - a)
        best = M[dist == dist.min()].max()  # the tie at 1.5 * 2^j goes up
        assert dec[j] == np.float32(np.sign(x[j]) * best)
    x64, q64 = x.astype(np.float64), dec.astype(np.float64)
    assert np.linalg.norm(x64 - q64) <= 0.5 * np.linalg.norm(x64) + 2.0 ** k * np.sqrt(d)
    assert q.message_bits(d) == d * 4
    # exact midpoints 1.5 * 2^j between two levels go up; just below them go down
    mid = np.array([1.5 * 2.0 ** j for j in range(k, K)], np.float32)
    qm = O.Quantizer(O.Q_POW2, bits, O.group_offsets(len(mid), 0), pow2_k=k, pow2_K=K)
    np.testing.assert_array_equal(qm.quantize(mid)[2], (2 * mid / 1.5).astype(np.float32))
    below = np.nextafter(mid, np.float32(0))
    np.testing.assert_array_equal(qm.quantize(-below)[2], (-mid / 1.5).astype(np.float32))
    # The appendix bounds each coordinate's error by |x_j|/2, hence |Q(x)_j| <= 1.5 |x_j|, for
    # 2^(k-1) <= |x_j| <= 2^K + 2^(K-1).  Both hold from (2/3) 2^k upwards ...
    lo, hi = 2.0 ** k * 2.0 / 3.0, 2.0 ** K + 2.0 ** (K - 1)
    ok = (np.abs(x64) >= lo) & (np.abs(x64) <= hi)
    assert np.all(np.abs(x64[ok] - q64[ok]) <= 0.5 * np.abs(x64[ok]))
    assert np.all(np.abs(q64[ok]) <= 1.5 * np.abs(x64[ok]))
    # ... but not on [2^(k-1), (2/3) 2^k), nor below, where Q lifts |x_j| up to 2^k (a reading
    # recorded with the design): e.g. |x_j| = 2^(k-1) maps to 2^k, an error of |x_j|.
    xe = np.array([2.0 ** (k - 1), 0.6 * 2.0 ** k], np.float32)
    _, _, de = O.Quantizer(O.Q_POW2, bits, O.group_offsets(2, 0), pow2_k=k, pow2_K=K).quantize(xe)
    assert np.all(de == np.float32(2.0 ** k))
    assert np.all(np.abs(de.astype(np.float64)) > 1.5 * xe.astype(np.float64))


def test_identity_is_exact():
    rng = np.random.default_rng(0)
    x = rng.standard_normal(100).astype(np.float32)
    q = O.Quantizer(O.Q_IDENTITY, 32, O.group_offsets(100, 0))
    words, _, dec = q.quantize(x)
    np.testing.assert_array_equal(dec, x)
    np.testing.assert_array_equal(words[:100], x.view(np.uint32))
    assert q.message_bits(100) == 3200
