"""The floating-point facts the construction kernels rely on, checked on the
CPU in IEEE arithmetic (numpy float32 / Python float, exact rationals as the
reference).  Nothing here runs or imports GPU code: these pin the arithmetic
each kernel's exactness argument rests on.

- Centre sums (Eq. summary): a bf16 value x splits on the FP32 pipe as
  s = x + C1, h = s - C1, l = x - h, t = l + C2 (C1 = 1.5 * 2^8, C2 = 1.5 *
  2^-9), and bits(s) - bits(C1) = h * 2^15, bits(t) - bits(C2) = l * 2^32 give
  x * 2^32 exactly whenever x is a multiple of 2^-32 below 128; otherwise the
  check |t - C2 - l| != 0 or |x| >= 128 flags it.
- Centre means: RN(S / c) = fma(fma(-q0, c, S), y, q0) with y = RN(1 / c),
  q0 = RN(S y) (Markstein's correction) for the kernel's integer counts c.
- Lloyd assignment keys: a distance with a centre index in its 8 low
  significand bits is within 2^-15 |d| of it, and the fminf / fmaxf network
  keeps the three smallest keys.
"""
import random
from fractions import Fraction

import numpy as np

F32 = np.float32
C1 = F32(384.0)
C2 = F32(1.5 * 2.0 ** -9)


def _bits(x):
    return int(np.array([x], dtype=np.float32).view(np.uint32)[0])


def _bf16_exact(b):
    e, m7 = (b >> 7) & 0xFF, b & 0x7F
    if e == 255:
        return None
    v = Fraction(m7, 2 ** 133) if e == 0 else Fraction(m7 | 0x80) * Fraction(2) ** (e - 134)
    return -v if b & 0x8000 else v


def test_magic_split_is_exact_on_its_window_and_flags_the_rest():
    b = np.arange(65536, dtype=np.uint32)
    x = (b << 16).view(np.float32)
    with np.errstate(all="ignore"):
        s = x + C1
        h = s - C1
        l = x - h
        t = l + C2
        err = np.abs((t - C2) - l)
        ok = (err == 0) & (np.abs(x) < F32(128))
    hi = (s.view(np.uint32).astype(np.int64) - _bits(C1)) & 0xFFFFFFFF
    lo = (t.view(np.uint32).astype(np.int64) - _bits(C2)) & 0xFFFFFFFF
    hi = np.where(hi >= 2 ** 31, hi - 2 ** 32, hi)
    lo = np.where(lo >= 2 ** 31, lo - 2 ** 32, lo)
    n_ok = 0
    for i in range(65536):
        v = _bf16_exact(i)
        in_window = v is not None and abs(v) < 128 and (v * 2 ** 32).denominator == 1
        assert bool(ok[i]) == in_window, hex(i)
        if ok[i]:
            n_ok += 1
            assert abs(int(hi[i])) < 2 ** 22 and abs(int(lo[i])) <= 2 ** 16
            assert Fraction(int(hi[i]) * 2 ** 17 + int(lo[i]), 2 ** 32) == v, hex(i)
    # every bf16 multiple of 2^-32 below 128: exponents 102..133 in full, 95..101
    # with trailing zeros, and both zeros
    assert n_ok == 2 * (32 * 128 + 127) + 2


def test_mod_2_32_lane_sums_recover_64_terms():
    rng = random.Random(3)
    for _ in range(2000):
        terms = [rng.randint(-(2 ** 22) + 1, 2 ** 22 - 1) for _ in range(64)]
        c = rng.getrandbits(32)
        acc = sum((t + c) for t in terms) & 0xFFFFFFFF       # bits(s) summed mod 2^32
        got = (acc - 64 * c) & 0xFFFFFFFF
        got = got - 2 ** 32 if got >= 2 ** 31 else got
        assert got == sum(terms)


def _fma(a, b, c):
    return float(Fraction(a) * Fraction(b) + Fraction(c))


def test_markstein_corrected_quotient_is_correctly_rounded():
    rng = random.Random(5)
    cases = [(1, 3), (-1, 7), (2 ** 53 - 1, 3), (2 ** 53 + 1, 65535), (2 ** 62 - 1, 2 ** 17),
             ((2 ** 53 - 1) * 3, 98304), (-(2 ** 62), 131071)]
    for _ in range(20000):
        t = rng.randint(-(2 ** rng.choice([20, 40, 62])), 2 ** rng.choice([20, 40, 62]))
        cases.append((t, rng.choice([rng.randint(1, 131072), rng.randint(1, 64)])))
    for t, c in cases:
        S = float(t)                          # the integer sum, rounded once
        y = (1.0 / c) * 2.0 ** -32            # RN(1 / (c 2^32))
        b = float(c) * 2.0 ** 32
        q0 = S * y
        q = _fma(_fma(-q0, b, S), y, q0)
        assert q == (S * 2.0 ** -32) / c, (t, c)


def _key(d, col):
    return np.array([(_bits(F32(d)) & ~0xFF) | col], dtype=np.uint32).view(np.float32)[0]


def test_packed_keys_stay_close_and_the_network_keeps_the_best_three():
    rng = np.random.default_rng(11)
    for _ in range(400):
        n = int(rng.integers(3, 257))
        d = (rng.standard_normal(n) * 10.0 ** rng.integers(-3, 4)).astype(np.float32)
        keys = np.array([_key(d[j], j) for j in range(n)], dtype=np.float32)
        assert np.all(np.abs(keys.astype(np.float64) - d) <= 2.0 ** -15 * np.abs(d.astype(np.float64)))
        x0 = x1 = x2 = np.float32(np.inf)
        for k in keys:
            t0 = max(x0, k)
            x0 = min(x0, k)
            t1 = max(x1, t0)
            x1 = min(x1, t0)
            x2 = min(x2, t1)
        assert [x0, x1, x2] == sorted(keys.tolist())[:3]
        # distinct centres never tie, and the index is recoverable
        assert len(set(keys.tolist())) == n
        assert int(_bits(x0) & 0xFF) == int(np.argmin(keys))


def test_byte_permute_selector_places_the_centre_index():
    def perm(x, y, s):
        bs = [(x >> (8 * i)) & 255 for i in range(4)] + [(y >> (8 * i)) & 255 for i in range(4)]
        return sum(bs[(s >> (4 * i)) & 7] << (8 * i) for i in range(4))

    rng = random.Random(7)
    for _ in range(20000):
        x = rng.getrandbits(32)
        k, m, b = rng.randrange(16), rng.randrange(4), rng.randrange(4)
        cols = (16 * k * 0x01010101 + 0x03020100 + 4 * m * 0x01010101) & 0xFFFFFFFF
        assert perm(x, cols, 0x3214 + b) == ((x & ~0xFF) | (16 * k + 4 * m + b))
