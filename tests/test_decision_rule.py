"""The quantize kernel decides a code with one comparison instead of a division:
code != 0 iff |w| > s/2 (for s >= 2^-100). The correctly rounded fp32 quotient
|w| / s exceeds 0.5 exactly when the real quotient exceeds the midpoint
0.5 + 2^-25 (the tie goes to the even 0.5), i.e. when |w| > s (1/2 + 2^-25); for
a normal s that threshold lies strictly between s/2 and the next fp32 value
above it, so the two conditions agree on every fp32 |w|. This checks, on the CPU
in numpy fp32, that the rule agrees bit for bit with the quotient test that
§3.1's round(clip(w/s)) implies — on random pairs, on every fp32 value around
the tie, and on every 16-bit-prefix mantissa of s."""
import numpy as np


def rule(w, s):
    w = w.astype(np.float32)
    s = s.astype(np.float32)
    return np.abs(w) > s * np.float32(0.5)  # 0.5 * s is exact for s >= 2^-125


def division(w, s):
    with np.errstate(divide="ignore", invalid="ignore"):
        return np.abs(w.astype(np.float32) / s.astype(np.float32)) > np.float32(0.5)


def test_rule_matches_division_random():
    rs = np.random.default_rng(0)
    s = np.exp(rs.uniform(np.log(2.0 ** -90), np.log(2.0 ** 90), 2_000_000)).astype(np.float32)
    q = rs.uniform(-3, 3, s.size)
    w = (q * s).astype(np.float32)
    assert np.array_equal(rule(w, s), division(w, s))


def test_rule_matches_division_at_the_tie():
    rs = np.random.default_rng(1)
    s = np.exp(rs.uniform(np.log(2.0 ** -90), np.log(2.0 ** 90), 20000)).astype(np.float32)
    half = (s * np.float32(0.5)).astype(np.float32)
    ws = []
    w = half.copy()
    for _ in range(8):  # 8 fp32 steps on each side of s/2
        w = np.nextafter(w, np.float32(np.inf))
        ws.append(w.copy())
    w = half.copy()
    for _ in range(8):
        w = np.nextafter(w, np.float32(0))
        ws.append(w.copy())
    ws.append(half)
    for w in ws:
        for sign in (1, -1):
            assert np.array_equal(rule(sign * w, s), division(sign * w, s))
    # the exact tie itself is a zero code
    assert not rule(half, s).any()


def test_rule_extremes():
    s = np.array([2.0 ** -100, 1.0, 3.0e38, 0.015625], dtype=np.float32)
    for w in (np.zeros(4, np.float32), s * np.float32(0.25), s, s * np.float32(4)):
        w = w.astype(np.float32)
        assert np.array_equal(rule(w, s), division(w, s))


def test_rule_every_scale_mantissa():
    # every s = (1 + i / 2^16) * 2^e, with w on the four fp32 values nearest s/2
    i = np.arange(1 << 16, dtype=np.float64)
    for e in (-100, -7, 0, 20):
        s = ((1.0 + i / 65536.0) * 2.0 ** e).astype(np.float32)
        half = (s * np.float32(0.5)).astype(np.float32)
        up = np.nextafter(half, np.float32(np.inf))
        down = np.nextafter(half, np.float32(0))
        for w in (half, up, down, np.nextafter(up, np.float32(np.inf))):
            assert np.array_equal(rule(w, s), division(w, s))
