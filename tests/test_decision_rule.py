"""The quantize kernel decides a code with a fused multiply-add instead of a
division: code != 0 iff |w| - s/2 > s * 2^-25 (for s >= 2^-100). This checks,
on the CPU in numpy fp32, that the rule agrees bit for bit with the correctly
rounded fp32 quotient |w| / s > 0.5 that §3.1's round(clip(w/s)) implies —
on random pairs and on pairs placed on every fp32 value around the tie."""
import numpy as np


def rule(w, s):
    w = w.astype(np.float32)
    s = s.astype(np.float32)
    # fma(-0.5, s, |w|): 0.5*s is exact; the difference rounded once to fp32
    d = (np.abs(w).astype(np.float64) - 0.5 * s.astype(np.float64)).astype(np.float32)
    t = (s * np.float32(2.0 ** -25)).astype(np.float32)
    return d > t


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
