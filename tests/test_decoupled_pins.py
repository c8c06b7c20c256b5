"""Pins of the decoupled-quantizer oracle (oracle/decoupled_oracle.py): reduction
to the standard quantizer at factor 1, the Gaussian zero ratio at a lowered
threshold (closed form), brute force on tiny inputs, and closed forms of the
magnitude's gradient."""
import math

import numpy as np

from oracle import decoupled_oracle as D
from oracle import tq_oracle as O
from paper_2606_18114_gb300 import synth


def test_factor_one_is_the_standard_quantizer():
    w = synth.latent_weights(96, 1024, seed=3)
    for g in (32, 128, 512):
        codes, s, z, c, tau = D.quantize_decoupled(w, g)
        ref = O.quantize(w, g)
        assert np.array_equal(codes, ref[0]) and np.array_equal(s, ref[1])
        assert np.array_equal(z, ref[2]) and np.array_equal(tau, s)


def test_lowered_threshold_gaussian_zero_ratio():
    """Zero iff |w| < f s / 2 and s -> sigma sqrt(2/pi): the zero ratio of N(0, sigma^2)
    weights tends to P(|z| < (f / 2) sqrt(2 / pi)) = erf(f / (2 sqrt(pi))) (0.2505 at
    f = 0.8, 0.3101 at f = 1)."""
    w = synth.latent_weights(2048, 2048, seed=4)
    g = 512  # a long group keeps the absmean close to its expectation
    for f in (0.8, 1.0):
        _, _, z, _, _ = D.quantize_decoupled(w, g, np.full(2048, f, np.float32))
        ratio = z.sum() / w.size
        assert abs(ratio - math.erf(f / (2 * math.sqrt(math.pi)))) < 3e-3, (f, ratio)


def test_asymmetric_rows():
    """The paper's gate rows (the first half of the rows here) at 0.8 x absmean,
    the rest at 1: fewer zeros on the lowered rows, the other rows untouched."""
    w = synth.latent_weights(256, 1024, seed=5)
    f = np.ones(256, np.float32)
    f[:128] = 0.8
    _, s, z, c, tau = D.quantize_decoupled(w, 128, f)
    ref = O.quantize(w, 128)
    assert np.array_equal(z[128:], ref[2][128:]) and np.array_equal(c[128:], ref[3][128:])
    assert z[:128].sum() < ref[2][:128].sum()
    np.testing.assert_array_equal(tau[:128], (s[:128] * np.float32(0.8)).astype(np.float32))


def test_brute_force_tiny():
    rs = np.random.default_rng(6)
    n, k, g = 3, 64, 32
    w = (rs.standard_normal((n, k)) * 0.02).astype(np.float32)
    f = np.array([0.8, 1.0, 0.5], np.float32)
    dw = rs.standard_normal((n, k))
    codes, s, z, c, tau = D.quantize_decoupled(w, g, f)
    da = D.alpha_grad(dw, codes, g)
    for r in range(n):
        for j in range(k // g):
            grp = [float(w[r, j * g + i]) for i in range(g)]
            s_ = sum(abs(v) for v in grp) / g
            t_ = float(np.float32(np.float32(s_) * f[r]))
            cs = []
            for v in grp:
                q = float(np.float32(v) / np.float32(t_))
                q = max(-1.0, min(1.0, q))
                cs.append(int(round(q)) if abs(abs(q) - 0.5) > 0 else 0)
            assert abs(float(s[r, j]) - s_) <= 1e-7 * s_
            assert cs == [int(x) for x in c[r, j * g:(j + 1) * g]]
            assert z[r, j] == cs.count(0)
            assert abs(da[r, j] - sum(float(dw[r, j * g + i]) * cs[i] for i in range(g))) < 1e-12


def test_alpha_grad_closed_forms():
    """With dW^ = c the gradient counts the non-zero codes; with dW^ = 1 it sums them."""
    w = synth.latent_weights(64, 512, seed=7)
    codes, _, z, c, _ = D.quantize_decoupled(w, 128)
    cnt = D.alpha_grad(c.astype(np.float64), codes, 128)
    np.testing.assert_array_equal(cnt, 128 - z)
    tot = D.alpha_grad(np.ones(c.shape), c, 128)
    np.testing.assert_array_equal(tot, c.reshape(64, 4, 128).sum(axis=2))
