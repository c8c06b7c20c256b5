"""Pins of the learnable-scale oracle (oracle/learnable_oracle.py) against what the
mathematics fixes independently of its formulas: the reduction to §3.1's
quantizer at the absmean, the sign symmetry of the scale, torch autograd of the
straight-through surrogate, finite differences of that surrogate, closed forms
at the extremes of the scale, and pure-Python brute force."""
import numpy as np
import torch

from oracle import adamw_oracle as A
from oracle import learnable_oracle as L
from oracle import tq_oracle as O
from paper_2606_18114_gb300 import synth


def _scales(w, g, seed, lo=0.5, hi=2.0):
    """The absmean times a random factor per group (a trained scale drifts from it)."""
    n, k = w.shape
    s = O.quantize(w, g)[1]
    f = np.random.default_rng(seed).uniform(lo, hi, size=s.shape).astype(np.float32)
    return (s * f).astype(np.float32)


def test_absmean_scales_reduce_to_the_standard_quantizer():
    w = synth.latent_weights(64, 1024, seed=11)
    for g in (32, 128, 512):
        codes, s, z, c = O.quantize(w, g)
        lc, lz, lcc = L.quantize_with_scales(w, g, s)
        assert np.array_equal(lc, codes) and np.array_equal(lz, z) and np.array_equal(lcc, c)


def test_negative_scales_flip_the_codes():
    """s -> -s negates every code, so s * c (the dequantized weight) is unchanged."""
    w = synth.latent_weights(32, 512, seed=12)
    s = _scales(w, 128, seed=1)
    _, z1, c1 = L.quantize_with_scales(w, 128, s)
    _, z2, c2 = L.quantize_with_scales(w, 128, -s)
    assert np.array_equal(c2, -c1) and np.array_equal(z1, z2)
    sr = np.repeat(s, 128, axis=1)
    assert np.array_equal(sr * c1, (-sr) * c2)


def test_zero_and_special_scales():
    """s = 0: the sign of w (0 for w = 0); an infinite scale: every code 0."""
    w = synth.latent_weights(4, 64, seed=13)
    w[0, :5] = 0.0
    s = np.zeros((4, 2), np.float32)
    s[3, :] = np.inf
    _, z, c = L.quantize_with_scales(w, 32, s)
    assert np.array_equal(c[:3], np.sign(w[:3]).astype(np.int8))
    assert np.all(c[3] == 0) and np.all(z[3] == 32)
    assert z[0, 0] == 5


def _surrogate_grad_torch(w, dw, c, s, g):
    """ds by torch autograd (fp64) of W^ = s * (clip(w / s) + const), const =
    c - clip(w / s) held fixed: the straight-through rounding."""
    n, k = w.shape
    wt = torch.tensor(w, dtype=torch.float64)
    st = torch.tensor(s, dtype=torch.float64, requires_grad=True)
    sr = st.repeat_interleave(g, dim=1)
    q = (wt / sr).clamp(-1.0, 1.0)
    ct = torch.tensor(c, dtype=torch.float64)
    w_hat = sr * (q + (ct - q).detach())
    (w_hat * torch.tensor(dw, dtype=torch.float64)).sum().backward()
    return st.grad.numpy()


def test_scale_grad_matches_torch_autograd():
    rs = np.random.default_rng(14)
    for g in (32, 128):
        w = synth.latent_weights(48, 512, seed=15 + g)
        s = _scales(w, g, seed=g)
        s[0, 0] = -s[0, 0]  # one negative scale
        dw = rs.standard_normal(w.shape)
        _, _, c = L.quantize_with_scales(w, g, s)
        got = L.scale_grad(w, dw, c, s, g)
        ref = _surrogate_grad_torch(w, dw, c, s, g)
        np.testing.assert_allclose(got, ref, rtol=1e-10, atol=1e-12)


def test_scale_grad_matches_finite_differences():
    """Central differences of F(s) = sum dW * (s (c - clip(w/s0)) + s clip(w/s)) at s0."""
    rs = np.random.default_rng(16)
    g = 64
    w = synth.latent_weights(8, 256, seed=17).astype(np.float64)
    s0 = _scales(w.astype(np.float32), g, seed=3).astype(np.float64)
    dw = rs.standard_normal(w.shape)
    _, _, c = L.quantize_with_scales(w.astype(np.float32), g, s0.astype(np.float32))
    got = L.scale_grad(w.astype(np.float32), dw, c, s0.astype(np.float32), g)
    n, k = w.shape
    const = c.astype(np.float64) - np.clip(w / np.repeat(s0, g, 1), -1, 1)

    def F(s):
        sr = np.repeat(s, g, 1)
        return (dw * (sr * const + sr * np.clip(w / sr, -1, 1))).reshape(n, k // g, g).sum(axis=2)

    h = 1e-7 * np.abs(s0)
    fd = np.zeros_like(s0)
    for j in range(k // g):
        e = np.zeros_like(s0)
        e[:, j] = h[:, j]
        fd[:, j] = ((F(s0 + e) - F(s0 - e)) / (2 * h))[:, j]
    np.testing.assert_allclose(got, fd, rtol=1e-5, atol=1e-9)


def test_scale_grad_closed_forms():
    """All |w| >= |s| (a tiny scale): every code is sign(w) and no weight is inside
    the clip, ds = sum dW sign(w). A huge scale: every code 0 and every weight
    inside, ds = -sum dW w / s."""
    rs = np.random.default_rng(18)
    w = synth.latent_weights(16, 256, seed=19)
    w[np.abs(w) < 1e-6] = 1e-3
    dw = rs.standard_normal(w.shape)
    tiny = np.full((16, 2), 1e-7, np.float32)
    _, _, c = L.quantize_with_scales(w, 128, tiny)
    assert np.array_equal(c, np.sign(w).astype(np.int8))
    np.testing.assert_allclose(L.scale_grad(w, dw, c, tiny, 128),
                               (dw * np.sign(w)).reshape(16, 2, 128).sum(2), rtol=1e-12)
    huge = np.full((16, 2), 10.0, np.float32)
    _, z, c = L.quantize_with_scales(w, 128, huge)
    assert np.all(c == 0) and np.all(z == 128)
    np.testing.assert_allclose(L.scale_grad(w, dw, c, huge, 128),
                               -(dw * w.astype(np.float64)).reshape(16, 2, 128).sum(2) / 10.0,
                               rtol=1e-12)


def test_brute_force_tiny():
    rs = np.random.default_rng(20)
    n, k, g = 3, 64, 32
    w = (rs.standard_normal((n, k)) * 0.02).astype(np.float32)
    s = np.array([[0.01, -0.02], [0.0, 0.03], [0.015, 1e-9]], np.float32)
    dw = rs.standard_normal((n, k))
    codes, z, c = L.quantize_with_scales(w, g, s)
    ds = L.scale_grad(w, dw, codes, s, g)
    for r in range(n):
        for j in range(k // g):
            sv = float(s[r, j])
            cs, acc = [], 0.0
            for i in range(g):
                x = float(w[r, j * g + i])
                if sv == 0.0:
                    q = float("nan") if x == 0.0 else (float("inf") if x > 0 else float("-inf"))
                else:
                    q = float(np.float32(x) / np.float32(sv))
                cc = 0 if q != q else int(round(max(-1.0, min(1.0, q)))) if abs(abs(q) - 0.5) > 0 else 0
                cs.append(cc)
                d = float(dw[r, j * g + i])
                acc += d * cc
                if abs(x) < abs(sv):
                    acc -= d * x / sv
            assert cs == [int(v) for v in c[r, j * g:(j + 1) * g]], (r, j)
            assert z[r, j] == cs.count(0)
            assert abs(ds[r, j] - acc) <= 1e-9 * (1 + abs(acc)), (r, j, ds[r, j], acc)


def test_fused_step_is_adamw_then_quantize():
    w = synth.latent_weights(32, 256, seed=21)
    rs = np.random.default_rng(22)
    gr = (rs.standard_normal(w.shape) * 1e-3).astype(np.float32)
    z = np.zeros_like(w)
    c = A.step_constants(lr=2.5e-4, beta1=0.9, beta2=0.95, eps=1e-8, weight_decay=0.01, step=1)
    s = _scales(w, 64, seed=5)
    w1, m1, v1, codes, zc = L.adamw_requantize_with_scales(w, gr, z, z, 64, c, s)
    w_ref, m_ref, v_ref = A.adamw_step(w, gr, z, z, c)
    assert np.array_equal(w1, w_ref) and np.array_equal(m1, m_ref) and np.array_equal(v1, v_ref)
    assert np.array_equal(codes, L.quantize_with_scales(w_ref, 64, s)[0])
