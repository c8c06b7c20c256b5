"""Pins of the AdamW + requantize oracle (oracle/adamw_oracle.py) against what the
optimizer's definition fixes: the closed form of the first step from zero
moments, the decay of the moments under a zero gradient, and agreement with an
independent implementation (torch.optim.AdamW) over several steps."""
import math

import numpy as np
import pytest
import torch

from oracle import adamw_oracle as A
from oracle import tq_oracle as O

HP = dict(lr=2.5e-4, beta1=0.9, beta2=0.95, eps=1e-8, weight_decay=0.01)  # §3.3


def _rand(shape, seed, std=1.0):
    return (np.random.default_rng(seed).standard_normal(shape) * std).astype(np.float32)


def test_first_step_closed_form():
    """From m = v = 0 at t = 1: m = (1 - b1) g, v = (1 - b2) g^2 and the step is
    lr * g / (|g| + eps): each weight moves by about lr against its gradient."""
    w0 = _rand((64, 256), 1, 0.02)
    g = _rand((64, 256), 2, 1e-3)
    c = A.step_constants(step=1, **HP)
    w1, m1, v1 = A.adamw_step(w0, g, np.zeros_like(w0), np.zeros_like(w0), c)
    g64 = g.astype(np.float64)
    np.testing.assert_allclose(m1, (1 - HP["beta1"]) * g64, rtol=2e-7, atol=0)
    np.testing.assert_allclose(v1, (1 - HP["beta2"]) * g64 ** 2, rtol=5e-7, atol=0)
    expect = w0.astype(np.float64) * (1 - HP["lr"] * HP["weight_decay"]) - \
        HP["lr"] * g64 / (np.abs(g64) + HP["eps"])
    err = np.abs(w1.astype(np.float64) - expect)
    assert err.max() <= 4 * np.spacing(np.float32(0.1)), err.max()
    # the step is lr in magnitude wherever |g| >> eps
    step = w0.astype(np.float64) * (1 - HP["lr"] * HP["weight_decay"]) - w1
    big = np.abs(g64) > 1e-5
    np.testing.assert_allclose(np.abs(step[big]), HP["lr"], rtol=2e-3)
    assert np.all(np.sign(step[big]) == np.sign(g64[big]))


def test_zero_gradient_decays_moments():
    """With g = 0 the moments decay by beta1, beta2 and the weights move by the
    bias-corrected ratio of the decayed moments, plus the weight decay."""
    w0 = _rand((32, 128), 3, 0.02)
    m0 = _rand((32, 128), 4, 1e-4)
    v0 = np.abs(_rand((32, 128), 5, 1e-8)) + np.float32(1e-9)
    t = 7
    c = A.step_constants(step=t, **HP)
    w1, m1, v1 = A.adamw_step(w0, np.zeros_like(w0), m0, v0, c)
    np.testing.assert_allclose(m1, HP["beta1"] * m0.astype(np.float64), rtol=2e-7)
    np.testing.assert_allclose(v1, HP["beta2"] * v0.astype(np.float64), rtol=2e-7)
    mh = HP["beta1"] * m0.astype(np.float64) / (1 - HP["beta1"] ** t)
    vh = HP["beta2"] * v0.astype(np.float64) / (1 - HP["beta2"] ** t)
    expect = w0 * (1 - HP["lr"] * HP["weight_decay"]) - HP["lr"] * mh / (np.sqrt(vh) + HP["eps"])
    np.testing.assert_allclose(w1, expect, rtol=0, atol=4e-9)


def test_agrees_with_torch_adamw_over_steps():
    """Five steps against torch.optim.AdamW (fp32 CPU, an independent
    implementation with its own rounding order): weights, moments and the
    accumulated update agree to fp32 rounding."""
    shape = (48, 384)
    w = _rand(shape, 6, 0.02)
    tw = torch.nn.Parameter(torch.from_numpy(w.copy()))
    opt = torch.optim.AdamW([tw], lr=HP["lr"], betas=(HP["beta1"], HP["beta2"]),
                            eps=HP["eps"], weight_decay=HP["weight_decay"], foreach=False)
    m = np.zeros(shape, np.float32)
    v = np.zeros(shape, np.float32)
    for t in range(1, 6):
        g = _rand(shape, 100 + t, 1e-3)
        tw.grad = torch.from_numpy(g.copy())
        opt.step()
        w, m, v = A.adamw_step(w, g, m, v, A.step_constants(step=t, **HP))
    st = opt.state[tw]
    # absolute slack of a few fp32 ulps of the largest moment (entries that cancel
    # to nearly zero differ relatively, not absolutely)
    np.testing.assert_allclose(m, st["exp_avg"].numpy(), rtol=1e-5, atol=1e-6 * np.abs(m).max())
    np.testing.assert_allclose(v, st["exp_avg_sq"].numpy(), rtol=1e-5, atol=1e-6 * np.abs(v).max())
    w0 = _rand(shape, 6, 0.02).astype(np.float64)
    np.testing.assert_allclose(w - w0, tw.detach().numpy() - w0, rtol=2e-4, atol=2e-9)


def test_grad_scale_is_a_gradient_multiplier():
    """grad_scale (the clip coefficient) is the same as scaling the gradient."""
    w0 = _rand((16, 128), 7, 0.02)
    g = _rand((16, 128), 8, 1e-3)
    z = np.zeros_like(w0)
    a = A.adamw_step(w0, g, z, z, A.step_constants(step=3, grad_scale=0.5, **HP))
    b = A.adamw_step(w0, g * np.float32(0.5), z, z, A.step_constants(step=3, **HP))
    for x, y in zip(a, b):
        np.testing.assert_array_equal(x, y)


def test_requantize_uses_the_updated_weights():
    """The codes, scales and zero counts are those of the updated weights (the
    scale is recomputed from the weights every step, §3.1)."""
    w0 = _rand((8, 256), 9, 0.02)
    g = _rand((8, 256), 10, 1e-3)
    z = np.zeros_like(w0)
    c = A.step_constants(step=1, **HP)
    w1, _, _, codes, s, zc = A.adamw_requantize(w0, g, z, z, 128, c)
    s_ref = np.abs(w1.astype(np.float64)).reshape(8, 2, 128).mean(axis=2)
    np.testing.assert_allclose(s, s_ref, rtol=1e-6)
    assert not np.array_equal(s, O.quantize(w0, 128)[1])
    cc = O.unpack(codes, 256)
    assert set(np.unique(cc)) <= {-1, 0, 1}
    assert np.array_equal(zc, (cc.reshape(8, 2, 128) == 0).sum(axis=2))


def test_step_must_count_from_one():
    with pytest.raises(ValueError):
        A.step_constants(step=0, **HP)
    assert math.isclose(float(A.step_constants(step=1, **HP)["step_size"]),
                        HP["lr"] / (1 - HP["beta1"]), rel_tol=1e-7)
