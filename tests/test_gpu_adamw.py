"""GPU parity of the fused AdamW step + requantize (tq_adamw_requantize) against
oracle/adamw_oracle.py: w, m and v bit for bit (both sides run the same fp32
operations in the same order), then codes / scales / zero counts of the new
weights under the quantizer's bar (codes and zero counts exact outside
near-ties, scales within 1e-6)."""
import numpy as np
import pytest
import torch

from oracle import adamw_oracle as A
from paper_2606_18114_gb300 import synth
from parity import check_quantize, to_np

pytestmark = pytest.mark.gpu

HP = dict(lr=2.5e-4, beta1=0.9, beta2=0.95, eps=1e-8, weight_decay=0.01)  # §3.3


@pytest.fixture(scope="module")
def tq():
    from paper_2606_18114_gb300 import tq as _tq
    _tq.load()
    return _tq


def _state(n, k, seed, dist="gauss"):
    """Latent weights, a gradient, and moments as a few earlier steps leave them."""
    rs = np.random.default_rng(seed)
    w = synth.latent_weights(n, k, seed=seed, dist=dist)
    grad = (rs.standard_normal((n, k)) * 1e-3).astype(np.float32)
    m = (rs.standard_normal((n, k)) * 3e-4).astype(np.float32)
    v = (np.abs(rs.standard_normal((n, k))) * 1e-7 + 1e-9).astype(np.float32)
    return w, grad, m, v


def _run(tq, w, grad, m, v, g, step, **kw):
    wd, gd, md, vd = (torch.from_numpy(a.copy()).cuda() for a in (w, grad, m, v))
    codes, s, z = tq.adamw_requantize(wd, gd, md, vd, g, step=step, **{**HP, **kw})
    tq.device_status()
    return wd, md, vd, codes, s, z


def _check(w_new, m_new, v_new, wd, md, vd, g, codes, s, z):
    for name, ref, got in (("w", w_new, wd), ("m", m_new, md), ("v", v_new, vd)):
        got = to_np(got)
        bad = np.flatnonzero(got.view(np.uint32) != ref.view(np.uint32))
        assert bad.size == 0, f"{name}: {bad.size} elements differ, first {bad[:4]}"
    flips, ties = check_quantize(w_new, g, codes, s, z)
    assert flips <= ties


@pytest.mark.parametrize("n,k,g", [
    (512, 256, 128),      # the single grouped ternary linear's shape
    (200, 192, 64),       # ragged: 200 * 192 is not a multiple of the 4096-weight stage
    (136, 320, 32),
    (264, 512, 256),
    (128, 1024, 512),
    (7, 96, 32),          # smaller than one stage
])
def test_adamw_requantize_parity(tq, n, k, g):
    w, grad, m, v = _state(n, k, seed=n + k + g)
    step = 5
    w1, m1, v1 = A.adamw_step(w, grad, m, v, A.step_constants(step=step, **HP))
    wd, md, vd, codes, s, z = _run(tq, w, grad, m, v, g, step)
    _check(w1, m1, v1, wd, md, vd, g, codes, s, z)


@pytest.mark.parametrize("dist", ["gauss", "t3"])
def test_adamw_requantize_in_proj(tq, dist):
    """The full Mamba-2 1.3B in_proj matrix [8512, 2048], g = 128."""
    n, k = synth.MAMBA2_1P3B["in_proj"]
    w, grad, m, v = _state(n, k, seed=21, dist=dist)
    w1, m1, v1 = A.adamw_step(w, grad, m, v, A.step_constants(step=100, **HP))
    wd, md, vd, codes, s, z = _run(tq, w, grad, m, v, 128, 100)
    _check(w1, m1, v1, wd, md, vd, 128, codes, s, z)


def test_adamw_requantize_chained_steps(tq):
    """Three consecutive steps from zero moments on the device, each compared
    with the oracle's chain."""
    n, k, g = 264, 1024, 128
    w, _, _, _ = _state(n, k, seed=3)
    m = np.zeros((n, k), np.float32)
    v = np.zeros((n, k), np.float32)
    wd, md, vd = (torch.from_numpy(a.copy()).cuda() for a in (w, m, v))
    rs = np.random.default_rng(4)
    for t in range(1, 4):
        grad = (rs.standard_normal((n, k)) * 1e-3).astype(np.float32)
        w, m, v = A.adamw_step(w, grad, m, v, A.step_constants(step=t, **HP))
        codes, s, z = tq.adamw_requantize(wd, torch.from_numpy(grad).cuda(), md, vd, g, step=t, **HP)
        tq.device_status()
        _check(w, m, v, wd, md, vd, g, codes, s, z)


def test_adamw_grad_scale_and_zero_gradient(tq):
    n, k, g = 96, 512, 64
    w, grad, m, v = _state(n, k, seed=8)
    for gs, gr in ((0.25, grad), (1.0, np.zeros_like(grad))):
        c = A.step_constants(step=2, grad_scale=gs, **HP)
        w1, m1, v1 = A.adamw_step(w, gr, m, v, c)
        wd, md, vd, codes, s, z = _run(tq, w, gr, m, v, g, 2, grad_scale=gs)
        _check(w1, m1, v1, wd, md, vd, g, codes, s, z)
