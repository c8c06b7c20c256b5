"""GPU parity of the decoupled quantizer (tq_quantize_decoupled) and its magnitude
gradient (tq_alpha_grad) against oracle/decoupled_oracle.py, and of a decoupled
linear step (forward, dX with the magnitudes alpha as the scales, dalpha)."""
import numpy as np
import pytest
import torch

from oracle import decoupled_oracle as D
from oracle import tq_oracle as O
from paper_2606_18114_gb300 import synth
from parity import check_close, codes_u32, to_np

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def tq():
    from paper_2606_18114_gb300 import tq as _tq
    _tq.load()
    return _tq


def _check_codes(w, g, f, codes, s, z):
    """Codes and zero counts exact outside elements within 1e-5 of the tie
    |w / tau| = 1/2; scales (the absmean) within 1e-6."""
    n, k = w.shape
    ref_codes, ref_s, ref_z, ref_c, tau = D.quantize_decoupled(w, g, f)
    s, z = to_np(s), to_np(z)
    np.testing.assert_allclose(s, ref_s, rtol=1e-6, atol=0)
    c = O.unpack(codes_u32(codes), k)
    ties = O.near_tie_mask(w, tau, g, 1e-5)
    assert not ((c != ref_c) & ~ties).any()
    grp_ties = ties.reshape(n, k // g, g).sum(axis=2)
    assert np.all(np.abs(z.astype(np.int64) - ref_z) <= grp_ties)
    return ref_c, tau


@pytest.mark.parametrize("n,k,g", [(512, 256, 128), (200, 192, 64), (136, 320, 32),
                                   (264, 512, 256), (128, 1024, 512)])
def test_quantize_decoupled_parity(tq, n, k, g):
    w = synth.latent_weights(n, k, seed=n + g)
    f = np.random.default_rng(n).uniform(0.5, 1.5, n).astype(np.float32)
    codes, s, z = tq.quantize_decoupled(torch.from_numpy(w).cuda(), g, torch.from_numpy(f).cuda())
    tq.device_status()
    _check_codes(w, g, f, codes, s, z)


def test_quantize_decoupled_null_factor_is_quantize(tq):
    w = torch.from_numpy(synth.latent_weights(264, 1024, seed=2)).cuda()
    a = tq.quantize_decoupled(w, 128)
    b = tq.quantize(w, 128)
    tq.device_status()
    for x, y in zip(a, b):
        assert torch.equal(x, y)


@pytest.mark.parametrize("dist", ["gauss", "t3"])
def test_asymmetric_gate_in_proj(tq, dist):
    """The paper's asymmetric gate on the full in_proj: rows 0..4095 at 0.8 x absmean."""
    n, k = synth.MAMBA2_1P3B["in_proj"]
    w = synth.latent_weights(n, k, seed=12, dist=dist)
    f = np.ones(n, np.float32)
    f[:4096] = 0.8
    codes, s, z = tq.quantize_decoupled(torch.from_numpy(w).cuda(), 128, torch.from_numpy(f).cuda())
    tq.device_status()
    _check_codes(w, 128, f, codes, s, z)
    zr = to_np(z)
    assert zr[:4096].mean() < zr[4096:].mean()  # the gate rows keep more weights


@pytest.mark.parametrize("n,k,g", [(512, 256, 128), (136, 320, 32), (128, 1024, 512), (8512, 2048, 128)])
def test_alpha_grad_parity(tq, n, k, g):
    w = synth.latent_weights(n, k, seed=k + g)
    dw = np.random.default_rng(g).standard_normal((n, k)).astype(np.float32)
    codes, _, _ = tq.quantize(torch.from_numpy(w).cuda(), g)
    da = tq.alpha_grad(torch.from_numpy(dw).cuda(), codes, g)
    tq.device_status()
    check_close(to_np(da), D.alpha_grad(dw, codes_u32(codes), g), f"dalpha {n}x{k} g={g}")


def test_decoupled_linear_step(tq):
    """Forward and dX take the magnitudes alpha as their scales; dalpha comes from
    the dW of the same backward."""
    n, k, m, g = 520, 1024, 300, 128
    w = synth.latent_weights(n, k, seed=31)
    x = synth.activations_bf16(m, k, seed=31, stream="x")
    dy = synth.activations_bf16(m, n, seed=31, std=1e-2, stream="dy")
    f = np.full(n, 0.8, np.float32)
    codes, s, z = tq.quantize_decoupled(torch.from_numpy(w).cuda(), g, torch.from_numpy(f).cuda())
    alpha = s * torch.linspace(0.9, 1.1, k // g, device="cuda")[None, :]  # a learned-looking alpha
    xd, dyd = x.cuda(), dy.cuda()
    y = tq.linear_fwd(xd, codes, alpha, g)
    dx, dw = tq.linear_bwd(dyd, xd, codes, alpha, k, g)
    da = tq.alpha_grad(dw, codes, g)
    tq.device_status()
    w_hat = O.dequantize(codes_u32(codes), to_np(alpha), k, g)
    check_close(to_np(y), O.linear_fwd(x, w_hat), "Y (alpha)")
    check_close(to_np(dx), O.linear_bwd_dx(dy, w_hat), "dX (alpha)")
    dw_ref = O.linear_bwd_dw(dy, x)
    check_close(to_np(da), D.alpha_grad(dw_ref, codes_u32(codes), g), "dalpha")
