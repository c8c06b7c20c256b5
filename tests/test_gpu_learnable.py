"""GPU parity of the learnable-scale variant against oracle/learnable_oracle.py:
codes and zero counts against given scales (bit for bit: both sides decide on the
same fp32 quotient), the scale gradient (within the fp32 summation bound), the
fused AdamW step with requantization against given scales and the plain AdamW
step (bit for bit), and one learnable-scale QAT step end to end."""
import numpy as np
import pytest
import torch

from oracle import adamw_oracle as A
from oracle import learnable_oracle as L
from oracle import tq_oracle as O
from paper_2606_18114_gb300 import synth
from parity import check_close, codes_u32, to_np

pytestmark = pytest.mark.gpu

HP = dict(lr=2.5e-4, beta1=0.9, beta2=0.95, eps=1e-8, weight_decay=0.01)  # §3.3


@pytest.fixture(scope="module")
def tq():
    from paper_2606_18114_gb300 import tq as _tq
    _tq.load()
    return _tq


def _scales(w, g, seed, special=True):
    """Absmean times a random factor in [0.5, 2]; with ``special`` also a negative,
    a zero and a tiny scale."""
    s = O.quantize(w, g)[1]
    f = np.random.default_rng(seed).uniform(0.5, 2.0, size=s.shape).astype(np.float32)
    s = (s * f).astype(np.float32)
    if special and s.size >= 4:
        s.flat[0] = -s.flat[0]
        s.flat[1] = 0.0
        s.flat[2] = np.float32(1e-35)
        s.flat[3] = -s.flat[3]
    return s


def _check_codes(codes_gpu, zeros_gpu, ref_codes, ref_z):
    assert np.array_equal(codes_u32(codes_gpu), ref_codes)
    assert np.array_equal(to_np(zeros_gpu), ref_z)


def _check_ds(got, w, dw, c, s, g):
    ref = L.scale_grad(w, dw, c, s, g)
    n, k = w.shape
    cg = c.reshape(n, k // g, g).astype(np.float64)
    wg = w.reshape(n, k // g, g).astype(np.float64)
    dg = np.asarray(dw, np.float64).reshape(n, k // g, g)
    s64 = s.astype(np.float64)
    with np.errstate(divide="ignore", invalid="ignore"):
        scale = np.abs(dg * cg).sum(2) + np.where(s64 != 0, np.abs(dg * wg).sum(2) / np.abs(s64), 0)
    err = np.abs(to_np(got).astype(np.float64) - ref)
    assert np.all(err <= 1e-5 * scale + 1e-30), f"worst {np.max(err / (scale + 1e-30)):.3e}"


@pytest.mark.parametrize("n,k,g", [(512, 256, 128), (200, 192, 64), (136, 320, 32),
                                   (264, 512, 256), (128, 1024, 512), (7, 96, 32)])
def test_quantize_with_scales_parity(tq, n, k, g):
    w = synth.latent_weights(n, k, seed=n + k + g)
    s = _scales(w, g, seed=g)
    codes, z = tq.quantize_with_scales(torch.from_numpy(w).cuda(), g, torch.from_numpy(s).cuda())
    tq.device_status()
    ref_codes, ref_z, _ = L.quantize_with_scales(w, g, s)
    _check_codes(codes, z, ref_codes, ref_z)


@pytest.mark.parametrize("n,k,g", [(512, 256, 128), (200, 192, 64), (136, 320, 32),
                                   (128, 1024, 512)])
def test_scale_grad_parity(tq, n, k, g):
    w = synth.latent_weights(n, k, seed=3 * n + g)
    s = _scales(w, g, seed=n)
    dw = (np.random.default_rng(n).standard_normal((n, k)) * 1e-2).astype(np.float32)
    ref_codes, _, c = L.quantize_with_scales(w, g, s)
    wd, dwd, sd = (torch.from_numpy(a).cuda() for a in (w, dw, s))
    codes = torch.from_numpy(ref_codes.view(np.int32)).cuda()
    ds = tq.scale_grad(wd, dwd, codes, sd, g)
    tq.device_status()
    _check_ds(ds, w, dw, c, s, g)


@pytest.mark.parametrize("dist", ["gauss", "t3"])
def test_learnable_in_proj(tq, dist):
    """The full Mamba-2 1.3B in_proj matrix [8512, 2048], g = 128."""
    n, k = synth.MAMBA2_1P3B["in_proj"]
    w = synth.latent_weights(n, k, seed=23, dist=dist)
    s = _scales(w, 128, seed=24)
    dw = (np.random.default_rng(25).standard_normal((n, k)) * 1e-3).astype(np.float32)
    wd, dwd, sd = (torch.from_numpy(a).cuda() for a in (w, dw, s))
    codes, z = tq.quantize_with_scales(wd, 128, sd)
    ds = tq.scale_grad(wd, dwd, codes, sd, 128)
    tq.device_status()
    ref_codes, ref_z, c = L.quantize_with_scales(w, 128, s)
    _check_codes(codes, z, ref_codes, ref_z)
    _check_ds(ds, w, dw, c, s, 128)


@pytest.mark.parametrize("n,k,g", [(512, 256, 128), (200, 192, 64), (7, 96, 32)])
def test_adamw_requantize_with_scales_parity(tq, n, k, g):
    rs = np.random.default_rng(n + g)
    w = synth.latent_weights(n, k, seed=n * g)
    grad = (rs.standard_normal((n, k)) * 1e-3).astype(np.float32)
    m = (rs.standard_normal((n, k)) * 3e-4).astype(np.float32)
    v = (np.abs(rs.standard_normal((n, k))) * 1e-7 + 1e-9).astype(np.float32)
    s = _scales(w, g, seed=7)
    w1, m1, v1, ref_codes, ref_z = L.adamw_requantize_with_scales(
        w, grad, m, v, g, A.step_constants(step=4, **HP), s)
    wd, gd, md, vd, sd = (torch.from_numpy(a.copy()).cuda() for a in (w, grad, m, v, s))
    codes, z = tq.adamw_requantize_with_scales(wd, gd, md, vd, g, sd, step=4, **HP)
    tq.device_status()
    for name, ref, got in (("w", w1, wd), ("m", m1, md), ("v", v1, vd)):
        assert np.array_equal(to_np(got).view(np.uint32), ref.view(np.uint32)), name
    _check_codes(codes, z, ref_codes, ref_z)


@pytest.mark.parametrize("count", [16, 4096, 136192, 100000 * 16 + 16])
def test_plain_adamw_parity(tq, count):
    rs = np.random.default_rng(count % 1000)
    p = (rs.standard_normal(count) * 2e-2).astype(np.float32)
    grad = (rs.standard_normal(count) * 1e-3).astype(np.float32)
    m = (rs.standard_normal(count) * 3e-4).astype(np.float32)
    v = (np.abs(rs.standard_normal(count)) * 1e-7 + 1e-9).astype(np.float32)
    p1, m1, v1 = A.adamw_step(p, grad, m, v, A.step_constants(step=9, **HP))
    pd, gd, md, vd = (torch.from_numpy(a.copy()).cuda() for a in (p, grad, m, v))
    tq.adamw(pd, gd, md, vd, step=9, **HP)
    tq.device_status()
    for name, ref, got in (("p", p1, pd), ("m", m1, md), ("v", v1, vd)):
        assert np.array_equal(to_np(got).view(np.uint32), ref.view(np.uint32)), name


def test_plain_adamw_rejects_ragged_count(tq):
    t = torch.zeros(24, device="cuda")
    with pytest.raises(tq.TqError):
        tq.adamw(t, t, t, t, lr=1e-3, step=1)


def test_learnable_qat_step(tq):
    """One step of the learnable-scale variant on the library's kernels: codes against
    s, Y, dW, ds, the AdamW step of s and the fused step of w against the new s."""
    n, k, m, g = 264, 512, 300, 128
    rs = np.random.default_rng(31)
    w = synth.latent_weights(n, k, seed=32)
    s = O.quantize(w, g)[1]
    x = synth.activations_bf16(m, k, seed=33)
    dy = synth.activations_bf16(m, n, seed=34, std=1e-2, stream="dy")
    wd, sd = torch.from_numpy(w.copy()).cuda(), torch.from_numpy(s.copy()).cuda()
    codes, _ = tq.quantize_with_scales(wd, g, sd)
    y = tq.linear_fwd(x.cuda(), codes, sd, g)
    _, dw = tq.linear_bwd(dy.cuda(), x.cuda(), codes, sd, k, g, want_dx=False)
    ds = tq.scale_grad(wd, dw, codes, sd, g)
    ms, vs = torch.zeros_like(sd), torch.zeros_like(sd)
    tq.adamw(sd.view(-1), ds.view(-1), ms.view(-1), vs.view(-1), step=1, **HP)
    mw, vw = torch.zeros_like(wd), torch.zeros_like(wd)
    codes1, z1 = tq.adamw_requantize_with_scales(wd, dw, mw, vw, g, sd, step=1, **HP)
    tq.device_status()
    # oracle chain on the same inputs
    ref_codes, _, c = L.quantize_with_scales(w, g, s)
    assert np.array_equal(codes_u32(codes), ref_codes)
    w_hat = np.repeat(s.astype(np.float64), g, axis=1) * c
    check_close(y, O.linear_fwd(x, w_hat), "Y")
    dw_ref = O.linear_bwd_dw(dy, x)
    check_close(dw, dw_ref, "dW")
    dwg = to_np(dw)  # the GPU dW drives the rest, as in training
    _check_ds(ds, w, dwg, c, s, g)
    cst = A.step_constants(step=1, **HP)
    s1, _, _ = A.adamw_step(s, to_np(ds), np.zeros_like(s), np.zeros_like(s), cst)
    assert np.array_equal(to_np(sd).view(np.uint32), s1.view(np.uint32))
    w1, _, _, ref_codes1, ref_z1 = L.adamw_requantize_with_scales(
        w, dwg, np.zeros_like(w), np.zeros_like(w), g, cst, s1)
    assert np.array_equal(to_np(wd).view(np.uint32), w1.view(np.uint32))
    _check_codes(codes1, z1, ref_codes1, ref_z1)


def test_zero_ratio_tracking_runs(tq):
    """The synthetic tracking driver: both parameterizations start from the same
    codes (the absmean of the teacher's weights, ~31 % zeros for Gaussian weights),
    stay finite, and only the learnable run moves its scales off the absmean."""
    from paper_2606_18114_gb300 import qat
    a = qat.track_zero_ratio(tq, 256, 512, 256, 128, 20, learnable=False, seed=3, every=10)
    b = qat.track_zero_ratio(tq, 256, 512, 256, 128, 20, learnable=True, seed=3, every=10)
    assert [r["step"] for r in a] == [0, 10, 20] == [r["step"] for r in b]
    assert a[0]["zero_ratio"] == b[0]["zero_ratio"] and a[0]["loss"] == b[0]["loss"]
    assert abs(a[0]["zero_ratio"] - 0.31) < 0.02
    for r in a + b:
        assert 0.0 <= r["zero_ratio"] <= 1.0 and np.isfinite(r["loss"])
    assert all(abs(r["scale_ratio"] - 1.0) < 1e-3 for r in a)
    assert b[-1]["scale_ratio"] != b[0]["scale_ratio"]
