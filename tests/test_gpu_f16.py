"""fp16 activations (the paper's A16 is FP16, §3.3): forward, dX and dW on fp16 x
and dY through the same kernels (TQ_IN_F16), against the fp64 oracle on the same
fp16 values."""
import numpy as np
import pytest
import torch

from oracle import tq_oracle as O
from paper_2606_18114_gb300 import synth
from parity import check_close, to_np, validated_w_hat

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def tq():
    from paper_2606_18114_gb300 import tq as _tq
    _tq.load()
    return _tq


def _setup(tq, n, k, m, g, seed, dy_std=1.0):
    w = synth.latent_weights(n, k, seed=seed)
    x = synth.activations_f16(m, k, seed=seed, stream="x")
    dy = synth.activations_f16(m, n, seed=seed, std=dy_std, stream="dy")
    codes, s, z = tq.quantize(torch.from_numpy(w).cuda(), g)
    return x, dy, validated_w_hat(w, g, codes, s, z), codes, s


@pytest.mark.parametrize("n,k,m,g", [
    (512, 256, 64, 128),
    (200, 192, 300, 64),
    (136, 320, 257, 32),
    (264, 512, 17, 256),
    (128, 1024, 256, 512),
    (520, 1024, 1, 128),     # decode
    (520, 1024, 3, 64),
    (520, 1024, 12, 128),    # decode, two token tiles
])
def test_linear_f16_parity(tq, n, k, m, g):
    x, dy, w_hat, codes, s = _setup(tq, n, k, m, g, seed=n + m + g)
    xd, dyd = x.cuda(), dy.cuda()
    y = tq.linear_fwd(xd, codes, s, g)
    dx, dw = tq.linear_bwd(dyd, xd, codes, s, k, g)
    dxt, _ = tq.linear_bwd(dyd, xd, codes, s, k, g, want_dw=False, codes_t=tq.codes_transpose(codes, k))
    tq.device_status()
    check_close(y, O.linear_fwd(x, w_hat), "Y f16")
    check_close(dx, O.linear_bwd_dx(dy, w_hat), "dX f16")
    check_close(dxt, O.linear_bwd_dx(dy, w_hat), "dX f16 (codes_t)")
    check_close(dw, O.linear_bwd_dw(dy, x), "dW f16")


def test_batched_decode_f16(tq):
    items, refs = [], []
    for i, (n, k, g) in enumerate([(300, 512, 128), (1024, 2048, 64), (64, 256, 32)]):
        x, _, w_hat, codes, s = _setup(tq, n, k, 5, g, seed=70 + i)
        items.append(dict(x=x.cuda(), codes=codes, scales=s, g=g, y=torch.empty((5, n), device="cuda")))
        refs.append(O.linear_fwd(x, w_hat))
    tq.linear_fwd_batched(tq.fwd_batch(items), 5)
    tq.device_status()
    for it, ref in zip(items, refs):
        check_close(it["y"], ref, "batched Y f16")


def test_prefill_f16_in_proj_sampled(tq):
    n, k = synth.MAMBA2_1P3B["in_proj"]
    m, g = 16384, 128
    x, dy, w_hat, codes, s = _setup(tq, n, k, m, g, seed=9, dy_std=1e-2)
    xd, dyd = x.cuda(), dy.cuda()
    y = tq.linear_fwd(xd, codes, s, g)
    dx, dw = tq.linear_bwd(dyd, xd, codes, s, k, g, codes_t=tq.codes_transpose(codes, k))
    tq.device_status()
    rs = np.random.default_rng(2)
    rows = np.sort(rs.choice(m, 32, replace=False))
    nrows = np.sort(rs.choice(n, 32, replace=False))
    sel = torch.from_numpy(rows).cuda()
    check_close(to_np(y[sel]), O.linear_fwd(x, w_hat, rows), "Y rows f16")
    check_close(to_np(dx[sel]), O.linear_bwd_dx(dy, w_hat, rows), "dX rows f16")
    check_close(to_np(dw[torch.from_numpy(nrows).cuda()]), O.linear_bwd_dw(dy, x, nrows), "dW rows f16")
