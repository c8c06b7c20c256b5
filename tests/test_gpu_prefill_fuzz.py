"""Prefill (m > 16) products on seeded random shapes against the oracle (needs a GB300).

Shapes drawn once from a fixed seed: every group size, k any multiple of 64 and of g up
to 4096, n a multiple of 8 up to 1400 (the backward's requirement), m from 17 to
2500 tokens (ragged token tiles); the forward, dX from the codes and from the
transposed codes (bit-identical to each other), dW overwritten and accumulated.
"""
import numpy as np
import pytest
import torch

from oracle import tq_oracle as O
from paper_2606_18114_gb300 import synth
from parity import check_close, to_np, validated_w_hat

pytestmark = pytest.mark.gpu


def _cases(seed, count):
    rs = np.random.default_rng(seed)
    out = []
    for i in range(count):
        g = int(rs.choice([32, 64, 128, 256, 512]))
        step = max(64, g)
        k = step * int(rs.integers(1, 4096 // step + 1))
        n = 8 * int(rs.integers(1, 176))
        m = int(rs.integers(17, 2501))
        out.append((i, n, k, g, m))
    return out


@pytest.fixture(scope="module")
def tq():
    if not torch.cuda.is_available():
        pytest.fail("the gpu tests need a CUDA device")
    from paper_2606_18114_gb300 import build, tq as _tq
    build.build()
    _tq.load()
    return _tq


@pytest.mark.parametrize("case", _cases(99, 20), ids=lambda c: f"n{c[1]}k{c[2]}g{c[3]}m{c[4]}")
def test_prefill_random_shapes(tq, case):
    i, n, k, g, m = case
    w = synth.latent_weights(n, k, seed=8000 + i)
    x_h = synth.activations_bf16(m, k, seed=8000 + i, stream="x")
    dy_h = synth.activations_bf16(m, n, seed=8000 + i, std=1e-2, stream="dy")
    x, dy = x_h.cuda(), dy_h.cuda()
    codes, s, z = tq.quantize(torch.from_numpy(w).cuda(), g)
    w_hat = validated_w_hat(w, g, codes, s, z)
    y = tq.linear_fwd(x, codes, s, g)
    dx_t, dw = tq.linear_bwd(dy, x, codes, s, k, g, codes_t=tq.codes_transpose(codes, k))
    dx, _ = tq.linear_bwd(dy, x, codes, s, k, g, want_dw=False)
    dw_acc = torch.full((n, k), 0.25, device="cuda")
    tq.linear_bwd(dy, x, codes, s, k, g, want_dx=False, dw=dw_acc, accumulate_dw=True)
    tq.device_status()
    what = f"n={n} k={k} g={g} m={m}"
    check_close(y, O.linear_fwd(x_h, w_hat), f"Y {what}")
    check_close(dx, O.linear_bwd_dx(dy_h, w_hat), f"dX {what}")
    assert torch.equal(dx, dx_t), f"dX from the transposed codes differs, {what}"
    ref_dw = O.linear_bwd_dw(dy_h, x_h)
    check_close(dw, ref_dw, f"dW {what}")
    check_close(to_np(dw_acc) - 0.25, ref_dw, f"dW accumulated {what}")
