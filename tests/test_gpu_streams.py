"""Ordering of dW launches across streams (needs a GB300).

dW launches of one device share the library's stream-K workspace and tile
counters; the library orders each launch after the previous one whatever stream
either was issued on. Shape: 4160 x 1280 at 640 tokens cuts the tiles past the
last whole wave into pieces, so both launches use the workspace.
"""
import numpy as np
import pytest
import torch

from oracle import tq_oracle as O
from paper_2606_18114_gb300 import synth
from parity import check_close, to_np

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def tq():
    if not torch.cuda.is_available():
        pytest.fail("the gpu tests need a CUDA device")
    from paper_2606_18114_gb300 import build, tq as _tq
    build.build()
    _tq.load()
    return _tq


def test_dw_default_then_side_stream(tq):
    """dW on the legacy default stream, then at once on a new non-blocking torch
    stream with no synchronisation between: both equal the single-stream result
    bit for bit, and match the oracle."""
    n, k, m, g = 4160, 1280, 640, 128
    w = torch.from_numpy(synth.latent_weights(n, k, seed=61)).cuda()
    x_h = synth.activations_bf16(m, k, seed=61, stream="x")
    dy_h = synth.activations_bf16(m, n, seed=61, std=1e-2, stream="dy")
    x, dy = x_h.cuda(), dy_h.cuda()
    codes, s, _ = tq.quantize(w, g)
    ref_dw = torch.empty((n, k), device="cuda")
    tq.linear_bwd(dy, x, codes, s, k, g, want_dx=False, dw=ref_dw)
    tq.device_status()
    default = torch.cuda.default_stream()
    side = torch.cuda.Stream()
    for _ in range(3):
        a = torch.full((n, k), float("nan"), device="cuda")
        b = torch.full((n, k), float("nan"), device="cuda")
        torch.cuda.synchronize()
        with torch.cuda.stream(default):
            tq.linear_bwd(dy, x, codes, s, k, g, want_dx=False, dw=a)
        with torch.cuda.stream(side):
            tq.linear_bwd(dy, x, codes, s, k, g, want_dx=False, dw=b)
        torch.cuda.synchronize()
        tq.device_status()
        assert torch.equal(a, ref_dw) and torch.equal(b, ref_dw)
    rows = np.sort(np.random.default_rng(61).choice(n, 64, replace=False))
    check_close(to_np(ref_dw[torch.from_numpy(rows).cuda()]), O.linear_bwd_dw(dy_h, x_h, rows),
                "dW rows")
