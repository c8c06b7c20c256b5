"""dX past one whole wave of tiles (needs a GB300): n = 4096 (32 k-blocks of the
reduction), k = 2048 (16 row tiles), m = 2560 (10 token tiles) is 160 tiles on the 152
CTAs of a GB300, so 8 CTAs run a second tile. The whole dX is compared with the oracle,
on both dX paths (transposed and plain codes) and with fp32 and bf16 outputs; repeated
launches are bit-identical, also with dW launches on another stream in between."""
import numpy as np
import pytest
import torch

from oracle import tq_oracle as O
from paper_2606_18114_gb300 import synth
from parity import check_close, to_np, validated_w_hat

pytestmark = pytest.mark.gpu

N, K, M, G = 4096, 2048, 2560, 128


@pytest.fixture(scope="module")
def tq():
    if not torch.cuda.is_available():
        pytest.fail("the gpu tests need a CUDA device")
    from paper_2606_18114_gb300 import build, tq as _tq
    build.build()
    _tq.load()
    return _tq


@pytest.fixture(scope="module")
def case(tq):
    w_h = synth.latent_weights(N, K, seed=71)
    w = torch.from_numpy(w_h).cuda()
    x_h = synth.activations_bf16(M, K, seed=71, stream="x")
    dy_h = synth.activations_bf16(M, N, seed=71, std=1e-2, stream="dy")
    codes, s, z, codes_t = tq.quantize_with_transpose(w, G)
    w_hat = validated_w_hat(w_h, G, codes, s, z)
    return dict(x=x_h.cuda(), dy=dy_h.cuda(), codes=codes, s=s, codes_t=codes_t,
                ref=O.linear_bwd_dx(dy_h, w_hat))


@pytest.mark.parametrize("transposed", [True, False])
@pytest.mark.parametrize("out", [torch.float32, torch.bfloat16])
def test_dx_past_one_wave_matches_the_oracle(tq, case, transposed, out):
    ct = case["codes_t"] if transposed else None
    dx, _ = tq.linear_bwd(case["dy"], case["x"], case["codes"], case["s"], K, G, want_dw=False,
                          codes_t=ct, dx_dtype=out)
    tq.device_status()
    check_close(dx, case["ref"], f"dX ({'codes_t' if transposed else 'codes'}, {out})")


def test_dx_repeatable_between_dw_on_another_stream(tq, case):
    side = torch.cuda.Stream()
    first, _ = tq.linear_bwd(case["dy"], case["x"], case["codes"], case["s"], K, G,
                             want_dw=False, codes_t=case["codes_t"])
    torch.cuda.synchronize()
    for _ in range(3):
        dx = torch.full_like(first, float("nan"))
        with torch.cuda.stream(side):
            tq.linear_bwd(case["dy"], case["x"], case["codes"], case["s"], K, G, want_dx=False)
        tq.linear_bwd(case["dy"], case["x"], case["codes"], case["s"], K, G, want_dw=False,
                      dx=dx, codes_t=case["codes_t"])
        torch.cuda.synchronize()
        tq.device_status()
        assert torch.equal(dx, first)
