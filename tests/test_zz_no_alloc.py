"""tq_linear_bwd_noalloc: the transposed-codes dX path with the library's own
scratch for the transposed codes. CPU: rejections before any launch. GPU: the
results equal tq_linear_bwd with a caller-provided codes_t, bit for bit, and the
oracle within the parity bars."""
import pytest
import torch

from oracle import tq_oracle as O
from paper_2606_18114_gb300 import synth
from parity import check_close, validated_w_hat

FAKE = 1 << 20


@pytest.fixture(scope="module")
def lib():
    from paper_2606_18114_gb300 import build, tq as _tq
    return _tq.load(build.build())


@pytest.fixture(scope="module")
def tq():
    if not torch.cuda.is_available():
        pytest.fail("the gpu tests need a CUDA device")
    from paper_2606_18114_gb300 import build, tq as _tq
    build.build()
    _tq.load()
    return _tq


def test_noalloc_rejects_before_launch(lib):
    args = lambda n, k, dxd=0: (FAKE, FAKE, 64, n, k, FAKE, FAKE, 128, FAKE, dxd, FAKE, 0, None)
    assert lib.tq_linear_bwd_noalloc(*args(1 << 20, 4096)) == 2   # scratch too small
    assert b"codes_t" in lib.tq_last_error()
    assert lib.tq_linear_bwd_noalloc(*args(60, 256)) == 2         # n % 8
    assert lib.tq_linear_bwd_noalloc(*args(64, 256, 5)) == 1      # dx dtype


@pytest.mark.gpu
@pytest.mark.parametrize("n,k,m", [(512, 256, 64), (8512, 2048, 300), (2048, 4096, 129),
                                   (136, 192, 17)])
def test_noalloc_matches_explicit_codes_t(tq, n, k, m):
    g = 64 if k % 128 else 128
    w = torch.from_numpy(synth.latent_weights(n, k, seed=n)).cuda()
    x = synth.activations_bf16(m, k, seed=n, stream="x").cuda()
    dy = synth.activations_bf16(m, n, seed=n, std=1e-2, stream="dy").cuda()
    codes, s, z = tq.quantize(w, g)
    codes_t = tq.codes_transpose(codes, k)
    dx1, dw1 = tq.linear_bwd(dy, x, codes, s, k, g, codes_t=codes_t)
    dx2, dw2 = tq.linear_bwd_noalloc(dy, x, codes, s, k, g)
    tq.device_status()
    assert torch.equal(dx1, dx2) and torch.equal(dw1, dw2)
    # and the oracle, on the dequantised weights
    w_hat = validated_w_hat(w.cpu().numpy(), g, codes, s, z)
    check_close(dx2, O.linear_bwd_dx(dy.float().cpu(), w_hat), "dX (no-alloc)")


@pytest.mark.gpu
def test_noalloc_accumulates_dw_and_skips_dx(tq):
    n, k, m = 256, 512, 96
    w = torch.from_numpy(synth.latent_weights(n, k, seed=3)).cuda()
    x = torch.randn(m, k, device="cuda").to(torch.bfloat16)
    dy = torch.randn(m, n, device="cuda").to(torch.bfloat16)
    codes, s, _ = tq.quantize(w, 128)
    dw = torch.ones(n, k, device="cuda")
    dx, dw = tq.linear_bwd_noalloc(dy, x, codes, s, k, 128, want_dx=False, dw=dw,
                                   accumulate_dw=True)
    _, dw_ref = tq.linear_bwd(dy, x, codes, s, k, 128, want_dx=False)
    tq.device_status()
    assert dx is None
    assert torch.allclose(dw, dw_ref + 1.0, rtol=0, atol=1e-5)
