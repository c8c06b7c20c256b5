"""TernaryLinear as a torch autograd function and module (needs a GB300).

Through autograd the layer must give exactly what the C-ABI calls give (same kernels,
same inputs): y from tq_quantize_with_transpose + tq_linear_fwd, dX and dW from
tq_linear_bwd on the transposed codes, bit for bit; and, against the oracle, the §3.1
forward and STE backward within the parity bars. A batch dimension is flattened and
restored; fp16 activations work the same way; an optimizer step moves the latent
weights; the zero-ratio monitor reads the group zero counts of the last forward."""
import numpy as np
import pytest
import torch

from oracle import tq_oracle as O
from paper_2606_18114_gb300 import synth
from parity import check_close, to_np, validated_w_hat

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def tq():
    if not torch.cuda.is_available():
        pytest.fail("the gpu tests need a CUDA device")
    from paper_2606_18114_gb300 import build, tq as _tq
    build.build()
    _tq.load()
    return _tq


def _inputs(n, k, m, seed, act=torch.bfloat16):
    w = torch.from_numpy(synth.latent_weights(n, k, seed=seed)).cuda()
    x_h = synth.activations_bf16(m, k, seed=seed, stream="x")
    dy_h = synth.activations_bf16(m, n, seed=seed, std=1e-2, stream="dy")
    return w, x_h.cuda().to(act), dy_h.cuda().to(act), x_h, dy_h


@pytest.mark.parametrize("n,k,m,g", [(520, 256, 300, 128), (136, 512, 40, 64), (264, 1024, 17, 256)])
def test_autograd_equals_the_c_abi_calls(tq, n, k, m, g):
    from paper_2606_18114_gb300.ternary_linear import TernaryLinearFunction
    w, x, dy, _, _ = _inputs(n, k, m, seed=n + k)
    xb = x.reshape(1, m, k).clone().requires_grad_(True)  # a leading batch dimension
    wp = w.clone().requires_grad_(True)
    y, zeros = TernaryLinearFunction.apply(xb, wp, g, torch.float32)
    y.backward(dy.float().reshape(1, m, n))
    codes, s, z, codes_t = tq.quantize_with_transpose(w, g)
    y_ref = tq.linear_fwd(x, codes, s, g)
    dx_ref, dw_ref = tq.linear_bwd(dy, x, codes, s, k, g, codes_t=codes_t,
                                   dx_dtype=torch.bfloat16)
    tq.device_status()
    assert y.shape == (1, m, n) and torch.equal(y.reshape(m, n), y_ref)
    assert torch.equal(zeros, z)
    assert xb.grad.dtype == torch.bfloat16 and torch.equal(xb.grad.reshape(m, k), dx_ref)
    assert torch.equal(wp.grad, dw_ref)


def test_autograd_matches_the_oracle(tq):
    from paper_2606_18114_gb300.ternary_linear import TernaryLinearFunction
    n, k, m, g = 520, 256, 300, 128
    w, x, dy, x_h, dy_h = _inputs(n, k, m, seed=7)
    xr = x.clone().requires_grad_(True)
    wp = w.clone().requires_grad_(True)
    y, _ = TernaryLinearFunction.apply(xr, wp, g, torch.float32)
    y.backward(dy.float())
    codes, s, z, _ = tq.quantize_with_transpose(w, g)
    w_hat = validated_w_hat(to_np(w), g, codes, s, z)
    check_close(y, O.linear_fwd(x_h, w_hat), "Y")
    check_close(xr.grad.float(), O.linear_bwd_dx(dy_h, w_hat), "dX (bf16)")
    check_close(wp.grad, O.linear_bwd_dw(dy_h, x_h), "dW")


def test_fp16_activations(tq):
    from paper_2606_18114_gb300.ternary_linear import TernaryLinearFunction
    n, k, m, g = 264, 512, 64, 128
    w, x, dy, _, _ = _inputs(n, k, m, seed=9, act=torch.float16)
    xr = x.clone().requires_grad_(True)
    y, _ = TernaryLinearFunction.apply(xr, w.clone().requires_grad_(True), g, None)
    assert y.dtype == torch.float32  # fp32 by default for fp16 activations
    y.backward(dy.float())
    codes, s, _, codes_t = tq.quantize_with_transpose(w, g)
    dx_ref, _ = tq.linear_bwd(dy, x, codes, s, k, g, want_dw=False, codes_t=codes_t)
    tq.device_status()
    assert xr.grad.dtype == torch.float16
    assert torch.equal(xr.grad, dx_ref.to(torch.float16))


def test_module_step_and_zero_ratio(tq):
    from paper_2606_18114_gb300.ternary_linear import TernaryLinear
    torch.manual_seed(0)
    layer = TernaryLinear(1024, 520, g=128)
    assert layer.weight.dtype == torch.float32 and layer.weight.shape == (520, 1024)
    opt = torch.optim.AdamW(layer.parameters(), lr=1e-4)
    x = torch.randn(4, 128, 1024, device="cuda").to(torch.bfloat16)
    target = torch.randn(4, 128, 520, device="cuda")
    w0 = layer.weight.detach().clone()
    y = layer(x)
    assert y.shape == (4, 128, 520) and y.dtype == torch.bfloat16
    # Gaussian weights: share of zero codes near 2 Phi(0.5 sqrt(2/pi)) - 1 = 0.310
    assert abs(layer.zero_ratio() - 0.310) < 0.01
    loss = ((y.float() - target) ** 2).mean()
    loss.backward()
    assert layer.weight.grad is not None and torch.isfinite(layer.weight.grad).all()
    opt.step()
    tq.device_status()
    assert not torch.equal(layer.weight.detach(), w0)


@pytest.mark.parametrize("m", [3, 300])
def test_packed_inference_equals_the_training_forward(tq, m):
    """TernaryLinear.pack(): the codes and scales of the current weights, 2-bit
    storage, the same forward kernels (decode up to 16 tokens, the GEMM beyond)."""
    from paper_2606_18114_gb300.ternary_linear import PackedTernaryLinear, TernaryLinear
    torch.manual_seed(m)
    layer = TernaryLinear(1024, 520, g=128)
    packed = layer.pack()
    assert isinstance(packed, PackedTernaryLinear)
    nbytes = sum(b.numel() * b.element_size() for b in packed.buffers())
    assert nbytes == 520 * 1024 // 4 + 520 * (1024 // 128) * 4  # 0.25 + 4/g bytes per weight
    x = torch.randn(2, m, 1024, device="cuda").to(torch.bfloat16)
    with torch.no_grad():
        y_train = layer(x)
    y_packed = packed(x)
    tq.device_status()
    assert y_packed.shape == (2, m, 520) and y_packed.dtype == torch.bfloat16
    assert torch.equal(y_packed, y_train)
