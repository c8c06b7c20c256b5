"""TernaryLinear's argument checks, which run before anything reaches the library
(no GPU)."""
import pytest
import torch

from paper_2606_18114_gb300.ternary_linear import TernaryLinear, TernaryLinearFunction


@pytest.mark.parametrize("k,n,g", [(100, 8, 32), (256, 8, 96), (256, 12, 128)])
def test_module_rejects_unsupported_shapes(k, n, g):
    with pytest.raises(ValueError):
        TernaryLinear(k, n, g=g, device="cpu")


def test_function_rejects_activation_and_weight_types():
    w = torch.zeros(8, 32)
    with pytest.raises(TypeError):
        TernaryLinearFunction.apply(torch.zeros(4, 32), w, 32, None)  # fp32 activations
    with pytest.raises(TypeError):
        TernaryLinearFunction.apply(torch.zeros(4, 32, dtype=torch.bfloat16), w.double(), 32, None)
    with pytest.raises(ValueError):
        TernaryLinearFunction.apply(torch.zeros(4, 16, dtype=torch.bfloat16), w, 32, None)
    with pytest.raises(TypeError):
        TernaryLinearFunction.apply(torch.zeros(4, 32, dtype=torch.bfloat16), w, 32, torch.float16)


def test_module_rejects_k_not_a_multiple_of_64():
    with pytest.raises(ValueError):
        TernaryLinear(96, 8, g=32, device="cpu")  # a multiple of g and of 16, not of 64


def test_packed_module_checks_its_buffers_and_inputs():
    from paper_2606_18114_gb300.ternary_linear import PackedTernaryLinear
    codes = torch.zeros(8, 256 // 16, dtype=torch.int32)
    scales = torch.zeros(8, 256 // 128)
    layer = PackedTernaryLinear(codes, scales, 256, g=128)
    assert layer.out_features == 8 and dict(layer.named_buffers()).keys() == {"codes", "scales"}
    with pytest.raises(ValueError):
        PackedTernaryLinear(codes[:, :8], scales, 256, g=128)        # codes of another k
    with pytest.raises(ValueError):
        PackedTernaryLinear(codes, scales.double(), 256, g=128)      # fp64 scales
    with pytest.raises(ValueError):
        PackedTernaryLinear(codes.long(), scales, 256, g=128)        # int64 codes
    with pytest.raises(TypeError):
        PackedTernaryLinear(codes, scales, 256, g=128, out_dtype=torch.float16)
    with pytest.raises(TypeError):
        layer(torch.zeros(2, 256))                                   # fp32 activations
    with pytest.raises(ValueError):
        layer(torch.zeros(2, 128, dtype=torch.bfloat16))             # wrong feature count
