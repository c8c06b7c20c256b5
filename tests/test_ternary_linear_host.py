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
