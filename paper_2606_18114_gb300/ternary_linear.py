"""TernaryLinear (§3.1) as a torch autograd function and module over libtq.

The forward quantises the fp32 latent weights at every call (per-group absmean scale,
recomputed and not learned; ternary codes; 2-bit packing) and multiplies bf16 or fp16
activations by the dequantised weights (W1.58A16); the backward is the straight-through
estimator: dX = dY·Ŵ and dW = dYᵀ·X, handed to the latent weights unchanged. Every step
runs in libtq's kernels (``tq.quantize_with_transpose``, ``tq.linear_fwd``,
``tq.linear_bwd``); this module only marshals tensors. No bias (the paper's layer has
none).

Shapes: ``x [..., in_features]`` (bf16 or fp16, last dimension contiguous after a
reshape), ``weight [out_features, in_features]`` fp32; in_features a multiple of 64 and of
the group size g, out_features a multiple of 8 (the backward kernels' requirement).
``PackedTernaryLinear`` (from ``TernaryLinear.pack()``) is the inference form: only the
2-bit codes and group scales, no latent weights, no gradient.
"""
from __future__ import annotations

import torch

from . import tq

_OUT_TYPES = (torch.float32, torch.bfloat16)


class TernaryLinearFunction(torch.autograd.Function):
    """y = x Ŵᵀ with Ŵ = s·c the grouped ternary quantisation of ``weight``; STE backward.

    ``out_dtype`` is the dtype of y (fp32 or bf16; default: x's dtype when bf16, else
    fp32). dX comes back in x's dtype when that is bf16 and in fp32 otherwise, cast to x's
    dtype as autograd requires; dW is fp32."""

    @staticmethod
    def forward(ctx, x: torch.Tensor, weight: torch.Tensor, g: int, out_dtype=None):
        if x.dtype not in (torch.bfloat16, torch.float16):
            raise TypeError(f"x must be bf16 or fp16, not {x.dtype}")
        if weight.dtype != torch.float32:
            raise TypeError(f"weight must be fp32, not {weight.dtype}")
        n, k = weight.shape
        if x.shape[-1] != k:
            raise ValueError(f"x has {x.shape[-1]} features, weight {k}")
        if out_dtype is None:
            out_dtype = torch.bfloat16 if x.dtype == torch.bfloat16 else torch.float32
        if out_dtype not in _OUT_TYPES:
            raise TypeError(f"out_dtype must be fp32 or bf16, not {out_dtype}")
        x2 = x.reshape(-1, k).contiguous()
        w = weight.detach().contiguous()
        codes, scales, zeros, codes_t = tq.quantize_with_transpose(w, g)
        y = tq.linear_fwd(x2, codes, scales, g, out_dtype=out_dtype)
        ctx.save_for_backward(x2, codes, scales, codes_t)
        ctx.g, ctx.n, ctx.k, ctx.x_shape, ctx.x_dtype = g, n, k, x.shape, x.dtype
        ctx.mark_non_differentiable(zeros)
        return y.reshape(*x.shape[:-1], n), zeros

    @staticmethod
    def backward(ctx, dy: torch.Tensor, _dzeros):
        x2, codes, scales, codes_t = ctx.saved_tensors
        g, n, k = ctx.g, ctx.n, ctx.k
        want_dx, want_dw = ctx.needs_input_grad[0], ctx.needs_input_grad[1]
        if not (want_dx or want_dw):
            return None, None, None, None
        dy2 = dy.reshape(-1, n).to(ctx.x_dtype).contiguous()
        dx_dtype = torch.bfloat16 if ctx.x_dtype == torch.bfloat16 else torch.float32
        dx, dw = tq.linear_bwd(dy2, x2, codes, scales, k, g, want_dx=want_dx, want_dw=want_dw,
                               codes_t=codes_t, dx_dtype=dx_dtype)
        if dx is not None:
            dx = dx.to(ctx.x_dtype).reshape(ctx.x_shape)
        return dx, dw, None, None


class TernaryLinear(torch.nn.Module):
    """Drop-in linear layer with grouped ternary weights (§3.1): fp32 latent weights
    ``[out_features, in_features]`` trained through the straight-through estimator, no
    bias. ``zero_ratio()`` is the share of zero codes in the last forward (§4's zero-ratio
    monitor; it reads the group zero counts back from the device)."""

    def __init__(self, in_features: int, out_features: int, g: int = 128, out_dtype=None,
                 device="cuda", init_std: float = 0.02):
        super().__init__()
        if in_features % 64 or in_features % g:
            raise ValueError("in_features must be a multiple of 64 and of g")
        if out_features % 8:
            raise ValueError("out_features must be a multiple of 8")
        self.in_features, self.out_features, self.g, self.out_dtype = (
            in_features, out_features, g, out_dtype)
        self.weight = torch.nn.Parameter(
            torch.randn(out_features, in_features, device=device, dtype=torch.float32) * init_std)
        self._zeros = None

    def forward(self, x: torch.Tensor) -> torch.Tensor:
        y, zeros = TernaryLinearFunction.apply(x, self.weight, self.g, self.out_dtype)
        self._zeros = zeros
        return y

    def zero_ratio(self) -> float:
        if self._zeros is None:
            raise RuntimeError("no forward has run yet")
        return float(self._zeros.sum(dtype=torch.int64)) / self.weight.numel()

    @torch.no_grad()
    def pack(self) -> "PackedTernaryLinear":
        """The inference form of the current weights: their 2-bit codes and group scales
        (quantised once, here), without the fp32 latent weights."""
        codes, scales, _ = tq.quantize(self.weight.detach().contiguous(), self.g)
        return PackedTernaryLinear(codes, scales, self.in_features, self.g, self.out_dtype)

    def extra_repr(self) -> str:
        return f"in_features={self.in_features}, out_features={self.out_features}, g={self.g}"


class PackedTernaryLinear(torch.nn.Module):
    """Inference form of TernaryLinear (§8, storage): the weights held only as packed
    ternary codes (uint32-as-int32 ``[out_features, in_features / 16]``, 16 codes per
    word) and fp32 group scales ``[out_features, in_features / g]`` — 0.25 + 4/g bytes
    per weight — and the forward y = x Ŵᵀ run on them: the decode kernel up to 16
    tokens, the tensor-core GEMM beyond. No gradient flows through it."""

    def __init__(self, codes: torch.Tensor, scales: torch.Tensor, in_features: int, g: int = 128,
                 out_dtype=None):
        super().__init__()
        n = codes.shape[0]
        if codes.dtype != torch.int32 or codes.shape != (n, in_features // 16):
            raise ValueError("codes must be int32 [out_features, in_features / 16]")
        if scales.dtype != torch.float32 or scales.shape != (n, in_features // g):
            raise ValueError("scales must be fp32 [out_features, in_features / g]")
        if in_features % 64 or in_features % g:
            raise ValueError("in_features must be a multiple of 64 and of g")
        if out_dtype is not None and out_dtype not in _OUT_TYPES:
            raise TypeError(f"out_dtype must be fp32 or bf16, not {out_dtype}")
        self.in_features, self.out_features, self.g, self.out_dtype = in_features, n, g, out_dtype
        self.register_buffer("codes", codes.contiguous())
        self.register_buffer("scales", scales.contiguous())

    @torch.no_grad()
    def forward(self, x: torch.Tensor) -> torch.Tensor:
        if x.dtype not in (torch.bfloat16, torch.float16):
            raise TypeError(f"x must be bf16 or fp16, not {x.dtype}")
        if x.shape[-1] != self.in_features:
            raise ValueError(f"x has {x.shape[-1]} features, the layer {self.in_features}")
        out_dtype = self.out_dtype
        if out_dtype is None:
            out_dtype = torch.bfloat16 if x.dtype == torch.bfloat16 else torch.float32
        x2 = x.reshape(-1, self.in_features).contiguous()
        y = tq.linear_fwd(x2, self.codes, self.scales, self.g, out_dtype=out_dtype)
        return y.reshape(*x.shape[:-1], self.out_features)

    def extra_repr(self) -> str:
        return f"in_features={self.in_features}, out_features={self.out_features}, g={self.g}"
