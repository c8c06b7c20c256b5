"""Oracle for the learnable-scale variant — TEST INFRASTRUCTURE.

Only the tests, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU legs may
import this module; the product path never calls it.

§4 of the paper ("Zero-Ratio Collapse", Table 1) contrasts the fixed absmean
scale of §3.1 with a scale trained as a parameter (``nn.Parameter``), which let
the zero ratio run away to 90 %. The quantizer is the one of §3.1 with the
scale taken from the parameter instead of the weights; the paper does not write
out the gradient that reaches the scale. Restated, with the readings this
oracle takes:

* c_i  = round(clip(w_i / s_g, -1, 1)), the quotient in fp32 as §3.1's code
         decision, round half to even; for a scale of either sign (a negative
         scale flips the codes, s * c still approximates w); a NaN quotient
         (0 / 0) gives 0.
* W^_i = s_g * c_i (the forward and backward products are §3.1's).
* ds_g: the chain rule through W^ = s * round(clip(w / s)) with the rounding
  passed straight through (derivative 1, the rule §3.1 applies to the latent
  weights) and the clip's derivative 1 inside (-1, 1), 0 outside:
         dW^_i / ds = c_i - q_i [|q_i| < 1],   q_i = w_i / s,
         ds_g = sum_i dW^_i c_i - (1 / s) sum_{|w_i| < |s|} dW^_i w_i
  in fp64; the test |w| < |s| (the same as |q| < 1 for s != 0) compares the
  fp32 inputs exactly; for s = 0 the second sum is empty.
* The latent weights keep §3.1's identity straight-through gradient (dW
  unchanged), so the two parameterizations differ only in the scale; both the
  weights and the scales take the AdamW step of §3.3 (``adamw_oracle``).

Parity: pinned by ``tests/test_learnable_pins.py`` (reduction to §3.1 at the
absmean, sign symmetry, torch autograd of the straight-through surrogate, its
finite differences, closed forms, pure-Python brute force).
"""
from __future__ import annotations

import numpy as np

from oracle import adamw_oracle, tq_oracle

__all__ = ["quantize_with_scales", "scale_grad", "adamw_requantize_with_scales"]


def quantize_with_scales(w, g: int, s):
    """Codes of ``w`` (fp32 ``[N, K]``) against the scales ``s`` (fp32 ``[N, K/g]``).
    Returns ``(codes uint32 [N, K/16], zero_counts int32 [N, K/g], c int8 [N, K])``."""
    w = np.asarray(w, dtype=np.float32)
    s = np.asarray(s, dtype=np.float32)
    n, k = w.shape
    if k % g or k % 16:
        raise ValueError("K must be a multiple of g and of 16")
    wg = w.reshape(n, k // g, g)
    with np.errstate(invalid="ignore", divide="ignore", over="ignore"):
        q = wg / s[:, :, None]  # fp32 quotient
    c = np.rint(np.clip(q, np.float32(-1.0), np.float32(1.0)))
    c = np.where(np.isnan(c), np.float32(0.0), c).astype(np.int8).reshape(n, k)
    zero_counts = (c.reshape(n, k // g, g) == 0).sum(axis=2).astype(np.int32)
    return tq_oracle.pack(c), zero_counts, c


def scale_grad(w, dw, c, s, g: int) -> np.ndarray:
    """ds[n][j] of the straight-through reading above (fp64). ``c``: int8 codes
    ``[N, K]`` or packed uint32 ``[N, K/16]``."""
    w32 = np.asarray(w, dtype=np.float32)
    n, k = w32.shape
    s32 = np.asarray(s, dtype=np.float32)
    c = np.asarray(c)
    if c.dtype == np.uint32:
        c = tq_oracle.unpack(c, k)
    dwg = np.asarray(dw, dtype=np.float64).reshape(n, k // g, g)
    wg = w32.reshape(n, k // g, g)
    inside = np.abs(wg) < np.abs(s32)[:, :, None]  # fp32 comparison, exact
    a = (dwg * c.reshape(n, k // g, g).astype(np.float64)).sum(axis=2)
    b = (dwg * wg.astype(np.float64) * inside).sum(axis=2)
    s64 = s32.astype(np.float64)
    with np.errstate(invalid="ignore", divide="ignore"):
        return np.where(s64 == 0.0, a, a - b / s64)


def adamw_requantize_with_scales(w, grad, m, v, g: int, consts, s):
    """AdamW on the latent weights (``adamw_oracle.adamw_step``), then their codes
    against the given (already updated) scales. Returns ``(w, m, v, codes, zeros)``."""
    w_new, m_new, v_new = adamw_oracle.adamw_step(w, grad, m, v, consts)
    codes, zeros, _ = quantize_with_scales(w_new, g, s)
    return w_new, m_new, v_new, codes, zeros
