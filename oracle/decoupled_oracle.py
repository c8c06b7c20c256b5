"""Oracle for the decoupled (threshold / magnitude) quantizer — TEST INFRASTRUCTURE.

Only the tests, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU legs may
import this module; the product path never calls it.

The decoupled-quantization ablation of the paper's appendix separates the two
roles the absmean plays in the standard TernaryLinear (§3.1): a fixed threshold
tau_g, which decides which weights become zero, and a learnable magnitude
alpha_g, which scales the non-zero codes; the asymmetric-gate variant lowers the
threshold to 0.8 x absmean on the gate rows (rows 0..4095 of in_proj). Restated:

* s_g   = (1/g) * sum_{i in group} |w_i|              (fp64 mean, stored fp32)
* tau_g = f_n * s_g                                   (row factor f_n; fp32 product)
* c_i   = round(clip(w_i / tau_g, -1, 1))             (decided in fp32, as §3.1's codes)
* W^    = alpha_g * c                                 (forward and dX with alpha as the scale)
* dalpha_g = sum_{i in group} dW^_i * c_i             (the magnitude's gradient; dW^ = dY^T X,
                                                       the same matrix the STE hands to W)

Readings: the threshold factor multiplies the fp32
absmean in fp32; with f_n = 1 everything reduces to ``tq_oracle.quantize``; the
magnitude's gradient is the plain chain rule of W^ = alpha * c with c held fixed
(the codes do not depend on alpha), accumulated in fp64.

Parity: pinned by ``tests/test_decoupled_pins.py`` (reduction to the standard
quantizer, the Gaussian zero ratio at a lowered threshold, brute force).
"""
from __future__ import annotations

import numpy as np

from oracle import tq_oracle

__all__ = ["quantize_decoupled", "alpha_grad"]


def quantize_decoupled(w: np.ndarray, g: int, row_factor=None):
    """Codes decided against tau = f_n * absmean. ``row_factor``: fp32 [N] or None
    (all ones). Returns ``(codes uint32 [N, K/16], absmean fp32 [N, K/g],
    zero_counts int32 [N, K/g], c int8 [N, K], tau fp32 [N, K/g])``."""
    w = np.asarray(w, dtype=np.float32)
    n, k = w.shape
    if k % g or k % 16:
        raise ValueError("K must be a multiple of g and of 16")
    wg = w.reshape(n, k // g, g)
    s32 = (np.abs(wg.astype(np.float64)).sum(axis=2) / g).astype(np.float32)
    f = np.ones(n, np.float32) if row_factor is None else np.asarray(row_factor, np.float32)
    tau = (s32 * f[:, None]).astype(np.float32)  # one fp32 product
    with np.errstate(invalid="ignore", divide="ignore"):
        q = wg / tau[:, :, None]
    c = np.rint(np.clip(q, np.float32(-1.0), np.float32(1.0)))
    c = np.where(np.isnan(c), np.float32(0.0), c)  # tau = 0: every code is 0
    c = c.astype(np.int8).reshape(n, k)
    zero_counts = (c.reshape(n, k // g, g) == 0).sum(axis=2).astype(np.int32)
    return tq_oracle.pack(c), s32, zero_counts, c, tau


def alpha_grad(dw, c: np.ndarray, g: int) -> np.ndarray:
    """dalpha[n][j] = sum over group j of row n of dW * c (fp64). ``c``: int8 codes
    [N, K] (or packed uint32 [N, K/16])."""
    dw = np.asarray(dw, dtype=np.float64)
    n, k = dw.shape
    c = np.asarray(c)
    if c.dtype == np.uint32:
        c = tq_oracle.unpack(c, k)
    return (dw * c.astype(np.float64)).reshape(n, k // g, g).sum(axis=2)
