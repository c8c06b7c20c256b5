"""Oracle for the grouped ternary (W1.58A16) linear layer — TEST INFRASTRUCTURE.

Only the tests, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` may import this module. The product
path (``paper_2606_18114_gb300``) never calls it and has no CPU fallback.

It is a plain, slow, obviously-correct restatement of §3.1 ("TernaryLinear
Module") of the paper, in numpy, in fp64 except where noted:

* per-group absmean scale, groups of ``g`` consecutive weights along the input
  dimension K of one output row:        s = (1/g) * sum_{i in group} |w_i|
* ternary code:                          c_i = round(clip(w_i / s, -1, 1))
* dequantised weight:                    w^_i = s * c_i
* forward:                               Y  = X W^T          (W1.58A16)
* straight-through backward (§3.1, and the STE remark of the HG-GSQ appendix):
                                         dX = dY W^
                                         dW = dY^T X         (to the latent W)

Readings of points the paper leaves open:

* "round" is round-half-to-even (``np.rint``). Only |w/s| = 0.5 is a tie that
  matters (1.5 rounds to 2, which the clip maps to 1 like 1.49 does).
* The code decision ``w / s`` is taken in fp32 — the precision of the stored
  scale and of the kernel — with ``s`` the fp64 mean rounded to fp32.
* An all-zero group has s = 0; 0/0 is undefined, and every code of that group
  is 0 (so its zero count is g).
* Straight-through estimator = identity: no clip mask, no gradient to s
  (the scale is "not a learned parameter", §3.1).
* Group-scale storage is fp32; products use that fp32 value exactly.

The packed code layout is the one ``include/tq.h`` documents; it is restated
here from that description, not shared with the CUDA sources:
16 codes per uint32 word, word ``k // 16`` of row n holds k in [16w, 16w+16);
code ``i = k % 16`` sits at bit ``2*(i//2)`` when i is even and at bit
``16 + 2*(i//2)`` when i is odd; the 2-bit values are 0b00 -> 0, 0b01 -> +1,
0b11 -> -1 (0b10 is never written).

Parity: every function here is pinned by ``tests/test_oracle_pins.py``
(hand-worked example, tie and zero groups, invariants, closed-form zero
ratios, pure-Python brute force, dense-matmul special cases).
"""
from __future__ import annotations

import numpy as np

__all__ = [
    "quantize",
    "pack",
    "unpack",
    "dequantize",
    "near_tie_mask",
    "linear_fwd",
    "linear_bwd_dx",
    "linear_bwd_dw",
    "ENCODE",
]

# 2-bit encoding of a ternary value (format of include/tq.h).
ENCODE = {0: 0b00, 1: 0b01, -1: 0b11}


def _code_bit(i: np.ndarray) -> np.ndarray:
    """Bit offset of code ``i = k % 16`` inside its word (format of include/tq.h)."""
    return 16 * (i & 1) + 2 * (i >> 1)


def quantize(w: np.ndarray, g: int):
    """§3.1: per-group absmean scale, ternary codes, zero count per group.

    ``w``: fp32 ``[N, K]`` with ``K % g == 0`` and ``K % 16 == 0``.
    Returns ``(codes uint32 [N, K/16], scales fp32 [N, K/g],
    zero_counts int32 [N, K/g], c int8 [N, K])``.
    """
    w = np.asarray(w, dtype=np.float32)
    n, k = w.shape
    if k % g or k % 16:
        raise ValueError("K must be a multiple of g and of 16")
    wg = w.reshape(n, k // g, g)
    # s_g = (1/g) * sum |w_i|   — accumulated in fp64, stored as fp32.
    s64 = np.abs(wg.astype(np.float64)).sum(axis=2) / g
    s32 = s64.astype(np.float32)
    # w~_i = round(clip(w_i / s_g, -1, 1)), the division in fp32.
    with np.errstate(invalid="ignore", divide="ignore"):
        q = wg / s32[:, :, None]
    c = np.rint(np.clip(q, np.float32(-1.0), np.float32(1.0)))
    c = np.where(np.isnan(c), np.float32(0.0), c)  # s = 0: every code is 0
    c = c.astype(np.int8).reshape(n, k)
    zero_counts = (c.reshape(n, k // g, g) == 0).sum(axis=2).astype(np.int32)
    return pack(c), s32, zero_counts, c


def near_tie_mask(w: np.ndarray, scales: np.ndarray, g: int, tol: float = 1e-5) -> np.ndarray:
    """Elements whose |w/s| lies within ``tol`` of the rounding tie 0.5 (fp64).

    Two correct implementations may decide these differently when their fp32
    scales differ by an ulp; parity tests count them instead of comparing them.
    """
    w = np.asarray(w, dtype=np.float64)
    n, k = w.shape
    s = np.repeat(np.asarray(scales, dtype=np.float64), g, axis=1)
    with np.errstate(invalid="ignore", divide="ignore"):
        r = np.abs(w / s)
    return np.abs(r - 0.5) <= tol


def pack(c: np.ndarray) -> np.ndarray:
    """Ternary codes int8 ``[N, K]`` -> packed uint32 ``[N, K/16]``."""
    c = np.asarray(c)
    n, k = c.shape
    if k % 16:
        raise ValueError("K must be a multiple of 16")
    v = np.zeros(c.shape, dtype=np.uint32)
    v[c == 1] = ENCODE[1]
    v[c == -1] = ENCODE[-1]
    if np.any((c != 0) & (c != 1) & (c != -1)):
        raise ValueError("codes must be in {-1, 0, 1}")
    shifts = _code_bit(np.arange(16, dtype=np.uint32))
    v = v.reshape(n, k // 16, 16) << shifts[None, None, :]
    return np.bitwise_or.reduce(v, axis=2).astype(np.uint32)


def unpack(codes: np.ndarray, k: int) -> np.ndarray:
    """Packed uint32 ``[N, K/16]`` -> int8 ``[N, K]``; rejects the unused 0b10."""
    codes = np.asarray(codes, dtype=np.uint32)
    n = codes.shape[0]
    shifts = _code_bit(np.arange(16, dtype=np.uint32))
    v = (codes[:, :, None] >> shifts[None, None, :]) & np.uint32(3)
    v = v.reshape(n, k)
    if np.any(v == 0b10):
        raise ValueError("invalid 2-bit code 0b10")
    out = np.zeros((n, k), dtype=np.int8)
    out[v == ENCODE[1]] = 1
    out[v == ENCODE[-1]] = -1
    return out


def dequantize(codes: np.ndarray, scales: np.ndarray, k: int, g: int) -> np.ndarray:
    """§3.1: w^_i = s_g * w~_i, fp64 ``[N, K]`` (the fp32 scale taken exactly)."""
    c = unpack(codes, k).astype(np.float64)
    s = np.repeat(np.asarray(scales, dtype=np.float32).astype(np.float64), g, axis=1)
    return s * c


def _f64(a) -> np.ndarray:
    """bf16/fp32 torch tensor or numpy array -> fp64 numpy (exact)."""
    if hasattr(a, "detach"):
        return a.detach().to("cpu").float().double().numpy()
    return np.asarray(a, dtype=np.float64)


def linear_fwd(x, w_hat: np.ndarray, rows=None) -> np.ndarray:
    """W1.58A16 forward Y = X W^T in fp64; ``rows`` selects rows of X (and Y)."""
    x = _f64(x)
    if rows is not None:
        x = x[np.asarray(rows)]
    return x @ w_hat.T


def linear_bwd_dx(dy, w_hat: np.ndarray, rows=None) -> np.ndarray:
    """STE backward to the input: dX = dY W^ (fp64); ``rows`` selects tokens."""
    dy = _f64(dy)
    if rows is not None:
        dy = dy[np.asarray(rows)]
    return dy @ w_hat


def linear_bwd_dw(dy, x, out_rows=None) -> np.ndarray:
    """STE backward to the latent weights: dW = dY^T X (fp64).

    ``out_rows`` selects output features n (rows of dW).
    """
    dy = _f64(dy)
    x = _f64(x)
    if out_rows is not None:
        dy = dy[:, np.asarray(out_rows)]
    return dy.T @ x
