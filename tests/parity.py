"""Comparison helpers shared by the GPU parity tests (test infrastructure).

Bars (the floating-point ones are the parity target of this project):
* codes and zero counts bit-exact, except elements with |w/s| within 1e-5 of
  the rounding tie 0.5, which are counted and reported;
* scales within 1e-6 relative;
* Y, dX, dW: relative Frobenius error <= 5e-3 and max element error
  <= 2e-2 * rms of the oracle output.
"""
from __future__ import annotations

import numpy as np
import torch

from oracle import tq_oracle as O

REL_FROB = 5e-3
MAX_REL_RMS = 2e-2
SCALE_RTOL = 1e-6
TIE_TOL = 1e-5


def to_np(t: torch.Tensor) -> np.ndarray:
    t = t.detach().to("cpu")
    if t.dtype == torch.bfloat16:
        t = t.float()
    return t.numpy()


def codes_u32(t: torch.Tensor) -> np.ndarray:
    return to_np(t).view(np.uint32)


def check_quantize(w: np.ndarray, g: int, codes_gpu, scales_gpu, zeros_gpu, ref=None):
    """Compare the GPU quantiser with the oracle; returns the near-tie count."""
    n, k = w.shape
    ref_codes, ref_s, ref_z, ref_c = ref if ref is not None else O.quantize(w, g)
    s = to_np(scales_gpu)
    z = to_np(zeros_gpu)
    cw = codes_u32(codes_gpu)
    assert s.shape == ref_s.shape and z.shape == ref_z.shape and cw.shape == ref_codes.shape
    # scales
    rel = np.abs(s.astype(np.float64) - ref_s) / np.maximum(ref_s.astype(np.float64), 1e-300)
    bad = (rel > SCALE_RTOL) & ~((ref_s == 0) & (s == 0))
    assert not bad.any(), f"{bad.sum()} scales off; worst rel {rel[bad].max()}"
    # codes: decode the GPU words and compare outside near-ties
    c = O.unpack(cw, k)
    ties = O.near_tie_mask(w, ref_s, g, TIE_TOL)
    diff = c != ref_c
    assert not (diff & ~ties).any(), f"{(diff & ~ties).sum()} code mismatches away from ties"
    # whole words without a near-tie element are bit-identical
    word_ties = ties.reshape(n, k // 16, 16).any(axis=2)
    assert np.array_equal(cw[~word_ties], ref_codes[~word_ties])
    # zero counts: exact except groups with a near-tie, where they differ by
    # at most the number of near-ties of that group
    grp_ties = ties.reshape(n, k // g, g).sum(axis=2)
    dz = np.abs(z.astype(np.int64) - ref_z)
    assert np.all(dz <= grp_ties), "zero counts differ beyond near-ties"
    assert np.array_equal(z[grp_ties == 0], ref_z[grp_ties == 0])
    return int(diff.sum()), int(ties.sum())


def check_close(got, ref: np.ndarray, what: str, rel_frob=REL_FROB, max_rel_rms=MAX_REL_RMS):
    g = got if isinstance(got, np.ndarray) else to_np(got)
    g = g.astype(np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert g.shape == ref.shape, f"{what}: shape {g.shape} vs {ref.shape}"
    assert np.all(np.isfinite(g)), f"{what}: non-finite output"
    err = g - ref
    nref = np.linalg.norm(ref)
    relf = np.linalg.norm(err) / nref if nref > 0 else np.linalg.norm(err)
    rms = np.sqrt(np.mean(ref * ref))
    mx = np.abs(err).max() if err.size else 0.0
    assert relf <= rel_frob, f"{what}: relative Frobenius error {relf:.3e} > {rel_frob}"
    assert mx <= max_rel_rms * rms, f"{what}: max error {mx:.3e} > {max_rel_rms} * rms {rms:.3e}"
    return relf, mx / rms if rms > 0 else 0.0


def validated_w_hat(w: np.ndarray, g: int, codes_gpu, scales_gpu, zeros_gpu) -> np.ndarray:
    """The dequantized weights the GPU products use, for comparing those products:
    the GPU codes are first checked against the oracle (identical outside
    near-ties, where either rounding is correct), then expanded with the oracle's
    fp64-exact scales. Building W^ from the oracle's own codes instead would charge
    a product with s * x for every near-tie weight the two sides round apart."""
    n, k = w.shape
    ref = O.quantize(w, g)
    check_quantize(w, g, codes_gpu, scales_gpu, zeros_gpu, ref=ref)
    return O.dequantize(codes_u32(codes_gpu), ref[1], k, g)
