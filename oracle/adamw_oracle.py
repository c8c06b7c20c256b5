"""Oracle for the fused AdamW update + requantize — TEST INFRASTRUCTURE.

Only the tests, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU legs may
import this module; the product path never calls it.

§3.3 of the paper trains the latent fp32 weights with AdamW (betas (0.9, 0.95),
weight decay 0.01, gradient clip 1.0; the training-hyperparameter table of the
appendix) and requantizes them every step (§3.1: the scale is recomputed from
the weights each forward pass). This module restates one optimizer step on one
weight matrix followed by that requantization:

* AdamW, decoupled weight decay with Adam's bias correction:
      g' = grad_scale * g                 (grad_scale folds in gradient clipping)
      m  = beta1 * m + (1 - beta1) * g'
      v  = beta2 * v + (1 - beta2) * g'^2
      w  = w * (1 - lr * wd) - (lr / (1 - beta1^t)) * m / (sqrt(v) / sqrt(1 - beta2^t) + eps)
* then ``tq_oracle.quantize`` of the new w (scales, ternary codes, zero counts).

Readings of points the paper leaves open:

* eps is not given; the default of the common AdamW implementation, 1e-8.
* The update runs in fp32, the precision of the latent weights, because the new
  weights decide integer codes: the oracle takes those decisions in the
  kernel's precision. Every operation below is one IEEE fp32 operation (no
  fused multiply-add), in the order written; the step constants are computed
  in fp64 from the hyperparameters and rounded once to fp32. With that order
  fixed, the oracle and the kernel agree bit for bit on w, m and v.
* Weight decay multiplies the weights before the step (w * (1 - lr * wd)),
  the bias-corrected step is lr / (1 - beta1^t) times m / denom, divided first.

Parity: pinned by ``tests/test_adamw_pins.py`` (closed form of the first step
from zero moments, zero-gradient decay, agreement with torch.optim.AdamW over
several steps).
"""
from __future__ import annotations

import math

import numpy as np

from oracle import tq_oracle

__all__ = ["step_constants", "adamw_step", "adamw_requantize"]

F32 = np.float32


def step_constants(lr, beta1, beta2, eps, weight_decay, step, grad_scale=1.0):
    """fp32 constants of step t (t >= 1), each computed in fp64 and rounded once."""
    if step < 1:
        raise ValueError("step counts from 1")
    return dict(
        b1=F32(beta1), omb1=F32(1.0 - beta1),
        b2=F32(beta2), omb2=F32(1.0 - beta2),
        decay=F32(1.0 - lr * weight_decay),
        step_size=F32(lr / (1.0 - beta1 ** step)),
        inv_bc2_sqrt=F32(1.0 / math.sqrt(1.0 - beta2 ** step)),
        eps=F32(eps), grad_scale=F32(grad_scale))


def adamw_step(w, grad, m, v, c):
    """One AdamW step in fp32 (operation order of the module docstring).
    Returns new (w, m, v) as fp32 arrays; inputs are not modified."""
    w = np.asarray(w, dtype=F32)
    gr = np.asarray(grad, dtype=F32) * c["grad_scale"]
    m = np.asarray(m, dtype=F32)
    v = np.asarray(v, dtype=F32)
    m_new = c["b1"] * m + c["omb1"] * gr
    v_new = c["b2"] * v + c["omb2"] * (gr * gr)
    denom = np.sqrt(v_new) * c["inv_bc2_sqrt"] + c["eps"]
    w_new = w * c["decay"] - c["step_size"] * (m_new / denom)
    return w_new.astype(F32), m_new.astype(F32), v_new.astype(F32)


def adamw_requantize(w, grad, m, v, g, c):
    """The fused step: AdamW, then the group-wise ternary quantization of the new
    weights. Returns (w, m, v, codes, scales, zeros)."""
    w_new, m_new, v_new = adamw_step(w, grad, m, v, c)
    codes, scales, zeros, _ = tq_oracle.quantize(w_new, g)
    return w_new, m_new, v_new, codes, scales, zeros
