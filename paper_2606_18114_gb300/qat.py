"""Zero-ratio tracking of the two scale parameterizations (§4, "Zero-Ratio
Collapse", Table 1) on a synthetic task, every step on libtq's kernels.

The paper contrasts the fixed absmean scale of §3.1 with a scale trained as a
parameter and reports the share of zero codes over training. Its experiment needs
the pretrained model, the distillation data and 50k steps; this driver runs the
same two quantized-layer updates on a synthetic teacher–student regression
instead and records the zero ratio as it goes:

* teacher: a dense fp32 weight W_t ~ N(0, 0.02^2); the student's latent weights
  start at W_t (QAT starts from the pretrained weights), its scales at their
  absmean;
* data: a fixed pool of bf16 activation batches X ~ N(0, 1); target Y_t = X W_t^T;
  loss mean((Y - Y_t)^2), whose gradient dY = 2 (Y - Y_t) / numel is the task's,
  not the method's (it is formed with torch elementwise operations, as a model
  above the layer would form it);
* a step: Y = tq_linear_fwd, dW = tq_linear_bwd (the STE of §3.1), then
  - fixed absmean: tq_adamw_requantize (AdamW on w, codes and scales of the new
    w from its absmean);
  - learnable scale: ds = tq_scale_grad, the scales' AdamW step (tq_adamw), then
    tq_adamw_requantize_with_scales against the new scales;
  AdamW with the hyperparameters of §3.3 on both w and s, and §3.3's schedule
  scaled to the run's length: a linear warm-up over the first 2 % of the steps
  (1k of 50k in the paper), then a cosine decay of the learning rate to zero.
"""
from __future__ import annotations

import math
from typing import Dict, List

import torch

__all__ = ["track_zero_ratio", "lr_at"]


def lr_at(t: int, steps: int, lr: float, warmup: int) -> float:
    """Learning rate of update t (0-based) of ``steps``: linear warm-up to ``lr`` over
    ``warmup`` updates, then cosine decay to zero at the last update."""
    if t < warmup:
        return lr * (t + 1) / warmup
    span = max(steps - warmup, 1)
    return lr * 0.5 * (1.0 + math.cos(math.pi * (t - warmup) / span))


def track_zero_ratio(tq, n: int, k: int, m: int, g: int, steps: int, learnable: bool,
                     seed: int = 0, lr: float = 2.5e-4, pool: int = 8,
                     every: int = 100, warmup: int = -1) -> List[Dict[str, float]]:
    """Run ``steps`` updates of one ternary linear layer [n, k] (group ``g``) on
    batches of ``m`` tokens with peak learning rate ``lr`` (warm-up of ``warmup``
    updates, default 2 % of ``steps``, then cosine decay); returns ``{"step",
    "zero_ratio", "loss", "scale_ratio"}`` every ``every`` steps (and at step 0),
    where ``scale_ratio`` is the mean scale over the mean |w| of the latent weights."""
    if warmup < 0:
        warmup = max(1, steps // 50)
    dev = torch.device("cuda")
    gen = torch.Generator(device=dev)
    gen.manual_seed(seed)
    w_t = torch.randn((n, k), generator=gen, device=dev) * 0.02
    xs = [torch.randn((m, k), generator=gen, device=dev).to(torch.bfloat16) for _ in range(pool)]
    ys = [x.float() @ w_t.t() for x in xs]
    w = w_t.clone()
    mw, vw = torch.zeros_like(w), torch.zeros_like(w)
    codes, s, z = tq.quantize(w, g)
    ms, vs = torch.zeros_like(s), torch.zeros_like(s)
    y = torch.empty((m, n), device=dev)
    dw = torch.empty((n, k), device=dev)
    ds = torch.empty_like(s)
    hp = dict(beta1=0.9, beta2=0.95, eps=1e-8, weight_decay=0.01)
    out: List[Dict[str, float]] = []
    for t in range(steps + 1):
        x, y_t = xs[t % pool], ys[t % pool]
        tq.linear_fwd(x, codes, s, g, y=y)
        diff = y - y_t
        if t % every == 0 or t == steps:
            out.append({"step": t, "zero_ratio": round(float(z.sum()) / (n * k), 4),
                        "loss": float((diff * diff).mean()),
                        "scale_ratio": round(float(s.mean()) / float(w.abs().mean()), 4)})
        if t == steps:
            break
        dy = (diff * (2.0 / diff.numel())).to(torch.bfloat16)
        hp["lr"] = lr_at(t, steps, lr, warmup)
        tq.linear_bwd(dy, x, codes, s, k, g, want_dx=False, dw=dw)
        if learnable:
            tq.scale_grad(w, dw, codes, s, g, out=ds)
            tq.adamw(s.view(-1), ds.view(-1), ms.view(-1), vs.view(-1), step=t + 1, **hp)
            tq.adamw_requantize_with_scales(w, dw, mw, vw, g, s, step=t + 1, out=(codes, z), **hp)
        else:
            tq.adamw_requantize(w, dw, mw, vw, g, step=t + 1, out=(codes, s, z), **hp)
    tq.device_status()
    return out
