"""Decode launches chained as a model's layers (needs a GB300).

Each layer's bf16 output is the next layer's input, and the launches follow each
other on one stream with no synchronisation: a decode launch may start before the
previous one has finished (dependent launch), so it must not read its input, nor
write its output, before then. Outputs start as NaN; the chain must equal, bit for
bit, the same chain with the device synchronised between launches, and every layer
must match the oracle applied to the input it actually received."""
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


@pytest.mark.parametrize("m", [1, 3, 12])
def test_chained_layers(tq, m):
    g = 128
    dims = [2048, 1024, 2048, 4096, 1024] * 4 + [2048]   # k of layer l, n of layer l - 1
    layers = []
    for i in range(len(dims) - 1):
        k, n = dims[i], dims[i + 1]
        w = synth.latent_weights(n, k, seed=400 + i)
        codes, s, z = tq.quantize(torch.from_numpy(w).cuda(), g)
        layers.append((codes, s, validated_w_hat(w, g, codes, s, z), n))
    x0 = synth.activations_bf16(m, dims[0], seed=399).cuda()

    def run(sync):
        ys = [torch.full((m, n), float("nan"), device="cuda", dtype=torch.bfloat16)
              for (_, _, _, n) in layers]
        torch.cuda.synchronize()
        x = x0
        for (codes, s, _, _), y in zip(layers, ys):
            tq.linear_fwd(x, codes, s, g, y=y)
            if sync:
                torch.cuda.synchronize()
            x = y
        torch.cuda.synchronize()
        tq.device_status()
        return ys

    chained = run(sync=False)
    serial = run(sync=True)
    for i, (a, b) in enumerate(zip(chained, serial)):
        assert torch.equal(a, b), f"layer {i}: the chained launch differs from the serial one"
    x = x0.cpu()
    for i, ((_, _, w_hat, _), y) in enumerate(zip(layers, chained)):
        check_close(to_np(y), O.linear_fwd(x, w_hat), f"layer {i} m={m}", max_rel_rms=3e-2)
        x = y.cpu()
