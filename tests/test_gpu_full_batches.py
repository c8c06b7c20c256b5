"""The batched launches at their full size, against the oracle (needs a GB300).

Every in_proj [8512, 2048] and out_proj [2048, 4096] of the 48 blocks of Mamba-2
1.3B (96 matrices, 1.24 B weights) in one launch:

* the decode forward (``tq_linear_fwd_batched``) at 1, 4 and 16 tokens, g = 128 —
  the batch-1 decode that §8 calls bandwidth-bound; the launch claims its 256-row
  units longest-K first across matrices, thousands of units per launch;
* the per-step requantize (``tq_quantize_batched``, §3.1 recomputes the scale at
  every call) at every group size, half of the blocks drawn from N(0, 0.02^2) and
  half from the Student-t(3) of the same standard deviation.

The weights (5 GB) are drawn on the device by torch's generator and the sampled
rows copied back for the oracle; the oracle sees only those inputs.
"""
import numpy as np
import pytest
import torch

from oracle import tq_oracle as O
from paper_2606_18114_gb300 import synth
from parity import check_close, check_quantize, to_np, validated_w_hat

pytestmark = pytest.mark.gpu

N_LAYERS = synth.MAMBA2_1P3B["n_layers"]
SHAPES = [synth.MAMBA2_1P3B["in_proj"], synth.MAMBA2_1P3B["out_proj"]] * N_LAYERS


@pytest.fixture(scope="module")
def tq():
    if not torch.cuda.is_available():
        pytest.fail("the gpu tests need a CUDA device")
    from paper_2606_18114_gb300 import build, tq as _tq
    build.build()
    _tq.load()
    return _tq


def _student_t3(shape, gen, std):
    """Student-t(3) scaled to standard deviation std: z / sqrt(chi2_3 / 3) * std / sqrt(3)."""
    z = torch.randn(shape, generator=gen, device="cuda")
    c = sum(torch.randn(shape, generator=gen, device="cuda") ** 2 for _ in range(3)) / 3.0
    return z / c.sqrt() * (std / 3.0 ** 0.5)


def _sample_rows(n, rs):
    """Eight random rows, plus the last row (the ragged last 256-row unit of in_proj
    ends at row 8511, 64 rows into its unit)."""
    rows = set(rs.choice(n, 8, replace=False).tolist()) | {n - 1}
    return np.array(sorted(rows))


@pytest.fixture(scope="module")
def weights():
    """The 96 latent matrices on the device, even blocks Gaussian, odd blocks t3."""
    gen = torch.Generator(device="cuda")
    gen.manual_seed(2024)
    ws = []
    for i, shape in enumerate(SHAPES):
        block = i // 2
        ws.append(torch.randn(shape, generator=gen, device="cuda") * 0.02 if block % 2 == 0
                  else _student_t3(shape, gen, 0.02))
    yield ws
    del ws
    torch.cuda.empty_cache()


@pytest.mark.parametrize("g", [32, 64, 128, 256, 512])
def test_quantize_batched_96_projections(tq, weights, g):
    """One tq_quantize_batched over the 96 projections; nine rows of every matrix
    checked against the oracle (codes and zero counts exact outside near-ties,
    scales to 1e-6)."""
    items = [(w, torch.empty((w.shape[0], w.shape[1] // 16), dtype=torch.int32, device="cuda"),
              torch.empty((w.shape[0], w.shape[1] // g), device="cuda"),
              torch.empty((w.shape[0], w.shape[1] // g), dtype=torch.int32, device="cuda"))
             for w in weights]
    tq.quantize_batched(items, g)
    tq.device_status()
    rs = np.random.default_rng(g)
    for i, (w, codes, s, z) in enumerate(items):
        rows = torch.from_numpy(_sample_rows(w.shape[0], rs)).cuda()
        flips, ties = check_quantize(to_np(w[rows]), g, codes[rows], s[rows], z[rows])
        assert flips <= ties, f"matrix {i}"
    del items


@pytest.fixture(scope="module")
def quantized(tq, weights):
    """Codes and scales (g = 128) of the 96 matrices, and nine sampled rows of each
    with their validated dequantized weights."""
    rs = np.random.default_rng(7)
    out = []
    for w in weights:
        codes, s, z = tq.quantize(w, 128)
        rows = _sample_rows(w.shape[0], rs)
        sel = torch.from_numpy(rows).cuda()
        w_rows = to_np(w[sel])
        w_hat = validated_w_hat(w_rows, 128, codes[sel], s[sel], z[sel])
        out.append(dict(codes=codes, scales=s, rows=rows, w_hat=w_hat))
    tq.device_status()
    return out


@pytest.mark.parametrize("m", [1, 4, 16])
def test_decode_batched_96_projections(tq, quantized, m):
    """Config 4: one tq_linear_fwd_batched over all 96 projections at m tokens; the
    sampled rows' outputs of every matrix against the oracle (relative Frobenius
    5e-3, max 2e-2 * rms), every output finite. Two launches in a row, so the second
    runs on the scheduler state the first one left."""
    items = []
    for i, q in enumerate(quantized):
        n = q["codes"].shape[0]
        k = q["codes"].shape[1] * 16
        x = synth.activations_bf16(m, k, seed=300 + i, stream="x_decode")
        items.append(dict(x=x.cuda(), x_host=x, codes=q["codes"], scales=q["scales"], g=128,
                          y=torch.full((m, n), float("nan"), device="cuda")))
    arr = tq.fwd_batch(items)
    for rep in range(2):
        for it in items:
            it["y"].fill_(float("nan"))
        tq.linear_fwd_batched(arr, m)
        tq.device_status()
        for i, (it, q) in enumerate(zip(items, quantized)):
            y = it["y"]
            assert torch.isfinite(y).all(), f"matrix {i} rep {rep}: unwritten or non-finite outputs"
            got = to_np(y[:, torch.from_numpy(q["rows"]).cuda()])
            check_close(got, O.linear_fwd(it["x_host"], q["w_hat"]), f"Y matrix {i} m={m} rep {rep}")
