"""tq_quantize_with_transpose (needs a GB300): one cooperative launch that quantises
and then transposes the codes it wrote. Its four outputs must equal tq_quantize
followed by tq_codes_transpose bit for bit (those two are checked against the oracle
and against the transposed layout's definition in test_gpu_parity.py); the codes are
also checked against the oracle directly here. Shapes: the Mamba-2 projections, ragged
rows (n % 64 != 0, a last 16-row group past n), a single row, every group size; the
transposed output starts filled with -1 so that every word, padding included, must be
written. Repeated launches on two streams cover more launches than the grid barrier
has slots (256), so every slot is reused after its reset."""
import numpy as np
import pytest
import torch

from paper_2606_18114_gb300 import synth
from parity import check_quantize, to_np

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def tq():
    if not torch.cuda.is_available():
        pytest.fail("the gpu tests need a CUDA device")
    from paper_2606_18114_gb300 import build, tq as _tq
    build.build()
    _tq.load()
    return _tq


def _outputs(n, k, g, fill=-1):
    return (torch.full((n, k // 16), fill, dtype=torch.int32, device="cuda"),
            torch.full((n, k // g), float("nan"), device="cuda"),
            torch.full((n, k // g), fill, dtype=torch.int32, device="cuda"),
            torch.full((k, 4 * ((n + 63) // 64)), fill, dtype=torch.int32, device="cuda"))


def _two_calls(tq, w, g):
    codes, s, z = tq.quantize(w, g)
    return codes, s, z, tq.codes_transpose(codes, w.shape[1])


@pytest.mark.parametrize("n,k,g", [
    (8512, 2048, 128),   # in_proj
    (2048, 4096, 32),    # out_proj, smallest group
    (200, 192, 64),      # ragged rows: 200 = 3 x 64 + 8
    (17, 64, 32),        # one 16-row group and one row past it
    (1, 512, 512),       # a single row, one stage shorter than a full one
    (130, 512, 256),
    (64, 128, 128),
    (100, 1088, 64),     # a last 1088 % 512 = 64 columns, a ragged last row group
])
def test_matches_quantize_then_transpose(tq, n, k, g):
    w = torch.from_numpy(synth.latent_weights(n, k, seed=n + k + g)).cuda()
    ref = _two_calls(tq, w, g)
    got = tq.quantize_with_transpose(w, g, out=_outputs(n, k, g))
    tq.device_status()
    for name, a, b in zip(("codes", "scales", "zeros", "codes_t"), got, ref):
        assert torch.equal(a, b), name
    rows = np.unique(np.r_[np.random.default_rng(n).choice(n, min(n, 8), replace=False), n - 1])
    sel = torch.from_numpy(rows).cuda()
    flips, ties = check_quantize(to_np(w[sel]), g, got[0][sel], got[1][sel], got[2][sel])
    assert flips <= ties


def test_repeated_launches_two_streams(tq):
    n, k, g = 4160, 1280, 128
    w = torch.from_numpy(synth.latent_weights(n, k, seed=91)).cuda()
    ref = _two_calls(tq, w, g)
    tq.device_status()
    streams = [torch.cuda.current_stream(), torch.cuda.Stream()]
    outs = [_outputs(n, k, g), _outputs(n, k, g)]
    torch.cuda.synchronize()
    for i in range(300):
        j = i % 2
        with torch.cuda.stream(streams[j]):
            tq.quantize_with_transpose(w, g, out=outs[j])
    torch.cuda.synchronize()
    tq.device_status()
    for out in outs:
        assert all(torch.equal(a, b) for a, b in zip(out, ref))
