"""Decode (m <= 16) on seeded random shapes against the oracle (needs a GB300).

Shapes drawn once from a fixed seed: every group size, k any multiple of 64 and of g
up to ~9000 (per-unit, per-window and per-segment scale fetches, ragged last
segments), n from 1 to 1200 (ragged blocks of 256 rows), 1 to 16 tokens, fp32 and
bf16 outputs, bf16 and fp16 activations. Single calls take pieces of k in clusters
when they leave SMs idle; the batched calls mix matrices of every kind in one launch.
"""
import numpy as np
import pytest
import torch

from oracle import tq_oracle as O
from paper_2606_18114_gb300 import synth
from parity import check_close, validated_w_hat

pytestmark = pytest.mark.gpu

_GROUPS = [32, 64, 128, 256, 512]


def _shape(rs):
    g = int(rs.choice(_GROUPS))
    step = max(64, g)
    k = step * int(rs.integers(1, 9000 // step + 1))
    n = int(rs.integers(1, 1201))
    return n, k, g


def _cases(seed, count):
    rs = np.random.default_rng(seed)
    out = []
    for i in range(count):
        n, k, g = _shape(rs)
        m = int(rs.integers(1, 17))
        out.append((i, n, k, g, m, bool(rs.integers(0, 2)), bool(rs.integers(0, 4) == 0)))
    return out


@pytest.fixture(scope="module")
def tq():
    if not torch.cuda.is_available():
        pytest.fail("the gpu tests need a CUDA device")
    from paper_2606_18114_gb300 import build, tq as _tq
    build.build()
    _tq.load()
    return _tq


def _matrix(tq, n, k, g, m, seed, f16):
    w = synth.latent_weights(n, k, seed=seed)
    codes, s, z = tq.quantize(torch.from_numpy(w).cuda(), g)
    x = (synth.activations_f16 if f16 else synth.activations_bf16)(m, k, seed=seed)
    return x, codes, s, O.linear_fwd(x, validated_w_hat(w, g, codes, s, z))


@pytest.mark.parametrize("case", _cases(2024, 40), ids=lambda c: f"n{c[1]}k{c[2]}g{c[3]}m{c[4]}")
def test_decode_random_shapes(tq, case):
    i, n, k, g, m, bf16_out, f16 = case
    x, codes, s, ref = _matrix(tq, n, k, g, m, 7000 + i, f16)
    out_dtype = torch.bfloat16 if bf16_out else torch.float32
    y = tq.linear_fwd(x.cuda(), codes, s, g, out_dtype=out_dtype)
    y2 = tq.linear_fwd(x.cuda(), codes, s, g, out_dtype=out_dtype)
    tq.device_status()
    check_close(y.float(), ref, f"Y n={n} k={k} g={g} m={m} f16={f16}",
                max_rel_rms=3e-2 if bf16_out else 2e-2)
    assert torch.equal(y, y2)


@pytest.mark.parametrize("seed", [11, 12, 13, 14])
def test_decode_random_batches(tq, seed):
    rs = np.random.default_rng(seed)
    m = int(rs.integers(1, 17))
    f16 = seed % 2 == 1
    items = []
    for j in range(int(rs.integers(2, 7))):
        n, k, g = _shape(rs)
        x, codes, s, ref = _matrix(tq, n, k, g, m, 9000 + 10 * seed + j, f16)
        items.append(dict(x=x.cuda(), codes=codes, scales=s, g=g,
                          y=torch.empty((m, n), device="cuda"), ref=ref))
    tq.linear_fwd_batched(items, m)
    tq.device_status()
    for j, it in enumerate(items):
        check_close(it["y"], it["ref"], f"batched Y[{j}] {tuple(it['codes'].shape)} g={it['g']} m={m}")
