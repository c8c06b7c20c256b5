"""CUDA path vs oracle, element by element, through the C ABI (needs a GB300).

Inputs come from ``paper_2606_18114_gb300.synth`` (seeded, host-side); the
oracle never sees a value produced by the CUDA path.
"""
import numpy as np
import pytest
import torch

from oracle import tq_oracle as O
from paper_2606_18114_gb300 import synth
from parity import check_close, check_quantize, codes_u32, to_np, validated_w_hat

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def tq():
    if not torch.cuda.is_available():
        pytest.fail("the gpu tests need a CUDA device")
    from paper_2606_18114_gb300 import build, tq as _tq
    build.build()
    _tq.load()
    return _tq


def _quant(tq, w_np, g):
    w = torch.from_numpy(w_np).cuda()
    codes, s, z = tq.quantize(w, g)
    tq.device_status()
    return codes, s, z


# ------------------------------------------------------------------ quantize
def test_quantize_hand_example_g128(tq, golden_dir):
    import json, os
    with open(os.path.join(golden_dir, "hand_2group.json")) as f:
        gd = json.load(f)
    w = np.repeat(np.array(gd["w"], dtype=np.float32).reshape(2, 4), 32, axis=1).reshape(1, 256)
    codes, s, z = _quant(tq, w, 128)
    assert to_np(s)[0].tolist() == gd["g128_embedding"]["scales"]
    assert to_np(z)[0].tolist() == gd["g128_embedding"]["zero_counts"]
    c = O.unpack(codes_u32(codes), 256)[0]
    assert c.reshape(2, 4, 32)[:, :, 0].reshape(-1).tolist() == gd["codes"]


def test_quantize_exact_tie_goes_to_zero(tq):
    # |w/s| = 0.5 exactly: round half to even gives 0 (tie reading of §3.1).
    w = np.tile(np.array([0.25, 0.75, 1.0, 0.0], dtype=np.float32), 8).reshape(1, 32)
    w = np.concatenate([w, -w], axis=0)
    codes, s, z = _quant(tq, w, 32)
    assert to_np(s).tolist() == [[0.5], [0.5]]
    c = O.unpack(codes_u32(codes), 32)
    assert c[0, :4].tolist() == [0, 1, 1, 0] and c[1, :4].tolist() == [0, -1, -1, 0]
    assert to_np(z).tolist() == [[16], [16]]


def test_quantize_zero_groups(tq):
    w = synth.latent_weights(4, 512, seed=1)
    w[1] = 0.0
    w[2, 128:256] = 0.0
    codes, s, z = _quant(tq, w, 128)
    check_quantize(w, 128, codes, s, z)
    assert to_np(z)[1].tolist() == [128] * 4 and to_np(s)[1].tolist() == [0.0] * 4


@pytest.mark.parametrize("n,k,g", [
    (512, 256, 128),   # single grouped ternary linear
    (7, 96, 32),       # partial warp unit
    (33, 320, 64),
    (3, 768, 256),     # half of the last unit
    (5, 1536, 512),
    (1, 32, 32),
    (1, 16 * 3 * 32, 32),
])
def test_quantize_shapes(tq, n, k, g):
    w = synth.latent_weights(n, k, seed=n + k + g)
    codes, s, z = _quant(tq, w, g)
    check_quantize(w, g, codes, s, z)


@pytest.mark.parametrize("g", [32, 64, 128, 256, 512])
@pytest.mark.parametrize("dist", ["gauss", "t3"])
def test_quantize_group_sizes(tq, g, dist):
    w = synth.latent_weights(96, 2048, seed=g, dist=dist)
    codes, s, z = _quant(tq, w, g)
    check_quantize(w, g, codes, s, z)


def test_quantize_scaled_values(tq):
    w = synth.latent_weights(64, 1024, seed=9) * np.float32(2.0 ** 20)
    codes, s, z = _quant(tq, w, 128)
    check_quantize(w, 128, codes, s, z)


@pytest.mark.parametrize("proj", ["in_proj", "out_proj"])
@pytest.mark.parametrize("dist", ["gauss", "t3"])
def test_quantize_mamba2_full(tq, proj, dist):
    n, k = synth.MAMBA2_1P3B[proj]
    w = synth.latent_weights(n, k, seed=0, dist=dist)
    codes, s, z = _quant(tq, w, 128)
    flips, ties = check_quantize(w, 128, codes, s, z)
    assert flips <= ties
    ratio = to_np(z).sum() / w.size
    assert (0.30 < ratio < 0.32) if dist == "gauss" else (0.36 < ratio < 0.39)


def _quant_batched(tq, ws, g):
    items = []
    for w_np in ws:
        w = torch.from_numpy(w_np).cuda()
        n, k = w.shape
        items.append((w, torch.empty((n, k // 16), dtype=torch.int32, device="cuda"),
                      torch.empty((n, k // g), device="cuda"),
                      torch.empty((n, k // g), dtype=torch.int32, device="cuda")))
    tq.quantize_batched(items, g)
    tq.device_status()
    return items


@pytest.mark.parametrize("g", [32, 128, 512])
def test_quantize_batched_mixed(tq, g):
    # shapes whose flat sizes end mid-stage, a one-group matrix and an empty one
    shapes = [(7, 1024), (1, g), (300, 512), (0, 1024), (33, 4096), (2, 8192)]
    ws = [synth.latent_weights(n, k, seed=i, dist="t3" if i % 2 else "gauss")
          for i, (n, k) in enumerate(shapes)]
    for w, (_, codes, s, z) in zip(ws, _quant_batched(tq, ws, g)):
        if w.size:
            check_quantize(w, g, codes, s, z)


def test_quantize_batched_matches_single(tq):
    ws = [synth.latent_weights(n, k, seed=40 + i) for i, (n, k) in
          enumerate([(512, 2048), (64, 4096), (96, 256)] * 3)]
    for w, (wt, codes, s, z) in zip(ws, _quant_batched(tq, ws, 64)):
        c1, s1, z1 = tq.quantize(wt, 64)
        tq.device_status()
        assert torch.equal(codes, c1) and torch.equal(s, s1) and torch.equal(z, z1)


def test_quantize_batched_48_layers_sampled(tq):
    # every in_proj and out_proj of the 48 blocks (5 GB of latent weights, drawn
    # on the device) in one launch; 8 rows of each matrix checked
    gen = torch.Generator(device="cuda")
    gen.manual_seed(1234)
    items = []
    for _ in range(48):
        for p in ("in_proj", "out_proj"):
            n, k = synth.MAMBA2_1P3B[p]
            w = torch.randn((n, k), generator=gen, device="cuda") * 0.02
            items.append((w, torch.empty((n, k // 16), dtype=torch.int32, device="cuda"),
                          torch.empty((n, k // 128), device="cuda"),
                          torch.empty((n, k // 128), dtype=torch.int32, device="cuda")))
    tq.quantize_batched(items, 128)
    tq.device_status()
    rs = np.random.default_rng(5)
    for w, codes, s, z in items:
        rows = torch.from_numpy(np.sort(rs.choice(w.shape[0], 8, replace=False))).cuda()
        check_quantize(to_np(w[rows]), 128, codes[rows], s[rows], z[rows])
    del items


# ------------------------------------------------------------------ linear
def _setup(tq, n, k, m, g, seed=0, dy_std=1.0, dist="gauss"):
    w = synth.latent_weights(n, k, seed=seed, dist=dist)
    x = synth.activations_bf16(m, k, seed=seed, stream="x")
    dy = synth.activations_bf16(m, n, seed=seed, std=dy_std, stream="dy")
    codes, s, z = _quant(tq, w, g)
    return w, x, dy, validated_w_hat(w, g, codes, s, z), codes, s


@pytest.mark.parametrize("n,k,m,g", [
    (512, 256, 64, 128),     # single grouped ternary linear (seed 0)
    (200, 192, 300, 64),     # ragged rows, tokens and reduction
    (136, 320, 257, 32),
    (264, 512, 17, 256),     # smallest GEMM token count
    (128, 1024, 256, 512),
    (520, 1024, 1, 128),     # decode
    (520, 1024, 3, 128),
    (520, 1024, 16, 128),
    (40, 64, 5, 32),         # one k-block
    (200, 64, 300, 64),      # 256-token tiles, one forward k-block, two dX k-blocks
    (104, 256, 400, 128),    # 256-token tiles, one dX k-block, a second half of 144 tokens
])
def test_linear_parity(tq, n, k, m, g):
    w, x, dy, w_hat, codes, s = _setup(tq, n, k, m, g, seed=n + k + m)
    xd, dyd = x.cuda(), dy.cuda()
    y = tq.linear_fwd(xd, codes, s, g)
    dx, dw = tq.linear_bwd(dyd, xd, codes, s, k, g)
    ct = tq.codes_transpose(codes, k)
    dxt, _ = tq.linear_bwd(dyd, xd, codes, s, k, g, want_dw=False, codes_t=ct)
    tq.device_status()
    check_close(y, O.linear_fwd(x, w_hat), "Y")
    check_close(dx, O.linear_bwd_dx(dy, w_hat), "dX")
    check_close(dxt, O.linear_bwd_dx(dy, w_hat), "dX (codes_t)")
    check_close(dw, O.linear_bwd_dw(dy, x), "dW")


@pytest.mark.parametrize("n,k", [(200, 192), (64, 64), (17, 16), (130, 528), (520, 1024),
                                 (1000, 2048), (2048, 4096), (8512, 2048)])
def test_codes_transpose_layout(tq, n, k):
    """tq_codes_transpose against the oracle's packing of the transposed codes; the
    output starts as all ones, so the zero padding past n is written, not assumed."""
    rs = np.random.default_rng(n + k)
    c = rs.choice(np.array([-1, 0, 1], dtype=np.int8), size=(n, k))
    codes = torch.from_numpy(O.pack(c).view(np.int32)).cuda()
    ct = torch.full((k, 4 * ((n + 63) // 64)), -1, dtype=torch.int32, device="cuda")
    tq.codes_transpose(codes, k, out=ct)
    tq.device_status()
    npad = 64 * ((n + 63) // 64)
    cpad = np.zeros((k, npad), dtype=np.int8)
    cpad[:, :n] = c.T
    assert np.array_equal(codes_u32(ct), O.pack(cpad))


def test_linear_bf16_outputs_are_rounded_fp32(tq):
    n, k, m, g = 264, 512, 300, 128
    w, x, dy, w_hat, codes, s = _setup(tq, n, k, m, g, seed=3)
    xd, dyd = x.cuda(), dy.cuda()
    y32 = tq.linear_fwd(xd, codes, s, g)
    y16 = tq.linear_fwd(xd, codes, s, g, out_dtype=torch.bfloat16)
    dx32, _ = tq.linear_bwd(dyd, xd, codes, s, k, g, want_dw=False)
    dx16, _ = tq.linear_bwd(dyd, xd, codes, s, k, g, want_dw=False, dx_dtype=torch.bfloat16)
    tq.device_status()
    assert torch.equal(y16, y32.to(torch.bfloat16))
    assert torch.equal(dx16, dx32.to(torch.bfloat16))
    check_close(y16, O.linear_fwd(x, w_hat), "Y bf16", max_rel_rms=3e-2)


def test_dw_accumulate_and_single_outputs(tq):
    n, k, m, g = 136, 256, 200, 64
    w, x, dy, w_hat, codes, s = _setup(tq, n, k, m, g, seed=4)
    xd, dyd = x.cuda(), dy.cuda()
    base = torch.randn(n, k, device="cuda", dtype=torch.float32)
    base_np = to_np(base).astype(np.float64)
    dw = base.clone()
    dx, dw = tq.linear_bwd(dyd, xd, codes, s, k, g, want_dx=False, dw=dw, accumulate_dw=True)
    assert dx is None
    dx2, dw2 = tq.linear_bwd(dyd, None, codes, s, k, g, want_dw=False)
    tq.device_status()
    assert dw2 is None
    check_close(to_np(dw) - base_np, O.linear_bwd_dw(dy, x), "dW accumulated")
    check_close(dx2, O.linear_bwd_dx(dy, w_hat), "dX only")


@pytest.mark.parametrize("m", [64, 1999, 2000])
@pytest.mark.parametrize("accumulate", [False, True])
def test_dw_stream_k_tail(tq, m, accumulate):
    """dW over more 256 x 256 pair tiles than CTA pairs (5 x 17 = 85 tiles on the 76
    pairs of 152 SMs): the 9 tiles past the whole wave are cut into equal runs of
    128-token k-blocks, one run per pair, and each CTA's half of a tile is summed in
    k order by the CTA that completes it. m = 64 leaves fewer tail k-blocks than
    pairs (every tile whole); m = 2000 (16 k-blocks) cuts every tail tile into 8 or
    9 pieces; m = 1999 does the same ending on a ragged k-block
    (tests/test_dw_schedule.py checks these counts on the host). Full comparison
    with the oracle."""
    n, k, g = 4160, 1280, 128
    w, x, dy, w_hat, codes, s = _setup(tq, n, k, m, g, seed=11, dy_std=1e-2)
    xd, dyd = x.cuda(), dy.cuda()
    base = torch.randn(n, k, device="cuda", dtype=torch.float32) if accumulate else None
    dw = base.clone() if accumulate else None
    for _ in range(2):  # the second launch reuses the reset tail counters
        out = base.clone() if accumulate else dw
        _, dw = tq.linear_bwd(dyd, xd, codes, s, k, g, want_dx=False, dw=out,
                              accumulate_dw=accumulate)
        tq.device_status()
        got = to_np(dw).astype(np.float64) - (to_np(base).astype(np.float64) if accumulate else 0)
        check_close(got, O.linear_bwd_dw(dy, x), f"dW m={m} accumulate={accumulate}")


def test_empty_sizes(tq):
    codes = torch.zeros((64, 256 // 16), dtype=torch.int32, device="cuda")
    s = torch.zeros((64, 2), dtype=torch.float32, device="cuda")
    x = torch.zeros((0, 256), dtype=torch.bfloat16, device="cuda")
    y = tq.linear_fwd(x, codes, s, 128)
    assert y.shape == (0, 64)
    dy = torch.zeros((0, 64), dtype=torch.bfloat16, device="cuda")
    dw = torch.full((64, 256), 7.0, device="cuda")
    tq.linear_bwd(dy, x, codes, s, 256, 128, want_dx=False, dw=dw)
    tq.device_status()
    assert float(dw.abs().max()) == 0.0   # M = 0: dW = empty sum = 0


@pytest.mark.parametrize("g", [32, 64, 128, 256, 512])
@pytest.mark.parametrize("m", [1, 5, 8, 9, 16])
def test_decode_parity(tq, g, m):
    """Few-token forward (decode kernel): ragged rows (200 = 12.5 units of 16)."""
    n, k = 200, 1024
    w, x, dy, w_hat, codes, s = _setup(tq, n, k, m, g, seed=g + m)
    y = tq.linear_fwd(x.cuda(), codes, s, g)
    yb = tq.linear_fwd(x.cuda(), codes, s, g, out_dtype=torch.bfloat16)
    tq.device_status()
    ref = O.linear_fwd(x, w_hat)
    check_close(y, ref, "Y decode")
    assert torch.equal(yb, y.to(torch.bfloat16))


@pytest.mark.parametrize("m", [1, 2, 3, 4, 6, 7])
@pytest.mark.parametrize("g", [128, 256, 512])
def test_decode_activation_ranges(tq, m, g):
    """Few-token forward with activations over most of the bf16 range: every token
    scaled by its own power of two from 2^-100 to 2^100, one 128-wide chunk all
    zero, one chunk spanning 2^-30 .. 2^8 inside itself; each token compared on its
    own (the oracle's output of that token alone), so that a small token is not
    hidden by a large one."""
    n, k = 264, 1536
    w, x, dy, w_hat, codes, s = _setup(tq, n, k, m, g, seed=700 + m + g)
    rs = np.random.default_rng(m * 1000 + g)
    xf = x.float().numpy().copy()
    for tok in range(m):
        e = rs.integers(-100, 101)
        xf[tok] *= np.float32(2.0 ** float(e))
    xf[0, 128:256] = 0.0                                         # a zero chunk
    xf[m - 1, 256:384] = (rs.choice([-1, 1], 128) *
                          2.0 ** rs.uniform(-30, 8, 128)).astype(np.float32)
    xb = torch.from_numpy(xf).to(torch.bfloat16)
    y = tq.linear_fwd(xb.cuda(), codes, s, g)
    tq.device_status()
    ref = O.linear_fwd(xb, w_hat)
    for tok in range(m):
        check_close(to_np(y[tok:tok + 1]), ref[tok:tok + 1], f"Y token {tok} m={m} g={g}")


def test_decode_token_chunk_scales_independent(tq):
    """Tokens at scales 2^-120 and 2^120 in one launch, and one token whose first half
    is 2^60 times its second: each within the parity bars of its own output."""
    n, k, g = 136, 1024, 128
    w, x, dy, w_hat, codes, s = _setup(tq, n, k, 4, g, seed=77)
    xf = x.float().numpy().copy()
    xf[0] *= np.float32(2.0 ** -120)
    xf[1] *= np.float32(2.0 ** 120)
    xf[2, :512] *= np.float32(2.0 ** 60)
    xb = torch.from_numpy(xf).to(torch.bfloat16)
    y = tq.linear_fwd(xb.cuda(), codes, s, g)
    tq.device_status()
    ref = O.linear_fwd(xb, w_hat)
    for tok in range(4):
        check_close(to_np(y[tok:tok + 1]), ref[tok:tok + 1], f"Y token {tok}")


def test_batched_decode_mixed(tq):
    """One launch over matrices with different shapes, group sizes and output types."""
    specs = [(520, 256, 128, torch.float32), (264, 512, 32, torch.bfloat16),
             (8, 64, 64, torch.float32), (136, 1024, 512, torch.float32)]
    items = []
    for i, (n, k, g, dt) in enumerate(specs):
        w = synth.latent_weights(n, k, seed=200 + i)
        x = synth.activations_bf16(11, k, seed=200 + i)
        codes, s, z = _quant(tq, w, g)
        items.append(dict(x=x.cuda(), codes=codes, scales=s, g=g,
                          y=torch.empty((11, n), device="cuda", dtype=dt),
                          ref=O.linear_fwd(x, validated_w_hat(w, g, codes, s, z))))
    tq.linear_fwd_batched(items, 11)
    tq.device_status()
    for i, it in enumerate(items):
        check_close(it["y"].float(), it["ref"], f"batched Y[{i}]",
                    max_rel_rms=3e-2 if it["y"].dtype == torch.bfloat16 else 2e-2)


def test_batched_decode_matches_single(tq):
    mats = []
    for i, (n, k) in enumerate([(520, 256), (256, 512), (520, 256), (136, 1024)]):
        w = synth.latent_weights(n, k, seed=100 + i)
        x = synth.activations_bf16(4, k, seed=100 + i)
        codes, s, z = _quant(tq, w, 128)
        w_hat = validated_w_hat(w, 128, codes, s, z)
        mats.append(dict(x=x.cuda(), codes=codes, scales=s, g=128,
                         y=torch.empty((4, n), device="cuda"), ref=O.linear_fwd(x, w_hat)))
    tq.linear_fwd_batched(mats, 4)
    tq.device_status()
    for i, it in enumerate(mats):
        check_close(it["y"], it["ref"], f"batched Y[{i}]")


# ------------------------------------------------------------------ full size
@pytest.mark.parametrize("proj", ["in_proj", "out_proj"])
def test_linear_mamba2_prefill_sampled(tq, proj):
    """Full Mamba-2 1.3B projection at batch 8 x seq 2048, checked on sampled rows."""
    n, k = synth.MAMBA2_1P3B[proj]
    m, g = 16384, 128
    w, x, dy, w_hat, codes, s = _setup(tq, n, k, m, g, seed=0, dy_std=1e-2)
    xd, dyd = x.cuda(), dy.cuda()
    y = tq.linear_fwd(xd, codes, s, g)
    dx, dw = tq.linear_bwd(dyd, xd, codes, s, k, g)
    ct = tq.codes_transpose(codes, k)
    dxt, _ = tq.linear_bwd(dyd, xd, codes, s, k, g, want_dw=False, codes_t=ct)
    tq.device_status()
    assert torch.equal(dxt, dx)  # same operands, same MMA order
    rs = np.random.default_rng(1)
    rows = np.sort(rs.choice(m, 64, replace=False))
    nrows = np.sort(rs.choice(n, 64, replace=False))
    check_close(to_np(y[torch.from_numpy(rows).cuda()]), O.linear_fwd(x, w_hat, rows), "Y rows")
    check_close(to_np(dx[torch.from_numpy(rows).cuda()]), O.linear_bwd_dx(dy, w_hat, rows),
                "dX rows")
    check_close(to_np(dw[torch.from_numpy(nrows).cuda()]), O.linear_bwd_dw(dy, x, nrows),
                "dW rows")
    # every output finite, and the sampled tail rows of the ragged N tile too
    assert torch.isfinite(y).all() and torch.isfinite(dx).all() and torch.isfinite(dw).all()
    tail = np.arange(n - 8, n)
    check_close(to_np(dw[torch.from_numpy(tail).cuda()]), O.linear_bwd_dw(dy, x, tail), "dW tail")


# ------------------------------------------------------------------ the g sweep at full size
_SWEEP = {}


def _sweep_inputs(proj, dist):
    """W of the projection's shape (per distribution) and one X / dY per projection,
    shared by the sweep's group sizes."""
    n, k = synth.MAMBA2_1P3B[proj]
    if (proj, "xdy") not in _SWEEP:
        _SWEEP.clear()  # one projection's inputs at a time (the host arrays are large)
        x = synth.activations_bf16(16384, k, seed=5, stream="x")
        dy = synth.activations_bf16(16384, n, seed=5, std=1e-2, stream="dy")
        _SWEEP[(proj, "xdy")] = (x, dy, x.cuda(), dy.cuda())
    if (proj, dist) not in _SWEEP:
        _SWEEP[(proj, dist)] = synth.latent_weights(n, k, seed=5, dist=dist)
    return (_SWEEP[(proj, dist)],) + _SWEEP[(proj, "xdy")]


@pytest.mark.parametrize("dist", ["gauss", "t3"])
@pytest.mark.parametrize("g", [32, 64, 128, 256, 512])
@pytest.mark.parametrize("proj", ["in_proj", "out_proj"])
def test_prefill_sweep_all_group_sizes(tq, proj, g, dist):
    """One full projection step (quantize, Y, dX on the transposed codes, dW) at
    M = 16384 for each projection, group size and weight distribution; outputs
    checked on sampled rows, every group's code and scale checked in full."""
    w, x, dy, xd, dyd = _sweep_inputs(proj, dist)
    n, k = w.shape
    ref = O.quantize(w, g)
    codes, s, z = _quant(tq, w, g)
    flips, ties = check_quantize(w, g, codes, s, z, ref=ref)
    assert flips <= ties
    w_hat = O.dequantize(codes_u32(codes), ref[1], k, g)  # the GPU codes, checked above
    y = tq.linear_fwd(xd, codes, s, g)
    ct = tq.codes_transpose(codes, k)
    dx, dw = tq.linear_bwd(dyd, xd, codes, s, k, g, codes_t=ct)
    tq.device_status()
    rs = np.random.default_rng(g)
    rows = np.sort(rs.choice(16384, 32, replace=False))
    nrows = np.sort(rs.choice(n, 32, replace=False))
    sel = torch.from_numpy(rows).cuda()
    check_close(to_np(y[sel]), O.linear_fwd(x, w_hat, rows), f"Y rows {proj} g={g} {dist}")
    check_close(to_np(dx[sel]), O.linear_bwd_dx(dy, w_hat, rows), f"dX rows {proj} g={g} {dist}")
    check_close(to_np(dw[torch.from_numpy(nrows).cuda()]), O.linear_bwd_dw(dy, x, nrows),
                f"dW rows {proj} g={g} {dist}")


# ------------------------------------------------------------------ extreme shapes
@pytest.mark.parametrize("m", [1, 5, 12])
def test_decode_long_reduction(tq, m):
    """Decode over a 16384-long reduction: 32 segments per 256-row unit, a ragged
    last unit of 44 rows."""
    n, k, g = 300, 16384, 128
    w, x, dy, w_hat, codes, s = _setup(tq, n, k, m, g, seed=51)
    y = tq.linear_fwd(x.cuda(), codes, s, g)
    tq.device_status()
    check_close(to_np(y), O.linear_fwd(x, w_hat), f"Y m={m} k={k}")


# k/g > 32 with k/g % 4 == 0: the scales arrive in windows of 32 groups of all the
# unit's rows (256 x 128 bytes, swizzled); each k ends inside a window (a partial last
# window whose groups past k/g read as zero).
_WINDOW_K = {32: 1664, 64: 2816, 128: 4608, 256: 9216, 512: 18432}  # k/g = 52, 44, 36, 36, 36


@pytest.mark.parametrize("g", [32, 64, 128, 256, 512])
@pytest.mark.parametrize("m", [1, 8, 9, 16])
def test_decode_scale_windows(tq, g, m):
    """Decode with the group scales in windows: every g, one to sixteen tokens, a
    ragged last unit (300 rows = 256 + 44)."""
    n, k = 300, _WINDOW_K[g]
    w, x, dy, w_hat, codes, s = _setup(tq, n, k, m, g, seed=900 + g + m)
    y = tq.linear_fwd(x.cuda(), codes, s, g)
    tq.device_status()
    check_close(to_np(y), O.linear_fwd(x, w_hat), f"Y windows g={g} m={m}")


def test_batched_decode_scale_modes_past_the_map_limit(tq):
    """One call over 70 window-mode matrices (two tensor maps each: more than one
    launch holds, so the call splits) mixed with unit-mode (k/g <= 32) and 4-byte-mode
    (k/g % 4 != 0) matrices, fp32 and bf16 outputs."""
    g, m = 128, 3
    specs = [(16 + 8 * (i % 5), 4608 if i % 2 else 8192) for i in range(70)]
    specs[10:10] = [(264, 1024), (40, 1152)]    # unit mode (k/g 8), 4-byte mode (k/g 9)
    specs.append((520, 640))                    # 4-byte mode (k/g 5)
    items = []
    for i, (n, k) in enumerate(specs):
        w = synth.latent_weights(n, k, seed=3000 + i)
        x = synth.activations_bf16(m, k, seed=3000 + i)
        codes, s, z = _quant(tq, w, g)
        dt = torch.bfloat16 if i % 3 == 0 else torch.float32
        items.append(dict(x=x.cuda(), codes=codes, scales=s, g=g,
                          y=torch.empty((m, n), device="cuda", dtype=dt),
                          ref=O.linear_fwd(x, validated_w_hat(w, g, codes, s, z))))
    tq.linear_fwd_batched(items, m)
    tq.device_status()
    for i, it in enumerate(items):
        check_close(it["y"].float(), it["ref"], f"batched Y[{i}] {specs[i]}",
                    max_rel_rms=3e-2 if it["y"].dtype == torch.bfloat16 else 2e-2)


# A launch with fewer 256-row blocks than SMs cuts k into P pieces (clusters of P
# CTAs, the first adding the others' partial sums): one matrix per call here, each
# scale mode, ragged k and rows, pieces that end inside a window of scales.
_SPLIT_SHAPES = [
    (8512, 2048, 128),   # Mamba-2 1.3B in_proj: 34 blocks, unit scales
    (2048, 4096, 128),   # out_proj: 8 blocks
    (520, 1088, 64),     # k/g = 17: per-segment scales; 3 segments, the last ragged
    (264, 4608, 128),    # k/g = 36: scale windows cut by the pieces
    (300, 18432, 512),   # k/g = 36 at g = 512, 36 segments
    (136, 2560, 32),     # k/g = 80 windows of 32 groups at g = 32
]


@pytest.mark.parametrize("n,k,g", _SPLIT_SHAPES)
@pytest.mark.parametrize("m", [1, 5, 8, 9, 16])
def test_decode_pieces_of_k(tq, n, k, g, m):
    w, x, dy, w_hat, codes, s = _setup(tq, n, k, m, g, seed=n + k + m)
    xd = x.cuda()
    y = tq.linear_fwd(xd, codes, s, g)
    yb = tq.linear_fwd(xd, codes, s, g, out_dtype=torch.bfloat16)
    y2 = tq.linear_fwd(xd, codes, s, g)
    tq.device_status()
    check_close(to_np(y), O.linear_fwd(x, w_hat), f"Y pieces n={n} k={k} g={g} m={m}")
    assert torch.equal(y, y2)                      # the same sums in the same order
    assert torch.equal(yb, y.to(torch.bfloat16))


def test_decode_persistent_160_blocks(tq):
    """A batch of 160 blocks of rows (no pieces: a persistent grid claiming units),
    compared in full."""
    g, m = 128, 6
    items = []
    for i in range(40):
        n, k = 1024 - 8 * (i % 3), 1024 + 512 * (i % 2)
        w = synth.latent_weights(n, k, seed=5000 + i)
        x = synth.activations_bf16(m, k, seed=5000 + i)
        codes, s, z = _quant(tq, w, g)
        items.append(dict(x=x.cuda(), codes=codes, scales=s, g=g,
                          y=torch.empty((m, n), device="cuda"),
                          ref=O.linear_fwd(x, validated_w_hat(w, g, codes, s, z))))
    tq.linear_fwd_batched(items, m)
    tq.device_status()
    for i, it in enumerate(items):
        check_close(it["y"], it["ref"], f"persistent Y[{i}]")


def test_prefill_few_rows_many_tokens(tq):
    """64 weight rows (half a tile) against 40000 tokens (157 token tiles with a
    ragged last one), all three products."""
    n, k, m, g = 64, 512, 40000, 64
    w, x, dy, w_hat, codes, s = _setup(tq, n, k, m, g, seed=52, dy_std=1e-2)
    xd, dyd = x.cuda(), dy.cuda()
    y = tq.linear_fwd(xd, codes, s, g)
    dx, dw = tq.linear_bwd(dyd, xd, codes, s, k, g, codes_t=tq.codes_transpose(codes, k))
    tq.device_status()
    rows = np.sort(np.random.default_rng(52).choice(m, 256, replace=False))
    sel = torch.from_numpy(rows).cuda()
    check_close(to_np(y[sel]), O.linear_fwd(x, w_hat, rows), "Y rows")
    check_close(to_np(dx[sel]), O.linear_bwd_dx(dy, w_hat, rows), "dX rows")
    check_close(to_np(dw), O.linear_bwd_dw(dy, x), "dW (40000-token reduction)")


def test_dw_long_token_reduction(tq):
    """dW over 131072 tokens (2048 k-blocks per tile, fewer tiles than SMs)."""
    n, k, m, g = 256, 384, 131072, 128
    w, x, dy, w_hat, codes, s = _setup(tq, n, k, m, g, seed=53, dy_std=1e-2)
    _, dw = tq.linear_bwd(dy.cuda(), x.cuda(), codes, s, k, g, want_dx=False)
    tq.device_status()
    check_close(to_np(dw), O.linear_bwd_dw(dy, x), "dW (131072 tokens)")
