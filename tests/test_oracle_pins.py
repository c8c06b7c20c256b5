"""Pins of the oracle against what the paper and the mathematics fix (no GPU).

Each test ties ``oracle.tq_oracle`` to something other than itself: a
hand-worked example (§3.1), the tie and zero-scale readings, invariants of the
quantiser, closed-form zero ratios, an independent pure-Python brute force, and
special cases that reduce to a dense matmul. ``test_planted_*`` check that a
plausible mistake in the oracle would be caught by these pins.
"""
import json
import math
import os

import numpy as np
import pytest
import torch

import brute
from oracle import tq_oracle as O
from paper_2606_18114_gb300 import synth

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")


def _load(golden_dir, name):
    with open(os.path.join(golden_dir, name)) as f:
        return json.load(f)


# ---------------------------------------------------------------- hand example
def test_hand_example_quantize(golden_dir):
    gd = _load(golden_dir, "hand_2group.json")
    w = np.array([gd["w"]], dtype=np.float32)
    pad = np.zeros((1, 8), dtype=np.float32)  # K must be a multiple of 16
    w16 = np.concatenate([w, pad], axis=1)
    codes, s, z, c = O.quantize(w16, gd["g"])
    assert s[0, :2].tolist() == gd["scales"]
    assert c[0, :8].tolist() == gd["codes"]
    assert z[0, :2].tolist() == gd["zero_counts"]
    # the padded all-zero groups: s = 0, every code 0, zero count = g
    assert s[0, 2:].tolist() == [0.0, 0.0]
    assert z[0, 2:].tolist() == [4, 4]
    w_hat = O.dequantize(codes, s, 16, gd["g"])
    assert w_hat[0, :8].tolist() == gd["w_hat"]


def test_hand_example_linear(golden_dir):
    gd = _load(golden_dir, "hand_2group.json")
    w = np.zeros((1, 16), dtype=np.float32)
    w[0, :8] = gd["w"]
    codes, s, z, _ = O.quantize(w, gd["g"])
    w_hat = O.dequantize(codes, s, 16, gd["g"])
    x = np.zeros((1, 16))
    x[0, :8] = gd["x"]
    y = O.linear_fwd(x, w_hat)
    assert y.shape == (1, 1) and y[0, 0] == gd["y"]
    dy = np.array([gd["dy"]])
    assert O.linear_bwd_dx(dy, w_hat)[0, :8].tolist() == gd["dx"]
    assert O.linear_bwd_dw(dy, x)[0, :8].tolist() == gd["dw"]


def test_hand_example_g128_embedding(golden_dir):
    gd = _load(golden_dir, "hand_2group.json")
    w = np.repeat(np.array(gd["w"], dtype=np.float32).reshape(2, 4), 32, axis=1).reshape(1, 256)
    codes, s, z, c = O.quantize(w, 128)
    assert s[0].tolist() == gd["g128_embedding"]["scales"]
    assert z[0].tolist() == gd["g128_embedding"]["zero_counts"]


def test_hand_example_packed_word(golden_dir):
    gd = _load(golden_dir, "hand_2group.json")["packed_k16"]
    c = np.array([gd["codes"]], dtype=np.int8)
    assert int(O.pack(c)[0, 0]) == gd["word"]
    assert O.unpack(np.array([[gd["word"]]], dtype=np.uint32), 16)[0].tolist() == gd["codes"]


def test_tie_group_half_even(golden_dir):
    gd = _load(golden_dir, "tie_group.json")
    w = np.zeros((1, 16), dtype=np.float32)
    w[0, :4] = gd["w"]
    _, s, z, c = O.quantize(w, gd["g"])
    assert s[0, 0] == gd["scales"][0]
    assert c[0, :4].tolist() == gd["codes"]
    assert z[0, 0] == gd["zero_counts"][0]


def test_negative_tie_and_signed_zero():
    # w/s = -0.5 exactly: half-even gives -0, which is code 0.
    w = np.zeros((1, 16), dtype=np.float32)
    w[0, :4] = [-0.25, 0.75, -1.0, 0.0]
    _, s, _, c = O.quantize(w, 4)
    assert s[0, 0] == 0.5
    assert c[0, :4].tolist() == [0, 1, -1, 0]


def test_unpack_rejects_invalid_code():
    with pytest.raises(ValueError):
        O.unpack(np.array([[0b10]], dtype=np.uint32), 16)


# ---------------------------------------------------------------- invariants
@pytest.mark.parametrize("g", [32, 64, 128, 256, 512])
@pytest.mark.parametrize("dist", ["gauss", "t3"])
def test_invariants(g, dist):
    w = synth.latent_weights(64, 1024, seed=3, dist=dist)
    codes, s, z, c = O.quantize(w, g)
    assert set(np.unique(c).tolist()) <= {-1, 0, 1}
    # s = mean |w| (math.fsum per group, independent of numpy's sum)
    for n in (0, 17, 63):
        for j in range(1024 // g):
            ref = math.fsum(abs(float(v)) for v in w[n, j * g:(j + 1) * g]) / g
            assert abs(float(s[n, j]) - ref) <= 1e-7 * ref
    # zero count = number of zero codes
    assert np.array_equal(z, (c.reshape(64, -1, g) == 0).sum(axis=2))
    # round trip of the packing
    assert np.array_equal(O.unpack(codes, 1024), c)
    # reconstruction: |w - w^| <= s/2 wherever |w| <= 1.5 s
    w_hat = O.dequantize(codes, s, 1024, g)
    srep = np.repeat(s.astype(np.float64), g, axis=1)
    inside = np.abs(w) <= 1.5 * srep
    err = np.abs(w.astype(np.float64) - w_hat)
    assert np.all(err[inside] <= 0.5 * srep[inside] * (1 + 1e-6))
    # outside that band every code is the sign of w (saturated)
    assert np.all(c[~inside] == np.sign(w[~inside]))
    # codes are odd in w: quantising -w flips every code, keeps s and z
    codes_n, s_n, z_n, c_n = O.quantize(-w, g)
    assert np.array_equal(s_n, s) and np.array_equal(z_n, z) and np.array_equal(c_n, -c)


def test_scale_invariance_powers_of_two():
    # Multiplying W by a power of two scales s exactly and leaves codes alone.
    w = synth.latent_weights(16, 256, seed=5)
    _, s1, z1, c1 = O.quantize(w, 128)
    _, s2, z2, c2 = O.quantize(w * np.float32(8.0), 128)
    assert np.array_equal(s2, s1 * np.float32(8.0))
    assert np.array_equal(c1, c2) and np.array_equal(z1, z2)


def test_zero_group_and_constant_magnitude():
    w = np.zeros((2, 32), dtype=np.float32)
    w[1, :16] = np.float32(0.3) * np.sign(np.arange(16) % 3 - 1 + 0.5).astype(np.float32)
    codes, s, z, c = O.quantize(w, 16)
    assert s[0].tolist() == [0.0, 0.0] and z[0].tolist() == [16, 16]
    # equal magnitudes: every code is the sign, and w^ == w exactly
    assert np.all(c[1, :16] == np.sign(w[1, :16]))
    assert np.array_equal(O.dequantize(codes, s, 32, 16)[1, :16], w[1, :16].astype(np.float64))


# ---------------------------------------------------------------- closed forms
def test_zero_ratio_gaussian_closed_form():
    # For w ~ N(0, sigma^2) and s -> E|w| = sigma*sqrt(2/pi) (large g),
    # P(code = 0) = P(|Z| <= 0.5*sqrt(2/pi)) = 2*Phi(0.5*sqrt(2/pi)) - 1 = 0.3101.
    from scipy.stats import norm
    p = 2 * norm.cdf(0.5 * math.sqrt(2 / math.pi)) - 1
    assert abs(p - 0.3101) < 1e-4
    w = synth.latent_weights(512, 4096, seed=11)
    _, _, z, _ = O.quantize(w, 512)
    ratio = z.sum() / w.size
    assert abs(ratio - p) < 3e-3, ratio


def test_zero_ratio_t3_closed_form():
    # Student-t(3): E|T| = 2*sqrt(3)/pi, P(|T| <= 0.5*E|T|) from its CDF (~0.380).
    from scipy.stats import t as student_t
    e_abs = 2 * math.sqrt(3) / math.pi
    p = 2 * student_t.cdf(0.5 * e_abs, 3) - 1
    assert abs(p - 0.380) < 2e-3
    w = synth.latent_weights(512, 4096, seed=12, dist="t3")
    _, _, z, _ = O.quantize(w, 512)
    ratio = z.sum() / w.size
    # finite-group bias: the sample mean of a heavy-tailed group is below E|T|
    # more often than above, so the measured ratio sits slightly under p.
    assert p - 1.5e-2 < ratio < p + 3e-3, ratio


# ---------------------------------------------------------------- brute force
@pytest.mark.parametrize("shape", [(3, 32, 5, 8), (5, 16, 4, 16), (2, 48, 7, 16), (1, 64, 3, 32)])
def test_brute_force_tiny(shape):
    n, k, m, g = shape
    rs = np.random.default_rng(sum(shape))
    w = rs.standard_normal((n, k)).astype(np.float32) * np.float32(0.02)
    x = torch.from_numpy(rs.standard_normal((m, k)).astype(np.float32)).to(torch.bfloat16)
    dy = torch.from_numpy(rs.standard_normal((m, n)).astype(np.float32)).to(torch.bfloat16)
    codes, s, z, c = O.quantize(w, g)
    assert not O.near_tie_mask(w, s, g, 1e-4).any()

    wl = [[float(v) for v in row] for row in w]
    bc, bs, bz = brute.quantize_rows(wl, g)
    assert c.tolist() == bc
    assert z.tolist() == bz
    assert np.allclose(s, np.array(bs), rtol=1e-7, atol=0)
    assert [row.tolist() for row in codes] == [brute.pack_row(r) for r in bc]

    w_hat = O.dequantize(codes, s, k, g)
    bw = brute.dequant_rows(bc, [[float(v) for v in row] for row in s], g)
    xl = x.float().tolist()
    dyl = dy.float().tolist()
    y_b = np.array(brute.matmul_nt(xl, bw))
    dx_b = np.array(brute.matmul_nn(dyl, bw))
    dw_b = np.array(brute.matmul_nn(brute.transpose(dyl), xl))
    assert np.allclose(O.linear_fwd(x, w_hat), y_b, rtol=1e-12, atol=1e-14)
    assert np.allclose(O.linear_bwd_dx(dy, w_hat), dx_b, rtol=1e-12, atol=1e-14)
    assert np.allclose(O.linear_bwd_dw(dy, x), dw_b, rtol=1e-12, atol=1e-14)
    # shapes catch a transposed operand
    assert O.linear_fwd(x, w_hat).shape == (m, n)
    assert O.linear_bwd_dx(dy, w_hat).shape == (m, k)
    assert O.linear_bwd_dw(dy, x).shape == (n, k)


def test_row_selection_matches_full():
    w = synth.latent_weights(40, 128, seed=2)
    x = synth.activations_bf16(24, 128, seed=2)
    dy = synth.activations_bf16(24, 40, seed=2, stream="dy")
    codes, s, _, _ = O.quantize(w, 32)
    w_hat = O.dequantize(codes, s, 128, 32)
    rows = [0, 5, 23]
    assert np.array_equal(O.linear_fwd(x, w_hat, rows), O.linear_fwd(x, w_hat)[rows])
    assert np.array_equal(O.linear_bwd_dx(dy, w_hat, rows), O.linear_bwd_dx(dy, w_hat)[rows])
    assert np.allclose(O.linear_bwd_dw(dy, x, [1, 39]), O.linear_bwd_dw(dy, x)[[1, 39]], rtol=1e-14)


def test_equal_magnitude_reduces_to_dense_matmul():
    # Groups whose elements all share one magnitude are reproduced exactly
    # (w^ = w), so Y and dX equal a dense fp64 matmul with the latent W.
    rs = np.random.default_rng(7)
    mags = rs.uniform(0.01, 0.03, size=(24, 4)).astype(np.float32)
    signs = rs.choice([-1.0, 1.0], size=(24, 128)).astype(np.float32)
    w = (np.repeat(mags, 32, axis=1) * signs).astype(np.float32)
    x = synth.activations_bf16(16, 128, seed=4)
    dy = synth.activations_bf16(16, 24, seed=4, stream="dy")
    codes, s, z, _ = O.quantize(w, 32)
    assert np.all(z == 0)
    w_hat = O.dequantize(codes, s, 128, 32)
    assert np.array_equal(w_hat, w.astype(np.float64))
    xd, dyd = x.double().numpy(), dy.double().numpy()
    assert np.allclose(O.linear_fwd(x, w_hat), np.matmul(xd, w.astype(np.float64).T), rtol=1e-13)
    assert np.allclose(O.linear_bwd_dx(dy, w_hat), np.matmul(dyd, w.astype(np.float64)), rtol=1e-13)


# ---------------------------------------------------------------- planted mistakes
def _pins_hold(quantize_fn, golden_dir):
    """Run the hand-example and tie pins against a (possibly broken) quantiser."""
    gd = _load(golden_dir, "hand_2group.json")
    tie = _load(golden_dir, "tie_group.json")
    w = np.zeros((1, 16), dtype=np.float32)
    w[0, :8] = gd["w"]
    _, s, z, c = quantize_fn(w, 4)
    ok = s[0, :2].tolist() == gd["scales"] and c[0, :8].tolist() == gd["codes"] \
        and z[0, :2].tolist() == gd["zero_counts"]
    w = np.zeros((1, 16), dtype=np.float32)
    w[0, :4] = tie["w"]
    _, s, z, c = quantize_fn(w, 4)
    return ok and c[0, :4].tolist() == tie["codes"]


def _broken_quantize(kind):
    def q(w, g):
        n, k = w.shape
        wg = w.reshape(n, k // g, g).astype(np.float64)
        if kind == "no_abs":
            s64 = wg.sum(axis=2) / g
        elif kind == "max_not_mean":
            s64 = np.abs(wg).max(axis=2)
        else:
            s64 = np.abs(wg).sum(axis=2) / g
        s32 = s64.astype(np.float32)
        with np.errstate(invalid="ignore", divide="ignore"):
            qv = w.reshape(n, k // g, g) / s32[:, :, None]
        if kind == "half_away":
            c = np.sign(qv) * np.floor(np.abs(np.clip(qv, -1, 1)) + 0.5)
        else:
            c = np.rint(np.clip(qv, -1, 1))
        c = np.nan_to_num(c).astype(np.int8).reshape(n, k)
        z = (c.reshape(n, k // g, g) == 0).sum(axis=2)
        return None, s32, z, c
    return q


@pytest.mark.parametrize("kind", ["no_abs", "max_not_mean", "half_away"])
def test_planted_quantizer_mistakes_are_caught(kind, golden_dir):
    assert _pins_hold(_broken_quantize("none"), golden_dir)
    assert not _pins_hold(_broken_quantize(kind), golden_dir)


def test_planted_layout_mistake_is_caught(golden_dir):
    gd = _load(golden_dir, "hand_2group.json")["packed_k16"]
    c = np.array([gd["codes"]], dtype=np.int8)
    # consecutive 2-bit fields (a natural but different layout) give another word
    v = np.array([O.ENCODE[int(x)] for x in gd["codes"]], dtype=np.uint64)
    naive = int(np.bitwise_or.reduce(v << (2 * np.arange(16, dtype=np.uint64))))
    assert naive != gd["word"] and int(O.pack(c)[0, 0]) == gd["word"]
