"""Bounded waits that run out (needs a GB300).

The failure is made on purpose without faulting, trapping or hanging anything:
a test-only flag makes one kernel role withhold one barrier arrival, and a short
wait limit (1 ms) makes the role waiting for it give up. The kernel then winds
down (every other wait bounded too, no copy left in flight), the device status
reports TQ_ERR_TIMEOUT, and the next normal call must give the clean result bit
for bit — for dW that proves that tq_device_status reset the stream-K tile
counters the abandoned launch left set.
"""
import pytest
import torch

from paper_2606_18114_gb300 import synth

pytestmark = pytest.mark.gpu

LIMIT_NS = 1_000_000


@pytest.fixture(scope="module")
def tq():
    if not torch.cuda.is_available():
        pytest.fail("the gpu tests need a CUDA device")
    from paper_2606_18114_gb300 import build, tq as _tq
    build.build()
    _tq.load()
    yield _tq
    _tq.test_hooks(0, 0)


def _expect_timeout(tq):
    with pytest.raises(tq.TqError) as e:
        tq.device_status()
    assert e.value.status == 4, str(e.value)


def test_quantize_withheld_release_times_out_then_recovers(tq):
    n, k, g = 4096, 2048, 128   # more stages than the first round of every CTA
    w = torch.from_numpy(synth.latent_weights(n, k, seed=81)).cuda()
    ref = tq.quantize(w, g)
    tq.device_status()
    try:
        tq.test_hooks(LIMIT_NS, 1)
        tq.quantize(w, g)
        _expect_timeout(tq)
    finally:
        tq.test_hooks(0, 0)
    for _ in range(2):
        got = tq.quantize(w, g)
        tq.device_status()
        assert all(torch.equal(a, b) for a, b in zip(got, ref))


def test_quantize_with_transpose_withheld_release_times_out_then_recovers(tq):
    """The fused quantize + transpose: CTA 0 gives up on its stages and reaches the
    grid barrier late, the others give up on the barrier; every CTA still passes the
    barrier's reset, so after the timeout 300 clean launches (every one of the 256
    barrier slots again) give the clean result."""
    n, k, g = 4096, 2048, 128
    w = torch.from_numpy(synth.latent_weights(n, k, seed=84)).cuda()
    ref = tq.quantize_with_transpose(w, g)
    tq.device_status()
    try:
        tq.test_hooks(LIMIT_NS, 1)
        tq.quantize_with_transpose(w, g)
        _expect_timeout(tq)
    finally:
        tq.test_hooks(0, 0)
    out = tuple(torch.empty_like(t) for t in ref)
    for _ in range(300):
        tq.quantize_with_transpose(w, g, out=out)
    tq.device_status()
    assert all(torch.equal(a, b) for a, b in zip(out, ref))


def test_dw_withheld_accumulator_times_out_then_recovers(tq):
    # in_proj shape at 640 tokens: 272 pair tiles on 76 pairs, so the first pair
    # reuses its first accumulator, and the tail tiles are cut into stream-K pieces
    n, k, m, g = 8512, 2048, 640, 128
    w = torch.from_numpy(synth.latent_weights(n, k, seed=82)).cuda()
    x = synth.activations_bf16(m, k, seed=82, stream="x").cuda()
    dy = synth.activations_bf16(m, n, seed=82, std=1e-2, stream="dy").cuda()
    codes, s, _ = tq.quantize(w, g)
    _, ref = tq.linear_bwd(dy, x, codes, s, k, g, want_dx=False)
    tq.device_status()
    try:
        tq.test_hooks(LIMIT_NS, 2)
        tq.linear_bwd(dy, x, codes, s, k, g, want_dx=False)
        _expect_timeout(tq)
    finally:
        tq.test_hooks(0, 0)
    for _ in range(2):
        _, got = tq.linear_bwd(dy, x, codes, s, k, g, want_dx=False)
        tq.device_status()
        assert torch.equal(got, ref)


def test_decode_pieces_withheld_partial_sums_time_out_then_recover(tq):
    """A decode cut into pieces of k (in_proj at one token: clusters of CTAs over each
    block of rows): CTA 1 sends no partial sums, the first CTA of its cluster gives up
    waiting for them, the others give up waiting for its release; every other cluster
    finishes. The next normal calls give the clean result bit for bit."""
    n, k, m, g = 8512, 2048, 1, 128
    w = torch.from_numpy(synth.latent_weights(n, k, seed=85)).cuda()
    x = synth.activations_bf16(m, k, seed=85).cuda()
    codes, s, _ = tq.quantize(w, g)
    ref = tq.linear_fwd(x, codes, s, g)
    tq.device_status()
    try:
        tq.test_hooks(LIMIT_NS, 4)
        tq.linear_fwd(x, codes, s, g)
        _expect_timeout(tq)
    finally:
        tq.test_hooks(0, 0)
    for _ in range(2):
        got = tq.linear_fwd(x, codes, s, g)
        tq.device_status()
        assert torch.equal(got, ref)


def test_hooks_off_by_default_after_reset(tq):
    """With the limit and flags reset, a normal launch reports no timeout."""
    tq.test_hooks(0, 0)
    w = torch.from_numpy(synth.latent_weights(512, 256, seed=83)).cuda()
    tq.quantize(w, 128)
    tq.device_status()
