"""libtq's launches inside CUDA graphs (needs a GB300).

A decode step or a training step captured once and replayed must give exactly what
the same calls give eagerly: the launch path may hold no state that a capture
freezes wrongly (scheduler slots, tensor maps, cluster sizes, cross-stream
ordering)."""
import pytest
import torch

from paper_2606_18114_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def tq():
    if not torch.cuda.is_available():
        pytest.fail("the gpu tests need a CUDA device")
    from paper_2606_18114_gb300 import build, tq as _tq
    build.build()
    _tq.load()
    return _tq


def _capture(fn, replays=3):
    """Run fn eagerly on a side stream, capture it, replay it `replays` times."""
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        fn(s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        fn(s)
    for _ in range(replays):
        g.replay()
    torch.cuda.synchronize()
    return g


def test_decode_layers_in_a_graph(tq):
    """Six single-matrix decodes in stream order (pieces of k in clusters) and one
    batched call over 160 blocks of rows (the persistent grid), replayed."""
    g, m = 128, 3
    shapes = [(8512, 2048), (2048, 4096)] * 3
    calls = []
    for i, (n, k) in enumerate(shapes):
        w = torch.from_numpy(synth.latent_weights(n, k, seed=60 + i)).cuda()
        codes, s, _ = tq.quantize(w, g)
        x = synth.activations_bf16(m, k, seed=60 + i).cuda()
        calls.append((x, codes, s, torch.empty((m, n), device="cuda")))
    batch = []
    for i in range(40):
        w = torch.from_numpy(synth.latent_weights(1024, 1024, seed=90 + i)).cuda()
        codes, s, _ = tq.quantize(w, g)
        x = synth.activations_bf16(m, 1024, seed=90 + i).cuda()
        batch.append(dict(x=x, codes=codes, scales=s, g=g, y=torch.empty((m, 1024), device="cuda")))
    arr = tq.fwd_batch(batch)

    def step(stream):
        for (x, codes, s, y) in calls:
            tq.linear_fwd(x, codes, s, g, y=y, stream=stream)
        tq.linear_fwd_batched(arr, m, stream=stream)

    step(torch.cuda.current_stream())
    torch.cuda.synchronize()
    eager = [y.clone() for (_, _, _, y) in calls] + [it["y"].clone() for it in batch]
    for (_, _, _, y) in calls:
        y.zero_()
    for it in batch:
        it["y"].zero_()
    _capture(step)
    tq.device_status()
    got = [y for (_, _, _, y) in calls] + [it["y"] for it in batch]
    for i, (a, b) in enumerate(zip(eager, got)):
        assert torch.equal(a, b), f"output {i} differs after replay"


def test_training_step_in_a_graph(tq):
    """Quantize (with the transposed codes), forward and both backward products of
    one layer, captured and replayed: the same outputs as eager calls."""
    n, k, m, g = 1032, 1024, 640, 128
    w = torch.from_numpy(synth.latent_weights(n, k, seed=3)).cuda()
    x = synth.activations_bf16(m, k, seed=3, stream="x").cuda()
    dy = synth.activations_bf16(m, n, seed=3, std=1e-2, stream="dy").cuda()
    out = {}

    def step(stream):
        codes, s, z, codes_t = tq.quantize_with_transpose(w, g, stream=stream)
        y = tq.linear_fwd(x, codes, s, g, stream=stream)
        dx, dw = tq.linear_bwd(dy, x, codes, s, k, g, codes_t=codes_t, stream=stream)
        out.update(codes=codes, z=z, y=y, dx=dx, dw=dw)

    step(torch.cuda.current_stream())
    torch.cuda.synchronize()
    eager = {key: v.clone() for key, v in out.items()}
    graph = _capture(step)
    tq.device_status()
    for key in eager:
        assert torch.equal(eager[key], out[key]), f"{key} differs after replay"
    del graph
