"""Host model of the dW kernel's work split (csrc/dw_gemm.cu, CTA pairs with a
stream-K tail), checked for every schedule shape it can meet: each (tile, k-block) is
computed exactly once, a split tile's pieces are contiguous and in k order, the
fixup reads each piece from the workspace slot its writer used, no run needs more
than its two slots, every counter and slot index stays inside the device arrays, and
the tail pieces run in the order that keeps every pair's token offset within
nkb - (run length) of the time spent on the tail. The model restates the scheduler's
integer arithmetic; no GPU is involved."""
import itertools

import pytest

MAX_CTAS = 160  # kDwMaxCtas: workspace of two half-tiles per CTA, a counter per tail half


class Sched:
    def __init__(self, tiles, grid, nkb):
        self.grid, self.nkb = grid, nkb
        self.rem = tiles % grid
        self.units = self.rem * nkb
        if self.units < grid:
            self.rem, self.units = 0, 0
        self.dp = tiles - self.rem

    def run_start(self, c):
        return c * self.units // self.grid

    def owner(self, b):
        return ((b + 1) * self.grid - 1) // self.units

    def whole_of(self, c):
        return (self.dp - 1 - c) // self.grid + 1 if c < self.dp else 0

    def items(self, c):
        nw = self.whole_of(c)
        out = [(c + i * self.grid, 0, self.nkb, -1) for i in range(nw)]
        # token direction of the whole tiles: the last one runs down to token 0
        self.rev = [(nw - 1 - i) % 2 == 0 for i in range(nw)]
        if self.rem:
            s0, s1 = self.run_start(c), self.run_start(c + 1)
            if s1 > s0:
                npieces = (s1 - 1) // self.nkb - s0 // self.nkb + 1
                # a run crossing into the next tile does that tile's piece first
                for j in ([1, 0] if npieces == 2 else range(npieces)):
                    r = s0 // self.nkb + j
                    b0 = r * self.nkb
                    out.append((self.dp + r, max(s0, b0) - b0, min(s1, b0 + self.nkb) - b0, j))
        return out


def _check(tiles, pairs, nkb):
    q = Sched(tiles, pairs, nkb)
    done = {}
    slot_of = {}  # (pair, tile) -> slot its piece was written to
    for c in range(pairs):
        its = q.items(c)
        nonwhole = [it for it in its if not (it[1] == 0 and it[2] == nkb)]
        assert len(nonwhole) <= 2, (tiles, pairs, nkb, c, its)
        for t, kb0, kb1, sk in its:
            assert 0 <= kb0 < kb1 <= nkb
            for kb in range(kb0, kb1):
                assert (t, kb) not in done, ("twice", t, kb)
                done[(t, kb)] = c
            if not (kb0 == 0 and kb1 == nkb):
                assert sk >= 0
                slot_of[(c, t)] = 0 if sk == 0 else 1
    assert len(done) == tiles * nkb, "some (tile, k-block) never computed"
    for c in range(pairs):  # directions alternate, the last whole tile ending at token 0
        q.items(c)
        assert all(q.rev[i] != q.rev[i + 1] for i in range(len(q.rev) - 1))
        assert not q.rev or q.rev[-1]
    for c in range(pairs):  # token offset minus time, over the pair's tail pieces
        if not q.rem:
            break
        run = q.run_start(c + 1) - q.run_start(c)
        tau = 0
        for t, kb0, kb1, sk in q.items(c)[q.whole_of(c):]:
            assert 0 <= kb0 - tau <= nkb - run, (tiles, pairs, nkb, c, q.items(c))
            tau += kb1 - kb0
    for r in range(q.rem):
        t = q.dp + r
        b0 = r * nkb
        c_first, c_last = q.owner(b0), q.owner(b0 + nkb - 1)
        pieces = c_last - c_first + 1
        for p in range(pieces):  # piece p from pair c_first + p, in k order
            pc = c_first + p
            kbs = sorted(kb for (tt, kb), c in done.items() if tt == t and c == pc)
            assert kbs, (t, p)
            if pieces > 1:
                # the slot the fixup reads is the one the writer used
                assert slot_of[(pc, t)] == (0 if q.run_start(pc) >= b0 else 1)
            if p > 0:
                prev = max(kb for (tt, kb), c in done.items() if tt == t and c == pc - 1)
                assert kbs[0] == prev + 1
        for rank in (0, 1):
            assert 2 * r + rank < MAX_CTAS  # completion counter
    for c in range(pairs):
        for rank in (0, 1):
            for j in (0, 1):
                assert 2 * (2 * c + rank) + j < 2 * MAX_CTAS  # workspace slot


@pytest.mark.parametrize("tiles,pairs,nkb", [
    (272, 76, 256),   # Mamba-2 in_proj: 34 x 8 pair tiles, 16384 tokens
    (128, 76, 256),   # out_proj: 8 x 16 pair tiles
    (76, 76, 256),    # exactly one wave
    (77, 76, 1),      # a tail with fewer k-blocks than pairs: whole tiles
    (3, 2, 5),
    (1, 1, 1),
    (1, 1, 2048),     # one tile, one pair: 131072 tokens
])
def test_dw_pair_schedule_shapes(tiles, pairs, nkb):
    _check(tiles, pairs, nkb)


def test_dw_pair_schedule_sweep():
    for tiles, pairs, nkb in itertools.product([1, 2, 5, 37, 75, 76, 77, 151, 152, 272],
                                               [1, 2, 3, 38, 75, 76, 80],
                                               [1, 2, 3, 7, 16, 64, 257]):
        if pairs <= tiles:
            _check(tiles, pairs, nkb)


def _pieces_per_tail_tile(q):
    return [q.owner(r * q.nkb + q.nkb - 1) - q.owner(r * q.nkb) + 1 for r in range(q.rem)]


@pytest.mark.parametrize("m,cut", [(64, False), (1999, True), (2000, True)])
def test_dw_stream_k_gpu_test_shapes(m, cut):
    """The tail cases the GPU test test_dw_stream_k_tail names, for its shape
    (n = 4160, k = 1280: 5 x 17 = 85 pair tiles) on the 76 pairs of 152 SMs: at 64
    tokens the 9 tail tiles have fewer k-blocks than pairs and stay whole; at 1999
    and 2000 tokens (16 k-blocks, the first ending on a ragged block) they are cut
    into pieces, several per tile."""
    tiles = ((1280 + 255) // 256) * ((4160 + 255) // 256)
    nkb = (m + 127) // 128
    q = Sched(tiles, 76, nkb)
    assert tiles == 85
    if not cut:
        assert q.rem == 0
        return
    assert q.rem == 9 and q.units == 9 * 16
    assert min(_pieces_per_tail_tile(q)) >= 8
    _check(tiles, 76, nkb)
