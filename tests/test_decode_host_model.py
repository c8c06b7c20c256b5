"""Host models of the decode kernel's index arithmetic (no GPU).

Each function restates, in Python, a formula of the decode kernel and its launcher
and checks the property the kernel relies on: the pieces of k of a launch cover every
(block of rows, segment) once with no empty piece and one cluster per block; the bytes
the first CTA of a cluster expects equal those the other CTAs' lanes send; the scale
windows, swizzled as the TMA writes them, give every lane the scale of its own row and
group, and a warp's eight rows fall on distinct banks."""
import itertools

import pytest

ROWS, SEG_K, WIN_GROUPS = 256, 512, 32


def pieces_of(mats, pieces):
    """(unit -> (matrix, block, piece, s0, s1)) as the producer decodes blockIdx.x."""
    unit0, u = [], 0
    for (n, k) in mats:
        unit0.append(u)
        u += ((n + ROWS - 1) // ROWS) * pieces
    out = []
    for uu in range(u):
        d = max(i for i in range(len(mats)) if unit0[i] <= uu)
        n, k = mats[d]
        nseg = (k + SEG_K - 1) // SEG_K
        local = uu - unit0[d]
        piece = local % pieces
        block = local // pieces
        out.append((d, block, piece, piece * nseg // pieces, (piece + 1) * nseg // pieces))
    return out


@pytest.mark.parametrize("mats", [
    [(8512, 2048)], [(2048, 4096)], [(200, 1024)], [(300, 18432)], [(8192, 8192)],
    [(520, 1088), (264, 4608), (40, 1152)], [(16, 2560)] * 3, [(1, 64 * 17)],
])
def test_pieces_cover_every_segment_once(mats):
    min_nseg = min((k + SEG_K - 1) // SEG_K for _, k in mats)
    for pieces in (1, 2, 4, 8):
        if pieces > min_nseg:
            continue  # the launcher keeps P <= every matrix's segment count
        units = pieces_of(mats, pieces)
        seen = set()
        for u, (d, block, piece, s0, s1) in enumerate(units):
            assert s1 > s0, "empty piece"
            assert u % pieces == piece, "cluster rank is the piece"
            assert (u - piece) // pieces == (u - u % pieces) // pieces
            for s in range(s0, s1):
                assert (d, block, s) not in seen
                seen.add((d, block, s))
        # one cluster (P consecutive CTAs) holds the P pieces of one block
        for c in range(len(units) // pieces):
            members = units[c * pieces:(c + 1) * pieces]
            assert len({(d, b) for d, b, *_ in members}) == 1
        want = {(d, b, s) for d, (n, k) in enumerate(mats)
                for b in range((n + ROWS - 1) // ROWS) for s in range((k + SEG_K - 1) // SEG_K)}
        assert seen == want


def slice_bytes(two_tiles, m):
    """The launcher's expected bytes per row warp and sending CTA."""
    return 8 * 32 * (((m if m < 8 else 8) + 1) // 2 + (((m - 8 + 1) // 2) if two_tiles and m > 8 else 0))


@pytest.mark.parametrize("m", range(1, 17))
def test_expected_bytes_equal_the_bytes_sent(m):
    two_tiles = m > 8
    sent = 0
    for lane in range(32):
        t = lane & 3
        v0 = 2 * t < m                       # tokens 2t, 2t + 1 of the first n-tile
        v1 = two_tiles and 8 + 2 * t < m     # tokens 8 + 2t, 9 + 2t
        sent += 2 * 16 * (v0 + v1)           # a float4 per row tile, two row tiles
    assert sent == slice_bytes(two_tiles, m)
    # every token below m is sent by some lane
    tokens = {tok for lane in range(32) for tok in (2 * (lane & 3), 2 * (lane & 3) + 1)
              if 2 * (lane & 3) < m} | {8 + tok for lane in range(32)
                                         for tok in (2 * (lane & 3), 2 * (lane & 3) + 1)
                                         if two_tiles and 8 + 2 * (lane & 3) < m}
    assert {t for t in tokens if t < m} == set(range(m))


def tma_swizzle_128b(row, q):
    """Float q (< 32) of a 128-byte row as the TMA's 128-byte swizzle places it in a
    1024-byte-aligned buffer: 16-byte chunk j of row r lands at chunk j ^ (r % 8)."""
    chunk, within = q // 4, q % 4
    return row * 32 + ((chunk ^ (row % 8)) * 4) + within


def kernel_window_index(row, q, g_lane):
    """The consumer's address: row * 32 + ((q & 31) ^ (g << 2)), g = lane / 4."""
    return row * 32 + ((q & 31) ^ (g_lane << 2))


def test_window_addressing_matches_the_swizzle():
    for wr, gl, r, h in itertools.product(range(8), range(8), range(2), range(2)):
        row = 32 * wr + gl + 16 * r + 8 * h          # the lane's rows are all g mod 8
        for q in range(64):                          # two windows' worth of groups
            assert kernel_window_index(row, q, gl) == tma_swizzle_128b(row, q % 32)


def test_window_float2_loads_stay_paired_and_bank_conflict_free():
    for q0 in range(0, 32, 2):                       # g = 128: the pair q0, q0 + 1
        for gl in range(8):
            a = kernel_window_index(gl, q0, gl)
            assert kernel_window_index(gl, q0 + 1, gl) == a + 1 and a % 2 == 0
        # one 8-byte load per lane: the eight rows of a warp (g = 0..7) on 16 banks
        banks = [kernel_window_index(gl, q0, gl) % 32 for gl in range(8)]
        words = {b for b in banks} | {b + 1 for b in banks}
        assert len(words) == 16


def producer_windows(s0, s1, log2g):
    """(segment, first group of the box) of every window load of a piece."""
    wmask = (1 << (log2g - 4)) - 1
    return [(s, (s >> (log2g - 4)) * WIN_GROUPS) for s in range(s0, s1)
            if s == s0 or (s & wmask) == 0]


def consumer_windows(s0, s1, log2g):
    """(segment opening, segment closing) of every window the consumer waits for."""
    wmask = (1 << (log2g - 4)) - 1
    opened, out = None, []
    for s in range(s0, s1):
        if s == s0 or (s & wmask) == 0:
            assert opened is None, "a window opened before the previous one closed"
            opened = s
        if (s & wmask) == wmask or s + 1 == s1:
            out.append((opened, s))
            opened = None
    assert opened is None
    return out


@pytest.mark.parametrize("log2g", [5, 6, 7, 8, 9])
def test_window_sequences_of_pieces_match(log2g):
    g = 1 << log2g
    for k in (g * 36, g * 64, g * 100 + 0):
        k -= k % 64
        nseg = (k + SEG_K - 1) // SEG_K
        for pieces in (1, 2, 4, 8):
            if pieces > nseg:
                continue
            for p in range(pieces):
                s0, s1 = p * nseg // pieces, (p + 1) * nseg // pieces
                loads = producer_windows(s0, s1, log2g)
                waits = consumer_windows(s0, s1, log2g)
                assert len(loads) == len(waits)           # one buffer use per window
                for (ls, q0), (a, b) in zip(loads, waits):
                    assert ls == a and q0 % 4 == 0         # TMA x: a multiple of 16 bytes
                    for s in range(a, b + 1):              # every group the segment reads
                        first = (s * SEG_K) >> log2g
                        last = min(((s + 1) * SEG_K - 1) >> log2g, k // g - 1)
                        assert q0 <= first and last < q0 + WIN_GROUPS
