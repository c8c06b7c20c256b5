"""Pure-Python brute force of §3.1 for tiny inputs (test helper).

Written from the paper's definition with Python floats (fp64) and explicit
loops, independently of ``oracle.tq_oracle`` (no numpy in the arithmetic), so
that the two can pin each other on small cases. Inputs must avoid the rounding
tie |w/s| = 0.5, where fp32 and fp64 decisions may differ.
"""
from __future__ import annotations

import math


def quantize_rows(w_rows, g):
    """Lists of floats -> (codes [[int]], scales [[float]], zeros [[int]])."""
    codes, scales, zeros = [], [], []
    for row in w_rows:
        if len(row) % g:
            raise ValueError("row length must be a multiple of g")
        crow, srow, zrow = [], [], []
        for start in range(0, len(row), g):
            grp = row[start:start + g]
            s = math.fsum(abs(v) for v in grp) / g
            nz = 0
            for v in grp:
                if s == 0.0:
                    c = 0
                else:
                    q = v / s
                    q = max(-1.0, min(1.0, q))
                    # round half to even, written out
                    f = math.floor(q)
                    frac = q - f
                    if frac > 0.5:
                        c = f + 1
                    elif frac < 0.5:
                        c = f
                    else:
                        c = f if f % 2 == 0 else f + 1
                    c = int(c)
                crow.append(c)
                nz += c == 0
            srow.append(s)
            zrow.append(nz)
        codes.append(crow)
        scales.append(srow)
        zeros.append(zrow)
    return codes, scales, zeros


def pack_row(code_row):
    """One row of ternary codes -> list of 32-bit words (include/tq.h layout)."""
    words = []
    for start in range(0, len(code_row), 16):
        word = 0
        for i in range(16):
            c = code_row[start + i]
            val = {0: 0, 1: 1, -1: 3}[c]
            bit = (16 if i % 2 else 0) + 2 * (i // 2)
            word |= val << bit
        words.append(word)
    return words


def dequant_rows(codes, scales, g):
    return [[scales[n][k // g] * codes[n][k] for k in range(len(codes[n]))]
            for n in range(len(codes))]


def matmul_nt(a, b):
    """a [M][K] times b [N][K] transposed -> [M][N] (fsum per entry)."""
    return [[math.fsum(a[m][k] * b[n][k] for k in range(len(a[m]))) for n in range(len(b))]
            for m in range(len(a))]


def matmul_nn(a, b):
    """a [M][R] times b [R][C] -> [M][C]."""
    cols = len(b[0])
    return [[math.fsum(a[m][r] * b[r][c] for r in range(len(b))) for c in range(cols)]
            for m in range(len(a))]


def transpose(a):
    return [list(col) for col in zip(*a)]
