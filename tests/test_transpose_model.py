"""Host model of the register transpose in csrc/quantize.cu (transpose_codes_kernel):
a 16 x 16 block of 2-bit codes (16 words, one per row n) loaded in the row order
i(q) = 2 (q % 8) + q / 8, four levels of block swaps (8 and 4 fields as byte permutes,
2 and 1 fields as masked shift-xors), word p stored as output row i(p). Checked against
the definition of the transposed layout (word of row k holds the codes of 16 rows n at
the same bit rule as the codes) on random blocks, including all-ones and single-field
blocks. No GPU is involved."""
import numpy as np

M32 = 0xFFFFFFFF


def code_pos(i):
    """Bit of code i (0..15) inside its word (include/tq.h)."""
    return 16 * (i & 1) + 2 * (i >> 1)


def prmt(x, y, sel):
    """CUDA __byte_perm: byte j of the result is byte (sel >> 4j) & 7 of {y:x}."""
    b = [(x >> (8 * j)) & 255 for j in range(4)] + [(y >> (8 * j)) & 255 for j in range(4)]
    return sum(b[(sel >> (4 * j)) & 7] << (8 * j) for j in range(4))


def transpose_block_model(rows):
    t = [rows[2 * (q & 7) + (q >> 3)] for q in range(16)]
    for w in range(8):
        a, c = t[w], t[w + 8]
        t[w], t[w + 8] = prmt(a, c, 0x5410), prmt(a, c, 0x7632)
    for w in range(16):
        if not w & 4:
            a, c = t[w], t[w + 4]
            t[w], t[w + 4] = prmt(a, c, 0x6240), prmt(a, c, 0x7351)
    for b, m in ((2, 0x0F0F0F0F), (1, 0x33333333)):
        for w in range(16):
            if not w & b:
                a, c = t[w], t[w + b]
                x = ((a >> (2 * b)) ^ c) & m
                t[w + b] = c ^ x
                t[w] = (a ^ (x << (2 * b))) & M32
    out = [0] * 16
    for p in range(16):
        out[2 * (p & 7) + (p >> 3)] = t[p]
    return out


def transpose_block_definition(rows):
    """Output word kk holds, at bit code_pos(j), the field of code kk of row j."""
    return [sum(((rows[j] >> code_pos(kk)) & 3) << code_pos(j) for j in range(16))
            for kk in range(16)]


def test_register_transpose_matches_the_layout():
    rs = np.random.default_rng(0)
    blocks = [[int(v) for v in rs.integers(0, 2 ** 32, 16, dtype=np.uint64)] for _ in range(300)]
    blocks.append([M32] * 16)
    blocks.append([0] * 16)
    for j in range(16):
        for i in range(16):
            one = [0] * 16
            one[j] = 3 << code_pos(i)
            blocks.append(one)
    for rows in blocks:
        assert transpose_block_model(rows) == transpose_block_definition(rows)


def test_single_field_moves_to_the_transposed_position():
    """Code i of row j lands as code j of output word i."""
    for j in range(16):
        for i in range(16):
            rows = [0] * 16
            rows[j] = 1 << code_pos(i)
            out = transpose_block_model(rows)
            assert out[i] == 1 << code_pos(j)
            assert all(w == 0 for k, w in enumerate(out) if k != i)
