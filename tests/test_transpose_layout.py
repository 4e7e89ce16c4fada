"""Host model of the X_u^T transpose kernel of the M accumulators (csrc/backward.cu transpose_bf16):
a 64 x 64 shared tile whose 8-element groups are stored XOR-swizzled by the row's group, written
with 16-byte row loads and read down columns for 16-byte stores. The model replays every thread's
indices and checks that the result is the transpose on ragged shapes, that every tile access stays
inside the tile, and that a warp's column reads fall on distinct banks."""
import numpy as np
import pytest


def transpose_model(inp):
    rows, cols = inp.shape
    out = np.full((cols, rows), -1, dtype=np.int64)
    for by in range((rows + 63) // 64):
        for bx in range((cols + 63) // 64):
            c0, r0 = bx * 64, by * 64
            t = np.full((64, 64), -7, dtype=np.int64)
            for ty in range(32):
                for tx in range(8):
                    for k in range(ty, 64, 32):
                        r, c = r0 + k, c0 + 8 * tx
                        v = np.zeros(8, dtype=np.int64)
                        if r < rows:
                            for e in range(8):
                                if c + e < cols:
                                    v[e] = inp[r, c + e]
                        g = tx ^ ((k >> 3) & 7)
                        assert 0 <= g < 8
                        t[k, 8 * g:8 * g + 8] = v
            for ty in range(32):
                for tx in range(8):
                    for k in range(ty, 64, 32):
                        c, r = c0 + k, r0 + 8 * tx
                        if c >= cols:
                            continue
                        for e in range(8):
                            kr = 8 * tx + e
                            col = 8 * ((k >> 3) ^ ((kr >> 3) & 7)) + (k & 7)
                            assert 0 <= col < 64
                            if r + e < rows:
                                out[c, r + e] = t[kr, col]
    return out


@pytest.mark.parametrize("rows,cols", [(64, 64), (130, 77), (5, 200), (71, 9), (128, 136)])
def test_swizzled_tile_transposes_ragged_shapes(rows, cols):
    inp = np.arange(rows * cols).reshape(rows, cols)
    assert np.array_equal(transpose_model(inp), inp.T)


def test_column_reads_of_a_warp_hit_distinct_banks():
    """A warp is tx = 0..7 for four consecutive ty (rows k .. k + 3 of the output tile); for each of
    its 8 reads the 32 lanes touch 32-bit words in distinct banks (two lanes may share a word)."""
    for k0 in range(0, 64, 4):
        for e in range(8):
            banks = {}
            for ty in range(4):
                k = k0 + ty
                for tx in range(8):
                    kr = 8 * tx + e
                    col = 8 * ((k >> 3) ^ ((kr >> 3) & 7)) + (k & 7)
                    word = (kr * 128 + col * 2) // 4
                    banks.setdefault(word % 32, set()).add(word)
            assert max(len(w) for w in banks.values()) == 1
