"""Host model of how the split-K tensor-core decode (csrc/decode_tc.cu) cuts a phase.

The weight matrix of a decode phase (R rows, K columns) is cut into units of 128 rows x one
K-slice and each unit into 64-column chunks; the chunks of all units, slice-major, are dealt to
the CTAs in equal contiguous ranges. The partial kernel writes a unit's head (the run that starts
at its chunk 0) to P and the rest, if another CTA holds it, to P2; a head that holds the whole
unit writes zeros to P2, and the reduce kernel adds P + P2 for every unit. These tests restate the
plan and the segment walk of that file in Python and check, for many shapes and grids, that every
chunk is computed once, that no unit has more than two parts, and that P and P2 of every unit are
written exactly once each.
"""
import pytest

TM, KB = 128, 64
GRID_MAX, MIN_CHUNKS = 512, 4


def make_plan(R, K, cap):
    nrb, nck = -(-R // TM), -(-K // KB)
    total = nrb * nck
    grid = max(1, min(cap, total // MIN_CHUNKS))
    u = max(1, min(total // grid, nck))
    ns = -(-nck // u)
    return dict(nrb=nrb, nck=nck, total=total, grid=grid, ncf=u, ns=ns, nclast=nck - (ns - 1) * u)


def seg_at(p, g, e):
    per = p["nrb"] * p["ncf"]
    s = min(g // per, p["ns"] - 1)
    rem = g - s * per
    n = p["ncf"] if s < p["ns"] - 1 else p["nclast"]
    rb, c0 = divmod(rem, n)
    return s, rb, c0, min(g - c0 + n, e) - g


def walk(p):
    """Per unit: the (cta, first chunk, chunks) parts the partial kernel computes."""
    parts = {}
    for b in range(p["grid"]):
        g0, g1 = b * p["total"] // p["grid"], (b + 1) * p["total"] // p["grid"]
        g = g0
        while g < g1:
            s, rb, c0, nc = seg_at(p, g, g1)
            assert nc >= 1
            parts.setdefault((s, rb), []).append((b, c0, nc))
            g += nc
    return parts


SHAPES = [(4096, 8192), (24576, 4096), (8192, 8192), (2048, 4096), (3072, 8192), (6144, 4096),
          (4096, 28672), (1, 1), (1, 64), (129, 65), (1000, 777), (130, 4096), (7, 100000),
          (65536, 128), (300, 64 * 13 + 5), (57344, 8192)]


@pytest.mark.parametrize("R,K", SHAPES)
@pytest.mark.parametrize("cap", [1, 2, 7, 296, 304, 512])
def test_every_chunk_once_and_at_most_two_parts(R, K, cap):
    p = make_plan(R, K, cap)
    assert 1 <= p["grid"] <= cap and 1 <= p["nclast"] <= p["ncf"] <= p["nck"]
    assert (p["ns"] - 1) * p["ncf"] + p["nclast"] == p["nck"]
    parts = walk(p)
    assert len(parts) == p["ns"] * p["nrb"]
    for (s, rb), ps in parts.items():
        n = p["ncf"] if s < p["ns"] - 1 else p["nclast"]
        # contiguous, in order, covering the unit exactly once
        assert ps[0][1] == 0 and sum(nc for _, _, nc in ps) == n
        for (b0, c0, nc), (b1, c1, _) in zip(ps, ps[1:]):
            assert b1 == b0 + 1 and c1 == c0 + nc
        assert len(ps) <= 2, (s, rb, ps)
        # writers of P and of P2, by the epilogue's rule: head -> P (and zeros to P2 if whole),
        # a segment starting past chunk 0 -> P2
        writes_p = [b for b, c0, nc in ps if c0 == 0]
        writes_p2 = [b for b, c0, nc in ps if c0 > 0 or nc == n]
        assert len(writes_p) == 1 and len(writes_p2) == 1


@pytest.mark.parametrize("R,K", SHAPES)
def test_ranges_balanced_and_plan_bounds_workspace(R, K):
    """Every CTA holds floor or ceil of total/grid chunks, and no grid up to GRID_MAX gives more
    slices (partial-sum bytes) than the plan the workspace size is computed for."""
    big = make_plan(R, K, GRID_MAX)
    for cap in (1, 3, 152, 296, 304, GRID_MAX):
        p = make_plan(R, K, cap)
        sizes = {(b + 1) * p["total"] // p["grid"] - b * p["total"] // p["grid"] for b in range(p["grid"])}
        assert sizes <= {p["total"] // p["grid"], -(-p["total"] // p["grid"])}
        assert p["ns"] <= big["ns"]


def test_headline_cut():
    """70B gate/up (28672 x 8192, r = 4096) on 304 CTAs: phase 1 (W_p, 4096 x 8192) in 10 slices
    of 13 chunks (the last 11), phase 2 (C, 24576 x 4096) in 2 slices of 40 chunks (the last 24)."""
    p1, p2 = make_plan(4096, 8192, 304), make_plan(24576, 4096, 304)
    assert (p1["grid"], p1["ncf"], p1["ns"], p1["nclast"]) == (304, 13, 10, 11)
    assert (p2["grid"], p2["ncf"], p2["ns"], p2["nclast"]) == (304, 40, 2, 24)


def make_plan_fixed(R, K, grid):
    nrb, nck = -(-R // TM), -(-K // KB)
    total = nrb * nck
    u = max(1, min(total // grid, nck))
    ns = -(-nck // u)
    return dict(nrb=nrb, nck=nck, total=total, grid=grid, ncf=u, ns=ns, nclast=nck - (ns - 1) * u)


@pytest.mark.parametrize("R,K", [(24576, 4096), (19456, 8192), (38912, 520), (24577, 4100), (152 * 128, 64)])
def test_whole_row_plan_gives_each_cta_one_row_block(R, K):
    """The whole-row plan (grid = the phase's 128-row blocks) cuts K into one slice, and every
    CTA's range is exactly one unit: no unit is split, so the epilogue's sums are the outputs."""
    nrb = -(-R // TM)
    p = make_plan_fixed(R, K, nrb)
    assert p["ns"] == 1 and p["ncf"] == p["nclast"] == p["nck"]
    parts = walk(p)
    assert len(parts) == nrb
    for (s, rb), ps in parts.items():
        assert ps == [(rb, 0, p["nck"])]
