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


def pick_cs(nrb, nck, cap):
    """CTAs per row block in the row-block plan (0: the balanced plan with a reduce kernel); cap is
    the CTA slots (two per SM)."""
    if nrb > cap:
        return 0
    cs = 1
    while cs < 8 and nrb * cs * 2 <= cap and cs * 2 <= nck:
        cs *= 2
    return cs


def make_plan_rows(R, K, cs):
    nrb, nck = -(-R // TM), -(-K // KB)
    ncf = -(-nck // cs)
    ns = -(-nck // ncf)
    return dict(nrb=nrb, nck=nck, total=nrb * nck, grid=nrb * cs, ncf=ncf, ns=ns, nclast=nck - (ns - 1) * ncf)


ROW_SHAPES = [(4096, 8192), (24576, 4096), (2048, 4096), (2048, 11008), (8960, 2048), (8192, 4096),
              (19456, 8192), (38912, 520), (24577, 4100), (152 * 128, 64), (1, 1), (129, 65), (300, 837),
              (264, 520), (64, 128), (40, 1), (1400, 1000)]


@pytest.mark.parametrize("R,K", ROW_SHAPES)
@pytest.mark.parametrize("cap", [296, 304])
def test_row_block_plan_gives_each_cta_one_slice_of_its_cluster_block(R, K, cap):
    """The row-block plan: cs CTAs (a cluster) per 128-row block, cs a power of two up to 8 with the
    grid within the cap and every slice non-empty; CTA b takes slice b % cs of block b / cs (or
    nothing when the block has fewer slices), as the segment walk finds it from its (g0, g1). Every
    chunk of every block is computed once, inside the block's own cluster, and the cluster's
    row shares (128 / cs rows each) cover the block's 128 rows once."""
    nrb, nck = -(-R // TM), -(-K // KB)
    cs = pick_cs(nrb, nck, cap)
    if cs == 0:  # more blocks than CTA slots: the balanced plan
        assert nrb > cap
        return
    assert cs in (1, 2, 4, 8) and nrb * cs <= cap and cs <= nck
    assert cs == 8 or nrb * cs * 2 > cap or cs * 2 > nck   # the largest such cs
    p = make_plan_rows(R, K, cs)
    assert (p["ns"] - 1) * p["ncf"] + p["nclast"] == nck and 1 <= p["nclast"] <= p["ncf"] and p["ns"] <= cs
    seen = {}
    for b in range(p["grid"]):
        rb, k = divmod(b, cs)
        if k >= p["ns"]:
            continue
        n = p["ncf"] if k < p["ns"] - 1 else p["nclast"]
        g0 = k * nrb * p["ncf"] + rb * n
        g1 = g0 + n
        assert seg_at(p, g0, g1) == (k, rb, 0, n)
        assert (k, rb) not in seen
        seen[(k, rb)] = n
    assert len(seen) == nrb * p["ns"]
    for rb in range(nrb):
        assert sum(seen[(k, rb)] for k in range(p["ns"])) == nck
    rpr = TM // cs
    assert sorted(r for k in range(cs) for r in range(k * rpr, (k + 1) * rpr)) == list(range(TM))


def test_row_block_plan_on_the_llama_phases():
    """On 152 SMs (304 CTA slots): 70B gate/up phase 1 (32 blocks) and both 70B q/o phases take
    clusters of 8 (256 CTAs of 16 chunks), its phase 2 (192 blocks) one CTA per block, the 7B
    phases of 16 blocks clusters of 8 (128 CTAs), the 7B gate's phase 2 (70 blocks) clusters of 4;
    longer phases (more than 304 blocks) keep the balanced plan."""
    assert pick_cs(32, 128, 304) == 8 and pick_cs(192, 64, 304) == 1 and pick_cs(32, 64, 304) == 8
    assert pick_cs(16, 64, 304) == 8 and pick_cs(70, 32, 304) == 4 and pick_cs(311, 5, 304) == 0
    p = make_plan_rows(4096, 8192, 8)
    assert (p["grid"], p["ncf"], p["ns"], p["nclast"]) == (256, 16, 8, 16)


@pytest.mark.parametrize("tnt", [16, 32, 64, 128])
@pytest.mark.parametrize("nb", [1, 2])
def test_cluster_sums_fit_the_ring_and_tensor_memory(tnt, nb):
    """Per CTA (two per SM): the stage ring (112 KB less 1.5 KB) holds at least two stages and the
    cluster's [T][128] fp32 sums; tensor memory holds the accumulators in its 256 columns: two
    segments of 128 / (tnt nb) accumulators each up to 64 tokens, one accumulator of tnt nb columns
    at 128 tokens (the row-block plan's single segment)."""
    stage = TM * KB * 2 + nb * tnt * KB * 2
    stages = min(10, (112 * 1024 - 1536) // stage)
    assert stages >= 2 and TM * tnt * 4 <= stages * stage
    nacc = 1 if tnt * nb >= 128 else 128 // (tnt * nb)
    segments = 2 if tnt <= 64 else 1
    assert segments * nacc * tnt * nb <= 256
    assert 16 <= tnt * nb <= 256 and (tnt * nb) % 16 == 0          # an MMA's N for M = 128


# ---- the split prefill's choice of tile width and K-slices (csrc/prefill.cu pick_shape) ----------
def pick_bn_slots(M, T, bnmax, slots):
    mt = -(-M // 128)
    best, best_cost = bnmax, None
    for bn in range(bnmax, 15, -16):
        tiles = mt * -(-T // bn)
        cost = -(-tiles // slots) * (432 + bn)
        if best_cost is None or cost < best_cost:
            best, best_cost = bn, cost
    return best


def pick_shape(M, T, ksteps, sms=152):
    """(config, tokens per tile, K-slices per tile)."""
    mt = -(-M // 128)
    bnw = 256 if T >= 256 else -(-T // 16) * 16
    tiles_w = mt * -(-T // bnw)
    bn0 = pick_bn_slots(M, T, 256, sms)
    if tiles_w * 2 <= sms and bn0 <= 64:
        ks = 1
        while ks < 4 and tiles_w * ks * 2 <= sms and ksteps // (ks * 2) >= 16:
            ks *= 2
        if ks > 1:
            return 0, bnw, ks
    waves0 = -(-(mt * -(-T // bn0)) // sms)
    if waves0 < 3:
        return 0, bn0, 1
    return 1, pick_bn_slots(M, T, 160, 2 * sms), 1


def test_prefill_split_k_choice_on_the_llama_gemms():
    """GEMM 1 (M = r, K = n) and GEMM 2 (M = m - r, two passes over K = r): split into clusters of 4
    where the plain plan would run tiles of 64 tokens or fewer (7B attention and 70B layers at
    T = 256), kept whole where it fills the SMs with wider tiles (7B attention T = 2048, the
    r = 1024 layer at T = 2048, 70B q/o at T = 512)."""
    assert pick_shape(2048, 256, 64) == (0, 256, 4) and pick_shape(2048, 256, 64) == pick_shape(2048, 256, 2 * 32)
    assert pick_shape(4096, 256, 128) == (0, 256, 4)                  # 70B GEMM 1
    assert pick_shape(24576, 256, 128)[2] == 1                       # 70B gate/up GEMM 2: 192 tiles
    assert pick_shape(2048, 2048, 64) == (0, 240, 1)                 # 7B attention prefill
    assert pick_shape(1024, 2048, 64)[2] == 1                        # r = 1024 GEMM 1: 152 tiles of 112
    assert pick_shape(4096, 512, 128)[2] == 1                        # 70B q/o T = 512
    assert pick_shape(4096, 200, 128) == (0, 208, 4)                 # one ragged 208-token tile
    assert pick_shape(1100, 200, 32) == (0, 208, 2) and pick_shape(1900, 200, 36) == (0, 208, 2)


@pytest.mark.parametrize("ksteps,ks", [(64, 4), (36, 2), (128, 4), (33, 2), (16, 2)])
def test_prefill_k_slices_cover_every_step_once(ksteps, ks):
    """CTA z of a tile's cluster accumulates K-steps [z ksteps / ks, (z + 1) ksteps / ks)."""
    steps = [i for z in range(ks) for i in range(z * ksteps // ks, (z + 1) * ksteps // ks)]
    assert steps == list(range(ksteps))


@pytest.mark.parametrize("ks,bn,ntok", [(2, 256, 256), (4, 256, 200), (4, 208, 200), (2, 208, 17)])
def test_prefill_cluster_sums_cover_the_tile_once(ks, bn, ntok):
    """The split prefill's cluster epilogue: every CTA stores its partial tile as [token][128 rows]
    (bn tokens, within the ring); CTA z of ks then finishes rows [z 128 / ks, (z + 1) 128 / ks) for
    the tile's ntok tokens, thread idx taking token idx / rpc and row z rpc + idx % rpc. Every
    (token, row) of the tile is finished exactly once, and every read stays inside the stored
    partial tile."""
    rpc = 128 // ks
    seen = set()
    for z in range(ks):
        for idx in range(rpc * ntok):
            t, rr = idx // rpc, z * rpc + idx % rpc
            assert 0 <= t < ntok <= bn and 0 <= rr < 128
            off = t * 128 + rr
            assert 0 <= off < bn * 128
            assert (t, rr) not in seen
            seen.add((t, rr))
    assert len(seen) == ntok * 128
    assert bn * 128 * 4 <= 4 * (16 * 1024 + 256 * 128)          # the one-CTA shape's 4-stage ring
