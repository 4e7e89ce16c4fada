"""GPU parity: pifa_forward (through the C ABI) against the fp64 oracle on the same bf16 operands.

Tolerance (bf16 operands, fp32 accumulation, bf16 output): relative Frobenius error <= 5e-3 and
|err| <= 2e-2 * (|ref| + 1) per element. Large outputs are checked on a seeded sample of token
rows (rows of Y are independent in Algorithm 2). Every call runs with guard bands around Y
(sentinel rows before and after, sentinel padding columns when ldy > m) and Y pre-filled with
NaN, so a missed or stray write fails the test.

Layers: the oracle's own compression where it is quick (tiny: plain greedy loop; up to
4096 x 4096: the LAPACK pivoted-QR route); the library's host compression for the 7B MLP and
70B q/o shapes and the library's GPU compression for the 28672 x 8192 shape, each checked against
Eq. 1 and Eq. 2 in fp64 on sampled rows; and randomly drawn layers (inputs.synthetic_layer) where
only the kernels' tiling matters (many tiles, ragged K, grouped layers).
"""
import functools

import numpy as np
import pytest
import torch

import oracle
from paper_2501_19090_gb300 import inputs
from paper_2501_19090_gb300 import pifa as P

pytestmark = pytest.mark.gpu

REL_FRO = 5e-3
ELEM = 2e-2
SENTINEL = -16384.0   # exactly representable in bf16 (a power of two)


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    P.load()
    yield


DEV = torch.device("cuda:0")


class Layer:
    def __init__(self, pivots, nonpivots, Wp, C, name, c_dtype="bf16"):
        self.pivots = np.asarray(pivots, np.int64)
        self.nonpivots = np.asarray(nonpivots, np.int64)
        self.Wp = inputs.round_bf16(Wp)          # the exact operand values both sides use
        self.c_dtype = c_dtype
        self.C = inputs.round_bf16(C) if c_dtype == "bf16" else inputs.round_fp16(C)
        self.m = self.pivots.size + self.nonpivots.size
        self.r, self.n = self.Wp.shape
        self.name = name
        self._dev = None

    def dev(self, ldwp=None, ldc=None):
        """Device copies (bf16 / int32); optional padded pitches with NaN in the padding."""
        Wp = _pad_dev(self.Wp, ldwp)
        cdt = torch.bfloat16 if self.c_dtype == "bf16" else torch.float16
        C = _pad_dev(self.C, ldc, cdt) if self.C.size else torch.empty((0, self.r), dtype=cdt, device=DEV)
        piv = torch.from_numpy(self.pivots.astype(np.int32)).to(DEV)
        nonp = torch.from_numpy(self.nonpivots.astype(np.int32)).to(DEV)
        return Wp, C, piv, nonp


def _round8(v):
    return (v + 7) // 8 * 8


def _pad_dev(a32, ld=None, dtype=torch.bfloat16):
    """Device copy (bf16 or fp16; values already exact in that type) with row pitch ld (default:
    cols rounded up to 8, the 16-byte rule) and NaN in the padding."""
    rows, cols = a32.shape
    ld = ld or _round8(cols)
    buf = torch.full((rows, ld), float("nan"), dtype=dtype, device=DEV)
    buf[:, :cols] = torch.from_numpy(np.ascontiguousarray(a32)).to(DEV).to(dtype)
    return buf[:, :cols]


@functools.lru_cache(maxsize=None)
def _compressed(m, n, r, seed, source):
    U, V, _ = inputs.make_factors(m, n, r, seed)
    if source == "oracle_greedy":
        L = oracle.compress(U, V, r, "greedy")
        return L.pivots, L.nonpivots, L.Wp, L.C
    if source == "oracle_lapack":
        L = oracle.compress(U, V, r, "lapack")
        return L.pivots, L.nonpivots, L.Wp, L.C
    if source == "library":
        piv, nonp, Wp, C, _ = P.pifa_compress(U, V, r)
        # the oracle checks Eq. 1 and Eq. 2 on a sample of rows of W' = U V^T
        rows = inputs.random_rows(m - r, 64, seed) if m > r else np.zeros(0, np.int64)
        Vd = V.astype(np.float64)
        Wnp_s = U[nonp[rows]].astype(np.float64) @ Vd.T
        Wp_ref = U[piv].astype(np.float64) @ Vd.T
        assert np.abs(Wp - Wp_ref).max() <= 1e-12 * np.abs(Wp_ref).max()
        if rows.size:
            err = np.linalg.norm(C[rows] @ Wp - Wnp_s) / np.linalg.norm(Wnp_s)
            assert err <= 1e-10
        assert P.pifa_validate_indices(piv, nonp, m, r) == P.PIFA_OK
        return piv, nonp, Wp, C
    if source == "gpu":
        # the library's GPU compression (Algorithm 1 on the device); Eq. 1 and Eq. 2 checked in fp64
        # on the host on sampled rows
        Ud = torch.from_numpy(U.astype(np.float64)).to(DEV)
        Vd = torch.from_numpy(V.astype(np.float64)).to(DEV)
        piv_d, nonp_d, Wp_d, C_d, _ = P.pifa_compress_device(Ud, Vd)
        piv, nonp = piv_d.cpu().numpy(), nonp_d.cpu().numpy()
        Wp, C = Wp_d.cpu().numpy(), C_d.cpu().numpy()
        del Ud, Vd, Wp_d, C_d
        assert P.pifa_validate_indices(piv, nonp, m, r) == P.PIFA_OK
        rows = inputs.random_rows(m - r, 48, seed)
        Vd64 = V.astype(np.float64)
        Wnp_s = U[nonp[rows]].astype(np.float64) @ Vd64.T
        pr = inputs.random_rows(r, 16, seed)
        Wp_ref = U[piv[pr]].astype(np.float64) @ Vd64.T
        assert np.abs(Wp[pr] - Wp_ref).max() <= 1e-12 * np.abs(Wp_ref).max()
        assert np.linalg.norm(C[rows] @ Wp - Wnp_s) / np.linalg.norm(Wnp_s) <= 1e-10
        return piv, nonp, Wp, C
    if source == "synthetic":
        return inputs.synthetic_layer(m, n, r, seed)
    raise ValueError(source)


@functools.lru_cache(maxsize=None)
def layer_for(m, n, r, seed, source, c_dtype="bf16"):
    piv, nonp, Wp, C = _compressed(m, n, r, seed, source)
    return Layer(piv, nonp, Wp, C, f"{m}x{n}r{r}/{source}/C-{c_dtype}", c_dtype)


def acts(T, n, seed):
    rng = np.random.default_rng(1000 + seed)
    return inputs.make_activations(rng, T, n, "bf16")


def run(layer, X32, variant=P.PIFA_VARIANT_AUTO, ldx=None, ldy_pad=8, guard_rows=3, ldwp=None, ldc=None,
        stream=None, workspace_tensor=None):
    """pifa_forward with NaN-filled Y inside sentinel guard bands; returns Y (T x m) as float32."""
    T = X32.shape[0]
    m = layer.m
    Wp, C, piv, nonp = layer.dev(ldwp, ldc)
    X = _pad_dev(X32, ldx) if T else torch.empty((0, layer.n), dtype=torch.bfloat16, device=DEV)
    ldy = _round8(m + ldy_pad)
    big = torch.full((T + 2 * guard_rows, ldy), SENTINEL, dtype=torch.bfloat16, device=DEV)
    Y = big[guard_rows:guard_rows + T, :m]
    Y.fill_(float("nan"))
    P.pifa_forward(X, Wp, C, piv, nonp, Y=Y, variant=variant, stream=stream, workspace_tensor=workspace_tensor)
    st = P.pifa_device_status(stream)
    assert st == P.PIFA_OK, P.pifa_status_string(st)
    host = big.float().cpu().numpy()
    assert np.all(host[:guard_rows] == SENTINEL) and np.all(host[guard_rows + T:] == SENTINEL), "guard rows hit"
    assert np.all(host[:, m:] == SENTINEL), "padding columns of Y were written"
    out = host[guard_rows:guard_rows + T, :m]
    assert not np.isnan(out).any(), "some output element was never written"
    return out


def check(got, ref, what=""):
    got = got.astype(np.float64)
    denom = np.linalg.norm(ref)
    rel = np.linalg.norm(got - ref) / denom if denom > 0 else np.linalg.norm(got)
    elem = np.max(np.abs(got - ref) / (np.abs(ref) + 1.0)) if ref.size else 0.0
    assert rel <= REL_FRO and elem <= ELEM, f"{what}: rel_fro {rel:.3e} (<= {REL_FRO}), elem {elem:.3e} (<= {ELEM})"
    return rel, elem


def parity(layer, T, variant=P.PIFA_VARIANT_AUTO, sample=None, seed=0, **kw):
    X = acts(T, layer.n, seed)
    Y = run(layer, X, variant, **kw)
    rows = np.arange(T) if (sample is None or sample >= T) else inputs.random_rows(T, sample, seed)
    ref = oracle.forward(X[rows], layer.Wp, layer.C, layer.pivots, layer.nonpivots)
    return check(Y[rows], ref, f"{layer.name} T={T} variant={P.pifa_variant_name(variant)}")


# ---------------------------------------------------------------------------------------------
# the five workloads
# ---------------------------------------------------------------------------------------------
def test_tiny_layer_decode_and_prefill():
    L = layer_for(256, 256, 128, 0, "oracle_greedy")
    parity(L, 16, P.PIFA_VARIANT_DECODE)
    parity(L, 16, P.PIFA_VARIANT_PREFILL_SPLIT)
    parity(L, 16)


@pytest.mark.parametrize("T", [1, 8])
def test_attn7b_decode(T):
    L = layer_for(4096, 4096, 2048, 0, "oracle_lapack")
    assert P.pifa_select_variant(T, 4096, 4096, 2048) == P.PIFA_VARIANT_DECODE
    parity(L, T)


@pytest.mark.parametrize("T,sample", [(2048, None), (8192, 512)])
def test_attn7b_prefill(T, sample):
    L = layer_for(4096, 4096, 2048, 0, "oracle_lapack")
    parity(L, T, sample=sample)


@pytest.mark.parametrize("frac", [0.25, 0.4, 0.6, 0.75])
def test_rank_sweep_prefill(frac):
    r = int(np.floor(frac * 4096 + 0.5))
    L = layer_for(4096, 4096, r, 0, "oracle_lapack")
    parity(L, 2048, sample=768)


@pytest.mark.parametrize("T", [1, 2048])
def test_mlp7b_three_layers_back_to_back(T):
    gate = layer_for(11008, 4096, 2048, 0, "library")
    up = layer_for(11008, 4096, 2048, 1, "library")
    down = layer_for(4096, 11008, 2048, 2, "library")
    Xg = acts(T, 4096, 0)
    Xd = acts(T, 11008, 2)      # the down projection gets its own N(0,1) input (no SwiGLU here)
    stream = torch.cuda.Stream()
    outs = [run(gate, Xg, stream=stream), run(up, Xg, stream=stream), run(down, Xd, stream=stream)]
    rows = np.arange(T) if T <= 512 else inputs.random_rows(T, 384, 0)
    for L, X, Y in zip((gate, up, down), (Xg, Xg, Xd), outs):
        ref = oracle.forward(X[rows], L.Wp, L.C, L.pivots, L.nonpivots)
        check(Y[rows], ref, f"{L.name} T={T}")


@pytest.mark.parametrize("T", [1, 8, 16, 80, 128, 4096])
def test_llama70b_qo(T):
    L = layer_for(8192, 8192, 4096, 0, "library")
    parity(L, T, sample=256)


@pytest.mark.parametrize("T", [4, 16])
def test_llama70b_qo_persistent_grid(T):
    """The persistent decode grid forced on the 70B q/o layer: chunks on which some warps have no
    step, several chunks per tile, three or more tiles per cluster of up to eight CTAs (both
    receive buffers reused)."""
    L = layer_for(8192, 8192, 4096, 0, "library")
    P.pifa_set_decode_grid(P.PIFA_DECODE_GRID_PERSISTENT)
    try:
        parity(L, T, P.PIFA_VARIANT_DECODE)
    finally:
        P.pifa_set_decode_grid(P.PIFA_DECODE_GRID_AUTO)


@pytest.mark.parametrize("T", [1, 8, 16, 80, 128, 4096])
def test_llama70b_gate_up(T):
    """The 28672 x 8192, r = 4096 layer as Algorithm 1 makes it from Gaussian U V^T (compressed on
    the GPU): its C cancels heavily, the case that makes the hi + lo split of y_p necessary."""
    L = layer_for(28672, 8192, 4096, 0, "gpu")
    parity(L, T, sample=128)


@pytest.mark.parametrize("T", [1, 3, 8, 16])
@pytest.mark.parametrize("grid", [P.PIFA_DECODE_GRID_PERSISTENT, P.PIFA_DECODE_GRID_WAVES])
def test_decode_grids_many_tiles_ragged(T, grid):
    """Both decode layouts on a layer with more row tiles than co-resident clusters: the
    persistent grid (every cluster streaming several tiles through its TMA-filled stage ring) and
    waves of one-tile clusters; ragged K in both phases (520 and 264 columns), a partial last
    tile."""
    L = layer_for(40000, 520, 264, 3, "synthetic")
    P.pifa_set_decode_grid(grid)
    try:
        parity(L, T, P.PIFA_VARIANT_DECODE)
    finally:
        P.pifa_set_decode_grid(P.PIFA_DECODE_GRID_AUTO)


@pytest.mark.parametrize("T", [2, 8, 16])
def test_decode_persistent_grid_fp16_c_and_padding(T):
    """The persistent decode grid with C stored in fp16 (its TMA map in C's type), on padded
    pitches that hold NaN (the TMA boxes must not read past K)."""
    L = layer_for(3000, 1000, 600, 4, "synthetic", "fp16")
    P.pifa_set_decode_grid(P.PIFA_DECODE_GRID_PERSISTENT)
    try:
        parity(L, T, P.PIFA_VARIANT_DECODE, ldx=1000 + 24, ldwp=1000 + 40, ldc=600 + 16)
    finally:
        P.pifa_set_decode_grid(P.PIFA_DECODE_GRID_AUTO)


@pytest.mark.parametrize("T", [1, 3, 8, 16, 17, 33, 64, 65, 128])
def test_decode_splitk_tensor_cores_ragged(T):
    """The split-K tensor-core decode form forced on a layer with ragged K in both phases (520 and
    264 columns: partial 64-column chunks and K-slices), a partial last 128-row block in phase 1
    (264 rows) and many units per CTA in phase 2 (39736 rows). T = 17, 33 and 65 fill token tiles
    of 32, 64 and 128 rows only partly; T = 64 and 128 fill theirs. 128-token tiles need the
    row-block plan (at most 296 blocks per phase), so above T = 64 the layer has 30000 rows (233
    blocks in phase 2)."""
    L = layer_for(40000, 520, 264, 3, "synthetic") if T <= 64 else layer_for(30000, 520, 264, 3, "synthetic")
    P.pifa_set_decode_grid(P.PIFA_DECODE_GRID_SPLITK)
    try:
        parity(L, T, P.PIFA_VARIANT_DECODE)
    finally:
        P.pifa_set_decode_grid(P.PIFA_DECODE_GRID_AUTO)


@pytest.mark.parametrize("T", [1, 8, 16, 32, 64, 96, 128])
def test_decode_splitk_tensor_cores_compressed_layers(T):
    """The split-K form on compressed layers (C that cancels): 7B attention and the 70B gate/up
    layer, and C stored as fp16 (fp16 MMAs in phase 2, fp16 hi/lo planes) on padded pitches."""
    P.pifa_set_decode_grid(P.PIFA_DECODE_GRID_SPLITK)
    try:
        parity(layer_for(4096, 4096, 2048, 0, "oracle_lapack"), T, P.PIFA_VARIANT_DECODE)
        parity(layer_for(28672, 8192, 4096, 0, "gpu"), T, P.PIFA_VARIANT_DECODE, sample=128)
        parity(layer_for(3000, 1000, 600, 4, "synthetic", "fp16"), T, P.PIFA_VARIANT_DECODE,
               ldx=1000 + 24, ldwp=1000 + 40, ldc=600 + 16)
    finally:
        P.pifa_set_decode_grid(P.PIFA_DECODE_GRID_AUTO)


def test_decode_splitk_deterministic_and_r_equals_m():
    L = layer_for(4096, 4096, 2048, 0, "oracle_lapack")
    P.pifa_set_decode_grid(P.PIFA_DECODE_GRID_SPLITK)
    try:
        X = acts(16, 4096, 5)
        assert np.array_equal(run(L, X, P.PIFA_VARIANT_DECODE), run(L, X, P.PIFA_VARIANT_DECODE))
        parity(layer_for(64, 128, 64, 4, "oracle_greedy"), 9, P.PIFA_VARIANT_DECODE)
        parity(layer_for(40, 48, 1, 5, "oracle_greedy"), 12, P.PIFA_VARIANT_DECODE)
        X = acts(48, 4096, 5)
        assert np.array_equal(run(L, X, P.PIFA_VARIANT_DECODE), run(L, X, P.PIFA_VARIANT_DECODE))
        parity(layer_for(64, 128, 64, 4, "oracle_greedy"), 40, P.PIFA_VARIANT_DECODE)
        parity(layer_for(40, 48, 1, 5, "oracle_greedy"), 64, P.PIFA_VARIANT_DECODE)
        X = acts(128, 4096, 5)
        assert np.array_equal(run(L, X, P.PIFA_VARIANT_DECODE), run(L, X, P.PIFA_VARIANT_DECODE))
        parity(layer_for(64, 128, 64, 4, "oracle_greedy"), 100, P.PIFA_VARIANT_DECODE)
        parity(layer_for(40, 48, 1, 5, "oracle_greedy"), 128, P.PIFA_VARIANT_DECODE)
    finally:
        P.pifa_set_decode_grid(P.PIFA_DECODE_GRID_AUTO)


@pytest.mark.parametrize("m,n,r,T,forced", [
    (8192, 4096, 4096, 8, P.PIFA_DECODE_GRID_SPLITK),  # both phases 4096 rows, T > 2
    (8192, 4096, 4096, 16, P.PIFA_DECODE_GRID_SPLITK),
    (4096, 4096, 2048, 8, P.PIFA_DECODE_GRID_WAVES),   # 2048-row phases, at most two waves each
])
def test_decode_selector_matches_the_form_it_picks(m, n, r, T, forced):
    """The automatic decode choice is keyed on each phase's rows and T: split-K on the tensor cores
    for phases of at least 32 blocks of 128 rows when T > 2, waves of one-tile clusters for a
    phase that fits two waves. Its output equals, bit for bit, that of the form it should pick,
    forced."""
    L = layer_for(m, n, r, 6, "synthetic")
    X = acts(T, n, 6)
    auto = run(L, X, P.PIFA_VARIANT_DECODE)
    P.pifa_set_decode_grid(forced)
    try:
        assert np.array_equal(auto, run(L, X, P.PIFA_VARIANT_DECODE))
    finally:
        P.pifa_set_decode_grid(P.PIFA_DECODE_GRID_AUTO)


def test_launch_count_per_call():
    """pifa_launch_count: a split-K decode call whose phases take the row-block plan (both phases
    of 4096 rows, T = 8: clusters of 8 CTAs that add up their K-slices themselves) enqueues two
    kernels, one whose phase 2 has more 128-row blocks than the grid holds (39736 rows) three (a
    partial and a reduce kernel for it), a waves decode call on 2048-row phases two; replaying a
    captured call launches nothing through the library."""
    big, small = layer_for(8192, 4096, 4096, 6, "synthetic"), layer_for(4096, 4096, 2048, 6, "synthetic")
    long_ = layer_for(40000, 520, 264, 3, "synthetic")
    for L, n_k in ((big, 2), (small, 2), (long_, 3)):
        X = acts(8, L.n, 6)
        run(L, X, P.PIFA_VARIANT_DECODE)  # first call: per-shape setup out of the way
        c0 = P.pifa_launch_count()
        run(L, X, P.PIFA_VARIANT_DECODE)
        assert P.pifa_launch_count() - c0 == n_k, L.name
    Wp, C, piv, nonp = small.dev(None, None)
    Xd = torch.from_numpy(acts(8, small.n, 7)).to(DEV, torch.bfloat16)
    Y = torch.empty((8, small.m), dtype=torch.bfloat16, device=DEV)
    ws = P.workspace(P.pifa_workspace_size(8, small.m, small.n, small.r, P.PIFA_VARIANT_DECODE), DEV)
    stream = torch.cuda.Stream()
    P.pifa_forward(Xd, Wp, C, piv, nonp, Y=Y, variant=P.PIFA_VARIANT_DECODE, workspace_tensor=ws, stream=stream)
    stream.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        P.pifa_forward(Xd, Wp, C, piv, nonp, Y=Y, variant=P.PIFA_VARIANT_DECODE, workspace_tensor=ws, stream=stream)
    c0 = P.pifa_launch_count()
    with torch.cuda.stream(stream):
        for _ in range(3):
            g.replay()
    stream.synchronize()
    assert P.pifa_launch_count() == c0
    assert P.pifa_device_status(stream) == P.PIFA_OK


# ---------------------------------------------------------------------------------------------
# edge cases
# ---------------------------------------------------------------------------------------------
@pytest.mark.parametrize("T", [1, 3, 13, 16, 17, 40, 64, 65, 100, 128, 129, 300])
def test_ragged_shapes_all_variants(T):
    L = layer_for(300, 200, 77, 3, "oracle_greedy")
    variants = [P.PIFA_VARIANT_PREFILL_SPLIT] + ([P.PIFA_VARIANT_DECODE] if T <= 128 else [])
    for v in variants:
        parity(L, T, v)


@pytest.mark.parametrize("variant", [P.PIFA_VARIANT_DECODE, P.PIFA_VARIANT_PREFILL_SPLIT])
def test_full_rank_r_equals_m(variant):
    L = layer_for(64, 128, 64, 4, "oracle_greedy")
    assert L.C.shape == (0, 64)
    parity(L, 9, variant)


@pytest.mark.parametrize("variant", [P.PIFA_VARIANT_DECODE, P.PIFA_VARIANT_PREFILL_SPLIT])
def test_rank_one(variant):
    L = layer_for(40, 48, 1, 5, "oracle_greedy")
    parity(L, 12, variant)


@pytest.mark.parametrize("variant", [P.PIFA_VARIANT_DECODE, P.PIFA_VARIANT_PREFILL_SPLIT])
def test_padded_pitches_ignore_padding(variant):
    """ldx > n, ldwp > n, ldc > r and ldy > m with NaN in the input padding: never read."""
    L = layer_for(256, 256, 128, 0, "oracle_greedy")
    parity(L, 11, variant, ldx=264, ldwp=272, ldc=136, ldy_pad=24)


def test_zero_tokens_is_a_noop():
    L = layer_for(256, 256, 128, 0, "oracle_greedy")
    Wp, C, piv, nonp = L.dev()
    X = torch.empty((0, 256), dtype=torch.bfloat16, device=DEV)
    Y = torch.empty((0, 256), dtype=torch.bfloat16, device=DEV)
    P.pifa_forward(X, Wp, C, piv, nonp, Y=Y)
    assert P.pifa_device_status() == P.PIFA_OK


def test_deterministic_bitwise():
    L = layer_for(4096, 4096, 2048, 0, "oracle_lapack")
    X = acts(300, 4096, 7)
    for v in (P.PIFA_VARIANT_PREFILL_SPLIT,):
        a = run(L, X, v)
        b = run(L, X, v)
        assert np.array_equal(a, b)
    Xs = acts(8, 4096, 7)
    assert np.array_equal(run(L, Xs, P.PIFA_VARIANT_DECODE), run(L, Xs, P.PIFA_VARIANT_DECODE))


@pytest.mark.parametrize("variant", [P.PIFA_VARIANT_DECODE, P.PIFA_VARIANT_PREFILL_SPLIT])
def test_out_of_range_index_is_reported_not_written(variant):
    """A pivot index >= m is caught by the kernels' own bounds check: the write is skipped and
    PIFA_ERR_DEVICE_INDEX is latched; nothing outside Y changes."""
    L = layer_for(256, 256, 128, 0, "oracle_greedy")
    Wp, C, piv, nonp = L.dev()
    bad = piv.clone()
    bad[5] = 256                              # == m: out of range
    X = _pad_dev(acts(4, 256, 0))
    big = torch.full((4 + 6, 256 + 8), SENTINEL, dtype=torch.bfloat16, device=DEV)
    Y = big[3:7, :256]
    P.pifa_forward(X, Wp, C, bad, nonp, Y=Y, variant=variant)
    assert P.pifa_device_status() == P.PIFA_ERR_DEVICE_INDEX
    assert P.pifa_device_status() == P.PIFA_OK           # cleared by the read
    host = big.float().cpu().numpy()
    assert np.all(host[:3] == SENTINEL) and np.all(host[7:] == SENTINEL) and np.all(host[:, 256:] == SENTINEL)


def test_prefill_variants_agree_with_decode_at_t16():
    L = layer_for(4096, 4096, 2048, 0, "oracle_lapack")
    X = acts(16, 4096, 3)
    a = run(L, X, P.PIFA_VARIANT_DECODE)
    b = run(L, X, P.PIFA_VARIANT_PREFILL_SPLIT)
    ref = oracle.forward(X, L.Wp, L.C, L.pivots, L.nonpivots)
    check(a, ref, "decode")
    check(b, ref, "prefill_split")


# ---------------------------------------------------------------------------------------------
# C stored as fp16: decode and split prefill (hi + lo planes of fp16)
# ---------------------------------------------------------------------------------------------
SPLIT = P.PIFA_VARIANT_PREFILL_SPLIT


def test_fp16_c_tiny_all_variants():
    L = layer_for(256, 256, 128, 0, "oracle_greedy", "fp16")
    for v in (P.PIFA_VARIANT_DECODE, SPLIT):
        parity(L, 16, v)


@pytest.mark.parametrize("T", [1, 8, 16])
def test_fp16_c_attn7b_decode(T):
    parity(layer_for(4096, 4096, 2048, 0, "oracle_lapack", "fp16"), T)


def test_selector_picks_split_prefill():
    assert P.pifa_select_variant(2048, 4096, 4096, 2048, P.PIFA_DTYPE_FP16) == SPLIT, P.pifa_last_error()
    assert P.pifa_select_variant(2048, 4096, 4096, 2048, P.PIFA_DTYPE_BF16) == SPLIT, P.pifa_last_error()
    assert P.pifa_select_variant(16, 4096, 4096, 2048, P.PIFA_DTYPE_BF16) == P.PIFA_VARIANT_DECODE
    assert P.pifa_select_variant(64, 4096, 4096, 2048, P.PIFA_DTYPE_BF16) == P.PIFA_VARIANT_DECODE
    assert P.pifa_select_variant(96, 4096, 4096, 2048, P.PIFA_DTYPE_BF16) == SPLIT      # 16 non-pivot blocks
    assert P.pifa_select_variant(128, 28672, 8192, 4096, P.PIFA_DTYPE_BF16) == P.PIFA_VARIANT_DECODE  # 192
    assert P.pifa_select_variant(129, 28672, 8192, 4096, P.PIFA_DTYPE_BF16) == SPLIT
    assert P.pifa_select_variant(100, 40000, 520, 264, P.PIFA_DTYPE_BF16) == SPLIT  # 311 row blocks


@pytest.mark.parametrize("T,sample", [(2048, None), (8192, 512), (300, None), (17, None)])
def test_fp16_c_attn7b_split(T, sample):
    parity(layer_for(4096, 4096, 2048, 0, "oracle_lapack", "fp16"), T, SPLIT, sample=sample)


@pytest.mark.parametrize("frac", [0.25, 0.4, 0.6, 0.75])
def test_fp16_c_rank_sweep_split(frac):
    r = int(np.floor(frac * 4096 + 0.5))
    parity(layer_for(4096, 4096, r, 0, "oracle_lapack", "fp16"), 2048, SPLIT, sample=512)


@pytest.mark.parametrize("T", [1, 2048])
def test_fp16_c_mlp7b(T):
    for m, n, seed in ((11008, 4096, 0), (4096, 11008, 2)):
        parity(layer_for(m, n, 2048, seed, "library", "fp16"), T, sample=384)


@pytest.mark.parametrize("T", [16, 4096])
def test_fp16_c_llama70b(T):
    parity(layer_for(8192, 8192, 4096, 0, "library", "fp16"), T, sample=256)
    parity(layer_for(28672, 8192, 4096, 0, "gpu", "fp16"), T, sample=128)


@pytest.mark.parametrize("T", [1, 17, 40, 64, 100, 128, 300, 513])
def test_fp16_c_ragged_split_and_decode(T):
    L = layer_for(300, 200, 77, 3, "oracle_greedy", "fp16")
    for v in ([SPLIT] if T > 128 else [P.PIFA_VARIANT_DECODE, SPLIT]):
        parity(L, T, v)


@pytest.mark.parametrize("variant", [P.PIFA_VARIANT_DECODE, SPLIT])
def test_fp16_c_full_rank_and_rank_one(variant):
    parity(layer_for(64, 128, 64, 4, "oracle_greedy", "fp16"), 16 if variant == P.PIFA_VARIANT_DECODE else 40,
           variant)
    parity(layer_for(40, 48, 1, 5, "oracle_greedy", "fp16"), 12, variant)


def test_fp16_c_split_deterministic_and_padded():
    L = layer_for(4096, 4096, 2048, 0, "oracle_lapack", "fp16")
    X = acts(600, 4096, 7)
    a = run(L, X, SPLIT)
    b = run(L, X, SPLIT, ldx=4104, ldwp=4112, ldc=2056, ldy_pad=24)
    assert np.array_equal(a, b)


# ---------------------------------------------------------------------------------------------
# failure detection without a GPU fault
# ---------------------------------------------------------------------------------------------
def test_wait_timeout_is_reported_and_recoverable():
    """Failure detection without a GPU fault: a kernel waits, with a 2 ms bound, on an mbarrier
    that nothing arrives on. The wait runs out, PIFA_ERR_TIMEOUT is latched and read back, the
    context stays usable, and a forward pass right after is correct."""
    L = layer_for(256, 256, 128, 0, "oracle_greedy")
    try:
        P.pifa_set_wait_timeout(2_000_000)
        P.pifa_selftest_wait_timeout()
        assert P.pifa_device_status() == P.PIFA_ERR_TIMEOUT
        assert P.pifa_device_status() == P.PIFA_OK       # read-and-clear
    finally:
        P.pifa_set_wait_timeout(0)
    for v in (P.PIFA_VARIANT_DECODE, P.PIFA_VARIANT_PREFILL_SPLIT):
        parity(L, 16, v)


def test_workspace_needs_no_initialisation_and_is_shared():
    """One caller workspace, filled with 0xFF bytes (NaN as bf16 and fp16) and never cleared, serves
    decode at several T, then prefill, then decode again: no call depends on its contents."""
    L = layer_for(300, 200, 77, 3, "oracle_greedy")
    cases = ((8, P.PIFA_VARIANT_DECODE), (1, P.PIFA_VARIANT_DECODE), (100, SPLIT), (16, P.PIFA_VARIANT_DECODE),
             (300, SPLIT), (3, P.PIFA_VARIANT_DECODE))
    need = max(P.pifa_workspace_size(T, L.m, L.n, L.r, v) for T, v in cases)
    ws = torch.full((need,), 0xFF, dtype=torch.uint8, device=DEV)
    for T, v in cases:
        parity(L, T, v, workspace_tensor=ws)


# ---------------------------------------------------------------------------------------------
# grouped layers sharing X (pifa_forward_grouped)
# ---------------------------------------------------------------------------------------------
def run_grouped(layers, X32, pad=8):
    """pifa_forward_grouped over `layers` (one shape) stacked by rows; Y (T x G m) inside a
    NaN-filled buffer whose padding columns hold a sentinel. Returns Y as float32."""
    G = len(layers)
    L0 = layers[0]
    m, r = L0.m, L0.r
    Wp = torch.cat([L.dev()[0] for L in layers])
    C = torch.cat([L.dev()[1] for L in layers])
    piv = torch.cat([L.dev()[2] + g * m for g, L in enumerate(layers)])
    nonp = torch.cat([L.dev()[3] + g * m for g, L in enumerate(layers)])
    T = X32.shape[0]
    X = _pad_dev(X32)
    ldy = _round8(G * m + pad)
    big = torch.full((T, ldy), SENTINEL, dtype=torch.bfloat16, device=DEV)
    Y = big[:, :G * m]
    Y.fill_(float("nan"))
    P.pifa_forward_grouped(G, X, Wp, C, piv, nonp, Y=Y)
    st = P.pifa_device_status(None)
    assert st == P.PIFA_OK, P.pifa_status_string(st)
    host = big.float().cpu().numpy()
    assert np.all(host[:, G * m:] == SENTINEL), "padding columns of Y were written"
    out = host[:, :G * m]
    assert not np.isnan(out).any(), "some output element was never written"
    return out


def grouped_parity(layers, T, sample=None, seed=0):
    X = acts(T, layers[0].n, seed)
    Y = run_grouped(layers, X)
    m = layers[0].m
    rows = np.arange(T) if (sample is None or sample >= T) else inputs.random_rows(T, sample, seed)
    for g, L in enumerate(layers):
        ref = oracle.forward(X[rows], L.Wp, L.C, L.pivots, L.nonpivots)
        check(Y[rows, g * m:(g + 1) * m], ref, f"group {g} of {len(layers)} ({L.name}) T={T}")


@pytest.mark.parametrize("G", [2, 3])
@pytest.mark.parametrize("T", [1, 3, 8, 16, 40, 64, 100, 128, 300])
def test_grouped_layers_match_per_layer_oracle(G, T):
    """G synthetic layers of one shape (m - r = 7 x 128, ragged n) sharing X: each group's block of
    Y equals the oracle's forward of that layer alone (decode for T <= 64, split prefill above)."""
    layers = [layer_for(1408, 1000, 512, 10 + g, "synthetic") for g in range(G)]
    grouped_parity(layers, T)


@pytest.mark.parametrize("T", [2, 8, 16, 48])
@pytest.mark.parametrize("grid", [P.PIFA_DECODE_GRID_PERSISTENT, P.PIFA_DECODE_GRID_WAVES,
                                  P.PIFA_DECODE_GRID_SPLITK])
def test_grouped_layers_both_decode_grids(T, grid):
    """Grouped decode under both layouts; the persistent grid keeps every group's K range of y_p
    resident (T <= 2) or stages the tile's group's columns (T > 2)."""
    layers = [layer_for(1408, 1000, 512, 20 + g, "synthetic") for g in range(2)]
    P.pifa_set_decode_grid(grid)
    try:
        grouped_parity(layers, T)
    finally:
        P.pifa_set_decode_grid(P.PIFA_DECODE_GRID_AUTO)


@pytest.mark.parametrize("T,sample", [(1, None), (8, None), (2048, 256)])
def test_grouped_mlp7b_gate_up(T, sample):
    """The 7B MLP's gate and up projections (11008 x 4096, r = 2048, m - r = 70 x 128) as one grouped
    call on a shared X."""
    layers = [layer_for(11008, 4096, 2048, 0, "library"), layer_for(11008, 4096, 2048, 1, "library")]
    grouped_parity(layers, T, sample=sample)


# ---------------------------------------------------------------------------------------------
# split prefill: many tiles per GEMM
# ---------------------------------------------------------------------------------------------
@pytest.mark.parametrize("T", [17, 300, 1000])
def test_prefill_many_tiles_ragged(T):
    """Split prefill on a layer whose GEMM 2 spans several waves of tiles (m - r = 39736 rows: 311
    row tiles, the last one partial); ragged K in both GEMMs (520 and 264)."""
    L = layer_for(40000, 520, 264, 3, "synthetic")
    parity(L, T, P.PIFA_VARIANT_PREFILL_SPLIT, sample=192)


@pytest.mark.parametrize("T", [40, 700])
def test_prefill_fp16_c_padding_rank_not_multiple_of_64(T):
    """Split prefill with C in fp16 (the single fp16 y_p pass, range check in the GEMM 1 epilogue)
    on padded pitches holding NaN, with a rank (600) that leaves a partial 64-column K chunk."""
    L = layer_for(3000, 1000, 600, 4, "synthetic", "fp16")
    parity(L, T, P.PIFA_VARIANT_PREFILL_SPLIT, ldx=1000 + 24, ldwp=1000 + 40, ldc=600 + 16)


def test_prefill_two_waves_deterministic():
    """Bitwise-identical Y over repeated calls where both GEMMs take two waves of tiles (70B q/o
    layer, T = 2048: 288 tiles each on 152 SMs), with the next GEMM launched programmatically
    while the previous one drains."""
    L = layer_for(8192, 8192, 4096, 0, "library")
    X = acts(2048, 8192, 9)
    first = run(L, X, P.PIFA_VARIANT_PREFILL_SPLIT)
    for _ in range(2):
        assert np.array_equal(run(L, X, P.PIFA_VARIANT_PREFILL_SPLIT), first)
    rows = inputs.random_rows(2048, 96, 9)
    check(first[rows], oracle.forward(X[rows], L.Wp, L.C, L.pivots, L.nonpivots), "70B q/o T=2048")


@pytest.mark.parametrize("T", [300, 1200])
def test_grouped_layers_prefill_three_groups(T):
    """Grouped prefill, three groups: GEMM 2 tiles read their group's hi/lo column range."""
    layers = [layer_for(1408, 1000, 512, 30 + g, "synthetic") for g in range(3)]
    grouped_parity(layers, T, sample=160)


# ---------------------------------------------------------------------------------------------
# back-to-back calls in a CUDA graph (the chained kernels of one call overlap the next call's)
# ---------------------------------------------------------------------------------------------
@pytest.mark.parametrize("m,n,r,T", [(4096, 4096, 2048, 8), (8192, 8192, 4096, 1), (8192, 8192, 4096, 16),
                                     (28672, 8192, 4096, 16), (4096, 4096, 2048, 40), (28672, 8192, 4096, 64),
                                     (8192, 8192, 4096, 128), (4096, 4096, 2048, 300)])
def test_graph_replay_back_to_back_matches_single_calls(m, n, r, T):
    """64 calls captured in one CUDA graph and replayed, on four rotating (X, Y) pairs that share one
    workspace: every call's kernels launch while the previous call's still run (programmatic
    dependent launch), so a call that read the shared y_p planes or partial sums too early, or
    wrote them too late, would change some output. Each Y must equal, bit for bit, the same call
    made alone. Covers the wave, split-K tensor-core and persistent decode forms (the latter with
    token tiles of 64 and 128 rows at T = 40, 64 and 128) and the prefill."""
    variant = P.PIFA_VARIANT_DECODE if T <= 128 else P.PIFA_VARIANT_PREFILL_SPLIT
    piv, nonp, Wp32, C32 = inputs.synthetic_layer(m, n, r, 40)
    L = Layer(piv, nonp, Wp32, C32, f"{m}x{n}r{r}/graph")
    Wp, C, pd, nd = L.dev()
    copies = 4
    Xs = [_pad_dev(acts(T, n, 50 + j)) for j in range(copies)]
    Ys = [torch.full((T, m), float("nan"), dtype=torch.bfloat16, device=DEV) for _ in range(copies)]
    ws = torch.empty(P.pifa_workspace_size(T, m, n, r, variant) + 512, dtype=torch.uint8, device=DEV)
    stream = torch.cuda.Stream()
    torch.cuda.synchronize()
    ref = []
    for j in range(copies):
        Yj = torch.empty((T, m), dtype=torch.bfloat16, device=DEV)
        P.pifa_forward(Xs[j], Wp, C, pd, nd, Y=Yj, workspace_tensor=ws, stream=stream, variant=variant)
        stream.synchronize()
        ref.append(Yj)

    def step(i):
        P.pifa_forward(Xs[i % copies], Wp, C, pd, nd, Y=Ys[i % copies], workspace_tensor=ws, stream=stream,
                       variant=variant)

    with torch.cuda.stream(stream):
        for i in range(4):
            step(i)
    stream.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for i in range(64):
            step(i)
    for _ in range(2):
        for Y in Ys:
            Y.fill_(float("nan"))
        torch.cuda.synchronize()
        with torch.cuda.stream(stream):
            g.replay()
        stream.synchronize()
        assert P.pifa_device_status(stream) == P.PIFA_OK
        for j in range(copies):
            assert torch.equal(Ys[j].view(torch.int16), ref[j].view(torch.int16)), f"copy {j} differs"
    del g


# ---------------------------------------------------------------------------------------------
# split prefill with split-K clusters: GEMMs of too few 256-token tiles to fill the GPU
# ---------------------------------------------------------------------------------------------
@pytest.mark.parametrize("T", [256, 200])
def test_prefill_split_k_clusters_llama70b(T):
    """70B gate/up at T = 256 (GEMM 1: 32 tiles of 256 tokens, four CTAs each over K = 8192, the
    partial tiles added in a cluster) and 70B q/o with C in fp16 at T = 200 (both GEMMs split in
    four, one 208-token tile holding 200 tokens; fp16 hi/lo planes written by the cluster sum)."""
    if T == 256:
        parity(layer_for(28672, 8192, 4096, 0, "gpu"), T, P.PIFA_VARIANT_PREFILL_SPLIT, sample=96)
    else:
        parity(layer_for(8192, 8192, 4096, 0, "library", "fp16"), T, P.PIFA_VARIANT_PREFILL_SPLIT, sample=96)


def test_prefill_split_k_clusters_ragged_and_deterministic():
    """A layer with a partial last row tile in both GEMMs (1100 and 1900 rows) and ragged K (2000 and
    1100 columns) at T = 200: each GEMM split over two CTAs (GEMM 2's slices are its hi and its lo
    pass); the same call twice gives the same bits (the slices are added in rank order)."""
    L = layer_for(3000, 2000, 1100, 4, "synthetic")
    parity(L, 200, P.PIFA_VARIANT_PREFILL_SPLIT)
    X = acts(200, 2000, 9)
    assert np.array_equal(run(L, X, P.PIFA_VARIANT_PREFILL_SPLIT), run(L, X, P.PIFA_VARIANT_PREFILL_SPLIT))
