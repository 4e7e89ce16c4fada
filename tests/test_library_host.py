"""Host-only checks of libpifa.so (no GPU): the library loads and exports every symbol that
include/pifa.h declares, the host compression (Algorithm 1) agrees with the oracle, and
argument errors are reported as status codes before anything touches a device."""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle
from paper_2501_19090_gb300 import inputs
from paper_2501_19090_gb300 import pifa as P

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "pifa.h")


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(P.LIB_PATH):
        from paper_2501_19090_gb300 import build
        build.build()
    return P.load()


def header_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?(?:int|int64_t|char|void)\s*\**\s*(pifa_\w+)\s*\(",
                                 src, flags=re.M)))


def test_exports_every_declared_symbol(lib):
    names = header_functions()
    assert len(names) >= 10
    assert set(names) == set(P.EXPORTS)
    for name in names:
        assert hasattr(lib, name), name
        assert ctypes.cast(getattr(lib, name), ctypes.c_void_p).value


def test_status_and_variant_strings(lib):
    assert P.pifa_status_string(P.PIFA_OK) == "PIFA_OK"
    assert P.pifa_status_string(P.PIFA_ERR_TIMEOUT) == "PIFA_ERR_TIMEOUT"
    assert P.pifa_variant_name(P.PIFA_VARIANT_DECODE) == "decode"
    assert "sm_103a" in P.pifa_version()


def test_decode_grid_setter(lib):
    """The decode layout knob takes the four declared modes and rejects anything else (no GPU
    work: the mode only steers later launches)."""
    for mode in (P.PIFA_DECODE_GRID_WAVES, P.PIFA_DECODE_GRID_PERSISTENT, P.PIFA_DECODE_GRID_SPLITK,
                 P.PIFA_DECODE_GRID_AUTO):
        assert lib.pifa_set_decode_grid(mode) == P.PIFA_OK
    for bad in (-1, 4, 99):
        assert lib.pifa_set_decode_grid(bad) == P.PIFA_ERR_INVALID_ARG
    assert lib.pifa_set_decode_grid(P.PIFA_DECODE_GRID_AUTO) == P.PIFA_OK


def test_grouped_workspace_and_argument_rules(lib):
    """pifa_workspace_size_grouped: y_p scratch for all groups; the grouped shape rules."""
    one = P.pifa_workspace_size(8, 1408, 1000, 512)
    assert P.pifa_workspace_size_grouped(1, 8, 1408, 1000, 512) == one
    assert P.pifa_workspace_size_grouped(3, 8, 1408, 1000, 512) > one
    assert P.pifa_workspace_size_grouped(2, 2048, 11008, 4096, 2048) >= 2 * 2048 * 4096 * 2
    assert lib.pifa_workspace_size_grouped(0, 8, 1408, 1000, 512, P.PIFA_DTYPE_BF16) == P.PIFA_ERR_INVALID_ARG
    assert lib.pifa_workspace_size_grouped(2, 8, 1400, 1000, 512, P.PIFA_DTYPE_BF16) == P.PIFA_ERR_UNSUPPORTED
    assert lib.pifa_workspace_size_grouped(2, 8, 1412, 1000, 516, P.PIFA_DTYPE_BF16) == P.PIFA_ERR_UNSUPPORTED
    assert lib.pifa_workspace_size_grouped(2, 8, 512, 1000, 512, P.PIFA_DTYPE_BF16) == P.PIFA_ERR_UNSUPPORTED
    assert lib.pifa_workspace_size_grouped(2, 0, 1408, 1000, 512, P.PIFA_DTYPE_BF16) == 0


def test_selector(lib):
    assert P.pifa_select_variant(1, 4096, 4096, 2048) == P.PIFA_VARIANT_DECODE
    assert P.pifa_select_variant(16, 28672, 8192, 4096) == P.PIFA_VARIANT_DECODE
    assert P.pifa_select_variant(2048, 4096, 4096, 2048) == P.PIFA_VARIANT_PREFILL_SPLIT
    assert P.pifa_select_variant(64, 256, 256, 128) == P.PIFA_VARIANT_DECODE
    assert P.pifa_select_variant(128, 256, 256, 128) == P.PIFA_VARIANT_PREFILL_SPLIT  # 1 non-pivot block
    assert P.pifa_select_variant(129, 256, 256, 128) == P.PIFA_VARIANT_PREFILL_SPLIT
    # 64 < T <= 128 decodes where the non-pivot rows make 148 to 296 blocks of 128 (and the pivot
    # rows at most 296)
    assert P.pifa_select_variant(100, 28672, 8192, 4096) == P.PIFA_VARIANT_DECODE       # 32 and 192
    assert P.pifa_select_variant(128, 8192, 8192, 4096) == P.PIFA_VARIANT_PREFILL_SPLIT  # 32 and 32
    assert P.pifa_select_variant(100, 40000, 520, 264) == P.PIFA_VARIANT_PREFILL_SPLIT  # 3 and 311
    assert P.pifa_select_variant(64, 40000, 520, 264) == P.PIFA_VARIANT_DECODE
    # grouped layers count their stacked rows: 70B gate + up (2 x 192 non-pivot blocks) prefill
    ws_dec = P.pifa_workspace_size(100, 28672, 8192, 4096, P.PIFA_VARIANT_DECODE)
    ws_pre = P.pifa_workspace_size(100, 28672, 8192, 4096, P.PIFA_VARIANT_PREFILL_SPLIT)
    assert P.pifa_workspace_size(100, 28672, 8192, 4096) == ws_dec
    assert ws_dec != ws_pre
    assert P.pifa_select_variant(4096, 4096, 4096, 2048, P.PIFA_DTYPE_FP16) == P.PIFA_VARIANT_PREFILL_SPLIT
    with pytest.raises(P.PifaError):
        P.pifa_select_variant(1, 100, 50, 60)      # r > n


def test_workspace_sizes(lib):
    # decode: fp32 y_p, T rows of pitch round_up(r, 8)
    # every size includes the 256 reserved bytes at the head of the workspace
    # decode: the y_p planes (two 2-byte T x round_up(r, 8) matrices), then room for the split-K
    # form's fp32 partial sums: at least one T x rows block per phase
    assert P.pifa_workspace_size(8, 4096, 4096, 2048, P.PIFA_VARIANT_DECODE) >= 256 + 8 * 2048 * 4 + 8 * 2048 * 4
    assert P.pifa_workspace_size(3, 4096, 4096, 1638, P.PIFA_VARIANT_DECODE) % 256 == 0
    assert P.pifa_workspace_size(3, 4096, 4096, 1638, P.PIFA_VARIANT_DECODE) >= 256 + 3 * 1640 * 4 + 3 * 2458 * 4
    # split prefill: Y_p hi and lo, two 2-byte T x round_up(r, 8) matrices
    assert P.pifa_workspace_size(2048, 4096, 4096, 2048, P.PIFA_VARIANT_PREFILL_SPLIT) == 256 + 2 * 2048 * 2048 * 2
    assert P.pifa_workspace_size(2048, 4096, 4096, 2048, P.PIFA_VARIANT_PREFILL_SPLIT,
                                 P.PIFA_DTYPE_FP16) == 256 + 2 * 2048 * 2048 * 2
    assert P.pifa_workspace_size(2048, 4096, 4096, 1638, P.PIFA_VARIANT_PREFILL_SPLIT,
                                 P.PIFA_DTYPE_FP16) == 256 + 2 * 2048 * 1640 * 2
    assert P.pifa_workspace_size(0, 4096, 4096, 2048, P.PIFA_VARIANT_AUTO) == 0
    with pytest.raises(P.PifaError) as e:
        P.pifa_workspace_size(4, 10, 10, 11, P.PIFA_VARIANT_AUTO)   # r > min(m, n)
    assert e.value.status == P.PIFA_ERR_INVALID_ARG


def test_validate_indices(lib):
    piv = np.array([1, 3], np.int32)
    nonp = np.array([0, 2, 4], np.int32)
    assert P.pifa_validate_indices(piv, nonp, 5, 2) == P.PIFA_OK
    assert P.pifa_validate_indices(np.array([3, 1], np.int32), nonp, 5, 2) == P.PIFA_ERR_INVALID_ARG
    assert P.pifa_validate_indices(np.array([1, 2], np.int32), nonp, 5, 2) == P.PIFA_ERR_INVALID_ARG
    assert P.pifa_validate_indices(np.array([1, 5], np.int32), np.array([0, 2, 3], np.int32), 5, 2) \
        == P.PIFA_ERR_INVALID_ARG
    assert P.pifa_validate_indices(np.arange(4, dtype=np.int32), np.zeros(0, np.int32), 4, 4) == P.PIFA_OK


def _fwd_raw(lib, **kw):
    """pifa_forward_variant with fake (never dereferenced) pointers, for argument checks only."""
    a = dict(X=0x10000, T=4, n=64, ldx=64, Wp=0x20000, r=16, ldwp=64, C=0x30000, m=48, ldc=16,
             cdt=P.PIFA_DTYPE_BF16, piv=0x40000, nonpiv=0x50000, Y=0x60000, ldy=48, ws=0x70000,
             wsb=1 << 20, variant=P.PIFA_VARIANT_AUTO)
    a.update(kw)
    return lib.pifa_forward_variant(a["X"], a["T"], a["n"], a["ldx"], a["Wp"], a["r"], a["ldwp"], a["C"],
                                    a["m"], a["ldc"], a["cdt"], a["piv"], a["nonpiv"], a["Y"], a["ldy"],
                                    a["ws"], a["wsb"], a["variant"], None)


def test_forward_argument_errors(lib):
    E = P
    assert _fwd_raw(lib, r=0) == E.PIFA_ERR_INVALID_ARG
    assert _fwd_raw(lib, r=65) == E.PIFA_ERR_INVALID_ARG            # r > n
    assert _fwd_raw(lib, T=-1) == E.PIFA_ERR_INVALID_ARG
    assert _fwd_raw(lib, X=None) == E.PIFA_ERR_INVALID_ARG
    assert _fwd_raw(lib, C=None) == E.PIFA_ERR_INVALID_ARG
    assert _fwd_raw(lib, ldx=32) == E.PIFA_ERR_INVALID_ARG
    assert _fwd_raw(lib, ldy=40) == E.PIFA_ERR_INVALID_ARG
    assert _fwd_raw(lib, X=0x10002) == E.PIFA_ERR_ALIGNMENT
    assert _fwd_raw(lib, ldwp=68) == E.PIFA_ERR_ALIGNMENT
    assert _fwd_raw(lib, Y=0x10000 + 64) == E.PIFA_ERR_INVALID_ARG   # Y overlaps X
    assert "overlap" in _last(lib)
    assert _fwd_raw(lib, variant=9) == E.PIFA_ERR_INVALID_ARG
    assert _fwd_raw(lib, cdt=7) == E.PIFA_ERR_INVALID_ARG
    assert _fwd_raw(lib, variant=P.PIFA_VARIANT_DECODE, T=129) == E.PIFA_ERR_UNSUPPORTED
    # 64 < T <= 128 only with at most 296 row blocks of 128 per phase (39984 non-pivot rows: 313)
    tall = dict(X=0x10000000, Wp=0x20000000, C=0x30000000, Y=0x40000000, ws=0x50000000, m=40000, ldy=40000,
                variant=P.PIFA_VARIANT_DECODE)
    assert _fwd_raw(lib, T=100, **tall) == E.PIFA_ERR_UNSUPPORTED
    assert "row blocks" in _last(lib)
    assert _fwd_raw(lib, T=64, wsb=0, **tall) == E.PIFA_ERR_WORKSPACE   # T <= 64 passes that rule
    assert _fwd_raw(lib, wsb=16) == E.PIFA_ERR_WORKSPACE
    assert _fwd_raw(lib, ws=None) == E.PIFA_ERR_WORKSPACE
    assert _fwd_raw(lib, ws=0x70010) == E.PIFA_ERR_ALIGNMENT
    assert _fwd_raw(lib, T=0) == E.PIFA_OK                           # no-op, no device touched
    assert _fwd_raw(lib, wsb=256) == E.PIFA_ERR_WORKSPACE             # only the reserved head


def test_forward_rejects_a_workspace_overlapping_y_or_an_input(lib):
    """The kernels write y_p into the workspace, so it may share no byte with Y or an input; the
    check runs on the host before any device access (every call here fails validation)."""
    for ws in (0x60000, 0x5ff00, 0x10000, 0x20000, 0x30000):        # Y, ends inside Y, X, W_p, C
        assert _fwd_raw(lib, ws=ws) == P.PIFA_ERR_INVALID_ARG, hex(ws)
        assert "workspace overlaps" in _last(lib)


def _last(lib):
    return lib.pifa_last_error().decode()


def test_compress_argument_errors(lib):
    U = np.zeros((4, 2))
    V = np.zeros((3, 2))
    with pytest.raises(P.PifaError) as e:
        P.pifa_compress(U, V, 2)                                      # W' = 0: rank 0 < 2
    assert e.value.status == P.PIFA_ERR_RANK_DEFICIENT
    st = lib.pifa_compress(None, None, 4, 3, 2, None, None, None, 3, None, 2, None)
    assert st == P.PIFA_ERR_INVALID_ARG


def _compare_with_oracle(m, n, r, seed, rule="greedy"):
    U, V, _ = inputs.make_factors(m, n, r, seed)
    ref = oracle.compress(U, V, r, rule)
    piv, nonp, Wp, C, info = P.pifa_compress(U, V, r)
    assert np.array_equal(piv, ref.pivots), "pivot indices differ from the oracle"
    assert np.array_equal(nonp, ref.nonpivots)
    W = oracle.form_weight(U, V)
    scale = np.abs(W).max()
    assert np.abs(Wp - ref.Wp).max() <= 1e-12 * scale
    if m > r:
        assert np.abs(C - ref.C).max() <= 1e-10 * max(1.0, np.abs(ref.C).max())
        # Eq. 2 holds for the library's own C, judged by the oracle's definition
        lay = oracle.PifaLayer(piv.astype(np.int64), nonp.astype(np.int64), Wp, C, ref.info)
        assert oracle.lossless_error(W, lay) <= 1e-10
    return info, ref


@pytest.mark.parametrize("m,n,r,seed", [(256, 256, 128, 0), (300, 200, 100, 1), (96, 160, 96, 2),
                                        (64, 64, 64, 3), (129, 77, 33, 4), (40, 40, 1, 5)])
def test_compress_matches_oracle(lib, m, n, r, seed):
    info, ref = _compare_with_oracle(m, n, r, seed)
    assert info.threads >= 1
    if ref.info.gaps.size:
        assert abs(info.min_pivot_gap - ref.info.gaps.min()) <= 1e-6


def test_compress_golden_example(lib):
    """The hand-derived example of tests/golden (rank 2, W' given directly as U V^T with V = I_3[:, :2]
    mapping): pivots {1, 3} and the rational C rows."""
    W = np.array([[1, 0, 0], [0, 2, 0], [1, 2, 0], [2, 2, 0], [0, 0, 0]], dtype=np.float64)
    U = W[:, :2].copy()                     # W' = U V^T with V = [[1,0],[0,1],[0,0]]
    V = np.array([[1.0, 0.0], [0.0, 1.0], [0.0, 0.0]])
    piv, nonp, Wp, C, _ = P.pifa_compress(U, V, 2)
    assert list(piv) == [1, 3] and list(nonp) == [0, 2, 4]
    assert np.allclose(C, [[-0.5, 0.5], [0.5, 0.5], [0.0, 0.0]], atol=1e-14)
    assert np.array_equal(Wp, W[[1, 3]])


@pytest.mark.slow
def test_compress_matches_oracle_lapack_attention_shape(lib):
    """4096 x 4096, r = 2048 (LLaMA-2-7B attention projection): pivots bit-exact with the oracle's
    LAPACK route (skipped unless -m slow)."""
    _compare_with_oracle(4096, 4096, 2048, 0, "lapack")


def _header_prototypes():
    """name -> (return category, [parameter categories]) for every pifa_* function in pifa.h."""
    import re
    src = open(os.path.join(ROOT, "include", "pifa.h")).read()
    src = re.sub(r"/\*.*?\*/", " ", src, flags=re.S)
    src = re.sub(r"//[^\n]*", " ", src)
    src = re.sub(r"#[^\n]*", " ", src)
    src = re.sub(r"\s+", " ", src)

    def cat(decl):
        decl = decl.strip()
        if "*" in decl:
            return "ptr"
        words = set(re.findall(r"\w+", decl))
        if "int64_t" in words:
            return "i64"
        if words & {"int", "int32_t"}:
            return "i32"
        if "double" in words:
            return "f64"
        if "float" in words:
            return "f32"
        raise AssertionError(f"unmapped C type: {decl!r}")

    out = {}
    for ret, name, params in re.findall(r"([\w\s\*]+?)\b(pifa_\w+)\s*\(([^;{()]*)\)\s*;", src):
        params = params.strip()
        plist = [] if params in ("", "void") else [cat(p) for p in params.split(",")]
        out[name] = (cat(ret), plist)
    return out


def test_binding_argtypes_match_the_header(lib):
    """Every declared function's ctypes prototype in the binding matches pifa.h in arity and in
    each argument's width (pointer / int64_t / int): a mismatch would corrupt arguments silently."""
    import ctypes
    protos = _header_prototypes()
    assert set(P.EXPORTS) <= set(protos), sorted(set(P.EXPORTS) - set(protos))

    def cat(t):
        if t is ctypes.c_int64 or t is ctypes.c_longlong or t is ctypes.c_long:
            return "i64"
        if t is ctypes.c_int or t is ctypes.c_int32:
            return "i32"
        if t is ctypes.c_double:
            return "f64"
        if t is ctypes.c_float:
            return "f32"
        if t in (ctypes.c_void_p, ctypes.c_char_p) or (isinstance(t, type) and issubclass(t, ctypes._Pointer)):
            return "ptr"
        raise AssertionError(f"unmapped ctypes type {t}")

    for name in P.EXPORTS:
        fn = getattr(lib, name)
        ret, params = protos[name]
        assert [cat(t) for t in fn.argtypes] == params, name
        assert cat(fn.restype) == ret, name


def _documented_choice(T, G, m, r):
    """pifa.h's rule: decode for T <= 64; for 64 < T <= 128 when the G (m - r) non-pivot rows make
    148 to 296 blocks of 128 and the G r pivot rows at most 296; the split prefill otherwise."""
    if T <= 64:
        return P.PIFA_VARIANT_DECODE
    bp, bnp = -(-G * r // 128), -(-G * (m - r) // 128)
    if T <= 128 and bp <= 296 and 148 <= bnp <= 296:
        return P.PIFA_VARIANT_DECODE
    return P.PIFA_VARIANT_PREFILL_SPLIT


def test_selector_and_forced_decode_follow_the_documented_rule(lib):
    """Random shapes and token counts: the selector's variant (single layers) and the workspace the
    grouped entry point sizes (its own choice) follow the documented rule; a forced decode call is
    refused exactly where 64 < T <= 128 and a phase has more than 296 blocks, or T > 128."""
    rng = np.random.default_rng(5)
    for _ in range(400):
        r = int(rng.integers(1, 9000))
        m = r + int(rng.integers(0, 45000))
        n = int(rng.integers(r, r + 9000))
        T = int(rng.choice([1, 16, 64, 65, 96, 128, 129, 500]))
        assert P.pifa_select_variant(T, m, n, r) == _documented_choice(T, 1, m, r), (T, m, n, r)
        fits = T <= 64 or (T <= 128 and -(-r // 128) <= 296 and -(-(m - r) // 128) <= 296)
        X, Wp, C, Y = 1 << 36, 2 << 36, 3 << 36, 4 << 36
        p8 = lambda v: (v + 7) // 8 * 8
        st = lib.pifa_forward_variant(X, T, n, p8(n), Wp, r, p8(n), C, m, p8(r), P.PIFA_DTYPE_BF16, 0x50000, 0x60000,
                                      Y, p8(m), None, 0, P.PIFA_VARIANT_DECODE, None)
        # buffers 64 GB apart never overlap at these sizes; a fitting shape fails on the missing workspace
        assert st == (P.PIFA_ERR_WORKSPACE if fits else P.PIFA_ERR_UNSUPPORTED), (T, m, n, r, st)
    # grouped layers whose stacked non-pivot rows make fewer than 148 or more than 296 blocks take
    # the split prefill above T = 64: the workspace the grouped entry point sizes is the prefill's,
    # 256 reserved bytes and the hi and lo planes (T x pad8(G r) bf16 each, 256-byte rounded)
    for G, m, r in ((2, 11008, 2048), (2, 28672, 4096), (3, 1408, 512)):
        for T in (100, 128):
            assert _documented_choice(T, G, m, r) == P.PIFA_VARIANT_PREFILL_SPLIT
            plane = -(-(T * -(-G * r // 8) * 8 * 2) // 256) * 256
            assert lib.pifa_workspace_size_grouped(G, T, m, 4096, r, P.PIFA_DTYPE_BF16) == 256 + 2 * plane
