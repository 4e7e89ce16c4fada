"""pifa_forward_decode_noalloc: the decode entry point for callers that cannot allocate device
memory (for example a runtime that plans every device byte ahead and forbids a library's
cudaMalloc). It keeps its scratch in the library's static device data instead of a caller
workspace. Checked through the C ABI against pifa_forward's decode variant, on two calls in a
row (the shared static scratch keeps the first call's contents when the second one runs).

This file is named so pytest collects it last; it builds everything it needs itself, so it also
passes on its own in a fresh process.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2501_19090_gb300 import inputs
from paper_2501_19090_gb300 import pifa as P

pytestmark = pytest.mark.gpu

REL_FRO = 5e-3
ELEM = 2e-2
DEV = torch.device("cuda:0")


def _dev_bf16(a32):
    rows, cols = a32.shape
    ld = (cols + 7) // 8 * 8
    buf = torch.zeros((rows, ld), dtype=torch.bfloat16, device=DEV)
    buf[:, :cols] = torch.from_numpy(np.ascontiguousarray(a32)).to(DEV).to(torch.bfloat16)
    return buf[:, :cols]


def _close(got, ref):
    """The parity bar against the fp64 oracle: relative Frobenius and per-element bounds."""
    got = got.float().cpu().numpy().astype(np.float64)
    rel = np.linalg.norm(got - ref) / np.linalg.norm(ref)
    elem = np.max(np.abs(got - ref) / (np.abs(ref) + 1.0))
    assert rel <= REL_FRO and elem <= ELEM, f"rel_fro {rel:.3e}, elem {elem:.3e}"


def _layers():
    """A compressed tiny layer (the oracle's Algorithm 1) and a ragged random one (r = 301)."""
    U, V, _ = inputs.make_factors(256, 256, 128, 0)
    L = oracle.compress(U, V, 128)
    yield L.pivots, L.nonpivots, inputs.round_bf16(L.Wp), inputs.round_bf16(L.C)
    piv, nonp, Wp, C = inputs.synthetic_layer(1000, 776, 301, 3)
    yield piv, nonp, Wp, C


def test_noalloc_decode_matches_pifa_forward_twice():
    assert torch.cuda.is_available(), "GPU test needs CUDA"
    P.load()
    for piv, nonp, Wp32, C32 in _layers():
        Wp, C = _dev_bf16(Wp32), _dev_bf16(C32)
        pd = torch.from_numpy(np.asarray(piv, np.int32)).to(DEV)
        nd = torch.from_numpy(np.asarray(nonp, np.int32)).to(DEV)
        rng = np.random.default_rng(7)
        for T in (16, 5):                         # two calls in a row, different token counts
            X32 = inputs.make_activations(rng, T, Wp32.shape[1], "bf16")
            X = _dev_bf16(X32)
            ref = P.pifa_forward(X, Wp, C, pd, nd, variant=P.PIFA_VARIANT_DECODE)
            got = P.pifa_forward_decode_noalloc(X, Wp, C, pd, nd)
            assert P.pifa_device_status() == P.PIFA_OK
            # same kernels, same operands: the two entry points agree bit for bit (a read of stale
            # scratch left by the previous, larger call would show here)
            assert torch.equal(got.view(torch.int16), ref.view(torch.int16))
            _close(got, oracle.forward(X32, Wp32, C32, np.asarray(piv, np.int64), np.asarray(nonp, np.int64)))


def test_noalloc_rejects_output_overlapping_an_input():
    lib = P.load()
    base = 0x100000                              # never dereferenced: rejected before any launch
    # Y (4 x 64, pitch 64) placed over X (4 x 64): PIFA_ERR_INVALID_ARG, as pifa_forward
    st = lib.pifa_forward_decode_noalloc(base, 4, 64, 64, base + 0x10000, 16, 64, base + 0x20000, 48, 16,
                                         base + 0x30000, base + 0x31000, base + 64, 48, None)
    assert st == P.PIFA_ERR_INVALID_ARG
    assert "overlaps" in P.pifa_last_error()


def test_noalloc_rejects_sizes_beyond_the_static_scratch():
    lib = P.load()
    fake = 1 << 36                               # never dereferenced: rejected before any launch;
    # the buffers sit 64 GiB apart, so none overlaps another
    # 256 + T * round_up(r, 8) * 4 bytes must fit in 1 MiB: r = 16392 at T = 16 does not
    st = lib.pifa_forward_decode_noalloc(fake, 16, 20000, 20000, fake * 2, 16392, 20000, fake * 3,
                                         20000, 16392, fake * 4, fake * 5, fake * 6, 20000, None)
    assert st == P.PIFA_ERR_WORKSPACE
    assert "1 MiB" in P.pifa_last_error()
    st = lib.pifa_forward_decode_noalloc(fake, 17, 64, 64, fake * 2, 16, 64, fake * 3, 48, 16,
                                         fake * 4, fake * 5, fake * 6, 48, None)
    assert st == P.PIFA_ERR_UNSUPPORTED
