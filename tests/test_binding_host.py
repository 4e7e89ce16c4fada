"""The Python binding's operand checks, without a GPU: every call here is rejected before any
pointer reaches the library (the C ABI sees raw pointers and sizes only, so the binding checks
tensor type, dtype, shape and device)."""
import pytest
import torch

from paper_2501_19090_gb300 import pifa as P

T, n, m, r = 4, 64, 48, 16


def ops(**kw):
    """A well-formed operand set on the CPU (so the device check is the last one to fail)."""
    a = dict(X=torch.zeros((T, n), dtype=torch.bfloat16), Wp=torch.zeros((r, n), dtype=torch.bfloat16),
             C=torch.zeros((m - r, r), dtype=torch.bfloat16), piv=torch.arange(r, dtype=torch.int32),
             nonp=torch.arange(r, m, dtype=torch.int32), Y=torch.zeros((T, m), dtype=torch.bfloat16))
    a.update(kw)
    return a


def fwd(a, fn=P.pifa_forward):
    return fn(a["X"], a["Wp"], a["C"], a["piv"], a["nonp"], Y=a["Y"])


@pytest.mark.parametrize("bad,msg", [
    (dict(X=torch.zeros((T, n), dtype=torch.float32)), "X must be a 2-D bfloat16"),
    (dict(X=torch.zeros((T * n,), dtype=torch.bfloat16)), "X must be a 2-D bfloat16"),
    (dict(X=[[0.0] * n] * T), "X must be a torch tensor"),
    (dict(Wp=torch.zeros((r, n + 8), dtype=torch.bfloat16)), "Wp must be"),
    (dict(Wp=torch.zeros((r, n), dtype=torch.float16)), "Wp must be"),
    (dict(piv=torch.arange(r, dtype=torch.int64)), "pivot_idx must be a contiguous 1-D int32"),
    (dict(piv=torch.arange(2 * r, dtype=torch.int32)[::2]), "pivot_idx must be a contiguous 1-D int32"),
    (dict(nonp=torch.arange(r, m, dtype=torch.int64)), "nonpivot_idx must be a contiguous 1-D int32"),
    (dict(piv=torch.arange(r - 1, dtype=torch.int32)), "Wp must be|pivot_idx must hold"),
    (dict(C=torch.zeros((m - r, r + 8), dtype=torch.bfloat16)), "C must be"),
    (dict(C=torch.zeros((m - r, r), dtype=torch.float32)), "C must be"),
    (dict(Y=torch.zeros((T, m + 8), dtype=torch.bfloat16)), "Y must be"),
    (dict(Y=torch.zeros((T, m), dtype=torch.float32)), "Y must be"),
    ({}, "X must be a CUDA tensor"),
])
def test_forward_rejects_before_the_library(bad, msg):
    with pytest.raises(ValueError, match=msg):
        fwd(ops(**bad))


def test_noalloc_wants_bf16_c():
    a = ops(C=torch.zeros((m - r, r), dtype=torch.float16))
    with pytest.raises(ValueError, match="C must be a bfloat16 tensor"):
        fwd(a, P.pifa_forward_decode_noalloc)
    with pytest.raises(ValueError, match="X must be a CUDA tensor"):   # fp16 C is fine for pifa_forward
        fwd(a)


def test_grouped_shapes_and_groups():
    G = 2
    a = dict(X=torch.zeros((T, n), dtype=torch.bfloat16), Wp=torch.zeros((G * r, n), dtype=torch.bfloat16),
             C=torch.zeros((G * (m - r), r), dtype=torch.bfloat16), piv=torch.arange(G * r, dtype=torch.int32),
             nonp=torch.arange(G * (m - r), dtype=torch.int32), Y=torch.zeros((T, G * m), dtype=torch.bfloat16))
    call = lambda g, **kw: P.pifa_forward_grouped(g, **{**dict(X=a["X"], Wp=a["Wp"], C=a["C"], pivot_idx=a["piv"],
                                                                nonpivot_idx=a["nonp"], Y=a["Y"]), **kw})
    with pytest.raises(ValueError, match="groups must be"):
        call(0)
    with pytest.raises(ValueError, match="Y must be"):
        call(G, Y=torch.zeros((T, m), dtype=torch.bfloat16))
    with pytest.raises(ValueError, match="nonpivot_idx must hold the same number"):
        call(G, nonpivot_idx=torch.arange(G * (m - r) - 1, dtype=torch.int32))
    with pytest.raises(ValueError, match="X must be a CUDA tensor"):
        call(G)
