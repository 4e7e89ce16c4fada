"""GPU parity of the training-side paths through the C ABI, against the fp64 oracle:

* pifa_backward -- the gradients of Algorithm 2 (fine-tuning, Sec. 5.1; Sec. 6): dX, dW_p, dC
  against oracle.backward on the same bf16 operands;
* pifa_m_accumulate -- the online accumulators of the M reconstruction (Sec. 4, Algorithm 3):
  X X^T and Y_t X^T against oracle.m_accumulate, over two batches in a row (the online form).

Tolerance as the forward pass: relative Frobenius error <= 5e-3 and |err| <= 2e-2 (|ref| + 1) per
element (bf16 operands, fp32 accumulation, bf16 intermediates).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2501_19090_gb300 import inputs
from paper_2501_19090_gb300 import pifa as P

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")
REL_FRO = 5e-3
ELEM = 2e-2


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    P.load()


def check(got, ref, what):
    got = np.asarray(got, dtype=np.float64)
    rel = np.linalg.norm(got - ref) / max(np.linalg.norm(ref), 1e-300)
    elem = np.max(np.abs(got - ref) / (np.abs(ref) + 1.0)) if ref.size else 0.0
    assert rel <= REL_FRO and elem <= ELEM, f"{what}: rel_fro {rel:.3e}, elem {elem:.3e}"


def dev_bf16(a32):
    rows, cols = a32.shape
    ld = (cols + 7) // 8 * 8
    buf = torch.full((rows, ld), float("nan"), dtype=torch.bfloat16, device=DEV)
    buf[:, :cols] = torch.from_numpy(np.ascontiguousarray(a32, dtype=np.float32)).to(DEV).to(torch.bfloat16)
    return buf[:, :cols]


def compressed(m, n, r, seed, route):
    U, V, _ = inputs.make_factors(m, n, r, seed)
    L = oracle.compress(U, V, r, route)
    return L.pivots, L.nonpivots, inputs.round_bf16(L.Wp), inputs.round_bf16(L.C)


CASES = [
    ("tiny 256x256 r128", (256, 256, 128, 0, "greedy"), 64),
    ("ragged 300x200 r77", (300, 200, 77, 3, "greedy"), 37),
    ("r = m 64x128", (64, 128, 64, 4, "greedy"), 20),
    ("rank one 40x48", (40, 48, 1, 5, "greedy"), 13),
    ("7B attention 4096x4096 r2048", (4096, 4096, 2048, 0, "lapack"), 512),
    # T = 2048: dX and dW_p span more than one wave of tiles and run gemm_tc's two-CTA shape
    ("7B attention 4096x4096 r2048 T2048", (4096, 4096, 2048, 0, "lapack"), 2048),
]


@pytest.mark.parametrize("name,layer,T", CASES, ids=[c[0] for c in CASES])
def test_backward_matches_the_oracle(name, layer, T):
    piv, nonp, Wp32, C32 = compressed(*layer)
    m, n, r = piv.size + nonp.size, Wp32.shape[1], Wp32.shape[0]
    rng = np.random.default_rng(11)
    X32 = inputs.make_activations(rng, T, n, "bf16")
    dY32 = inputs.make_activations(rng, T, m, "bf16")
    X, Wp, dY = dev_bf16(X32), dev_bf16(Wp32), dev_bf16(dY32)
    C = dev_bf16(C32) if m > r else torch.empty((0, r), dtype=torch.bfloat16, device=DEV)
    pd = torch.from_numpy(piv.astype(np.int32)).to(DEV)
    nd = torch.from_numpy(nonp.astype(np.int32)).to(DEV)
    dX, dWp, dC = P.pifa_backward(X, Wp, C, pd, nd, dY)
    assert P.pifa_device_status() == P.PIFA_OK
    rX, rWp, rC = oracle.backward(X32, Wp32, C32, piv, nonp, dY32)
    check(dX.float().cpu().numpy(), rX, f"{name} dX")
    check(dWp.cpu().numpy(), rWp, f"{name} dW_p")
    if m > r:
        check(dC.cpu().numpy(), rC, f"{name} dC")
    else:
        assert dC is None


def test_backward_zero_tokens_gives_zero_weight_gradients():
    piv, nonp, Wp32, C32 = compressed(256, 256, 128, 0, "greedy")
    Wp, C = dev_bf16(Wp32), dev_bf16(C32)
    pd = torch.from_numpy(piv.astype(np.int32)).to(DEV)
    nd = torch.from_numpy(nonp.astype(np.int32)).to(DEV)
    X = torch.empty((0, 256), dtype=torch.bfloat16, device=DEV)
    dY = torch.empty((0, 256), dtype=torch.bfloat16, device=DEV)
    _, dWp, dC = P.pifa_backward(X, Wp, C, pd, nd, dY)
    assert P.pifa_device_status() == P.PIFA_OK
    assert torch.count_nonzero(dWp) == 0 and torch.count_nonzero(dC) == 0


def _macc_inputs(T, n, m, seed):
    rng = np.random.default_rng(seed)
    Xu = inputs.round_bf16(rng.standard_normal((T, n)))
    Xo = inputs.round_bf16(Xu + 0.1 * rng.standard_normal((T, n)))
    W = inputs.round_bf16(rng.standard_normal((m, n)) / np.sqrt(n))
    return Xo, Xu, W


def test_m_accumulate_two_batches_match_the_oracle():
    n, m, lam = 520, 1000, 0.25
    XXt = torch.zeros((n, n), dtype=torch.float32, device=DEV)
    YtXt = torch.zeros((m, n), dtype=torch.float32, device=DEV)
    ref = (None, None)
    for T, seed in ((300, 1), (77, 2)):
        Xo, Xu, W = _macc_inputs(T, n, m, seed)
        # one W for both batches (the same layer): the second draw's W is replaced by the first's
        if seed == 1:
            W0 = W
        P.pifa_m_accumulate(dev_bf16(Xo), dev_bf16(Xu), dev_bf16(W0), lam, XXt, YtXt)
        ref = oracle.m_accumulate(Xo, Xu, W0, lam, *ref)
    assert P.pifa_device_status() == P.PIFA_OK
    # X X^T is accumulated in its upper triangle (it is symmetric)
    check(np.triu(XXt.cpu().numpy()), np.triu(ref[0]), "X X^T")
    check(YtXt.cpu().numpy(), ref[1], "Y_t X^T")


def test_m_accumulate_xxt_only_and_lambda_edges():
    n = 256
    Xo, Xu, W = _macc_inputs(100, n, 128, 3)
    XXt = torch.zeros((n, n), dtype=torch.float32, device=DEV)
    P.pifa_m_accumulate(None, dev_bf16(Xu), None, 0.5, XXt)
    check(np.triu(XXt.cpu().numpy()), np.triu(oracle.m_accumulate(Xo, Xu, W, 0.5)[0]), "X X^T alone")
    for lam in (0.0, 1.0):
        XXt.zero_()
        Y = torch.zeros((128, n), dtype=torch.float32, device=DEV)
        P.pifa_m_accumulate(dev_bf16(Xo), dev_bf16(Xu), dev_bf16(W), lam, XXt, Y)
        check(Y.cpu().numpy(), oracle.m_accumulate(Xo, Xu, W, lam)[1], f"Y_t X^T lambda={lam}")
    assert P.pifa_device_status() == P.PIFA_OK


def test_m_accumulate_llama_shape_sampled_rows():
    """7B attention shape (n = m = 4096) with T = 512 samples; 48 sampled rows of each
    accumulator against the oracle restricted to those rows."""
    n = m = 4096
    Xo, Xu, W = _macc_inputs(512, n, m, 4)
    XXt = torch.zeros((n, n), dtype=torch.float32, device=DEV)
    YtXt = torch.zeros((m, n), dtype=torch.float32, device=DEV)
    P.pifa_m_accumulate(dev_bf16(Xo), dev_bf16(Xu), dev_bf16(W), 0.25, XXt, YtXt)
    assert P.pifa_device_status() == P.PIFA_OK
    rx, ry = inputs.random_rows(n, 48, 5), inputs.random_rows(m, 48, 6)
    a, b = oracle.m_accumulate(Xo, Xu, W, 0.25, rows=(rx, ry))
    upper = np.arange(n)[None, :] >= rx[:, None]  # the accumulated triangle of each sampled row
    check(np.where(upper, XXt[torch.from_numpy(rx)].cpu().numpy(), 0.0), np.where(upper, a, 0.0), "X X^T rows")
    check(YtXt[torch.from_numpy(ry)].cpu().numpy(), b, "Y_t X^T rows")


# ---------------------------------------------------------------------------------------------
# pifa_m_reconstruct: U_r (Eq. 4) and V_r (Eq. 8) from the accumulators, float64
# ---------------------------------------------------------------------------------------------
def _accumulated(T, n, m, r, seed):
    Xo, Xu, W = _macc_inputs(T, n, m, seed)
    XXt = torch.zeros((n, n), dtype=torch.float32, device=DEV)
    YtXt = torch.zeros((m, n), dtype=torch.float32, device=DEV)
    P.pifa_m_accumulate(dev_bf16(Xo), dev_bf16(Xu), dev_bf16(W), 0.25, XXt, YtXt)
    V = np.random.default_rng(seed + 100).standard_normal((n, r)) / np.sqrt(n)
    return Xo, Xu, W, XXt, YtXt, V


@pytest.mark.parametrize("m,n,r,T,alpha", [(300, 256, 64, 1000, 0.0), (300, 256, 64, 1000, 1e-3),
                                           (1024, 1024, 256, 3000, 1e-3)])
def test_m_reconstruct_matches_the_oracle_on_the_same_accumulators(m, n, r, T, alpha):
    """Same fp32 accumulators on both sides; both solve in float64 (the library by Cholesky and
    triangular inverses, the oracle by LAPACK solves): agreement to 1e-8 relative."""
    Xo, Xu, W, XXt, YtXt, V = _accumulated(T, n, m, r, 7)
    Wd = dev_bf16(W)
    U_r, V_r = P.pifa_m_reconstruct(XXt, YtXt, torch.from_numpy(V).to(DEV), W=Wd, alpha=alpha)
    A, B = XXt.double().cpu().numpy(), YtXt.double().cpu().numpy()
    A = np.triu(A) + np.triu(A, 1).T  # the library keeps X X^T's upper triangle; both sides see it whole
    rU, rV = oracle.m_reconstruct(A, B, V, W=W.astype(np.float64), alpha=alpha)
    for got, ref, what in ((U_r, rU, "U_r"), (V_r, rV, "V_r")):
        got = got.cpu().numpy()
        rel = np.linalg.norm(got - ref) / np.linalg.norm(ref)
        assert rel <= 1e-8, f"{what}: rel {rel:.3e}"


def test_m_path_end_to_end_against_the_oracle():
    """GPU accumulation then GPU reconstruction against the oracle's accumulation and
    reconstruction from the same bf16 samples: within the bf16 tolerance."""
    m, n, r, T = 300, 256, 64, 1000
    Xo, Xu, W, XXt, YtXt, V = _accumulated(T, n, m, r, 8)
    U_r, V_r = P.pifa_m_reconstruct(XXt, YtXt, torch.from_numpy(V).to(DEV), W=dev_bf16(W), alpha=1e-3)
    A, B = oracle.m_accumulate(Xo, Xu, W, 0.25)
    rU, rV = oracle.m_reconstruct(A, B, V, W=W.astype(np.float64), alpha=1e-3)
    check(U_r.cpu().numpy(), rU, "U_r")
    # the reconstructed layer U_r V_r^T is the product that matters downstream
    check((U_r @ V_r.t()).cpu().numpy(), rU @ rV.T, "U_r V_r^T")


def test_m_reconstruct_reports_a_singular_system():
    """Fewer samples than inputs (T < n) leave X X^T singular; without the regulariser
    (alpha = 0) Eq. 7 has no unique solution: PIFA_ERR_RANK_DEFICIENT."""
    m, n, r, T = 128, 256, 32, 100
    _, _, _, XXt, YtXt, V = _accumulated(T, n, m, r, 9)
    with pytest.raises(P.PifaError) as e:
        P.pifa_m_reconstruct(XXt, YtXt, torch.from_numpy(V).to(DEV), alpha=0.0)
    assert e.value.status == P.PIFA_ERR_RANK_DEFICIENT


def test_backward_and_m_accumulate_under_graph_capture():
    """The backward's and the M accumulators' independent products run on side streams forked from
    and joined back into the caller's stream. Captured into a CUDA graph (after a first eager call,
    which creates the side streams), a replay gives every output bit for bit equal to the eager
    call's."""
    m, n, r, T = 1024, 768, 384, 512
    piv, nonp, Wp32, C32 = inputs.synthetic_layer(m, n, r, 21)
    rng = np.random.default_rng(22)
    X = dev_bf16(inputs.make_activations(rng, T, n, "bf16"))
    dY = dev_bf16(inputs.make_activations(rng, T, m, "bf16"))
    Wp, C = dev_bf16(Wp32), dev_bf16(C32)
    pd = torch.from_numpy(piv.astype(np.int32)).to(DEV)
    nd = torch.from_numpy(nonp.astype(np.int32)).to(DEV)
    ws = torch.empty(P.pifa_backward_workspace_size(T, m, n, r) + 256, dtype=torch.uint8, device=DEV)
    st = torch.cuda.Stream()
    torch.cuda.synchronize()
    ref = P.pifa_backward(X, Wp, C, pd, nd, dY, workspace_tensor=ws, stream=st)
    st.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=st):
        got = P.pifa_backward(X, Wp, C, pd, nd, dY, workspace_tensor=ws, stream=st)
    for _ in range(2):
        g.replay()
    torch.cuda.synchronize()
    assert P.pifa_device_status() == P.PIFA_OK
    assert torch.equal(got[0].view(torch.int16), ref[0].view(torch.int16))
    assert torch.equal(got[1], ref[1]) and torch.equal(got[2], ref[2])
    del g

    Xo, Xu, W = _macc_inputs(T, n, m, 23)
    Xo, Xu, W = dev_bf16(Xo), dev_bf16(Xu), dev_bf16(W)
    wsm = torch.empty(P.pifa_m_accumulate_workspace_size(T, m, n) + 256, dtype=torch.uint8, device=DEV)
    XXt0 = torch.zeros((n, n), dtype=torch.float32, device=DEV)
    Y0 = torch.zeros((m, n), dtype=torch.float32, device=DEV)
    P.pifa_m_accumulate(Xo, Xu, W, 0.3, XXt0, Y0, workspace_tensor=wsm, stream=st)
    st.synchronize()
    XXt1 = torch.zeros_like(XXt0)
    Y1 = torch.zeros_like(Y0)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=st):
        P.pifa_m_accumulate(Xo, Xu, W, 0.3, XXt1, Y1, workspace_tensor=wsm, stream=st)
    XXt1.zero_()
    Y1.zero_()
    torch.cuda.synchronize()
    g.replay()
    torch.cuda.synchronize()
    assert P.pifa_device_status() == P.PIFA_OK
    assert torch.equal(torch.triu(XXt1), torch.triu(XXt0)) and torch.equal(Y1, Y0)
