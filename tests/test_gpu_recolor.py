"""hf_recolor_fit (Eq. 3-5, Newton-Schulz roots and polar factor in fp32)
against the oracle's Recolor fit (fp64 eigendecompositions and SVD)."""

import numpy as np
import pytest
import torch

from oracle import heterofold_oracle as O
from paper_2609_32259_gb300 import binding as B

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__ as g

    g.build()


def _data(seed, N, d_s, d_r, noise, dtype):
    g = torch.Generator(device="cpu").manual_seed(seed)
    X = torch.randn((N, d_s), generator=g) @ (torch.randn((d_s, d_s), generator=g) * 0.1) + 0.5
    A_true = torch.randn((d_s, d_r), generator=g) / np.sqrt(d_s)
    Y = X @ A_true + 0.3 + noise * torch.randn((N, d_r), generator=g)
    w = torch.rand((N,), generator=g) * 1.5 + 0.5
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    return X.to(tdt).cuda(), Y.to(tdt).cuda(), w.cuda()


def _fit(dtype, X, Y, w, reg):
    N, d_s = X.shape
    d_r = Y.shape[1]
    ws = torch.empty(B.recolor_workspace_size(N, d_s, d_r), dtype=torch.uint8, device="cuda")
    W_out = torch.empty((d_r, d_s), dtype=X.dtype, device="cuda")
    b_out = torch.empty((d_r,), dtype=torch.float32, device="cuda")
    r = B.recolor_fit(dtype, X, Y, w, W_out, b_out, ws, reg=reg)
    return W_out.double().cpu().numpy().T, b_out.double().cpu().numpy(), r


@pytest.mark.parametrize("dtype,tol", [("f32", 2e-3), ("bf16", 6e-3)])
def test_recolor_matches_oracle(dtype, tol):
    X, Y, w = _data(1, 4096, 192, 128, 0.5, dtype)
    A, b, r = _fit(dtype, X, Y, w, 1e-3)
    Xn, Yn, wn = X.double().cpu().numpy(), Y.double().cpu().numpy(), w.double().cpu().numpy()
    A_ref, b_ref, r_ref = O.recolor(Xn, Yn, wn, reg=1e-3)
    assert abs(r - r_ref) <= 1e-5 * r_ref
    rel = np.linalg.norm(A - A_ref) / np.linalg.norm(A_ref)
    assert rel <= tol, rel
    relb = np.linalg.norm(b - b_ref) / max(np.linalg.norm(b_ref), 1.0)
    assert relb <= tol, relb


def test_recolor_recovers_an_exact_rotation():
    """Y = Z Q + c with Q orthogonal: the fit returns A = Q, b = c."""
    g = torch.Generator(device="cpu").manual_seed(2)
    d = 64
    X = torch.randn((2048, d), generator=g, dtype=torch.float64) @ torch.randn((d, d), generator=g,
                                                                                dtype=torch.float64)
    w = torch.rand((2048,), generator=g, dtype=torch.float64) + 0.5
    Q, _ = torch.linalg.qr(torch.randn((d, d), generator=g, dtype=torch.float64))
    c = torch.randn((d,), generator=g, dtype=torch.float64)
    r = O.sender_rms(X.numpy(), w.numpy())
    Y = (X / r) @ Q + c
    A, b, r2 = _fit("f32", X.float().cuda(), Y.float().cuda(), w.float().cuda(), 0.0)
    assert abs(r2 - r) <= 1e-5 * r
    assert np.linalg.norm(A - Q.numpy()) / np.linalg.norm(Q.numpy()) < 2e-3
    assert np.abs(b - c.numpy()).max() < 5e-3


def test_recolor_rejects_bad_shapes():
    with pytest.raises(B.HFError):
        B.recolor_workspace_size(100, 64, 128)   # d_S < d_R


def test_recolor_at_the_benchmarked_shape():
    """One map of the 32K Llama -> Ministral-shaped direction: 32,768 weighted
    sample pairs, d_S = 3 x 1,024 (Eq. 2 input), d_R = 1,024, bf16 inputs,
    reg 1e-3 (the bench's workload): every Newton-Schulz iteration count the
    bench runs, against the oracle's fp64 eigendecompositions and SVD."""
    N, d_s, d_r = 32768, 3072, 1024
    g = torch.Generator(device="cuda").manual_seed(12)
    X = (torch.randn((N, d_s), generator=g, device="cuda")
         @ (torch.randn((d_s, d_s), generator=g, device="cuda") / d_s ** 0.5)).to(torch.bfloat16)
    A_true = torch.randn((d_s, d_r), generator=g, device="cuda") / d_s ** 0.5
    Y = (X.float() @ A_true + 0.5 * torch.randn((N, d_r), generator=g, device="cuda")
         ).to(torch.bfloat16)
    w = torch.rand((N,), generator=g, device="cuda") + 0.5
    ws = torch.empty(B.recolor_workspace_size(N, d_s, d_r), dtype=torch.uint8, device="cuda")
    W_out = torch.empty((d_r, d_s), dtype=torch.bfloat16, device="cuda")
    b_out = torch.empty((d_r,), dtype=torch.float32, device="cuda")
    r, its = B.recolor_fit("bf16", X, Y, w, W_out, b_out, ws, reg=1e-3, return_iters=True)
    A = W_out.double().cpu().numpy().T
    b = b_out.double().cpu().numpy()
    Xn, Yn, wn = X.double().cpu().numpy(), Y.double().cpu().numpy(), w.double().cpu().numpy()
    A_ref, b_ref, r_ref = O.recolor(Xn, Yn, wn, reg=1e-3)
    assert abs(r - r_ref) <= 1e-5 * r_ref
    assert all(0 < k < 80 for k in its), its
    rel = np.linalg.norm(A - A_ref) / np.linalg.norm(A_ref)
    assert rel <= 6e-3, rel   # bf16 rounding of A_final dominates (2^-9 relative)
    relb = np.linalg.norm(b - b_ref) / max(np.linalg.norm(b_ref), 1.0)
    assert relb <= 6e-3, relb
    print(f"recolor 32768 x 3072 -> 1024: iterations {its}, rel A {rel:.2e}, rel b {relb:.2e}")
