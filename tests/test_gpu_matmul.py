"""The fp32 product kernel behind hf_recolor_fit (tcgen05, three-way bf16
split of each operand) through its C-ABI test hook, against the plain fp64
product of the same inputs: indexing (exact small-integer products, every
transpose form, ragged sizes, split-K), and fp32 accuracy on random data
(a dropped split term shows as an error of 2^-16 or more)."""

import numpy as np
import pytest
import torch

from paper_2609_32259_gb300 import binding as B

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__ as g

    g.build()


def _views(M, N, K, ta, tb, gen, fill):
    """op(A) [M, K] and op(B) [K, N] as fp64 numpy, and the device matrices
    with the strides that express them (ta / tb: stored transposed)."""
    a = fill((M, K), gen)
    b = fill((K, N), gen)
    if ta:   # stored as A^T [K][M]: op(A)(i, k) = At[k][i]
        dA = torch.as_tensor(np.ascontiguousarray(a.T), dtype=torch.float32, device="cuda")
        sa = (1, M)
    else:
        dA = torch.as_tensor(a, dtype=torch.float32, device="cuda")
        sa = (K, 1)
    if tb:   # stored as B^T [N][K]: op(B)(k, j) = Bt[j][k]
        dB = torch.as_tensor(np.ascontiguousarray(b.T), dtype=torch.float32, device="cuda")
        sb = (1, K)
    else:
        dB = torch.as_tensor(b, dtype=torch.float32, device="cuda")
        sb = (N, 1)
    return a, b, dA, sa, dB, sb


def _ints(shape, gen):
    return gen.integers(-8, 9, size=shape).astype(np.float64)


def _randn(shape, gen):
    return gen.standard_normal(shape).astype(np.float32).astype(np.float64)


SHAPES = [(256, 256, 64), (300, 200, 500), (192, 192, 4096), (1024, 1024, 1024),
          (130, 257, 70), (512, 128, 8192)]


@pytest.mark.parametrize("M,N,K", SHAPES)
@pytest.mark.parametrize("ta,tb", [(False, False), (True, False), (False, True), (True, True)])
def test_matmul_exact_on_small_integers(M, N, K, ta, tb):
    """Small-integer operands: every product and partial sum is exact in
    fp32, so the result must equal the fp64 product exactly; a wrong row,
    column or K index anywhere changes it."""
    gen = np.random.default_rng(M * 7 + N * 3 + K + 11 * ta + 5 * tb)
    a, b, dA, sa, dB, sb = _views(M, N, K, ta, tb, gen, _ints)
    C = torch.full((M, N), 12345.0, dtype=torch.float32, device="cuda")
    assert B.debug_matmul_f32(dA, sa, dB, sb, C, M, N, K) == 0
    assert np.array_equal(C.cpu().numpy().astype(np.float64), a @ b)


@pytest.mark.parametrize("M,N,K", SHAPES)
def test_matmul_fp32_accuracy(M, N, K):
    gen = np.random.default_rng(M + 2 * N + 3 * K)
    a, b, dA, sa, dB, sb = _views(M, N, K, True, False, gen, _randn)
    C0 = gen.standard_normal((M, N)).astype(np.float32)
    C = torch.as_tensor(C0, device="cuda")
    assert B.debug_matmul_f32(dA, sa, dB, sb, C, M, N, K, alpha=-0.5, beta=1.5) == 0
    ref = -0.5 * (a @ b) + 1.5 * C0.astype(np.float64)
    got = C.cpu().numpy().astype(np.float64)
    # fp32 accumulation (one fp32 add per 16-deep MMA step and term): a few
    # 1e-7 relative; a missing second-order split term would add ~2^-16
    # (1.5e-5) relative, a missing first-order one ~2^-8
    scale = np.sqrt(K) * np.abs(a).max() * np.abs(b).max()
    assert np.abs(got - ref).max() <= 3e-6 * scale, np.abs(got - ref).max() / scale
    rel = np.linalg.norm(got - ref) / np.linalg.norm(ref)
    assert rel <= 5e-6, rel


def test_matmul_gram_shares_planes():
    """X^T X: both operands read the same matrix the same way (one set of
    planes); against the fp64 Gram matrix."""
    gen = np.random.default_rng(3)
    n, d = 5000, 320
    x = gen.standard_normal((n, d)).astype(np.float32)
    dX = torch.as_tensor(x, device="cuda")
    C = torch.empty((d, d), dtype=torch.float32, device="cuda")
    assert B.debug_matmul_f32(dX, (1, d), dX, (d, 1), C, d, d, n) == 0
    ref = x.astype(np.float64).T @ x.astype(np.float64)
    got = C.cpu().numpy().astype(np.float64)
    assert np.linalg.norm(got - ref) / np.linalg.norm(ref) <= 5e-6


def test_matmul_unbiased_on_positive_data():
    """Positive operands, K = 16,384: the tensor core's accumulator adds by
    truncation (a single accumulator over K came out 7.6e-5 low on average),
    so the kernel drains it into round-to-nearest fp32 sums every 64-wide K
    atom; the mean relative error must stay at the fp32 level."""
    M, K = 1024, 16384
    gen = np.random.default_rng(17)
    a = (1.0 + gen.random((M, K))).astype(np.float32)
    b = (1.0 + gen.random((K, M))).astype(np.float32)
    dA = torch.as_tensor(a, device="cuda")
    dB = torch.as_tensor(b, device="cuda")
    C = torch.empty((M, M), dtype=torch.float32, device="cuda")
    assert B.debug_matmul_f32(dA, (K, 1), dB, (M, 1), C, M, M, K) == 0
    ref = torch.as_tensor(a, dtype=torch.float64, device="cuda") @ torch.as_tensor(
        b, dtype=torch.float64, device="cuda")
    rel = ((C.double() - ref) / ref).cpu().numpy()
    assert abs(rel.mean()) <= 1e-6, rel.mean()
    assert np.abs(rel).max() <= 1e-5, np.abs(rel).max()
