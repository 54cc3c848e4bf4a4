"""The block step's tcgen05 GEMM (hcw_gemm_bf16) against the product's
definition, C = op(A) op(B), computed in fp64 on the host from the same bf16
values: every layout of the two operands, ragged tiles in M, N and K, boxes
smaller than a tile, K splits with their fixed-order sum, and the plain
kernel that takes the shapes TMA cannot read.

Tolerance: the products of two bf16 values are exact in fp32, so the only
error is the fp32 accumulation, bounded by gamma_K = K u (u = 2^-24) times
(|A| |B|)_ij; the test allows four times that, which a wrong element (an
operand read from the wrong row, a dropped K step) exceeds by orders of
magnitude."""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

U32 = 2.0 ** -24


@pytest.fixture(scope="module")
def H():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2609_18145_gb300 import hcw
    hcw.lib()
    return hcw


def operands(M, N, K, ta, tb, seed):
    g = torch.Generator().manual_seed(seed)
    A = torch.randn((K, M) if ta else (M, K), generator=g).to(torch.bfloat16)
    B = torch.randn((N, K) if tb else (K, N), generator=g).to(torch.bfloat16)
    return A, B


def reference(A, B, ta, tb):
    a = A.double().numpy()
    b = B.double().numpy()
    a = a.T if ta else a
    b = b.T if tb else b
    return a @ b, np.abs(a) @ np.abs(b)


def check(C, A, B, ta, tb):
    ref, absref = reference(A, B, ta, tb)
    K = A.shape[0] if ta else A.shape[1]
    got = C.double().cpu().numpy()
    tol = 4.0 * (K + 2) * U32 * absref + 1e-30
    bad = np.abs(got - ref) > tol
    assert not bad.any(), (int(bad.sum()), np.argwhere(bad)[:4].tolist())


CASES = [
    # M, N, K, ta, tb
    (300, 520, 200, False, True),     # both K-major; ragged M, N and K
    (256, 768, 136, False, False),    # B MN-major
    (192, 320, 1000, True, False),    # both MN-major; M a half tile past a whole one
    (384, 256, 4096, True, True),     # A MN-major, long K: split
    (128, 64, 512, False, False),     # B narrower than a tile (one 64-column block)
    (64, 11, 64, False, True),        # 11 output columns (head of an 11-symbol vocabulary)
    (2048, 256, 512, False, True),    # the head's shape: tokens x V x d
    (512, 1024, 16384, True, False),  # a weight gradient: d x h x tokens, split
    (37, 45, 29, False, False),       # plain kernel: rows TMA cannot read
    (11, 64, 32, True, False),        # plain kernel: MN-major A of 11 columns
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: "M%d_N%d_K%d_ta%d_tb%d" % c)
def test_gemm_matches_the_product(H, case):
    M, N, K, ta, tb = case
    A, B = operands(M, N, K, ta, tb, seed=M + 7 * N + 13 * K)
    C = H.hcw_gemm_bf16(A.cuda(), B.cuda(), ta=ta, tb=tb)
    torch.cuda.synchronize()
    assert H.hcw_sync_status() == H.HCW_OK
    check(C.cpu(), A, B, ta, tb)


def test_split_sums_are_deterministic_and_match_the_unsplit_product(H):
    M, N, K = 512, 1024, 16384
    assert H.hcw_gemm_workspace_bytes(M, N, K) > 0
    A, B = operands(M, N, K, True, False, seed=3)
    Ad, Bd = A.cuda(), B.cuda()
    C1 = H.hcw_gemm_bf16(Ad, Bd, ta=True)
    C2 = H.hcw_gemm_bf16(Ad, Bd, ta=True)
    C0 = H.hcw_gemm_bf16(Ad, Bd, ta=True, split=False)
    torch.cuda.synchronize()
    assert H.hcw_sync_status() == H.HCW_OK
    assert torch.equal(C1, C2)
    check(C0.cpu(), A, B, True, False)
    check(C1.cpu(), A, B, True, False)


def test_misaligned_operands_take_the_plain_kernel(H):
    """An operand view that starts 2 bytes past a 16-byte boundary cannot be a
    TMA source; the result is the same product."""
    M, N, K = 130, 256, 96
    A, B = operands(M, N, K + 1, False, True, seed=5)
    Ad = A.cuda()
    Bd = B.cuda()
    a = torch.empty(M * K + 1, dtype=torch.bfloat16, device="cuda")[1:].view(M, K)
    a.copy_(Ad[:, 1:])
    b = Bd[:, 1:].contiguous()
    C = H.hcw_gemm_bf16(a, b, tb=True)
    torch.cuda.synchronize()
    assert H.hcw_sync_status() == H.HCW_OK
    check(C.cpu(), A[:, 1:].contiguous(), B[:, 1:].contiguous(), False, True)


BATCHED = [
    # batch, M, N, K
    (3, 512, 1024, 2000),   # the FFN's dW2 shape, ragged K
    (4, 1024, 512, 640),    # dW1 shape
    (2, 192, 320, 1000),    # a half tile past a whole one in M
    (2, 100, 64, 96),       # M not a multiple of 64: one product at a time
]


@pytest.mark.parametrize("case", BATCHED, ids=lambda c: "b%d_M%d_N%d_K%d" % c)
def test_batched_products_match_each_product(H, case):
    """hcw_gemm_bf16_batched: C[b] = A[b]^T B[b] for every b, each against its
    own fp64 product, with a batch stride larger than one product (padding
    between them) for A."""
    nb, M, N, K = case
    g = torch.Generator().manual_seed(nb * 7 + M)
    A = torch.randn(nb, K + 3, M, generator=g).to(torch.bfloat16)[:, :K, :]
    B = torch.randn(nb, K, N, generator=g).to(torch.bfloat16)
    Ad = torch.empty(nb, K + 3, M, dtype=torch.bfloat16, device="cuda")
    Ad[:, :K, :] = A.cuda()
    Ad = Ad[:, :K, :]
    assert Ad.stride(0) == (K + 3) * M
    C = H.hcw_gemm_bf16_batched(Ad, B.cuda())
    torch.cuda.synchronize()
    for b in range(nb):
        check(C[b], A[b].contiguous(), B[b].contiguous(), True, False)
