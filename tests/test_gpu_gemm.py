"""The tcgen05 contraction under the head: every operand layout, ragged edges, accumulation.
Compared with a plain torch f32 product of the same bf16 values (products are exact in
f32; only the summation order differs)."""
import pytest
import torch

pytestmark = pytest.mark.gpu


def _ref(A, B, a_mn, b_mn):
    Am = (A.float().t() if a_mn else A.float())          # [M][K]
    Bm = (B.float() if b_mn else B.float().t())          # [K][N]
    return Am @ Bm


@pytest.mark.parametrize("pair", [0, 1, 2])
@pytest.mark.parametrize("a_mn,b_mn", [(0, 0), (0, 1), (1, 1), (1, 0)])
@pytest.mark.parametrize("M,N,K", [(128, 256, 64), (300, 520, 200), (1000, 777, 968), (64, 40, 8), (129, 257, 65),
                                   (513, 1300, 136)])
def test_layouts_and_ragged_edges(a_mn, b_mn, M, N, K, pair):
    from paper_2606_29758_gb300 import _binding as B
    g = torch.Generator(device="cuda").manual_seed(M * 7 + N * 3 + K + a_mn * 2 + b_mn)
    pad8 = lambda x: (x + 7) // 8 * 8  # noqa: E731  (leading dimensions must be multiples of 8)
    Afull = torch.randn((K, pad8(M)) if a_mn else (M, pad8(K)), device="cuda", generator=g).to(torch.bfloat16)
    Bfull = torch.randn((K, pad8(N)) if b_mn else (N, pad8(K)), device="cuda", generator=g).to(torch.bfloat16)
    A = Afull[:, :M] if a_mn else Afull[:, :K]
    Bt = Bfull[:, :N] if b_mn else Bfull[:, :K]
    ldc = (N + 3) // 4 * 4
    C = torch.full((M, ldc), float("nan"), device="cuda")
    ws = torch.empty(256, dtype=torch.uint8, device="cuda")
    B.ps_diag_gemm_bf16(M, N, K, a_mn, b_mn, Afull, Afull.shape[1], Bfull, Bfull.shape[1], C, ldc, 0, ws, pair)
    torch.cuda.synchronize()
    assert B.ps_workspace_status(ws)[0] == B.PS_OK
    ref = _ref(A, Bt, a_mn, b_mn)
    err = (C[:, :N] - ref).abs().max().item()
    assert err <= 1e-4 * max(1.0, ref.abs().max().item()), err
    # accumulate into the previous result
    B.ps_diag_gemm_bf16(M, N, K, a_mn, b_mn, Afull, Afull.shape[1], Bfull, Bfull.shape[1], C, ldc, 1, ws, pair)
    torch.cuda.synchronize()
    err2 = (C[:, :N] - 2 * ref).abs().max().item()
    assert err2 <= 2e-4 * max(1.0, ref.abs().max().item()), err2


@pytest.mark.parametrize("pair", [0, 1, 2])
def test_many_waves(pair):
    from paper_2606_29758_gb300 import _binding as B
    g = torch.Generator(device="cuda").manual_seed(5)
    M, N, K = 4096, 4096, 1024
    A = torch.randn(M, K, device="cuda", generator=g).to(torch.bfloat16)
    Bt = torch.randn(N, K, device="cuda", generator=g).to(torch.bfloat16)
    C = torch.empty(M, N, device="cuda")
    ws = torch.empty(256, dtype=torch.uint8, device="cuda")
    B.ps_diag_gemm_bf16(M, N, K, 0, 0, A, K, Bt, K, C, N, 0, ws, pair)
    torch.cuda.synchronize()
    ref = A.float() @ Bt.float().t()
    assert (C - ref).abs().max().item() <= 1e-4 * ref.abs().max().item()


def test_bounded_wait_reports_timeout_and_context_survives():
    from paper_2606_29758_gb300 import _binding as B
    ws = torch.empty(256, dtype=torch.uint8, device="cuda")
    B.ps_diag_wait_timeout(50_000_000, ws)   # 50 ms on a barrier nothing completes
    rc, bits = B.ps_workspace_status(ws)
    assert rc == B.PS_ERR_TIMEOUT and bits & B.PS_DEV_TIMEOUT
    # the context is still usable
    A = torch.ones(128, 64, device="cuda", dtype=torch.bfloat16)
    C = torch.empty(128, 256, device="cuda")
    Bt = torch.ones(256, 64, device="cuda", dtype=torch.bfloat16)
    B.ps_diag_gemm_bf16(128, 256, 64, 0, 0, A, 64, Bt, 64, C, 256, 0, ws)
    torch.cuda.synchronize()
    assert B.ps_workspace_status(ws)[0] == B.PS_OK
    assert torch.all(C == 64.0)
