"""The tcgen05 GEMM through the C ABI (ra_gemm_bf16, ra_gemm_bf16_epi) against a plain fp32
PyTorch matmul of the same bf16 operands on the CPU: single tile, ragged M/N/K tails, the
BERT/LLaMA shapes of the step, every fused epilogue of the step (bias, bias+GELU, the saved
GELU' factor, the multiply by it, the fp32 residual) and bitwise determinism."""
import numpy as np
import pytest

from paper_2502_19864_gb300 import ringada as R

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__
    __graft_entry__.build()


def _run(M, N, K, bias=False, gelu=False, seed=0):
    import torch
    g = torch.Generator(device="cpu").manual_seed(seed)
    A = torch.randn(M, K, generator=g).to(torch.bfloat16).cuda()
    B = (torch.randn(N, K, generator=g) * 0.05).to(torch.bfloat16).cuda()
    b = (torch.randn(N, generator=g) * 0.1).float().cuda() if bias else None
    C = torch.full((M, N), float("nan"), dtype=torch.bfloat16, device="cuda")
    G = torch.full((M, N), float("nan"), dtype=torch.bfloat16, device="cuda") if gelu else None
    R.ra_gemm_bf16(A.data_ptr(), B.data_ptr(), C.data_ptr(), M, N, K,
                   b.data_ptr() if bias else None, G.data_ptr() if gelu else None)
    torch.cuda.synchronize()
    ref = (A.float().cpu() @ B.float().cpu().T).cuda()
    if bias:
        ref = ref + b
    return C, G, ref


def _check(C, ref, tol=8e-3):
    c = C.float()
    assert not bool(c.isnan().any()), "unwritten outputs"
    err = (c - ref).abs().max().item()
    scale = ref.abs().max().item()
    # bf16 output rounding (2^-9 relative) plus fp32 accumulation-order differences
    assert err <= tol * scale, (err, scale)
    rel = ((c - ref).norm() / ref.norm()).item()
    assert rel <= 4e-3, rel


@pytest.mark.parametrize("M,N,K", [(128, 256, 64), (128, 128, 128), (256, 512, 192)])
def test_gemm_small_tiles(M, N, K):
    C, _, ref = _run(M, N, K)
    _check(C, ref)


@pytest.mark.parametrize("M,N,K", [(300, 200, 136), (77, 1000, 72), (1000, 8, 1024), (129, 264, 8)])
def test_gemm_ragged_tails(M, N, K):
    C, _, ref = _run(M, N, K)
    _check(C, ref)


@pytest.mark.parametrize("M,N,K", [(4096, 2304, 768), (4096, 768, 3072), (8192, 4096, 1024),
                                   (8192, 1024, 4096), (8192, 2048, 5632)])
def test_gemm_step_shapes(M, N, K):
    C, _, ref = _run(M, N, K)
    _check(C, ref)


# shapes whose tiles are 192 columns wide (N = 768 at 4096 rows; a ragged last tile,
# 760 = 3 x 192 + 184, with ragged rows), and N = 3072 at 8192 rows
@pytest.mark.parametrize("M,N,K", [(4096, 768, 768), (8192, 3072, 1024), (4000, 760, 200)])
def test_gemm_192_wide_tiles(M, N, K):
    C, _, ref = _run(M, N, K)
    _check(C, ref)


# (4096, 768): the bias+GELU epilogue on 192-wide tiles
@pytest.mark.parametrize("M,N,K", [(520, 384, 256), (4096, 768, 256)])
def test_gemm_bias_and_gelu_epilogue(M, N, K):
    import torch
    C, G, ref = _run(M, N, K, bias=True, gelu=True)
    _check(C, ref)
    _check(G, torch.nn.functional.gelu(ref), tol=1e-2)


def test_gemm_is_deterministic():
    C1, _, _ = _run(1024, 768, 768, seed=3)
    C2, _, _ = _run(1024, 768, 768, seed=3)
    assert bool((C1.view(-1).view(dtype=__import__("torch").int16) ==
                 C2.view(-1).view(dtype=__import__("torch").int16)).all())


def _operands(M, N, K, seed):
    import torch
    g = torch.Generator(device="cpu").manual_seed(seed)
    A = torch.randn(M, K, generator=g).to(torch.bfloat16)
    B = (torch.randn(N, K, generator=g) * 0.05).to(torch.bfloat16)
    acc = A.float() @ B.float().T          # CPU fp32 reference of the product
    return A.cuda(), B.cuda(), acc, g


@pytest.mark.parametrize("M,N,K", [(300, 264, 136), (8192, 4096, 1024)])
def test_gemm_gelu_factor_epilogue(M, N, K):
    """u = acc + bias: C2 = GELU(u), C = GELU'(u) (the factor the backward multiplies by)."""
    import torch
    A, B, acc, g = _operands(M, N, K, 5)
    b = torch.randn(N, generator=g) * 0.1
    C = torch.full((M, N), float("nan"), dtype=torch.bfloat16, device="cuda")
    G = torch.full((M, N), float("nan"), dtype=torch.bfloat16, device="cuda")
    bd = b.cuda()
    R.ra_gemm_bf16_epi(A.data_ptr(), B.data_ptr(), M, N, K, R.RA_EPI_BIAS_GELU_G, bd.data_ptr(),
                       None, C.data_ptr(), R.RA_BF16, G.data_ptr())
    torch.cuda.synchronize()
    u = (acc + b).double()
    phi = torch.exp(-0.5 * u * u) / (2 * torch.pi) ** 0.5
    Phi = 0.5 * (1 + torch.erf(u / 2 ** 0.5))
    _check(G, (u * Phi).float().cuda(), tol=1e-2)
    _check(C, (Phi + u * phi).float().cuda(), tol=1e-2)


@pytest.mark.parametrize("M,N,K", [(300, 264, 136), (8192, 4096, 1024)])
def test_gemm_multiply_epilogue(M, N, K):
    """C = acc * aux with a bf16 aux operand (the backward's dH GEMM)."""
    import torch
    A, B, acc, g = _operands(M, N, K, 6)
    aux = (torch.rand(M, N, generator=g) * 1.2).to(torch.bfloat16)
    C = torch.full((M, N), float("nan"), dtype=torch.bfloat16, device="cuda")
    auxd = aux.cuda()
    R.ra_gemm_bf16_epi(A.data_ptr(), B.data_ptr(), M, N, K, R.RA_EPI_MUL, None, auxd.data_ptr(),
                       C.data_ptr(), R.RA_BF16)
    torch.cuda.synchronize()
    _check(C, (acc * aux.float()).cuda())


@pytest.mark.parametrize("M,N,K", [(300, 264, 136), (8192, 1024, 3072)])
def test_gemm_residual_epilogue(M, N, K):
    """C = acc + aux, fp32 aux and output (the dX GEMM of the post-FFN adapter placement)."""
    import torch
    A, B, acc, g = _operands(M, N, K, 7)
    aux = torch.randn(M, N, generator=g)
    C = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
    auxd = aux.cuda()
    R.ra_gemm_bf16_epi(A.data_ptr(), B.data_ptr(), M, N, K, R.RA_EPI_RESID, None, auxd.data_ptr(),
                       C.data_ptr(), R.RA_F32)
    torch.cuda.synchronize()
    ref = (acc + aux).cuda()
    assert not bool(C.isnan().any())
    # fp32 output: only accumulation-order differences remain
    assert (C - ref).abs().max().item() <= 1e-4 * ref.abs().max().item()


def test_gemm_f32_store_epilogue():
    """C = acc in fp32 (the encoder's dX GEMMs), no bias."""
    import torch
    M, N, K = 8192, 1024, 4096
    A, B, acc, _ = _operands(M, N, K, 8)
    C = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
    R.ra_gemm_bf16_epi(A.data_ptr(), B.data_ptr(), M, N, K, R.RA_EPI_STORE, None, None,
                       C.data_ptr(), R.RA_F32)
    torch.cuda.synchronize()
    ref = acc.cuda()
    assert not bool(C.isnan().any())
    assert (C - ref).abs().max().item() <= 1e-4 * ref.abs().max().item()


# B given as stored [K, N] (a forward weight read by a dX GEMM, no transposed copy): tile
# widths 256 (N 1024), 192 (N 768 at 4096 rows), 128 (N 128), ragged N and K, and a
# multiply epilogue
@pytest.mark.parametrize("M,N,K,epi", [(8192, 1024, 4096, "store"), (4096, 768, 3072, "store"),
                                       (256, 128, 192, "store"), (300, 264, 136, "store"),
                                       (1000, 520, 72, "mul")])
def test_gemm_b_given_as_k_by_n(M, N, K, epi):
    import torch
    A, _, _, g = _operands(M, N, K, 9)
    Wkn = (torch.randn(K, N, generator=g) * 0.05).to(torch.bfloat16)
    acc = A.float().cpu() @ Wkn.float()
    aux = (torch.rand(M, N, generator=g) * 1.2).to(torch.bfloat16)
    Wd, auxd = Wkn.cuda(), aux.cuda()
    if epi == "mul":  # bf16 output, as the step's dH GEMM writes it
        C = torch.full((M, N), float("nan"), dtype=torch.bfloat16, device="cuda")
        R.ra_gemm_bf16_epi(A.data_ptr(), Wd.data_ptr(), M, N, K, R.RA_EPI_MUL | R.RA_EPI_B_KN, None,
                           auxd.data_ptr(), C.data_ptr(), R.RA_BF16)
        torch.cuda.synchronize()
        _check(C, (acc * aux.float()).cuda())
        return
    C = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
    R.ra_gemm_bf16_epi(A.data_ptr(), Wd.data_ptr(), M, N, K, R.RA_EPI_STORE | R.RA_EPI_B_KN, None,
                       None, C.data_ptr(), R.RA_F32)
    torch.cuda.synchronize()
    ref = acc.cuda()
    assert not bool(C.isnan().any())
    assert (C - ref).abs().max().item() <= 1e-4 * ref.abs().max().item()


# Stream-K: the k-blocks of the last, partial round of output tiles spread over all CTAs,
# their fp32 partials summed in a fixed order by the CTA that finishes each tile.  It applies
# where each CTA's share is at least 24 k-blocks: the BERT-large FFN-down / dY1 (K = 4096)
# and dX (K = 3072) shapes, 256 tiles of 128 x 256 on the SMs (1.7 rounds), with B as given
# or as stored [K, N], and ragged M, N and K; bias; bf16 and f32 outputs.  The K = 1024
# shapes (attention output, QKV) stay one tile per CTA, bitwise the result without scratch.
@pytest.mark.parametrize("M,N,K,bias,cdt,kn,sk", [
    (8192, 1024, 4096, False, "f32", False, True), (8192, 1024, 4096, False, "f32", True, True),
    (8192, 1024, 3072, False, "f32", True, True), (8192, 1024, 4096, True, "bf16", False, True),
    (8000, 1000, 4000, True, "f32", False, True), (8192, 1024, 1024, True, "f32", False, False),
    (8192, 3072, 1024, True, "f32", False, False)])
def test_gemm_stream_k(M, N, K, bias, cdt, kn, sk):
    import torch
    A, B, acc, g = _operands(M, N, K, 11)
    if kn:  # the same product with B handed over as stored [K, N]
        B = B.T.contiguous()
    b = (torch.randn(N, generator=g) * 0.1).float()
    ref = (acc + b if bias else acc).cuda()
    bd = b.cuda() if bias else None
    nbytes = R.ra_gemm_scratch_bytes()
    ws = torch.zeros(nbytes // 4, dtype=torch.int32, device="cuda")
    dt, rdt = (torch.bfloat16, R.RA_BF16) if cdt == "bf16" else (torch.float32, R.RA_F32)
    epi = R.RA_EPI_STORE | (R.RA_EPI_B_KN if kn else 0)

    def run(scratch, A_=A):
        C = torch.full((M, N), float("nan"), dtype=dt, device="cuda")
        R.ra_gemm_bf16_epi(A_.data_ptr(), B.data_ptr(), M, N, K, epi,
                           bd.data_ptr() if bias else None, None, C.data_ptr(), rdt, None,
                           ws.data_ptr() if scratch else None, nbytes if scratch else 0)
        torch.cuda.synchronize()
        return C

    # another product through the same scratch first: the flags it leaves must be clear
    # (160 slots x 12 epilogue warps of u32 flags at the start of the scratch)
    run(True, A_=torch.flip(A, [0]))
    assert int(ws[: 160 * 12].abs().sum().item()) == 0
    C1 = run(True)
    C2 = run(True)
    C0 = run(False)
    assert torch.equal(C1, C2), "stream-K result depends on timing"
    assert int(ws[: 160 * 12].abs().sum().item()) == 0
    if cdt == "bf16":
        _check(C1, ref)
    else:
        assert not bool(C1.isnan().any())
        assert (C1 - ref).abs().max().item() <= 1e-4 * ref.abs().max().item()
        # a split tile sums its k-blocks in another order than one accumulator does: some
        # fp32 outputs differ in their last bits where stream-K ran, none where it did not
        assert torch.equal(C1, C0) != sk
