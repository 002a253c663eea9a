"""The tcgen05 dual GEMM against float64 products of the same bf16 operands.

Shapes span several 128 x BN tiles, ragged M/N/K tails and every product-term mask the
sweep uses (primal, dual forward, dual input layer, weight-tangent sum)."""
import numpy as np
import pytest

from gpu_util import need_gpu, rel_l2

SHAPES = [(128, 128, 64), (256, 1024, 1024), (256, 10, 1024), (1024, 1024, 512),
          (77, 45, 136), (130, 300, 8), (512, 4096, 256), (300, 16, 40)]
MASKS = [1, 1 | 8 | 16, 1 | 16, 2 | 4, 4, 1 | 2 | 4 | 8 | 16, 1 | 32, 2 | 4 | 32]


def _ref(A0, A1, B0, B1, mask):
    a0, a1, b0, b1 = (x.double().cpu() for x in (A0, A1, B0, B1))
    c0 = None
    c1 = None
    terms0 = [(1, a0, b0), (2, a1, b0), (4, a0, b1), (32, a1, b1)]
    terms1 = [(8, a1, b0), (16, a0, b1)]
    for bit, a, b in terms0:
        if mask & bit:
            c0 = a @ b.T if c0 is None else c0 + a @ b.T
    for bit, a, b in terms1:
        if mask & bit:
            c1 = a @ b.T if c1 is None else c1 + a @ b.T
    return c0, c1


@pytest.mark.gpu
@pytest.mark.parametrize("shape", SHAPES)
@pytest.mark.parametrize("mask", MASKS)
def test_dual_gemm(shape, mask):
    torch, native = need_gpu()
    M, N, K = shape
    g = torch.Generator(device="cpu").manual_seed(M * 131 + N * 7 + K + mask)
    mk = lambda r: (torch.randn(r, K, generator=g)).to(torch.bfloat16).cuda()
    A0, A1, B0, B1 = mk(M), mk(M), mk(N), mk(N)
    C0 = torch.full((M, N), float("nan"), device="cuda")
    C1 = torch.full((M, N), float("nan"), device="cuda")
    bias0 = torch.randn(N, generator=g).cuda()
    bias1 = torch.randn(N, generator=g).cuda()
    native.mf_dual_gemm_bf16(M, N, K, A0, A1, B0, B1, C0, C1, mask, bias0, bias1)
    torch.cuda.synchronize()
    r0, r1 = _ref(A0, A1, B0, B1, mask)
    if r0 is not None:
        r0 = r0 + bias0.double().cpu()
        assert rel_l2(C0.cpu().numpy(), r0.numpy()) < 1e-5
    if r1 is not None:
        r1 = r1 + bias1.double().cpu()
        assert rel_l2(C1.cpu().numpy(), r1.numpy()) < 1e-5


@pytest.mark.gpu
def test_dual_gemm_strided_operands():
    """Leading dimensions larger than K (padded operand buffers)."""
    torch, native = need_gpu()
    M, N, K, ld = 200, 96, 72, 88
    g = torch.Generator(device="cpu").manual_seed(3)
    A0 = torch.randn(M, ld, generator=g).to(torch.bfloat16).cuda()
    B0 = torch.randn(N, ld, generator=g).to(torch.bfloat16).cuda()
    C0 = torch.zeros(M, N + 8, device="cuda")
    native.mf_dual_gemm_bf16(M, N, K, A0, None, B0, None, C0, None, 1)
    torch.cuda.synchronize()
    ref = A0[:, :K].double().cpu() @ B0[:, :K].double().cpu().T
    assert rel_l2(C0[:, :N].cpu().numpy(), ref.numpy()) < 1e-5
    assert float(C0[:, N:].abs().max()) == 0.0


def _set_pair_mode(native, value):
    """MF_OPT_GEMM_2SM is process-wide; any handle can set it."""
    from paper_2505_00793_gb300 import synth
    mf = native.MixFlow.for_workload(synth.WORKLOADS["tiny"])
    mf.set_option(native.MF_OPT_GEMM_2SM, value)
    mf.close()


PAIR_SHAPES = [(256, 1024, 1024), (1024, 1024, 512), (130, 300, 8), (512, 4096, 256),
               (300, 16, 40), (600, 520, 200), (256, 256, 64), (1000, 130, 1096)]


@pytest.mark.gpu
@pytest.mark.parametrize("shape", PAIR_SHAPES)
@pytest.mark.parametrize("mask", MASKS)
def test_dual_gemm_pair_tiles(shape, mask):
    """The same products on 256-row tiles computed by CTA pairs (tcgen05 cta_group::2)."""
    torch, native = need_gpu()
    _set_pair_mode(native, 2)
    try:
        test_dual_gemm(shape, mask)
    finally:
        _set_pair_mode(native, 1)


MN_SHAPES = [(256, 1024, 1024), (1025, 1024, 256), (300, 10, 72), (130, 200, 40), (1000, 520, 200)]


@pytest.mark.gpu
@pytest.mark.parametrize("shape", MN_SHAPES)
@pytest.mark.parametrize("layout", [1, 2, 3])
@pytest.mark.parametrize("mask", [1, 1 | 8 | 16, 2 | 4, 1 | 32])
@pytest.mark.parametrize("pair_mode", [1, 2])
def test_dual_gemm_mn_major(shape, layout, mask, pair_mode):
    """Operands stored MN-major ([K][rows], rows contiguous; layout bit 0 for A, bit 1 for B),
    on one-SM and CTA-pair tiles."""
    torch, native = need_gpu()
    M, N, K = shape
    g = torch.Generator(device="cpu").manual_seed(M * 17 + N * 3 + K + mask + layout)
    ld8 = lambda n: (n + 7) // 8 * 8
    def op(rows, mn):
        x = torch.randn(rows, K, generator=g).to(torch.bfloat16)
        if not mn:
            return x, x.cuda()
        store = torch.zeros(K, ld8(rows), dtype=torch.bfloat16)
        store[:, :rows] = x.t()
        return x, store.cuda()
    a_mn, b_mn = bool(layout & 1), bool(layout & 2)
    (a0, A0), (a1, A1) = op(M, a_mn), op(M, a_mn)
    (b0, B0), (b1, B1) = op(N, b_mn), op(N, b_mn)
    C0 = torch.full((M, N), float("nan"), device="cuda")
    C1 = torch.full((M, N), float("nan"), device="cuda")
    _set_pair_mode(native, pair_mode)
    try:
        native.mf_dual_gemm_bf16(M, N, K, A0, A1, B0, B1, C0, C1, mask | (layout << 8))
        torch.cuda.synchronize()
    finally:
        _set_pair_mode(native, 1)
    r0, r1 = _ref(a0, a1, b0, b1, mask)
    if r0 is not None:
        assert rel_l2(C0.cpu().numpy(), r0.numpy()) < 1e-5
    if r1 is not None:
        assert rel_l2(C1.cpu().numpy(), r1.numpy()) < 1e-5
