"""GPU parity of fc_gemm_bf16 (the decoder's GEMM, a tcgen05 kernel) against
fp64 products of the same bf16 operands.

The tolerance is derived, not tuned.  The products of two bf16 values are
exact in fp32; the tensor cores add them in fp32 in some order, which is off
from the exact sum by at most gamma_K * sum_k |a_ik b_kj| with
gamma_K = K u / (1 - K u), where u is taken as 2^-23 (the spacing of fp32
near 1, so that even truncating additions are covered); rounding the result
to bf16 (8 significant bits, round to nearest) adds at most 2^-8 of its
magnitude.  So, element by element,

    |c - exact| <= 2^-8 |exact| + (1 + 2^-8) gamma_K (|A| |B|).

A dropped 16-deep slice, a swapped operand or a misplaced tile breaks this
bound by orders of magnitude.  Shapes cover ragged M, N and K (tiles past
every edge), one row, and the decoder's own shapes at DeepSeek-Coder 1.3B's
width with 2048 tree rows, where each CTA runs many tiles and both tensor
memory accumulators.
"""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def fc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2502_17139_gb300 import build
    build.build()
    import paper_2502_17139_gb300.fastcoder as fcm
    return fcm


def bound_check(a, b, c):
    A = a.double().cpu().numpy()
    Bm = b.double().cpu().numpy()
    exact = A @ Bm
    mag = np.abs(A) @ np.abs(Bm)
    K = A.shape[1]
    u = 2.0 ** -23
    gamma = K * u / (1 - K * u)
    got = c.double().cpu().numpy()
    err = np.abs(got - exact)
    lim = 2.0 ** -8 * np.abs(exact) + (1 + 2.0 ** -8) * gamma * mag
    assert np.isfinite(got).all()
    bad = err > lim
    assert not bad.any(), (int(bad.sum()), float((err - lim).max()))
    return float(err.max())


def operands(M, N, K, seed, scale_b=None):
    g = torch.Generator().manual_seed(seed)
    a = torch.randn((M, K), generator=g).to(torch.bfloat16).cuda()
    b = (torch.randn((K, N), generator=g) * (scale_b or K ** -0.5)).to(torch.bfloat16).cuda()
    return a, b


@pytest.mark.parametrize("M,N,K", [(777, 392, 256), (129, 264, 72), (300, 520, 200), (1, 8, 8), (128, 256, 64),
                                   (255, 1032, 1000), (4100, 64, 520)])
def test_gemm_ragged_shapes(fc, M, N, K):
    a, b = operands(M, N, K, M * 7 + N)
    c = torch.full((M, N), float("nan"), dtype=torch.bfloat16, device="cuda")
    fc.fc_gemm_bf16(a, b, out=c)
    torch.cuda.synchronize()
    assert fc.fc_get_error() == "FC_OK"
    bound_check(a, b, c)


@pytest.mark.parametrize("K,N", [(2048, 2048), (2048, 4096), (2048, 11008), (5504, 2048), (2048, 32256)])
def test_gemm_decoder_shapes(fc, K, N):
    """The decoder's GEMMs over 2048 tree rows (32 sequences x 64 nodes):
    Q, fused K/V, output, fused gate/up and down projections, and the LM
    head."""
    M = 2048
    a, b = operands(M, N, K, K + N)
    c = fc.fc_gemm_bf16(a, b)
    torch.cuda.synchronize()
    assert fc.fc_get_error() == "FC_OK"
    bound_check(a, b, c)


def test_gemm_back_to_back_and_empty(fc):
    a, b = operands(640, 768, 384, 5)
    c1 = fc.fc_gemm_bf16(a, b)
    c2 = fc.fc_gemm_bf16(a, b)
    torch.cuda.synchronize()
    assert torch.equal(c1, c2)  # deterministic: the same tiles, the same order
    empty = torch.empty((0, 384), dtype=torch.bfloat16, device="cuda")
    assert fc.fc_gemm_bf16(empty, b).shape == (0, 768)
    bad = torch.empty((16, 12), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(fc.FastCoderError) as e:
        fc.fc_gemm_bf16(bad, torch.empty((12, 16), dtype=torch.bfloat16, device="cuda"))
    assert e.value.status == "FC_ERR_UNSUPPORTED"
    assert fc.fc_get_error() == "FC_OK"
