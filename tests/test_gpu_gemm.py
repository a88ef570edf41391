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


def gemm_magnitude(a, b):
    """Exact product and the fp32-accumulation error bound per element."""
    A = a.double().cpu().numpy()
    Bm = b.double().cpu().numpy()
    K = A.shape[1]
    u = 2.0 ** -23
    return A @ Bm, K * u / (1 - K * u) * (np.abs(A) @ np.abs(Bm))


@pytest.mark.parametrize("batch,n_pad,Hkv,K", [(3, 64, 2, 256), (2, 128, 1, 520), (5, 64, 3, 2048)])
def test_gemm_kv_heads(fc, orc, batch, n_pad, Hkv, K):
    """The K/V projection with RoPE and the head-major layout in its epilogue,
    against the exact product rotated by the oracle's RoPE (O12).  Bound per
    element: one bf16 rounding of the result, plus the accumulation bound of
    both members of the rotated pair, plus 2^-20 of their magnitudes for the
    fp32 rotation (angle to ~1e-7 rad)."""
    M, D = batch * n_pad, 128
    a, w = operands(M, 2 * Hkv * D, K, 11 * K + Hkv)
    rng = np.random.default_rng(K)
    pos = rng.integers(0, 70000, (batch, n_pad)).astype(np.int32)
    pos[:, -5:] = -1  # padding rows stay unrotated
    k_rot = torch.full((batch, Hkv, n_pad, D), float("nan"), dtype=torch.bfloat16, device="cuda")
    v_heads = torch.full_like(k_rot, float("nan"))
    fc.fc_gemm_kv_heads(a, w, batch, n_pad, Hkv, torch.from_numpy(pos).cuda(), 10000.0, k_rot, v_heads)
    torch.cuda.synchronize()
    assert fc.fc_get_error() == "FC_OK"
    exact, G = gemm_magnitude(a, w)
    kv = exact.reshape(batch, n_pad, 2, Hkv, D)
    Gk = G.reshape(batch, n_pad, 2, Hkv, D)
    kk = kv[:, :, 0]
    p = np.repeat(pos[:, :, None], Hkv, 2)
    want_k = orc.rope(kk, np.maximum(p, 0))
    want_k[p < 0] = kk[p < 0]
    pair = lambda x: x + np.concatenate([x[..., 64:], x[..., :64]], -1)  # |x_d| + |x_(d +- 64)|
    lim_k = 2.0 ** -8 * np.abs(want_k) + (1 + 2.0 ** -8) * pair(Gk[:, :, 0]) + 2.0 ** -20 * pair(np.abs(kk))
    got_k = k_rot.double().cpu().numpy().transpose(0, 2, 1, 3)
    assert (np.abs(got_k - want_k) <= lim_k).all()
    want_v = kv[:, :, 1]
    lim_v = 2.0 ** -8 * np.abs(want_v) + (1 + 2.0 ** -8) * Gk[:, :, 1]
    got_v = v_heads.double().cpu().numpy().transpose(0, 2, 1, 3)
    assert (np.abs(got_v - want_v) <= lim_v).all()


def test_interleave_gate_up(fc):
    K, inter = 72, 384
    w = torch.randn((K, 2 * inter)).to(torch.bfloat16).cuda()
    out = fc.fc_interleave_gate_up(w)
    torch.cuda.synchronize()
    g, u = w[:, :inter].cpu(), w[:, inter:].cpu()
    o = out.cpu().view(K, inter // 128, 2, 128)
    assert torch.equal(o[:, :, 0].reshape(K, inter), g) and torch.equal(o[:, :, 1].reshape(K, inter), u)


@pytest.mark.parametrize("M,K,inter", [(777, 512, 384), (2048, 2048, 5504)])
def test_gemm_silu_mul(fc, M, K, inter):
    """silu(A Wg) * (A Wu) from the fp32 accumulators, rounded once: within one
    bf16 rounding of the exact value, plus the accumulation bounds carried
    through (|d silu / dg| <= 1.1), plus 2^-10 of the value for the fp32
    evaluation with the hardware exponential."""
    a, w = operands(M, 2 * inter, K, M + inter)
    act = torch.empty((M, inter), dtype=torch.bfloat16, device="cuda")
    fc.fc_gemm_silu_mul(a, fc.fc_interleave_gate_up(w), act)
    torch.cuda.synchronize()
    assert fc.fc_get_error() == "FC_OK"
    exact, G = gemm_magnitude(a, w)
    g, u = exact[:, :inter], exact[:, inter:]
    silu = g / (1 + np.exp(-g))
    ref = silu * u
    lim = (2.0 ** -8 + 2.0 ** -10) * np.abs(ref) + 1.1 * np.abs(u) * G[:, :inter] + np.abs(silu) * G[:, inter:] \
        + G[:, :inter] * G[:, inter:] + 1e-30
    got = act.double().cpu().numpy()
    assert (np.abs(got - ref) <= lim).all()
