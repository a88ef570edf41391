"""GPU parity for rotary position embedding by node position: fc_rope
against the oracle's O12, fc_tree_attn_rope (the queries rotated inside the
attention kernel) against the oracle attention that rotates queries and tree
keys, and the step loop with RoPE (tree keys rotated once, used by the
attention and by the cache append).

fc_rope computes in fp32 with the angle held to ~1e-7 rad, then rounds to
bf16, so a rotated value is within one bf16 rounding of the fp64 result; the
attention keeps the step's max-abs 2e-2.
"""
import numpy as np
import pytest
import torch

import paper_2502_17139_gb300.synth as synth

pytestmark = pytest.mark.gpu
ATOL = 2e-2


@pytest.fixture(scope="module")
def fc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2502_17139_gb300 import build
    build.build()
    import paper_2502_17139_gb300.fastcoder as fcm
    return fcm


def dev(a):
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint32:
        a = a.view(np.int32)
    return torch.from_numpy(a.copy()).cuda()


def bits(t):
    return t.cpu().view(torch.int16).numpy().view(np.uint16)


def f64(b16):
    return (b16.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


@pytest.mark.parametrize("layout,D,base", [(0, 128, 10000.0), (1, 128, 10000.0), (0, 64, 100000.0),
                                           (1, 256, 500000.0), (0, 128, 1000000.0)])
def test_rope_kernel_parity(fc, orc, layout, D, base):
    rng = np.random.default_rng(6000 + D + layout)
    B, n_pad, heads = 3, 64, 5
    shape = (B, n_pad, heads, D) if layout == 0 else (B, heads, n_pad, D)
    x = synth.randn_bf16(shape, 6100 + D, "cuda")
    pos = rng.integers(0, 1 << 22, (B, n_pad)).astype(np.int32)
    pos[:, :4] = (0, 1, 17, 65535)
    pos[:, -3:] = -1  # padding rows: left as they are
    y = fc.fc_rope(x, dev(pos), base, layout=layout)
    torch.cuda.synchronize()
    assert fc.fc_get_error() == "FC_OK"
    xb = bits(x)
    p_rows = pos[:, :, None] if layout == 0 else pos[:, None, :]
    p_full = np.broadcast_to(p_rows, shape[:-1])
    ref = orc.rope(f64(xb), np.maximum(p_full, 0), base)
    got = f64(bits(y))
    valid = p_full >= 0
    err = np.abs(got - ref)[valid]
    tol = (2.0 ** -8) * np.abs(ref)[valid] + 1e-5
    assert (err <= tol).all(), float((err - tol).max())
    assert np.array_equal(bits(y)[~valid], xb[~valid])
    # in place gives the same
    z = x.clone()
    fc.fc_rope(z, dev(pos), base, layout=layout, out=z)
    assert torch.equal(z, y)


def _rope_attn_case(fc, orc, seed, B, n_pad, H, Hkv, kv_len, cap, base=10000.0, workspace="auto", pos_shift=0):
    rng = synth.rng_for(60, seed)
    par = np.full((B, n_pad), -1, np.int32)
    nn = rng.integers(1, n_pad + 1, B).astype(np.int32)
    for b in range(B):
        _, p = synth.random_tree(rng, int(nn[b]), 10, 4, 1000)
        par[b, :nn[b]] = p
    kvl = np.asarray(kv_len, np.int32)
    D = 128
    q = synth.randn_bf16((B, n_pad, H, D), 1100 + seed, "cuda")
    kc = synth.randn_bf16((B, Hkv, cap, D), 2100 + seed, "cuda")
    vc = synth.randn_bf16((B, Hkv, cap, D), 3100 + seed, "cuda")
    kt = synth.randn_bf16((B, Hkv, n_pad, D), 4100 + seed, "cuda")
    vt = synth.randn_bf16((B, Hkv, n_pad, D), 5100 + seed, "cuda")
    gm = fc.fc_tree_mask(dev(par), dev(nn), dev(kvl))
    pos = gm["pos"] + pos_shift if pos_shift else gm["pos"]
    k_rot = fc.fc_rope(kt, pos, base, layout=1)
    out = torch.full_like(q, float("nan"))
    fc.fc_tree_attn_rope(q, kc, vc, dev(kvl), k_rot, vt, gm["mask"], dev(nn), pos, base, out=out, workspace=workspace)
    torch.cuda.synchronize()
    assert fc.fc_get_error() == "FC_OK"
    rm = orc.tree_mask(par, nn, kvl, n_pad)
    ref_pos = rm["pos"] + pos_shift if pos_shift else rm["pos"]
    ref = orc.tree_attn(bits(q), bits(kc), bits(vc), kvl, bits(kt), bits(vt), rm["mask"], nn, pos=ref_pos,
                        rope_base=base)
    got = out.float().cpu().numpy()
    assert np.isfinite(got).all()
    err = np.abs(got - ref).max()
    assert err <= ATOL, err
    return err


def test_rope_attn_c5_shape(fc, orc):
    _rope_attn_case(fc, orc, 1, 4, 128, 32, 8, [300, 17, 1000, 0], 1024)


def test_rope_attn_mha_n64(fc, orc):
    _rope_attn_case(fc, orc, 2, 3, 64, 8, 8, [64, 129, 5], 160, base=100000.0)


def test_rope_attn_long_positions_and_split(fc, orc):
    # positions near 2^20 and a cache long enough for the key split to engage
    _rope_attn_case(fc, orc, 3, 2, 128, 16, 2, [4000, 2500], 4096, pos_shift=1 << 20)
    _rope_attn_case(fc, orc, 4, 2, 128, 16, 2, [4000, 2500], 4096, workspace=None)


def test_rope_attn_matches_plain_at_equal_positions(fc, orc):
    """All positions equal and no cached keys: the rotations cancel, so the
    rotated attention must match the plain kernel within the bf16 rounding of
    the rotated operands."""
    rng = synth.rng_for(61)
    B, n_pad, H, Hkv, D = 3, 64, 8, 4, 128
    par = np.full((B, n_pad), -1, np.int32)
    nn = rng.integers(1, n_pad + 1, B).astype(np.int32)
    for b in range(B):
        _, p = synth.random_tree(rng, int(nn[b]), 10, 4, 1000)
        par[b, :nn[b]] = p
    kvl = np.zeros(B, np.int32)
    q = synth.randn_bf16((B, n_pad, H, D), 71, "cuda")
    kc = synth.randn_bf16((B, Hkv, 16, D), 72, "cuda")
    kt = synth.randn_bf16((B, Hkv, n_pad, D), 73, "cuda")
    vt = synth.randn_bf16((B, Hkv, n_pad, D), 74, "cuda")
    gm = fc.fc_tree_mask(dev(par), dev(nn), dev(kvl))
    pos = torch.full((B, n_pad), 777, dtype=torch.int32, device="cuda")
    k_rot = fc.fc_rope(kt, pos, 10000.0, layout=1)
    a = fc.fc_tree_attn_rope(q, kc, kc, dev(kvl), k_rot, vt, gm["mask"], dev(nn), pos, 10000.0)
    b = fc.fc_tree_attn(q, kc, kc, dev(kvl), kt, vt, gm["mask"], dev(nn))
    torch.cuda.synchronize()
    assert (a.float() - b.float()).abs().max().item() <= ATOL


def test_step_loop_rope_first_step(fc, orc):
    """The step loop with RoPE: the first step's attention against the
    oracle's own retrieval, tree and rotated attention, and the cache rows the
    append wrote against the oracle's rotation of the accepted path's keys."""
    from paper_2502_17139_gb300.step import StepLoop
    rng = synth.rng_for(74)
    Tr, _ = synth.make_corpus(rng, 200_000, 1.3, synth.VOCAB, n_grams=500, len_range=(8, 64))
    Tc, _ = synth.make_corpus(rng, 1_000_000, 1.1, synth.VOCAB)
    B, n_pad, H, Hkv, D, kv0 = 4, 128, 8, 2, 128, 100
    stride = 128 + 24
    ctx, cl, _ = synth.make_contexts(rng, B, 128, 16, [Tr, Tc, None], [0.5, 0.25, 0.25], 1.1, ctx_stride=stride)
    plen, rtok = synth.argmax_draws(rng, B, n_pad)
    cap = kv0 + 16
    kc0 = synth.randn_bf16((B, Hkv, cap, D), 81, "cuda")
    vc0 = synth.randn_bf16((B, Hkv, cap, D), 82, "cuda")
    q = synth.randn_bf16((B, n_pad, H, D), 83, "cuda")
    kt = synth.randn_bf16((B, Hkv, n_pad, D), 84, "cuda")
    vt = synth.randn_bf16((B, Hkv, n_pad, D), 85, "cuda")
    srcs = [fc.fc_datastore_build(dev(Tr), synth.VOCAB), fc.fc_datastore_build(dev(Tc), synth.VOCAB)]
    loop = StepLoop(srcs, ctx, cl, fc.params(16, 2, 64, 10, 4096), n_pad, n_pad, [1, 1], H, Hkv, D, kv_cap=cap,
                    kv_len0=kv0, vocab=synth.VOCAB, k_cache=kc0.clone(), v_cache=vc0.clone(), rope_base=10000.0)
    zeros = torch.zeros(B, dtype=torch.int32, device="cuda")
    loop.step(q, kt, vt, zeros, dev(plen), dev(rtok))
    torch.cuda.synchronize()
    assert fc.fc_get_error() == "FC_OK"
    # the oracle's own first step
    res = [orc.retrieve(T, ctx, cl, 16, 2, 64, 10, 4096) for T in (Tr, Tc)]
    root = ctx[np.arange(B), cl - 1]
    kvl = np.full(B, kv0, np.int32)
    tr = orc.build_tree(res, [1, 1], root, kvl, n_pad, n_pad)
    ref = orc.tree_attn(bits(q), bits(kc0), bits(vc0), kvl, bits(kt), bits(vt), tr["mask"], tr["n_nodes"],
                        pos=tr["pos"])
    got = loop.attn_out.float().cpu().numpy()
    assert np.abs(got - ref).max() <= ATOL
    am = orc.synth_argmax(tr["tok"], tr["parent"], tr["n_nodes"], plen, rtok, synth.VOCAB)
    ac = orc.accept(tr["tok"], tr["parent"], tr["n_nodes"], am, 12)
    kcache = f64(bits(loop.k_cache))
    ktb = f64(bits(kt))
    for b in range(B):
        for t in range(int(ac["acc_len"][b]) + 1):
            node = int(ac["path"][b, t])
            want = orc.rope(ktb[b, :, node, :], np.full(Hkv, tr["pos"][b, node]), 10000.0)
            gotr = kcache[b, :, kv0 + t, :]
            assert (np.abs(gotr - want) <= (2.0 ** -8) * np.abs(want) + 1e-5).all(), (b, t)
