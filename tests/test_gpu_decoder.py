"""GPU parity for the decoder forward over a draft tree (paper_2502_17139_gb300/
decoder.py) against the fp64 oracle (oracle/decoder.py), on seeded
random-init weights of a small LLaMA-family shape.

The GPU keeps bf16 between operations (fp32 inside each).  Two checks follow
from that arithmetic instead of a hand-picked number:

* Op by op: every operation of the forward, applied by the oracle in fp64 to
  the GPU's own bf16 inputs, must match the GPU's output within that
  operation's rounding bound: a GEMM within 2^-8 |C| (the bf16 store) plus
  (1 + 2^-8) gamma_K (|A| |B|) (fp32 accumulation, gamma_K = K u / (1 - K u),
  u = 2^-23); an add or a norm within one bf16 rounding plus its fp32 error;
  SiLU * up within two bf16 roundings; the tree attention within its 2e-2.
* End to end: the oracle's forward with the GPU's bf16 storage points
  (store_bf16=True) moves the exact forward by the rounding alone.  The GPU
  rounds at the same points from fp32 values that differ only in the last
  bits, so its distance from the exact forward is of the same order; the test
  allows three times the mirror's distance, element by element in the worst
  case, for logits and the rotated keys and values.  Greedy predictions must
  agree wherever the oracle's top-2 logit gap exceeds that tolerance.
"""
import numpy as np
import pytest
import torch

import paper_2502_17139_gb300.synth as synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def fc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2502_17139_gb300 import build
    build.build()
    import paper_2502_17139_gb300.fastcoder as fcm
    return fcm


@pytest.fixture(scope="module")
def dec(orc):
    from oracle import decoder
    return decoder


def dev(a):
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint32:
        a = a.view(np.int32)
    return torch.from_numpy(a.copy()).cuda()


def f64(t):
    return t.float().cpu().numpy().astype(np.float64)


def test_blocks(fc, dec):
    rng = np.random.default_rng(7000)
    torch.manual_seed(7001)
    # GEMM, rows not a multiple of any tile
    a = torch.randn((777, 256)).to(torch.bfloat16).cuda()
    b = (torch.randn((256, 392)) / 16).to(torch.bfloat16).cuda()
    c = fc.fc_gemm_bf16(a, b)
    ref = f64(a) @ f64(b)
    assert np.abs(f64(c) - ref).max() <= 2.0 ** -7 * np.abs(ref).max()
    # embedding with padding ids
    table = torch.randn((300, 256)).to(torch.bfloat16).cuda()
    ids = rng.integers(0, 300, 64).astype(np.uint32)
    ids[[3, 9]] = 0xFFFFFFFF
    out = torch.empty((64, 256), dtype=torch.bfloat16, device="cuda")
    fc.fc_embed(dev(ids), table, out)
    want = f64(table)[np.minimum(ids, 299).astype(np.int64)]
    want[[3, 9]] = 0
    assert np.array_equal(f64(out), want)
    # residual add + RMSNorm
    x = torch.randn((50, 264)).to(torch.bfloat16).cuda()
    r = torch.randn((50, 264)).to(torch.bfloat16).cuda()
    w = (1 + 0.1 * torch.randn(264)).to(torch.bfloat16).cuda()
    x0 = f64(x)
    o = torch.empty_like(x)
    fc.fc_add_rmsnorm(x, r, w, o, 1e-6)
    xs = x0 + f64(r)
    assert np.abs(f64(x) - xs).max() <= 2.0 ** -8 * np.abs(xs).max()
    ref = dec.rmsnorm(f64(x), f64(w), 1e-6)
    assert np.abs(f64(o) - ref).max() <= 2.0 ** -7 * np.abs(ref).max()
    # SiLU * up
    gu = torch.randn((40, 2 * 96)).to(torch.bfloat16).cuda()
    act = torch.empty((40, 96), dtype=torch.bfloat16, device="cuda")
    fc.fc_silu_mul(gu, act)
    g = f64(gu)
    ref = dec.silu(g[:, :96]) * g[:, 96:]
    assert np.abs(f64(act) - ref).max() <= 2.0 ** -7 * np.abs(ref).max() + 1e-3
    assert fc.fc_get_error() == "FC_OK"


def test_rope_heads(fc, orc):
    rng = np.random.default_rng(7100)
    B, n_pad, Hkv, D = 2, 64, 3, 128
    kv = torch.randn((B * n_pad, 2 * Hkv * D)).to(torch.bfloat16).cuda()
    pos = rng.integers(0, 50000, (B, n_pad)).astype(np.int32)
    pos[0, -2:] = -1
    k = torch.empty((B, Hkv, n_pad, D), dtype=torch.bfloat16, device="cuda")
    v = torch.empty_like(k)
    fc.fc_rope_heads(kv, 0, 2 * Hkv * D, k, B, n_pad, Hkv, D, dev(pos), 10000.0)
    fc.fc_rope_heads(kv, Hkv * D, 2 * Hkv * D, v, B, n_pad, Hkv, D, dev(pos), 0.0)
    x = f64(kv).reshape(B, n_pad, 2, Hkv, D)
    want_v = x[:, :, 1].transpose(0, 2, 1, 3)
    assert np.array_equal(f64(v), want_v)
    kk = x[:, :, 0].transpose(0, 2, 1, 3)
    p = np.broadcast_to(pos[:, None, :], (B, Hkv, n_pad))
    want_k = orc.rope(kk, np.maximum(p, 0), 10000.0)
    want_k[p < 0] = kk[p < 0]
    assert (np.abs(f64(k) - want_k) <= 2.0 ** -8 * np.abs(want_k) + 1e-5).all()


SHAPES = [dict(hidden=256, layers=2, H=4, Hkv=2, inter=384, vocab=304),
          dict(hidden=512, layers=2, H=4, Hkv=4, inter=768, vocab=1000)]


U32 = 2.0 ** -23
BF = 2.0 ** -8


def gemm_bound_ok(a, b, c):
    exact = a @ b
    K = a.shape[1]
    gamma = K * U32 / (1 - K * U32)
    lim = BF * np.abs(exact) + (1 + BF) * gamma * (np.abs(a) @ np.abs(b))
    return bool((np.abs(c - exact) <= lim).all())


def chained_layer_checks(fc, dec, td, s, tok, nn, mask, pos, kvl):
    """Runs the decoder's operations one by one on the GPU (as TreeDecoder.forward
    does) and checks each against its fp64 definition on the GPU's own inputs."""
    B, n_pad = td.B, td.n_pad
    rows = np.concatenate([np.arange(b * n_pad, b * n_pad + int(nn[b])) for b in range(B)])
    W = td.W
    fc.fc_embed(dev(tok).reshape(-1), W["embed"], td.x)
    r = None
    checked = 0
    for l, Lw in enumerate(W["layers"]):
        x0 = f64(td.x)
        rr = None if r is None else f64(r)
        fc.fc_add_rmsnorm(td.x, r, Lw["attn_norm"], td.h, s.eps)
        xs = x0 if rr is None else x0 + rr
        assert (np.abs(f64(td.x) - xs) <= (BF + U32) * np.abs(xs)).all()
        ref = dec.rmsnorm(f64(td.x), f64(Lw["attn_norm"]), s.eps)
        d = s.hidden * U32 + 2.0 ** -18
        assert (np.abs(f64(td.h) - ref)[rows] <= (BF * (1 + d) + d) * np.abs(ref)[rows] + 1e-30).all()
        h = f64(td.h)
        fc.fc_gemm_bf16(td.h, Lw["wq"], out=td.q)
        assert gemm_bound_ok(h[rows], f64(Lw["wq"]), f64(td.q)[rows])
        # the K/V projection, rotated and laid out head-major in the GEMM's epilogue
        fc.fc_gemm_kv_heads(td.h, Lw["wkv"], B, n_pad, s.Hkv, pos, s.rope_base, td.k_rot[l], td.v_heads[l])
        wkv = f64(Lw["wkv"])
        K = wkv.shape[0]
        G = K * U32 / (1 - K * U32) * (np.abs(h) @ np.abs(wkv))
        kv = (h @ wkv).reshape(B, n_pad, 2, s.Hkv, s.D)
        Gk = G.reshape(B, n_pad, 2, s.Hkv, s.D)
        pp = np.repeat(pos.cpu().numpy()[:, :, None], s.Hkv, 2)
        from oracle import oracle as orc
        want_k = orc.rope(kv[:, :, 0], np.maximum(pp, 0), s.rope_base)
        want_k[pp < 0] = kv[:, :, 0][pp < 0]
        pair = lambda x: x + np.concatenate([x[..., 64:], x[..., :64]], -1)
        lim = BF * np.abs(want_k) + (1 + BF) * pair(Gk[:, :, 0]) + 2.0 ** -20 * pair(np.abs(kv[:, :, 0]))
        got_k = f64(td.k_rot[l]).transpose(0, 2, 1, 3)
        assert (np.abs(got_k - want_k) <= lim).all()
        got_v = f64(td.v_heads[l]).transpose(0, 2, 1, 3)
        assert (np.abs(got_v - kv[:, :, 1]) <= BF * np.abs(kv[:, :, 1]) + (1 + BF) * Gk[:, :, 1]).all()
        fc.fc_tree_attn_rope(td.q.view(B, n_pad, s.H, s.D), td.k_cache[l], td.v_cache[l], kvl, td.k_rot[l],
                             td.v_heads[l], mask, dev(nn), pos, s.rope_base, out=td.attn.view(B, n_pad, s.H, s.D))
        torch.cuda.synchronize()
        # the attention on the GPU's own bf16 inputs, every row, in fp64
        bits = lambda t: t.cpu().view(torch.int16).numpy().view(np.uint16)
        # fc_tree_attn_rope rotates Q while staging it (the tree keys arrive rotated):
        # rotate Q here and round it to bf16 as the kernel stores it
        qh = orc.rope(f64(td.q.view(B, n_pad, s.H, s.D)), np.repeat(pos.cpu().numpy()[:, :, None], s.H, 2))
        qb = dec.round_bf16(qh)  # the kernel keeps rotated Q in bf16 in shared memory
        qbits = (qb.astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)
        ref_a = orc.tree_attn(qbits, bits(td.k_cache[l]), bits(td.v_cache[l]), kvl.cpu().numpy(), bits(td.k_rot[l]),
                              bits(td.v_heads[l]), mask.cpu().numpy().view(np.uint64), nn)
        got_a = f64(td.attn.view(B, n_pad, s.H, s.D))
        for b in range(B):
            assert np.abs(got_a[b, :nn[b]] - ref_a[b, :nn[b]]).max() <= 2e-2
        a = f64(td.attn)
        fc.fc_gemm_bf16(td.attn, Lw["wo"], out=td.o)
        assert gemm_bound_ok(a[rows], f64(Lw["wo"]), f64(td.o)[rows])
        x0, o = f64(td.x), f64(td.o)
        fc.fc_add_rmsnorm(td.x, td.o, Lw["mlp_norm"], td.h, s.eps)
        assert (np.abs(f64(td.x) - (x0 + o)) <= (BF + U32) * np.abs(x0 + o)).all()
        h = f64(td.h)
        # the gate/up projection with SiLU * up in the GEMM's epilogue
        fc.fc_gemm_silu_mul(td.h, td.wgu[l], td.act)
        wgu = f64(Lw["wgu"])
        K = wgu.shape[0]
        G = K * U32 / (1 - K * U32) * (np.abs(h) @ np.abs(wgu))
        gu = h @ wgu
        g, u = gu[:, :s.inter], gu[:, s.inter:]
        silu = dec.silu(g)
        ref = silu * u
        lim = (BF + 2.0 ** -10) * np.abs(ref) + 1.1 * np.abs(u) * G[:, :s.inter] + np.abs(silu) * G[:, s.inter:] \
            + G[:, :s.inter] * G[:, s.inter:] + 1e-30
        assert (np.abs(f64(td.act) - ref)[rows] <= lim[rows]).all()
        act = f64(td.act)
        fc.fc_gemm_bf16(td.act, Lw["wd"], out=td.o)
        assert gemm_bound_ok(act[rows], f64(Lw["wd"]), f64(td.o)[rows])
        r = td.o
        checked += 1
    torch.cuda.synchronize()
    return checked


@pytest.mark.parametrize("shape", SHAPES, ids=["gqa", "mha"])
def test_decoder_forward_parity(fc, dec, orc, shape):
    from paper_2502_17139_gb300.decoder import DecoderShape, TreeDecoder
    s = DecoderShape(**shape)
    cfg = dec.DecoderConfig(**shape)
    Wt = synth.decoder_weights(s.hidden, s.layers, s.H, s.Hkv, s.D, s.inter, s.vocab, 77)
    Wd = {k: v.cuda() for k, v in Wt.items() if k != "layers"}
    Wd["layers"] = [{k: v.cuda() for k, v in Lw.items()} for Lw in Wt["layers"]]
    tobits = lambda t: t.view(torch.int16).numpy().view(np.uint16)
    Wb = {k: tobits(v) for k, v in Wt.items() if k != "layers"}
    Wb["layers"] = [{k: tobits(v) for k, v in Lw.items()} for Lw in Wt["layers"]]
    W = dec.widen_weights(Wb)
    B, n_pad, cap = 3, 64, 80
    rng = synth.rng_for(92)
    tok = np.full((B, n_pad), 0xFFFFFFFF, np.uint32)
    par = np.full((B, n_pad), -1, np.int32)
    nn = np.array([30, 64, 1], np.int32)
    for b in range(B):
        t, p = synth.random_tree(rng, int(nn[b]), 8, 4, s.vocab)
        tok[b, :nn[b]], par[b, :nn[b]] = t, p
    kvl = np.array([50, 3, 80], np.int32)
    m = orc.tree_mask(par, nn, kvl, n_pad)
    caches = [(synth.randn_bf16((B, s.Hkv, cap, s.D), 900 + l, "cuda"),
               synth.randn_bf16((B, s.Hkv, cap, s.D), 950 + l, "cuda")) for l in range(s.layers)]
    kc = [f64(c[0]) for c in caches]
    vc = [f64(c[1]) for c in caches]
    td = TreeDecoder(s, Wd, B, n_pad, cap, caches=caches)
    assert chained_layer_checks(fc, dec, td, s, tok, nn, dev(m["mask"].view(np.int64)), dev(m["pos"]),
                                dev(kvl)) == s.layers
    logits = td.forward(dev(tok), dev(nn), dev(m["mask"].view(np.int64)), dev(m["pos"]), dev(kvl))
    torch.cuda.synchronize()
    assert fc.fc_get_error() == "FC_OK"
    ref, k_new, v_new = dec.forward(cfg, W, tok, par, nn, kvl, kc, vc, m["pos"])
    mir, k_mir, v_mir = dec.forward(cfg, W, tok, par, nn, kvl, kc, vc, m["pos"], store_bf16=True)
    got = f64(logits)
    for b in range(B):
        n = int(nn[b])
        tol = 3 * np.abs(mir[b, :n] - ref[b, :n]).max()
        err = np.abs(got[b, :n] - ref[b, :n]).max()
        assert 0 < tol and err <= tol, (b, err, tol)
        top2 = np.sort(ref[b, :n], axis=1)[:, -2:]
        clear = top2[:, 1] - top2[:, 0] > tol
        assert (np.argmax(got[b, :n], 1)[clear] == np.argmax(ref[b, :n], 1)[clear]).all()
        for l in range(s.layers):
            gk = f64(td.k_rot[l])[b, :, :n].transpose(1, 0, 2)
            gv = f64(td.v_heads[l])[b, :, :n].transpose(1, 0, 2)
            tk = 3 * np.abs(k_mir[l, b, :n] - k_new[l, b, :n]).max()
            tv = 3 * np.abs(v_mir[l, b, :n] - v_new[l, b, :n]).max()
            assert np.abs(gk - k_new[l, b, :n]).max() <= tk
            assert np.abs(gv - v_new[l, b, :n]).max() <= max(tv, 2.0 ** -8 * np.abs(v_new[l, b, :n]).max())


def test_decoder_step_loop(fc):
    """The step loop verifying with the decoder: acceptance from its logits,
    every layer's cache grows by acc_len + 1 rows, and those rows are the
    tree's rotated keys and values along the accepted path."""
    from paper_2502_17139_gb300.decoder import DecoderShape, TreeDecoder
    from paper_2502_17139_gb300.step import StepLoop
    s = DecoderShape(hidden=256, layers=2, H=4, Hkv=2, inter=384, vocab=synth.VOCAB)
    Wt = synth.decoder_weights(s.hidden, s.layers, s.H, s.Hkv, s.D, s.inter, s.vocab, 78, device="cuda")
    rng = synth.rng_for(75)
    Tr, _ = synth.make_corpus(rng, 200_000, 1.3, synth.VOCAB, n_grams=500, len_range=(8, 64))
    B, n_pad, kv0, steps = 4, 64, 20, 5
    ctx, cl, _ = synth.make_contexts(rng, B, 128, 16, [Tr, None], [0.75, 0.25], 1.1, ctx_stride=128 + 12 * steps)
    cap = kv0 + 12 * steps + 8
    td = TreeDecoder(s, Wt, B, n_pad, cap)
    srcs = [fc.fc_datastore_build(dev(Tr), synth.VOCAB)]
    loop = StepLoop(srcs, ctx, cl, fc.params(16, 2, 16, 10, 4096), n_pad, n_pad, [1], s.H, s.Hkv, s.D, cap, kv0,
                    synth.VOCAB, k_cache=td.k_cache[0], v_cache=td.v_cache[0], decoder=td, cache_capacity=0)
    zeros = torch.zeros(B, dtype=torch.int32, device="cuda")
    for st in range(steps):
        kv_before = loop.kv_len_now.cpu().numpy().copy()
        loop.step(None, None, None, zeros, zeros, None)
        torch.cuda.synchronize()
        assert fc.fc_get_error() == "FC_OK"
        acc = loop.acc["acc_len"].cpu().numpy()
        path = loop.acc["path"].cpu().numpy()
        assert np.array_equal(loop.kv_len_now.cpu().numpy(), kv_before + acc + 1)
        for l in range(s.layers):
            kc = td.k_cache[l].cpu()
            kr = td.k_rot[l].cpu()
            vc = td.v_cache[l].cpu()
            vh = td.v_heads[l].cpu()
            for b in range(B):
                for t in range(int(acc[b]) + 1):
                    assert torch.equal(kc[b, :, kv_before[b] + t], kr[b, :, path[b, t]])
                    assert torch.equal(vc[b, :, kv_before[b] + t], vh[b, :, path[b, t]])
