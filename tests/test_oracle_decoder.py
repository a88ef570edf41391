"""Pins for the oracle's decoder forward over a draft tree (oracle/decoder.py).

Tree verification (Section IV-D, Eq. 4) must give every node the output it
would get from ordinary causal decoding of its own root-to-node path.  So:
  * a chain tree equals incremental causal decoding, written here as the
    textbook loop (one token at a time, each appending its rotated key and
    its value to the layer caches and attending over everything so far);
  * every node of a branching tree equals the last token of the chain made
    of its ancestors;
  * with the attention and MLP output projections zeroed, the logits are the
    final norm of the embedding times the LM head, whatever the tree or cache;
  * the numpy tree attention agrees with the pinned C++ attention oracle (O6
    with O12) on bf16-representable inputs.
"""
import numpy as np
import pytest
import torch

import paper_2502_17139_gb300.synth as synth


@pytest.fixture(scope="module")
def dec(orc):
    from oracle import decoder
    return decoder


CFG = dict(hidden=256, layers=2, H=4, Hkv=2, inter=384, vocab=300)


def setup(dec, seed, B=2, n_pad=64, cap=40, kv=(17, 5)):
    cfg = dec.DecoderConfig(**CFG)
    Wt = synth.decoder_weights(cfg.hidden, cfg.layers, cfg.H, cfg.Hkv, cfg.D, cfg.inter, cfg.vocab, seed)
    tobits = lambda t: t.view(torch.int16).numpy().view(np.uint16)
    Wb = {k: tobits(v) for k, v in Wt.items() if k != "layers"}
    Wb["layers"] = [{k: tobits(v) for k, v in Lw.items()} for Lw in Wt["layers"]]
    W = dec.widen_weights(Wb)
    rng = np.random.default_rng(seed)
    kc = [rng.standard_normal((B, cfg.Hkv, cap, cfg.D)) for _ in range(cfg.layers)]
    vc = [rng.standard_normal((B, cfg.Hkv, cap, cfg.D)) for _ in range(cfg.layers)]
    return cfg, W, kc, vc, np.asarray(kv, np.int32)


def incremental_decode(dec, orc, cfg, W, ids, kc, vc, L0):
    """Textbook causal decoding of one sequence's tokens ids after a cache of
    L0 rotated keys: returns the logits of every token."""
    kcache = [k[:, :L0].copy() for k in kc]
    vcache = [v[:, :L0].copy() for v in vc]
    out = []
    scale = 1.0 / np.sqrt(cfg.D)
    G = cfg.H // cfg.Hkv
    for t, tok in enumerate(ids):
        p = L0 + t
        x = W["embed"][tok].copy()
        for l, Lw in enumerate(W["layers"]):
            h = dec.rmsnorm(x, Lw["attn_norm"], cfg.eps)
            q = (h @ Lw["wq"]).reshape(cfg.H, cfg.D)
            kv = (h @ Lw["wkv"]).reshape(2, cfg.Hkv, cfg.D)
            kcache[l] = np.concatenate([kcache[l], orc.rope(kv[0], np.full(cfg.Hkv, p), cfg.rope_base)[:, None]], 1)
            vcache[l] = np.concatenate([vcache[l], kv[1][:, None]], 1)
            qr = orc.rope(q, np.full(cfg.H, p), cfg.rope_base)
            att = np.zeros((cfg.H, cfg.D))
            for hh in range(cfg.H):
                s = kcache[l][hh // G] @ qr[hh] * scale
                w = np.exp(s - s.max())
                att[hh] = (w / w.sum()) @ vcache[l][hh // G]
            x = x + att.reshape(-1) @ Lw["wo"]
            h = dec.rmsnorm(x, Lw["mlp_norm"], cfg.eps)
            gu = h @ Lw["wgu"]
            x = x + (dec.silu(gu[:cfg.inter]) * gu[cfg.inter:]) @ Lw["wd"]
        out.append(dec.rmsnorm(x, W["final_norm"], cfg.eps) @ W["lm_head"])
    return np.array(out)


def test_chain_tree_is_causal_decoding(dec, orc):
    cfg, W, kc, vc, kvl = setup(dec, 11, B=2)
    B, n_pad, n = 2, 64, 9
    rng = np.random.default_rng(12)
    tokens = np.full((B, n_pad), 0xFFFFFFFF, np.uint32)
    tokens[:, :n] = rng.integers(0, cfg.vocab, (B, n))
    parent = np.full((B, n_pad), -1, np.int32)
    parent[:, 1:n] = np.arange(n - 1)
    nn = np.full(B, n, np.int32)
    pos = np.full((B, n_pad), -1, np.int32)
    pos[:, :n] = kvl[:, None] + np.arange(n)
    logits, k_new, v_new = dec.forward(cfg, W, tokens, parent, nn, kvl, kc, vc, pos)
    for b in range(B):
        ref = incremental_decode(dec, orc, cfg, W, tokens[b, :n], [k[b] for k in kc], [v[b] for v in vc], int(kvl[b]))
        assert np.allclose(logits[b, :n], ref, atol=1e-9, rtol=1e-9)
    assert (logits[:, n:] == 0).all()


def test_branching_tree_equals_its_paths(dec, orc):
    cfg, W, kc, vc, kvl = setup(dec, 13, B=2)
    B, n_pad = 2, 64
    rng = synth.rng_for(90)
    tokens = np.full((B, n_pad), 0xFFFFFFFF, np.uint32)
    parent = np.full((B, n_pad), -1, np.int32)
    nn = np.array([14, 9], np.int32)
    pos = np.full((B, n_pad), -1, np.int32)
    for b in range(B):
        t, p = synth.random_tree(rng, int(nn[b]), 5, 3, cfg.vocab)
        tokens[b, :nn[b]], parent[b, :nn[b]] = t, p
        depth = np.zeros(nn[b], np.int32)
        for i in range(1, nn[b]):
            depth[i] = depth[p[i]] + 1
        pos[b, :nn[b]] = kvl[b] + depth
    logits, _, _ = dec.forward(cfg, W, tokens, parent, nn, kvl, kc, vc, pos)
    anc = [dec.ancestors_of(parent[b], int(nn[b])) for b in range(B)]
    for b in range(B):
        for i in range(int(nn[b])):
            path = anc[b][i]
            ref = incremental_decode(dec, orc, cfg, W, tokens[b, path], [k[b] for k in kc], [v[b] for v in vc],
                                     int(kvl[b]))
            assert np.allclose(logits[b, i], ref[-1], atol=1e-9, rtol=1e-9), (b, i)


def test_zero_output_projections_closed_form(dec, orc):
    cfg, W, kc, vc, kvl = setup(dec, 14, B=2)
    for Lw in W["layers"]:
        Lw["wo"][:] = 0.0
        Lw["wd"][:] = 0.0
    B, n_pad = 2, 64
    rng = np.random.default_rng(15)
    tokens = np.full((B, n_pad), 0xFFFFFFFF, np.uint32)
    tokens[:, :6] = rng.integers(0, cfg.vocab, (B, 6))
    parent = np.full((B, n_pad), -1, np.int32)
    parent[:, 1:6] = [0, 0, 1, 1, 3]
    nn = np.full(B, 6, np.int32)
    pos = np.full((B, n_pad), -1, np.int32)
    pos[:, :6] = kvl[:, None] + np.array([0, 1, 1, 2, 2, 3])
    logits, _, _ = dec.forward(cfg, W, tokens, parent, nn, kvl, kc, vc, pos)
    e = W["embed"][tokens[:, :6].astype(np.int64)]
    ref = e / np.sqrt((e * e).mean(-1, keepdims=True) + cfg.eps) * W["final_norm"] @ W["lm_head"]
    assert np.allclose(logits[:, :6], ref, atol=1e-9)


def test_numpy_attention_matches_the_c_oracle(dec, orc):
    cfg = dec.DecoderConfig(**CFG)
    rng = synth.rng_for(91)
    B, n_pad, cap = 2, 64, 30
    bf = lambda a: (a.astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)
    q = bf(rng.standard_normal((B, n_pad, cfg.H, cfg.D)))
    kc = bf(rng.standard_normal((B, cfg.Hkv, cap, cfg.D)))
    vc = bf(rng.standard_normal((B, cfg.Hkv, cap, cfg.D)))
    kt = bf(rng.standard_normal((B, cfg.Hkv, n_pad, cfg.D)))
    vt = bf(rng.standard_normal((B, cfg.Hkv, n_pad, cfg.D)))
    par = np.full((B, n_pad), -1, np.int32)
    nn = np.array([20, 7], np.int32)
    for b in range(B):
        _, p = synth.random_tree(rng, int(nn[b]), 6, 3, 100)
        par[b, :nn[b]] = p
    kvl = np.array([11, 30], np.int32)
    m = orc.tree_mask(par, nn, kvl, n_pad)
    ref = orc.tree_attn(q, kc, vc, kvl, kt, vt, m["mask"], nn, pos=m["pos"])
    w = dec.widen
    for b in range(B):
        n = int(nn[b])
        got = dec.tree_attention(w(q[b]), w(kc[b]), w(vc[b]), int(kvl[b]), w(kt[b]).transpose(1, 0, 2),
                                 w(vt[b]).transpose(1, 0, 2), dec.ancestors_of(par[b], n), n, m["pos"][b], cfg)
        assert np.allclose(got, ref[b, :n], atol=1e-10)


def test_round_bf16_matches_the_format(dec):
    """round_bf16 (used only for the bf16-storage variant of the forward) is
    round-to-nearest-even onto the bf16 grid: checked against torch's own
    conversion, and on hand values at and between grid points."""
    import torch
    rng = np.random.default_rng(3)
    x = np.concatenate([rng.standard_normal(20000) * 10.0 ** rng.integers(-30, 30, 20000),
                        [0.0, -0.0, 1.0, 1 + 2.0 ** -8, 1 + 3 * 2.0 ** -9, 1 + 2.0 ** -9, 3.0e38]])
    x = x.astype(np.float32).astype(np.float64)  # fp32 inputs: one rounding, as the GPU stores
    want = torch.from_numpy(x).float().to(torch.bfloat16).double().numpy()
    assert np.array_equal(dec.round_bf16(x), want)
    assert dec.round_bf16(np.array([1 + 2.0 ** -8]))[0] == 1.0          # a tie goes to the even neighbour
    assert dec.round_bf16(np.array([1 + 3 * 2.0 ** -8]))[0] == 1 + 2.0 ** -6


def test_store_bf16_forward_stays_near_the_exact_one(dec, orc):
    """The bf16-storage variant differs from the exact forward by rounding
    only: a few bf16 ulps of the logits' scale, never zero, never more."""
    cfg, W, kc, vc, kvl = setup(dec, 21, B=2)
    B, n_pad = 2, 64
    rng = synth.rng_for(91)
    tok = np.full((B, n_pad), 0xFFFFFFFF, np.uint32)
    par = np.full((B, n_pad), -1, np.int32)
    nn = np.array([20, 7], np.int32)
    pos = np.full((B, n_pad), -1, np.int32)
    for b in range(B):
        t, p = synth.random_tree(rng, int(nn[b]), 5, 3, cfg.vocab)
        tok[b, :nn[b]], par[b, :nn[b]] = t, p
        depth = np.zeros(nn[b], np.int32)
        for i in range(1, nn[b]):
            depth[i] = depth[p[i]] + 1
        pos[b, :nn[b]] = kvl[b] + depth
    ref = dec.forward(cfg, W, tok, par, nn, kvl, kc, vc, pos)[0]
    mir = dec.forward(cfg, W, tok, par, nn, kvl, kc, vc, pos, store_bf16=True)[0]
    d = np.abs(mir - ref).max()
    assert 0 < d <= 0.05 * np.abs(ref).max()
