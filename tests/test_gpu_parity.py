"""GPU parity: every kernel behind the C ABI against the CPU oracle, element
by element on the same seeded inputs.

Integer outputs (suffix arrays, buckets, retrieval results, trees, masks,
acceptance, cache append) must be bit-exact.  Tree attention (bf16 inputs,
fp32 accumulation and softmax on the GPU) must be within max-abs 2e-2 of the
fp64 oracle.
"""
import numpy as np
import pytest
import torch

import paper_2502_17139_gb300.synth as synth

pytestmark = pytest.mark.gpu
ATOL = 2e-2
PAD = 0xFFFFFFFF


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
    elif a.dtype == np.uint64:
        a = a.view(np.int64)
    return torch.from_numpy(a.copy()).cuda()


def host_u32(t):
    return t.cpu().numpy().view(np.uint32)


def bits_bf16(t):
    return t.cpu().view(torch.int16).numpy().view(np.uint16)


def check_no_error(fc):
    assert fc.fc_get_error() == "FC_OK"


# ------------------------------------------------------------ suffix array
@pytest.mark.parametrize("n,vocab,seed", [(1, 5, 0), (2, 2, 1), (3, 2, 2), (57, 2, 3), (4096, 3, 4),
                                          (4097, 8, 5), (8192 + 17, 4, 6), (50000, 2, 7), (70001, 300, 8)])
def test_sa_small_sweep(fc, orc, n, vocab, seed):
    rng = np.random.default_rng(seed)
    T = rng.integers(0, vocab, n).astype(np.uint32)
    if n > 100:
        T[n // 3:n // 3 + 60] = T[:60]  # a long repeat
    ds = fc.fc_datastore_build(dev(T), vocab)
    torch.cuda.synchronize()
    sa = orc.suffix_array(T)
    assert np.array_equal(host_u32(ds.sa), sa)
    assert np.array_equal(host_u32(ds.bucket), orc.bucket(T, sa, vocab))
    assert np.array_equal(ds.lcp.cpu().numpy(), orc.lcp(T, sa))


def test_sa_constant_corpus(fc, orc):
    T = np.full(10000, 7, np.uint32)
    ds = fc.fc_datastore_build(dev(T), 8)
    assert host_u32(ds.sa).tolist() == list(range(9999, -1, -1))


def test_sa_rejects_bad_token(fc):
    T = np.array([1, 2, 9, 3], np.uint32)
    with pytest.raises(fc.FastCoderError) as e:
        fc.fc_datastore_build(dev(T), 5)
    assert e.value.status == "FC_ERR_INVALID_ARG"


@pytest.fixture(scope="module")
def c1(fc, orc):
    cfg = synth.WORKLOADS[1]
    rng = synth.rng_for(1)
    T, _ = synth.build_corpus(rng, cfg["corpus"][0])
    ctx, cl, _ = synth.make_contexts(rng, cfg["batch"], cfg["ctx_len"], cfg["n_copy"], [T], [1.0], 1.1)
    ds = fc.fc_datastore_build(dev(T), synth.VOCAB)
    return dict(cfg=cfg, T=T, ctx=ctx, cl=cl, ds=ds)


def test_sa_c1_corpus(fc, orc, c1):
    sa = orc.suffix_array(c1["T"])
    assert np.array_equal(host_u32(c1["ds"].sa), sa)
    assert np.array_equal(host_u32(c1["ds"].bucket), orc.bucket(c1["T"], sa, synth.VOCAB))
    assert np.array_equal(c1["ds"].lcp.cpu().numpy(), orc.lcp(c1["T"], sa))


# --------------------------------------------------------------- retrieval
def compare_retrieval(gpu, ref, s=0):
    for name in ("drafts", "draft_len", "count", "n_drafts", "match_len"):
        g = gpu[name][s].cpu().numpy()
        r = ref[name]
        if r.dtype == np.uint32:
            g = g.view(np.uint32)
        assert np.array_equal(g, r), name


def test_retrieve_c1(fc, orc, c1):
    cfg = c1["cfg"]
    p = fc.params(cfg["n_max"], cfg["n_min"], cfg["top_k"], cfg["draft_len"], 4096)
    g = fc.fc_retrieve([c1["ds"]], dev(c1["ctx"]), dev(c1["cl"]), p)
    r = orc.retrieve(c1["T"], c1["ctx"], c1["cl"], cfg["n_max"], cfg["n_min"], cfg["top_k"], cfg["draft_len"], 4096)
    compare_retrieval(g, r)
    assert (r["match_len"] >= 8).mean() > 0.5  # most contexts end with a copied corpus span
    check_no_error(fc)


@pytest.mark.parametrize("keys", [True, False])
@pytest.mark.parametrize("seed", range(8))
def test_retrieve_tiny_sweep(fc, orc, seed, keys):
    """Tiny alphabets (2-6 tokens), so probes tie on their first eight tokens
    and the search reads the corpus; contexts copied from anywhere in the
    corpus, the end included; n_max up to 32.  With the suffix keys (one
    32-byte read per probe) and without them (suffix array, then corpus)."""
    rng = np.random.default_rng(500 + seed)
    N = int(rng.integers(2, 3000))
    vocab = int(rng.integers(2, 7))
    T = rng.integers(0, vocab, N).astype(np.uint32)
    B, stride = 40, 24
    ctx = rng.integers(0, vocab, (B, stride)).astype(np.uint32)
    cl = rng.integers(0, stride + 1, B).astype(np.int32)
    for b in range(0, B, 2):
        L = int(min(cl[b], N))
        if L:
            p0 = int(rng.integers(0, N - L + 1))
            ctx[b, cl[b] - L:cl[b]] = T[p0:p0 + L]
    n_max = int(rng.integers(1, 33))
    n_min = int(rng.integers(1, n_max + 1)) if seed % 2 else min(2, n_max)
    k, d = int(rng.integers(1, 257)), int(rng.integers(1, 17))
    max_occ = [1, 3, 4096, 17][seed % 4]
    ds = fc.fc_datastore_build(dev(T), vocab)
    assert ds.keys is not None
    g = fc.fc_retrieve([ds if keys else ds.without_keys()], dev(ctx), dev(cl), fc.params(n_max, n_min, k, d, max_occ))
    r = orc.retrieve(T, ctx, cl, n_max, n_min, k, d, max_occ)
    compare_retrieval(g, r)
    check_no_error(fc)


def test_suffix_keys_layout(fc):
    """Entry j of the suffix keys: sa[j], then the suffix's tokens 1..7
    (FC_PAD_TOKEN past the corpus end)."""
    rng = np.random.default_rng(31)
    T = rng.integers(0, 5, 3001).astype(np.uint32)
    ds = fc.fc_datastore_build(dev(T), 5)
    sa = host_u32(ds.sa)
    keys = host_u32(ds.keys).reshape(-1, 8)
    Tp = np.concatenate([T, np.full(8, PAD, np.uint32)])
    want = np.stack([sa] + [Tp[sa.astype(np.int64) + k] for k in range(1, 8)], 1)
    assert np.array_equal(keys, want)


def test_retrieve_two_sources_and_skip(fc, orc):
    rng = synth.rng_for(40)
    Tr, _ = synth.make_corpus(rng, 60000, 1.3, 500, n_grams=300, len_range=(8, 40))
    Tc, _ = synth.make_corpus(rng, 150000, 1.1, 500)
    ctx, cl, _ = synth.make_contexts(rng, 64, 40, 16, [Tr, Tc, None], [0.5, 0.25, 0.25], 1.1, 500)
    dsr, dsc = fc.fc_datastore_build(dev(Tr), 500), fc.fc_datastore_build(dev(Tc), 500)
    p = fc.params(16, 2, 64, 10, 4096)
    skip = np.zeros(64, np.int32)
    skip[::5] = 1
    out = fc.retrieve_outputs(2, 64, p)
    for v in out.values():
        v.fill_(-7)
    g = fc.fc_retrieve([dsr, dsc], dev(ctx), dev(cl), p, skip=dev(skip), out=out)
    for s, T in enumerate((Tr, Tc)):
        r = orc.retrieve(T, ctx, cl, 16, 2, 64, 10, 4096)
        keep = skip == 0
        for name in r:
            gg = g[name][s].cpu().numpy()
            if r[name].dtype == np.uint32:
                gg = gg.view(np.uint32)
            assert np.array_equal(gg[keep], r[name][keep]), name
            assert (g[name][s].cpu().numpy()[~keep] == -7).all()


def test_retrieve_bad_context_token(fc):
    T = np.arange(100, dtype=np.uint32) % 10
    ds = fc.fc_datastore_build(dev(T), 10)
    ctx = np.array([[1, 2, 3, 4], [1, 2, 99, 4]], np.uint32)
    g = fc.fc_retrieve([ds], dev(ctx), dev(np.array([4, 4], np.int32)), fc.params(4, 1, 4, 4, 64))
    assert fc.fc_get_error() == "FC_ERR_INVALID_ARG"
    assert int(g["match_len"][0, 0]) == 4 and int(g["match_len"][0, 1]) == 0


# -------------------------------------------------------------------- tree
def compare_tree(g, r):
    for name in ("tok", "parent", "depth", "pos", "n_nodes"):
        gg = g[name].cpu().numpy()
        if r[name].dtype == np.uint32:
            gg = gg.view(np.uint32)
        assert np.array_equal(gg, r[name]), name
    assert np.array_equal(g["mask"].cpu().numpy().view(np.uint64), r["mask"])


def test_tree_from_c1_retrieval(fc, orc, c1):
    cfg = c1["cfg"]
    p = fc.params(cfg["n_max"], cfg["n_min"], cfg["top_k"], cfg["draft_len"], 4096)
    g = fc.fc_retrieve([c1["ds"]], dev(c1["ctx"]), dev(c1["cl"]), p)
    r = orc.retrieve(c1["T"], c1["ctx"], c1["cl"], cfg["n_max"], cfg["n_min"], cfg["top_k"], cfg["draft_len"], 4096)
    root = c1["ctx"][np.arange(32), c1["cl"] - 1]
    kvl = np.full(32, 512, np.int32)
    for budget in (1, 17, 64):
        gt = fc.fc_build_tree(g, [1], dev(root), dev(kvl), budget, 64)
        rt = orc.build_tree([r], [1], root, kvl, budget, 64)
        compare_tree(gt, rt)
    check_no_error(fc)


def _random_sources(rng, S, B, k, d, vocab):
    res = []
    for s in range(S):
        o = dict(drafts=np.full((B, k, d), PAD, np.uint32), draft_len=np.zeros((B, k), np.int32),
                 count=np.zeros((B, k), np.uint32), n_drafts=np.zeros(B, np.int32), match_len=np.ones(B, np.int32))
        for b in range(B):
            nd = int(rng.integers(0, k + 1))
            seen, t = set(), 0
            while t < nd:
                L = int(rng.integers(1, d + 1))
                u = tuple(int(x) for x in rng.integers(0, vocab, L))
                if u in seen:
                    continue
                seen.add(u)
                o["drafts"][b, t, :L] = u
                o["draft_len"][b, t] = L
                o["count"][b, t] = int(rng.integers(1, 4097))
                t += 1
            o["n_drafts"][b] = nd
        res.append(o)
    return res


@pytest.mark.parametrize("S,k,d,vocab,n_pad", [(1, 16, 8, 3, 64), (2, 64, 10, 4, 128), (2, 64, 10, 32256, 64),
                                               (2, 256, 16, 2, 128), (4, 128, 12, 5, 128)])
def test_tree_random_drafts(fc, orc, S, k, d, vocab, n_pad):
    rng = np.random.default_rng(S * 1000 + k + d + vocab)
    B = 24
    res = _random_sources(rng, S, B, k, d, vocab)
    w = rng.integers(1, 5, S).astype(np.uint32)
    root = rng.integers(0, vocab, B).astype(np.uint32)
    kvl = rng.integers(0, 5000, B).astype(np.int32)
    g_res = {name: dev(np.stack([r[name] for r in res])) for name in res[0]}
    for budget in (1, 2, n_pad // 2 + 1, n_pad):
        gt = fc.fc_build_tree(g_res, w, dev(root), dev(kvl), budget, n_pad)
        rt = orc.build_tree(res, w, root, kvl, budget, n_pad)
        compare_tree(gt, rt)
    check_no_error(fc)


WEIGHTS = [(0, 1), (1, 0), (65535, 1), (1, 65535), (3, 1), (1, 3), (0, 0)]


@pytest.mark.parametrize("w", WEIGHTS, ids=[f"a{a}b{b}" for a, b in WEIGHTS])
def test_tree_weight_sweep(fc, orc, w):
    """Eq. 3 with alpha/beta away from 1, down to 0 and up to the largest
    weight, on two sources sharing many drafts (small vocabularies) so that
    merged weights decide which nodes are kept."""
    rng = np.random.default_rng(4200 + w[0] + 7 * w[1])
    B, k, d, n_pad = 24, 64, 10, 128
    res = _random_sources(rng, 2, B, k, d, 3)
    root = rng.integers(0, 3, B).astype(np.uint32)
    kvl = rng.integers(0, 5000, B).astype(np.int32)
    g_res = {name: dev(np.stack([r[name] for r in res])) for name in res[0]}
    wv = np.array(w, np.uint32)
    for budget in (2, 17, 64, 128):
        gt = fc.fc_build_tree(g_res, wv, dev(root), dev(kvl), budget, n_pad)
        rt = orc.build_tree(res, wv, root, kvl, budget, n_pad)
        compare_tree(gt, rt)
    check_no_error(fc)


def test_tree_handmade_on_gpu(fc):
    """The hand-worked trees of tests/golden/tree_handmade.json (weights
    (1,1), (3,1), (0,1), (1,0), (65535,1)) built by the GPU."""
    import json
    import os
    g = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "tree_handmade.json")))

    def src(drafts, lens, counts):
        k, d = 4, 3
        o = dict(drafts=np.full((1, k, d), PAD, np.uint32), draft_len=np.zeros((1, k), np.int32),
                 count=np.zeros((1, k), np.uint32), n_drafts=np.array([len(drafts)], np.int32),
                 match_len=np.ones(1, np.int32))
        for t, (u, L, c) in enumerate(zip(drafts, lens, counts)):
            o["drafts"][0, t, :L] = u[:L]
            o["draft_len"][0, t] = L
            o["count"][0, t] = c
        return o

    r = src(g["src_r"]["drafts"], [3, 3], g["src_r"]["count"])
    c = src(g["src_c"]["drafts"], g["src_c"]["len"], g["src_c"]["count"])
    g_res = {name: dev(np.stack([r[name], c[name]])) for name in r}
    for case in g["cases"]:
        t = fc.fc_build_tree(g_res, np.array(case["weights"], np.uint32), dev(np.array([9], np.uint32)),
                             dev(np.array([100], np.int32)), case["budget"], 64)
        n = int(t["n_nodes"].cpu()[0])
        assert n == len(case["tok"]), case["why"]
        assert t["tok"].cpu().numpy()[0, :n].tolist() == case["tok"], case["why"]
        assert t["parent"].cpu().numpy()[0, :n].tolist() == case["parent"], case["why"]
        assert t["depth"].cpu().numpy()[0, :n].tolist() == case["depth"], case["why"]
    check_no_error(fc)


@pytest.mark.parametrize("w", [(1, 1), (3, 1)])
def test_all_occurrence_trie_within_cap(fc, orc, w):
    """The trie over every retrieved continuation (the "top-k prefixes"
    reading of Section III-A and Eq. 3's occurrence counts over all of R_r and
    R_c): with max_occ <= 256 a source has at most 256 distinct
    continuations, so top_k = max_occ keeps all of them and the GPU tree
    equals the oracle's tree over its untruncated retrieval."""
    rng = synth.rng_for(42)
    Tr, _ = synth.make_corpus(rng, 60000, 1.3, 300, n_grams=300, len_range=(8, 40))
    Tc, _ = synth.make_corpus(rng, 150000, 1.05, 300)
    B, n_pad = 48, 128
    ctx, cl, _ = synth.make_contexts(rng, B, 40, 16, [Tr, Tc, None], [0.5, 0.25, 0.25], 1.1, 300)
    dsr, dsc = fc.fc_datastore_build(dev(Tr), 300), fc.fc_datastore_build(dev(Tc), 300)
    cap, d = 256, 10
    p = fc.params(16, 2, cap, d, cap)
    g = fc.fc_retrieve([dsr, dsc], dev(ctx), dev(cl), p)
    root = ctx[np.arange(B), cl - 1]
    kvl = np.full(B, 700, np.int32)
    wv = np.array(w, np.uint32)
    gt = fc.fc_build_tree(g, wv, dev(root), dev(kvl), n_pad, n_pad)
    res = [orc.retrieve(T, ctx, cl, 16, 2, 4096, d, cap) for T in (Tr, Tc)]
    assert max(int(r["n_drafts"].max()) for r in res) > 64  # more distinct continuations than a top-64 keeps
    assert all(int(r["n_drafts"].max()) <= cap for r in res)
    for r in res:  # the untruncated lists, cut to the slot count (every draft fits)
        for name in ("drafts", "draft_len", "count"):
            r[name] = np.ascontiguousarray(r[name][:, :cap])
    rt = orc.build_tree(res, wv, root, kvl, n_pad, n_pad)
    compare_tree(gt, rt)
    check_no_error(fc)


def _random_trees(rng, B, n_pad, vocab=32256, full=False):
    tok = np.full((B, n_pad), PAD, np.uint32)
    par = np.full((B, n_pad), -1, np.int32)
    nn = np.full(B, n_pad, np.int32) if full else rng.integers(1, n_pad + 1, B).astype(np.int32)
    for b in range(B):
        t, p = synth.random_tree(rng, int(nn[b]), 10, 4, vocab)
        tok[b, :nn[b]], par[b, :nn[b]] = t, p
    return tok, par, nn


def test_tree_mask_from_parents(fc, orc):
    rng = synth.rng_for(41)
    for n_pad in (64, 128):
        tok, par, nn = _random_trees(rng, 20, n_pad)
        kvl = rng.integers(0, 100, 20).astype(np.int32)
        g = fc.fc_tree_mask(dev(par), dev(nn), dev(kvl))
        r = orc.tree_mask(par, nn, kvl, n_pad)
        assert np.array_equal(g["mask"].cpu().numpy().view(np.uint64), r["mask"])
        assert np.array_equal(g["depth"].cpu().numpy(), r["depth"])
        assert np.array_equal(g["pos"].cpu().numpy(), r["pos"])


# --------------------------------------------------------------- attention
def _attn_case(fc, orc, seed, B, n_pad, H, Hkv, kv_len, cap, nn=None, full_rows=True, sample=None,
               workspace="auto", want_parts=None):
    rng = synth.rng_for(50, seed)
    tok, par, nn_r = _random_trees(rng, B, n_pad)
    if nn is not None:
        nn_r = np.asarray(nn, np.int32)
        for b in range(B):
            t, p = synth.random_tree(rng, int(nn_r[b]), 10, 4, 1000)
            par[b] = -1
            par[b, :nn_r[b]] = p
    kvl = np.asarray(kv_len, np.int32)
    D = 128
    q = synth.randn_bf16((B, n_pad, H, D), 1000 + seed, "cuda")
    kc = synth.randn_bf16((B, Hkv, cap, D), 2000 + seed, "cuda")
    vc = synth.randn_bf16((B, Hkv, cap, D), 3000 + seed, "cuda")
    kt = synth.randn_bf16((B, Hkv, n_pad, D), 4000 + seed, "cuda")
    vt = synth.randn_bf16((B, Hkv, n_pad, D), 5000 + seed, "cuda")
    gm = fc.fc_tree_mask(dev(par), dev(nn_r), dev(kvl))
    out = torch.full_like(q, float("nan"))
    fc.fc_tree_attn(q, kc, vc, dev(kvl), kt, vt, gm["mask"], dev(nn_r), out=out, workspace=workspace)
    torch.cuda.synchronize()
    check_no_error(fc)
    if want_parts is not None:  # the same call without a workspace: one CTA per row chunk
        ws = fc.attn_workspace(B, n_pad, H, Hkv, "cuda") if workspace == "auto" else workspace
        nbytes = 0 if ws is None else ws.numel()
        parts = fc.LIB.fc_tree_attn_parts(B, n_pad, H, Hkv, cap, nbytes)
        assert parts >= want_parts, parts
        single = torch.full_like(q, float("nan"))
        fc.fc_tree_attn(q, kc, vc, dev(kvl), kt, vt, gm["mask"], dev(nn_r), out=single, workspace=None)
        torch.cuda.synchronize()
        check_no_error(fc)
        assert torch.isfinite(out.float()).all()
        assert (out.float() - single.float()).abs().max().item() <= ATOL
    rm = orc.tree_mask(par, nn_r, kvl, n_pad)["mask"]
    args = [bits_bf16(x) for x in (q, kc, vc)] + [kvl] + [bits_bf16(x) for x in (kt, vt)] + [rm, nn_r]
    got = out.float().cpu().numpy()
    if full_rows:
        ref = orc.tree_attn(args[0], args[1], args[2], args[3], args[4], args[5], args[6], args[7])
        err = np.abs(got - ref).max()
        assert np.isfinite(got).all()
    else:
        rows = []
        for b in range(B):
            for i in sorted({0, int(nn_r[b]) - 1, int(rng.integers(0, nn_r[b])), min(n_pad - 1, int(nn_r[b]))}):
                for h in sorted({0, H - 1, int(rng.integers(0, H))}):
                    rows.append((b, i, h))
        if sample:
            rows = [rows[i] for i in rng.choice(len(rows), min(sample, len(rows)), replace=False)]
        rows = np.array(rows, np.int32)
        ref = orc.tree_attn(args[0], args[1], args[2], args[3], args[4], args[5], args[6], args[7], rows=rows)
        g = got[rows[:, 0], rows[:, 1], rows[:, 2]]
        err = np.abs(g - ref).max()
        assert np.isfinite(g).all()
    assert err <= ATOL, err
    return err


def test_attn_c1_shape_full(fc, orc):
    # c1: B=32, H=Hkv=32, D=128, KV 512, trees <= 64 nodes
    _attn_case(fc, orc, 1, 32, 64, 32, 32, [512] * 32, 512)


def test_attn_ragged_edges(fc, orc):
    B = 8
    kvl = [0, 1, 127, 128, 129, 300, 511, 512]
    _attn_case(fc, orc, 2, B, 64, 8, 8, kvl, 512, nn=[1, 2, 63, 64, 64, 5, 1, 33])


def test_attn_gqa_n128(fc, orc):
    B = 6
    kvl = [0, 5, 128, 1000, 2047, 2048]
    _attn_case(fc, orc, 3, B, 128, 32, 8, kvl, 2048, nn=[1, 20, 32, 33, 127, 128])


def test_attn_one_tile_chunks(fc, orc):
    # G = 4, 128-node trees whose second row chunk holds one tile (65..96
    # nodes): that CTA splits its KV blocks between its two softmax
    # warpgroups (odd and even block counts, an empty cache, one block)
    B = 8
    kvl = [0, 1, 128, 129, 383, 384, 2047, 2048]
    _attn_case(fc, orc, 10, B, 128, 32, 8, kvl, 2048, nn=[65, 70, 88, 96, 97, 30, 66, 96])


def test_attn_gqa_n64_group2(fc, orc):
    _attn_case(fc, orc, 4, 5, 64, 16, 8, [300, 0, 64, 700, 129], 777, nn=[64, 1, 40, 64, 2])


def test_attn_gqa_group8_n64(fc, orc):
    # G = 8 with 64-node trees: 512 rows per group, two row chunks of two tiles
    kvl = [0, 1, 300, 1000, 2048, 129]
    _attn_case(fc, orc, 8, 6, 64, 64, 8, kvl, 2048, nn=[64, 1, 33, 64, 17, 48], full_rows=False)


def test_attn_gqa_group16_n128(fc, orc):
    # G = 16 (the largest supported): up to 2048 rows per group, eight row chunks
    kvl = [700, 0, 2048, 1]
    _attn_case(fc, orc, 9, 4, 128, 32, 2, kvl, 2048, nn=[128, 3, 100, 65], full_rows=False)


def _units_over_sms(per_seq_units):
    """A batch whose row-chunk count is a little over one wave of CTAs: the
    chunks of the last sequence form a short second wave and have their keys
    split over several CTAs (the sampled rows always include that sequence)."""
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    return -(-(sms + 8) // per_seq_units)


def test_attn_kv_split_one_tile(fc, orc):
    # G = 1, 64-node trees: one 128-row tile per (sequence, kv head); ragged
    # caches (empty, one key, block edges) mixed with full ones
    B = _units_over_sms(8)
    rng = synth.rng_for(51)
    kvl = [[0, 1, 127, 128, 129, 2047, 2048][b % 7] if b < 14 else int(rng.integers(0, 2049)) for b in range(B)]
    _attn_case(fc, orc, 6, B, 64, 8, 8, kvl, 2048, full_rows=False, want_parts=2)


def test_attn_kv_split_two_tiles(fc, orc):
    # G = 4, 128-node trees: two row chunks per group, the first with two tiles
    B = _units_over_sms(16)
    rng = synth.rng_for(52)
    kvl = [int(rng.integers(0, 2049)) for _ in range(B)]
    nn = [int(rng.integers(1, 129)) if b % 3 else 128 for b in range(B)]
    _attn_case(fc, orc, 7, B, 128, 32, 8, kvl, 2048, nn=nn, full_rows=False, want_parts=2)


def test_attn_kv_split_deterministic(fc):
    """With the last wave's keys split over several CTAs, whichever CTA of a
    unit finishes last merges the parts; it sums them in part order, so
    repeated launches on the same inputs give the same bits.  The step loop's
    shape (32 sequences, GQA 32/8, 128-node padding, 16384-key caches, trees
    of 1 to 128 nodes), 12 launches."""
    B, n_pad, H, Hkv, cap = 32, 128, 32, 8, 16384
    rng = synth.rng_for(53)
    nn = rng.integers(1, n_pad + 1, B).astype(np.int32)
    kvl = rng.integers(cap - 200, cap + 1, B).astype(np.int32)
    par = np.full((B, n_pad), -1, np.int32)
    for b in range(B):
        _, p = synth.random_tree(rng, int(nn[b]), 10, 4, 1000)
        par[b, :nn[b]] = p
    D = 128
    q = synth.randn_bf16((B, n_pad, H, D), 61, "cuda")
    kc = synth.randn_bf16((B, Hkv, cap, D), 62, "cuda")
    vc = synth.randn_bf16((B, Hkv, cap, D), 63, "cuda")
    kt = synth.randn_bf16((B, Hkv, n_pad, D), 64, "cuda")
    vt = synth.randn_bf16((B, Hkv, n_pad, D), 65, "cuda")
    gm = fc.fc_tree_mask(dev(par), dev(nn), dev(kvl))
    ws = fc.attn_workspace(B, n_pad, H, Hkv, "cuda")
    assert fc.LIB.fc_tree_attn_parts(B, n_pad, H, Hkv, cap, ws.numel()) > 1
    out = torch.empty_like(q)
    first = None
    for _ in range(12):
        out.fill_(float("nan"))
        fc.fc_tree_attn(q, kc, vc, dev(kvl), kt, vt, gm["mask"], dev(nn), out=out, workspace=ws)
        torch.cuda.synchronize()
        if first is None:
            first = out.clone()
            assert not torch.isnan(first).any()
        else:
            assert torch.equal(out, first)
    check_no_error(fc)


def test_attn_stream_c1_shape(fc, orc):
    """The c1 launch (1024 one-tile groups, 512-key caches) runs on the
    streaming kernel: several groups per CTA."""
    assert fc.LIB.fc_tree_attn_streamed(32, 64, 32, 32, 512) == 1
    assert fc.LIB.fc_tree_attn_streamed(16, 64, 32, 32, 4096) == 0  # c3: long caches, per-group CTAs
    assert fc.LIB.fc_tree_attn_streamed(32, 128, 32, 8, 16384) == 0  # two-tile groups


def test_attn_stream_ragged(fc, orc):
    """Streaming kernel, one head per group: ragged caches (empty, one key,
    block edges) and trees (one node to full), every row against the oracle."""
    B, H = 40, 16
    assert fc.LIB.fc_tree_attn_streamed(B, 64, H, H, 512) == 1
    base_k, base_n = [0, 1, 127, 128, 129, 300, 511, 512], [1, 2, 63, 64, 64, 5, 1, 33]
    kvl = [base_k[b % 8] for b in range(B)]
    nn = [base_n[(b * 3) % 8] for b in range(B)]
    _attn_case(fc, orc, 21, B, 64, H, H, kvl, 512, nn=nn)


def test_attn_stream_gqa2(fc, orc):
    """Streaming kernel with two query heads per group (128 rows of 64-node
    trees) and caches up to 1000 keys."""
    B, H, Hkv = 80, 16, 8
    assert fc.LIB.fc_tree_attn_streamed(B, 64, H, Hkv, 1024) == 1
    rng = synth.rng_for(53)
    kvl = [int(rng.integers(0, 1001)) if b % 5 else [0, 1000][b % 2] for b in range(B)]
    _attn_case(fc, orc, 22, B, 64, H, Hkv, kvl, 1024, full_rows=False, sample=3000)


def test_attn_stream_matches_per_group_kernel(fc, orc):
    """The same sequences through the streaming kernel (40 sequences, 320
    groups) and through the per-group kernel (the first 19: 152 groups, one
    wave, no key split): bit-identical outputs."""
    B, H, n_pad, cap = 40, 8, 64, 512
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    Bs = sms // H
    assert fc.LIB.fc_tree_attn_streamed(B, n_pad, H, H, cap) == 1
    assert fc.LIB.fc_tree_attn_streamed(Bs, n_pad, H, H, cap) == 0
    rng = synth.rng_for(54)
    tok, par, nn = _random_trees(rng, B, n_pad)
    kvl = rng.integers(0, cap + 1, B).astype(np.int32)
    q = synth.randn_bf16((B, n_pad, H, 128), 61, "cuda")
    kc = synth.randn_bf16((B, H, cap, 128), 62, "cuda")
    vc = synth.randn_bf16((B, H, cap, 128), 63, "cuda")
    kt = synth.randn_bf16((B, H, n_pad, 128), 64, "cuda")
    vt = synth.randn_bf16((B, H, n_pad, 128), 65, "cuda")
    gm = fc.fc_tree_mask(dev(par), dev(nn), dev(kvl))
    out = fc.fc_tree_attn(q, kc, vc, dev(kvl), kt, vt, gm["mask"], dev(nn))
    part = fc.fc_tree_attn(q[:Bs].contiguous(), kc[:Bs].contiguous(), vc[:Bs].contiguous(), dev(kvl[:Bs]),
                           kt[:Bs].contiguous(), vt[:Bs].contiguous(), gm["mask"][:Bs].contiguous(), dev(nn[:Bs]))
    torch.cuda.synchronize()
    check_no_error(fc)
    assert torch.equal(out[:Bs], part)


def test_attn_stream_bad_length(fc, orc):
    """A node count out of range in one sequence: FC_ERR_INVALID_ARG, that
    sequence's rows all zero, every other sequence still right."""
    B, H, n_pad, cap = 40, 8, 64, 512
    assert fc.LIB.fc_tree_attn_streamed(B, n_pad, H, H, cap) == 1
    rng = synth.rng_for(55)
    tok, par, nn = _random_trees(rng, B, n_pad)
    kvl = rng.integers(0, cap + 1, B).astype(np.int32)
    q = synth.randn_bf16((B, n_pad, H, 128), 71, "cuda")
    kc = synth.randn_bf16((B, H, cap, 128), 72, "cuda")
    vc = synth.randn_bf16((B, H, cap, 128), 73, "cuda")
    kt = synth.randn_bf16((B, H, n_pad, 128), 74, "cuda")
    vt = synth.randn_bf16((B, H, n_pad, 128), 75, "cuda")
    gm = fc.fc_tree_mask(dev(par), dev(nn), dev(kvl))
    good = fc.fc_tree_attn(q, kc, vc, dev(kvl), kt, vt, gm["mask"], dev(nn))
    torch.cuda.synchronize()
    check_no_error(fc)
    bad_nn = nn.copy()
    bad_nn[17] = n_pad + 1
    out = torch.full_like(q, float("nan"))
    fc.fc_tree_attn(q, kc, vc, dev(kvl), kt, vt, gm["mask"], dev(bad_nn), out=out)
    torch.cuda.synchronize()
    assert fc.fc_get_error() == "FC_ERR_INVALID_ARG"
    assert (out[17] == 0).all()
    keep = [b for b in range(B) if b != 17]
    assert torch.equal(out[keep], good[keep])


def test_attn_c3_shape_full(fc, orc):
    # c3: B=16, H=Hkv=32, KV 4096, 64-node trees; every row against the fp64 oracle
    _attn_case(fc, orc, 5, 16, 64, 32, 32, [4096] * 16, 4096, nn=[64] * 16)


def test_attn_c5_shape_full(fc, orc):
    # c5: B=32, H=32, Hkv=8, KV 16384, trees <= 128 nodes; every row
    _attn_case(fc, orc, 6, 32, 128, 32, 8, [16384] * 32, 16384 + 256)


def test_attn_c5_subbatch_full(fc, orc):
    # the launch the step bench times: one sub-batch of 16 sequences (256 CTAs,
    # 1.7 waves, no KV split), KV lengths grown over the steps, trees of every
    # size; every row
    rng = synth.rng_for(53)
    kvl = [16384 + int(x) for x in rng.integers(0, 700, 16)]
    nn = [int(x) for x in rng.choice([1, 20, 40, 70, 97, 128], 16)]
    _attn_case(fc, orc, 11, 16, 128, 32, 8, kvl, 16384 + 768, nn=nn)


# ------------------------------------------------------- accept / append
def test_accept_and_synth_argmax(fc, orc):
    rng = synth.rng_for(60)
    for n_pad, vocab in ((64, 32256), (128, 4), (64, 3)):
        B = 64
        tok, par, nn = _random_trees(rng, B, n_pad, vocab=vocab)
        plen, rtok = synth.argmax_draws(rng, B, n_pad, vocab)
        g_am = fc.fc_synth_argmax(dev(tok), dev(par), dev(nn), dev(plen), dev(rtok), vocab)
        r_am = orc.synth_argmax(tok, par, nn, plen, rtok, vocab)
        assert np.array_equal(host_u32(g_am), r_am)
        # random predictions that often follow some child
        am = rng.integers(0, vocab, (B, n_pad)).astype(np.uint32)
        for b in range(B):
            for i in range(nn[b]):
                ch = [j for j in range(1, nn[b]) if par[b, j] == i]
                if ch and rng.random() < 0.85:
                    am[b, i] = tok[b, ch[int(rng.integers(0, len(ch)))]]
        for argmax in (r_am, am):
            g = fc.fc_accept(dev(tok), dev(par), dev(nn), dev(argmax), 12)
            r = orc.accept(tok, par, nn, argmax, 12)
            assert np.array_equal(g["acc_len"].cpu().numpy(), r["acc_len"])
            assert np.array_equal(g["path"].cpu().numpy(), r["path"])
            assert np.array_equal(host_u32(g["bonus"]), r["bonus"])
    check_no_error(fc)


def _logits_with_predictions(rng, pred, V, n_nodes, extras=True):
    """bf16 logits [B, Np, V] whose row argmax is `pred` (planted maxima; ties
    and NaNs placed so that the first index / first NaN rule decides)."""
    B, Np = pred.shape
    x = rng.standard_normal((B, Np, V)).astype(np.float32)
    for b in range(B):
        for i in range(Np):
            p = int(pred[b, i])
            x[b, i, p] = 8.0 + rng.random()  # clear winner
            if extras and V > 3 and rng.random() < 0.2:
                x[b, i, p:] = np.minimum(x[b, i, p:], x[b, i, p])  # later ties lose
                q = int(rng.integers(p, V))
                x[b, i, q] = x[b, i, p]
            if extras and rng.random() < 0.05:
                x[b, i, p] = np.nan                               # the first NaN wins
    h = (x.view(np.uint32) >> 16).astype(np.uint16)  # truncation: exact bf16 values
    return h


def test_argmax_accept_from_logits(fc, orc):
    rng = synth.rng_for(62)
    for n_pad, V, B in ((64, 32256, 8), (128, 1001, 6), (64, 7, 10)):
        tok, par, nn = _random_trees(rng, B, n_pad, vocab=V)
        plen, rtok = synth.argmax_draws(rng, B, n_pad, V)
        pred = orc.synth_argmax(tok, par, nn, plen, rtok, V)
        h = _logits_with_predictions(rng, pred, V, nn)
        # odd element offset: rows start off any 16-byte boundary
        flat = torch.zeros(h.size + 1, dtype=torch.int16, device="cuda")
        flat[1:] = torch.from_numpy(h.reshape(-1).view(np.int16)).cuda()
        logits = flat[1:].view(torch.bfloat16).view(B, n_pad, V)
        g = fc.fc_argmax_accept(logits, dev(tok), dev(par), dev(nn), 12)
        r_am = orc.argmax_rows(h, nn)
        assert np.array_equal(host_u32(g["argmax"]), r_am)
        r = orc.accept(tok, par, nn, r_am, 12)
        assert np.array_equal(g["acc_len"].cpu().numpy(), r["acc_len"])
        assert np.array_equal(g["path"].cpu().numpy(), r["path"])
        assert np.array_equal(host_u32(g["bonus"]), r["bonus"])
        if V == 32256:  # the planted predictions are the argmax where no NaN was planted
            assert (r["acc_len"] > 0).any()
    check_no_error(fc)


def test_kv_append_copy(fc, orc):
    rng = synth.rng_for(61)
    B, n_pad, Hkv, D, cap, stride = 16, 64, 8, 128, 300, 200
    tok, par, nn = _random_trees(rng, B, n_pad)
    plen, rtok = synth.argmax_draws(rng, B, n_pad, 32256)
    am = orc.synth_argmax(tok, par, nn, plen, rtok, 32256)
    acc = orc.accept(tok, par, nn, am, 12)
    kt = synth.randn_bf16((B, Hkv, n_pad, D), 7, "cuda")
    vt = synth.randn_bf16((B, Hkv, n_pad, D), 8, "cuda")
    kc = synth.randn_bf16((B, Hkv, cap, D), 9, "cuda")
    vc = synth.randn_bf16((B, Hkv, cap, D), 10, "cuda")
    kvl = rng.integers(0, 280, B).astype(np.int32)
    kvl[0] = cap - 1  # overflows unless nothing is accepted
    ctx = rng.integers(0, 32256, (B, stride)).astype(np.uint32)
    cl = rng.integers(1, 180, B).astype(np.int32)
    kc_h, vc_h, ctx_h = bits_bf16(kc).copy(), bits_bf16(vc).copy(), ctx.copy()
    gacc = dict(acc_len=dev(acc["acc_len"]), path=dev(acc["path"]), bonus=dev(acc["bonus"]))
    kvo, clo, root = (torch.empty(B, dtype=torch.int32, device="cuda") for _ in range(3))
    g_ctx = dev(ctx)
    fc.fc_kv_append(gacc, dev(tok), kt, vt, kc, vc, dev(kvl), kvo, g_ctx, dev(cl), clo, root)
    status = fc.fc_get_error()
    ok = kvl + acc["acc_len"] + 1 <= cap
    assert status == ("FC_OK" if ok.all() else "FC_ERR_CAPACITY")
    sel = np.nonzero(ok)[0]
    kc_s, vc_s, ctx_s = kc_h[sel].copy(), vc_h[sel].copy(), ctx_h[sel].copy()
    r_kvo, r_clo, r_root = orc.kv_append(acc["path"][sel], acc["acc_len"][sel], acc["bonus"][sel], tok[sel],
                                         bits_bf16(kt)[sel], bits_bf16(vt)[sel], kc_s, vc_s, kvl[sel], ctx_s, cl[sel])
    assert np.array_equal(bits_bf16(kc)[sel], kc_s) and np.array_equal(bits_bf16(vc)[sel], vc_s)
    assert np.array_equal(host_u32(g_ctx)[sel], ctx_s)
    assert np.array_equal(kvo.cpu().numpy()[sel], r_kvo) and np.array_equal(clo.cpu().numpy()[sel], r_clo)
    assert np.array_equal(host_u32(root)[sel], r_root)
    bad = np.nonzero(~ok)[0]
    assert np.array_equal(kvo.cpu().numpy()[bad], kvl[bad])


# ------------------------------------------------------------- step loop
def test_step_loop_matches_oracle(fc, orc):
    """c5-shaped loop on small corpora: two sources, replay cache with a
    seeded 50% hit pattern, 128-node trees, 24 steps."""
    from paper_2502_17139_gb300.step import StepLoop
    rng = synth.rng_for(70)
    Tr, _ = synth.make_corpus(rng, 200_000, 1.3, synth.VOCAB, n_grams=500, len_range=(8, 64))
    Tc, _ = synth.make_corpus(rng, 1_000_000, 1.1, synth.VOCAB)
    B, steps, n_pad, H, Hkv, D = 8, 24, 128, 8, 2, 128
    stride = 128 + steps * 12
    ctx, cl, _ = synth.make_contexts(rng, B, 128, 16, [Tr, Tc, None], [0.5, 0.25, 0.25], 1.1, ctx_stride=stride)
    hits = synth.cache_hit_pattern(rng, steps, B)
    plen = np.stack([synth.argmax_draws(rng, B, n_pad)[0] for _ in range(steps)])
    rtok = np.stack([synth.argmax_draws(rng, B, n_pad)[1] for _ in range(steps)])
    p = dict(n_max=16, n_min=2, top_k=64, draft_len=10, max_occ=4096, node_budget=128, n_pad=n_pad)
    no_hits = np.zeros_like(hits)
    cache = {}
    orc.step_loop([Tr, Tc], ctx, cl, steps, p, no_hits, plen, rtok, [1, 1], synth.VOCAB,
                  kv_len0=np.full(B, 100, np.int32), cache=cache)  # recording pass
    hist, r_ctx, r_cl, r_kvl = orc.step_loop([Tr, Tc], ctx, cl, steps, p, hits, plen, rtok, [1, 1], synth.VOCAB,
                                             kv_len0=np.full(B, 100, np.int32), cache=cache)
    srcs = [fc.fc_datastore_build(dev(Tr), synth.VOCAB), fc.fc_datastore_build(dev(Tc), synth.VOCAB)]
    loop = StepLoop(srcs, ctx, cl, fc.params(16, 2, 64, 10, 4096), 128, n_pad, [1, 1], H, Hkv, D,
                    kv_cap=100 + steps * 12, kv_len0=100, vocab=synth.VOCAB)
    q = synth.randn_bf16((B, n_pad, H, D), 1, "cuda")
    kt = synth.randn_bf16((B, Hkv, n_pad, D), 2, "cuda")
    vt = synth.randn_bf16((B, Hkv, n_pad, D), 3, "cuda")
    for st in range(steps):  # recording pass
        loop.step(q, kt, vt, dev(no_hits[st]), dev(plen[st]), dev(rtok[st]))
    loop.reset()
    for st in range(steps):
        loop.step(q, kt, vt, dev(hits[st]), dev(plen[st]), dev(rtok[st]))
        assert np.array_equal(loop.skip.cpu().numpy(), hist["hit"][st]), st
        assert np.array_equal(loop.acc["acc_len"].cpu().numpy(), hist["acc_len"][st]), st
        assert np.array_equal(host_u32(loop.acc["bonus"]), hist["bonus"][st]), st
        assert np.array_equal(loop.tree["n_nodes"].cpu().numpy(), hist["n_nodes"][st]), st
    check_no_error(fc)
    assert np.array_equal(host_u32(loop.ctx), r_ctx)
    assert np.array_equal(loop.ctx_len_now.cpu().numpy(), r_cl)
    assert np.array_equal(loop.kv_len_now.cpu().numpy(), r_kvl)
    served = sum(h.sum() for h in hist["hit"])
    assert 0.3 * hits.sum() < served <= hits.sum()  # the replay cache served the queries that asked for it
    assert np.mean(hist["n_nodes"]) > 20  # retrieval keeps finding drafts along the trajectory
