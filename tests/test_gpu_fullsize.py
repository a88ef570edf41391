"""Parity at the full benchmark sizes.

* Suffix arrays of 100M- and 1B-token corpora: the oracle's certificate (a
  permutation whose adjacent suffixes are strictly increasing), and the bucket
  table against its closed form bucket[v] = #{i : T[i] < v}.
* Retrieval and draft trees of every query of the two-source workload (256
  contexts, both sources; forward, reversed-corpus and all-occurrence
  variants) and of the 1B-token workload (1024 contexts), bit-exact against
  the oracle's linear corpus scans, which run on all host cores.
* The benchmarked step loop on the real 100M + 5M store (32 sequences in the
  bench's two sub-batch streams, GQA 32/8, KV 16384, 128-node trees, 50%
  replay hits) in lockstep with the oracle's step loop, and its tree
  attention on every row of one step against the fp64 oracle.
* The decoder forward at DeepSeek-Coder 1.3B's layer width against the fp64
  oracle on every node of two sequences, within three times the distance
  that bf16 storage alone puts between the oracle and the exact forward.
* Algorithm 1 on the default two-source store through properties that hold
  at any size (served drafts and their counts recounted in the stores, no
  longer match, missing-table keys absent from both corpora).
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


def dev(a):
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint32:
        a = a.view(np.int32)
    return torch.from_numpy(a).cuda()


def host_u32(t):
    return t.cpu().numpy().view(np.uint32)


def check_datastore(orc, ds, T, vocab):
    sa = host_u32(ds.sa)
    assert orc.sa_certificate(T, sa) == -1
    counts = np.bincount(T, minlength=vocab).astype(np.int64)
    closed = np.concatenate([[0], np.cumsum(counts)])
    assert np.array_equal(host_u32(ds.bucket).astype(np.int64), closed)
    # LCP of adjacent suffixes, from the definition, at sampled SA positions
    lcp = ds.lcp.cpu().numpy()
    assert lcp[0] == 0
    n = len(T)
    for j in synth.rng_for(99).integers(1, n, 2000):
        a, b = int(sa[j - 1]), int(sa[j])
        l = 0
        while l < 255 and a + l < n and b + l < n and T[a + l] == T[b + l]:
            l += 1
        assert lcp[j] == l, j


def compare_rows(g, r, rows):
    for name in r:
        gg = g[name].cpu().numpy()
        if r[name].dtype == np.uint32:
            gg = gg.view(np.uint32)
        elif r[name].dtype == np.uint64:
            gg = gg.view(np.uint64)
        assert np.array_equal(gg[rows], r[name]), name


def test_two_source_100m_5m(fc, orc):
    """Two-source workload: project store 5M (Zipf 1.3, planted repeats), general
    store 100M (Zipf 1.1), 256 contexts of 128 tokens, top-64 x 10, 64-node trees."""
    cfg = synth.WORKLOADS[2]
    rng = synth.rng_for(2)
    corpora = [synth.build_corpus(rng, spec, device="cuda")[0] for spec in cfg["corpus"]]
    Tr, Tc = corpora
    ctx, cl, _ = synth.make_contexts(rng, cfg["batch"], cfg["ctx_len"], cfg["n_copy"], [Tr, Tc, None], cfg["probs"],
                                     1.1)
    sources = []
    for T in corpora:
        ds = fc.fc_datastore_build(dev(T), synth.VOCAB)
        check_datastore(orc, ds, T, synth.VOCAB)
        sources.append(ds)
    p = fc.params(cfg["n_max"], cfg["n_min"], cfg["top_k"], cfg["draft_len"], 4096)
    g = fc.fc_retrieve(sources, dev(ctx), dev(cl), p)
    root = ctx[np.arange(cfg["batch"]), cl - 1]
    kvl = np.full(cfg["batch"], 4096, np.int32)
    gt = fc.fc_build_tree(g, [1, 1], dev(root), dev(kvl), cfg["node_budget"], cfg["n_pad"])
    assert fc.fc_get_error() == "FC_OK"
    every = np.arange(cfg["batch"])
    res = []
    for s, T in enumerate(corpora):
        r = orc.retrieve(T, ctx, cl, cfg["n_max"], cfg["n_min"], cfg["top_k"], cfg["draft_len"], 4096)
        compare_rows({k: v[s] for k, v in g.items()}, r, every)
        res.append(r)
    rt = orc.build_tree(res, [1, 1], root, kvl, cfg["node_budget"], cfg["n_pad"])
    compare_rows(gt, rt, every)
    # the reversed-corpus variant, every query
    revs = [fc.fc_datastore_build_reversed(dev(T), synth.VOCAB) for T in corpora]
    gr = fc.fc_retrieve_rev(sources, revs, dev(ctx), dev(cl), p)
    assert fc.fc_get_error() == "FC_OK"
    for s, r in enumerate(res):
        compare_rows({k: v[s] for k, v in gr.items()}, r, every)
    del revs, gr
    # the all-occurrence trie (every distinct continuation, up to 4096 per
    # source) of every query, against the oracle's untruncated lists
    pa = fc.params(cfg["n_max"], cfg["n_min"], 8, cfg["draft_len"], 4096)
    ga = fc.fc_retrieve_all(sources, dev(ctx), dev(cl), pa)
    ra = [orc.retrieve(T, ctx, cl, cfg["n_max"], cfg["n_min"], 4096, cfg["draft_len"], 4096) for T in corpora]
    gta = fc.fc_build_tree_all(ga, [1, 1], dev(root), dev(kvl), cfg["node_budget"], cfg["n_pad"])
    assert fc.fc_get_error() == "FC_OK"
    rta = orc.build_tree(ra, [1, 1], root, kvl, cfg["node_budget"], cfg["n_pad"])
    compare_rows(gta, rta, every)
    del ga, gta
    torch.cuda.empty_cache()
    # the workload has long project-store matches and short general ones
    ml = g["match_len"].cpu().numpy()
    assert (ml[0] == 16).mean() > 0.3 and (ml[1] > 0).mean() > 0.9


def test_one_billion_tokens(fc, orc):
    """Large datastore: 1B tokens (Zipf 1.1, 1% of positions in planted
    16-128-token repeats), 1024 contexts whose last 24 tokens are copied from
    the corpus (half from inside planted repeats), n 24 -> 2, top-64 x 12,
    128-node trees."""
    cfg = synth.WORKLOADS[4]
    rng = synth.rng_for(4)
    T, planted = synth.build_corpus(rng, cfg["corpus"][0], device="cuda")
    ctx, cl, _ = synth.make_contexts(rng, cfg["batch"], cfg["ctx_len"], cfg["n_copy"], [T], [1.0], 1.1,
                                     planted=[planted], planted_share=cfg["planted_share"])
    ds = fc.fc_datastore_build(dev(T), synth.VOCAB)
    check_datastore(orc, ds, T, synth.VOCAB)
    p = fc.params(cfg["n_max"], cfg["n_min"], cfg["top_k"], cfg["draft_len"], 4096)
    g = fc.fc_retrieve([ds], dev(ctx), dev(cl), p)
    root = ctx[np.arange(cfg["batch"]), cl - 1]
    kvl = np.zeros(cfg["batch"], np.int32)
    gt = fc.fc_build_tree(g, [1], dev(root), dev(kvl), cfg["node_budget"], cfg["n_pad"])
    assert fc.fc_get_error() == "FC_OK"
    every = np.arange(cfg["batch"])
    r = orc.retrieve(T, ctx, cl, cfg["n_max"], cfg["n_min"], cfg["top_k"], cfg["draft_len"], 4096)
    compare_rows({k: v[0] for k, v in g.items()}, r, every)
    rt = orc.build_tree([r], [1], root, kvl, cfg["node_budget"], cfg["n_pad"])
    compare_rows(gt, rt, every)
    assert (g["match_len"].cpu().numpy() == 24).mean() > 0.9


def bits_bf16(t):
    return t.cpu().view(torch.int16).numpy().view(np.uint16)


def test_step_loop_full_store_lockstep(fc, orc):
    """The benchmarked configuration at full size: the 100M + 5M two-source
    store, 32 sequences with 128-token contexts, n 16 -> 2, top-64 x 10 per
    source, 128-node trees, GQA 32/8, head dim 128, KV 16384, a seeded 50%
    replay-cache hit pattern, and the bench's launch configuration (four
    sub-batches of 8 sequences issued by the step executor, each on streams of
    its own with its own replay cache).  A recording pass fills the caches; the replayed pass is
    compared with the oracle's step loop step by step: which queries the
    cache served, tree sizes, accepted lengths, bonus tokens, and at the end
    every context, context length and KV length.  The last step's tree
    attention is compared on every row with the fp64 oracle."""
    import bench
    from paper_2502_17139_gb300.step import PipelinedStepLoop
    steps = 24
    inp = bench.make_inputs(1.0, 32, 0, steps + 1)
    cfg, B = inp["cfg"], inp["B"]
    H, Hkv, D, n_pad, d = cfg["H"], cfg["Hkv"], cfg["D"], cfg["n_pad"], cfg["draft_len"]
    kv0 = inp["kv0"]
    assert kv0 == 16384 and B == 32
    cap = kv0 + (steps + 1) * (d + 1) + 8
    sources = [fc.fc_datastore_build(dev(T), synth.VOCAB) for T in inp["corpora"]]
    p = fc.params(cfg["n_max"], cfg["n_min"], cfg["top_k"], d, 4096)
    kc = synth.randn_bf16((B, Hkv, cap, D), 501, "cuda")
    vc = synth.randn_bf16((B, Hkv, cap, D), 502, "cuda")
    acts = [(synth.randn_bf16((B, n_pad, H, D), 510 + i, "cuda"), synth.randn_bf16((B, Hkv, n_pad, D), 520 + i, "cuda"),
             synth.randn_bf16((B, Hkv, n_pad, D), 530 + i, "cuda")) for i in range(2)]
    loop = PipelinedStepLoop(4, sources, inp["ctx"], inp["cl"], p, cfg["node_budget"], n_pad, [1, 1], H, Hkv, D, cap,
                             kv0, synth.VOCAB, cache_capacity=1 << 14, k_cache=kc, v_cache=vc)
    # the per-step inputs stay resident: the sub-batch streams read them after
    # step() returns, so they must not be temporaries
    to_dev = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int32)).cuda()
    hits = inp["hits"][:steps]
    no_hits = np.zeros_like(hits)
    hits_d, no_hits_d = to_dev(hits), to_dev(no_hits)
    plen_d, rtok_d = to_dev(inp["plen"][:steps]), to_dev(inp["rtok"][:steps])
    for s in range(steps):  # recording pass
        loop.step(*acts[s % 2], no_hits_d[s], plen_d[s], rtok_d[s])
    loop.reset()
    got = dict(hit=[], acc_len=[], bonus=[], n_nodes=[])
    for s in range(steps):
        last = s == steps - 1
        if last:
            loop.join()
            kvl_before = loop.kv_len_now.cpu().numpy()
        loop.step(*acts[s % 2], hits_d[s], plen_d[s], rtok_d[s])
        loop.join()
        got["hit"].append(loop.skip.cpu().numpy())
        got["acc_len"].append(loop.acc["acc_len"].cpu().numpy())
        got["bonus"].append(host_u32(loop.acc["bonus"]))
        got["n_nodes"].append(loop.tree["n_nodes"].cpu().numpy())
    torch.cuda.synchronize()
    assert fc.fc_get_error() == "FC_OK" and loop.errors() == ["FC_OK"] * 4
    # the oracle, one sub-batch at a time with a replay cache of its own
    po = dict(n_max=cfg["n_max"], n_min=cfg["n_min"], top_k=cfg["top_k"], draft_len=d, max_occ=4096,
              node_budget=cfg["node_budget"], n_pad=n_pad)
    ref = dict(hit=[], acc_len=[], bonus=[], n_nodes=[])
    r_ctx, r_cl, r_kvl = [], [], []
    for sl in loop.slices:
        cache = {}
        args = (inp["corpora"], inp["ctx"][sl], inp["cl"][sl], steps, po)
        draws = (inp["plen"][:steps, sl], inp["rtok"][:steps, sl], [1, 1], synth.VOCAB)
        orc.step_loop(*args, no_hits[:, sl], *draws, kv_len0=np.full(sl.stop - sl.start, kv0, np.int32), cache=cache)
        hist, c_, l_, k_ = orc.step_loop(*args, hits[:, sl], *draws, kv_len0=np.full(sl.stop - sl.start, kv0, np.int32),
                                         cache=cache)
        for name in ref:
            ref[name].append(hist[name])
        r_ctx.append(c_)
        r_cl.append(l_)
        r_kvl.append(k_)
    for s in range(steps):
        for name in ("acc_len", "bonus", "n_nodes", "hit"):
            assert np.array_equal(got[name][s], np.concatenate([h[s] for h in ref[name]])), (name, s)
    assert np.array_equal(host_u32(loop.ctx), np.concatenate(r_ctx))
    assert np.array_equal(loop.ctx_len_now.cpu().numpy(), np.concatenate(r_cl))
    assert np.array_equal(loop.kv_len_now.cpu().numpy(), np.concatenate(r_kvl))
    served = sum(int(h.sum()) for h in got["hit"])
    assert 0.3 * hits.sum() < served <= hits.sum()
    nn_all = np.concatenate(got["n_nodes"])
    assert nn_all.mean() > 40 and (nn_all == 128).any() and (nn_all < 64).any()
    # the last step's attention, every row, against the fp64 oracle (the cache
    # rows it read, [0, kv_len), were not touched by that step's append)
    q, kt, vt = acts[(steps - 1) % 2]
    tree = loop.tree
    nn = tree["n_nodes"].cpu().numpy()
    mask = tree["mask"].cpu().numpy().view(np.uint64)
    out = loop.attn_out.float().cpu().numpy()
    ref_out = orc.tree_attn(bits_bf16(q), bits_bf16(kc), bits_bf16(vc), kvl_before, bits_bf16(kt), bits_bf16(vt),
                            mask, nn)
    assert np.isfinite(out).all()
    assert np.abs(out - ref_out).max() <= 2e-2


def test_decoder_full_width(fc, orc):
    """The decoder forward at DeepSeek-Coder 1.3B's layer width (hidden 2048,
    16 heads x 128, MLP 5504, vocab 32256; two layers of it) over 64-node
    trees and 2048-token caches, the shapes the decoder bench runs, against the
    fp64 oracle on every node of two sequences."""
    from oracle import decoder as dec
    from paper_2502_17139_gb300.decoder import DecoderShape, TreeDecoder
    shape = dict(hidden=2048, layers=2, H=16, Hkv=16, inter=5504, vocab=32256)
    s = DecoderShape(**shape)
    cfg = dec.DecoderConfig(**shape)
    Wt = synth.decoder_weights(s.hidden, s.layers, s.H, s.Hkv, s.D, s.inter, s.vocab, 79)
    Wd = {k: v.cuda() for k, v in Wt.items() if k != "layers"}
    Wd["layers"] = [{k: v.cuda() for k, v in Lw.items()} for Lw in Wt["layers"]]
    tobits = lambda t: t.view(torch.int16).numpy().view(np.uint16)
    Wb = {k: tobits(v) for k, v in Wt.items() if k != "layers"}
    Wb["layers"] = [{k: tobits(v) for k, v in Lw.items()} for Lw in Wt["layers"]]
    W = dec.widen_weights(Wb)
    B, n_pad, kv, cap = 2, 64, 2048, 2056
    rng = synth.rng_for(93)
    tok = np.full((B, n_pad), 0xFFFFFFFF, np.uint32)
    par = np.full((B, n_pad), -1, np.int32)
    nn = np.array([24, 9], np.int32)
    for b in range(B):
        t, p = synth.random_tree(rng, int(nn[b]), 10, 4, s.vocab)
        tok[b, :nn[b]], par[b, :nn[b]] = t, p
    kvl = np.array([kv, kv - 777], np.int32)
    m = orc.tree_mask(par, nn, kvl, n_pad)
    caches = [(synth.randn_bf16((B, s.Hkv, cap, s.D), 960 + l, "cuda"),
               synth.randn_bf16((B, s.Hkv, cap, s.D), 980 + l, "cuda")) for l in range(s.layers)]
    f64 = lambda t: t.float().cpu().numpy().astype(np.float64)
    kc = [f64(c[0]) for c in caches]
    vc = [f64(c[1]) for c in caches]
    td = TreeDecoder(s, Wd, B, n_pad, cap, caches=caches)
    logits = td.forward(dev(tok), dev(nn), dev(m["mask"].view(np.int64)), dev(m["pos"]), dev(kvl))
    torch.cuda.synchronize()
    assert fc.fc_get_error() == "FC_OK"
    ref, k_new, v_new = dec.forward(cfg, W, tok, par, nn, kvl, kc, vc, m["pos"])
    mir, k_mir, v_mir = dec.forward(cfg, W, tok, par, nn, kvl, kc, vc, m["pos"], store_bf16=True)
    got = f64(logits)
    # tolerance: three times the distance that bf16 storage alone puts between the
    # oracle's forward and the exact one (the derivation is in tests/test_gpu_decoder.py)
    for b in range(B):
        n = int(nn[b])
        tol = 3 * np.abs(mir[b, :n] - ref[b, :n]).max()
        assert 0 < tol and np.abs(got[b, :n] - ref[b, :n]).max() <= tol
        top2 = np.sort(ref[b, :n], axis=1)[:, -2:]
        clear = top2[:, 1] - top2[:, 0] > tol
        assert (np.argmax(got[b, :n], 1)[clear] == np.argmax(ref[b, :n], 1)[clear]).all()
        for l in range(s.layers):
            tk = 3 * np.abs(k_mir[l, b, :n] - k_new[l, b, :n]).max()
            tv = max(3 * np.abs(v_mir[l, b, :n] - v_new[l, b, :n]).max(), 2.0 ** -8 * np.abs(v_new[l, b, :n]).max())
            assert np.abs(f64(td.k_rot[l])[b, :, :n].transpose(1, 0, 2) - k_new[l, b, :n]).max() <= tk
            assert np.abs(f64(td.v_heads[l])[b, :, :n].transpose(1, 0, 2) - v_new[l, b, :n]).max() <= tv


def test_algorithm1_full_size_properties(fc):
    """Algorithm 1 on the default step loop's two-source store (100M + 5M
    tokens, 32 sequences, l = 50, 20-token pieces, 8192-word CACHEs) after 100
    steps, checked through properties that hold at any size: a draft the CACHE
    returns follows the matched context suffix inside one stored sequence, as
    often as its count says; no stored sequence holds a longer match; every
    sampled key of the missing table occurs in neither corpus followed by a
    token."""
    import bench
    from paper_2502_17139_gb300.step import StepLoop
    steps = 100
    inp = bench.make_inputs(1.0, 32, 0, steps + 1)
    cfg, B = inp["cfg"], inp["B"]
    d = cfg["draft_len"]
    sources = [fc.fc_datastore_build(dev(T), synth.VOCAB) for T in inp["corpora"]]
    p = fc.params(cfg["n_max"], cfg["n_min"], cfg["top_k"], d, 4096)
    seq = dict(capacity=8192, min_size=50, chunk=20, ctx_keep=16, missing_capacity=1 << 16, weight=1)
    kv0 = 64
    loop = StepLoop(sources, inp["ctx"], inp["cl"], p, 128, 128, [1, 1], 32, 8, 128, kv0 + (steps + 1) * (d + 1) + 8,
                    kv0, synth.VOCAB, seq_cache=seq)
    q = torch.zeros((B, 128, 32, 128), dtype=torch.bfloat16, device="cuda")
    kt = torch.zeros((B, 8, 128, 128), dtype=torch.bfloat16, device="cuda")
    zeros = torch.zeros(B, dtype=torch.int32, device="cuda")
    to_dev = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int32)).cuda()
    for s in range(steps):
        loop.step(q, kt, kt, zeros, to_dev(inp["plen"][s]), to_dev(inp["rtok"][s]), attention=False)
    # one more search on the final state, read back
    S = 2
    res = fc.retrieve_outputs(S + 1, B, p)
    state = torch.empty(B, dtype=torch.int32, device="cuda")
    fc.fc_cache_search(loop.seq_cache, loop.missing, loop.ctx, loop.ctx_len_now, p, S, res, state)
    torch.cuda.synchronize()
    assert fc.fc_get_error() == "FC_OK"
    words = host_u32(loop.seq_cache.words)
    meta = loop.seq_cache.meta.cpu().numpy()
    ctx = host_u32(loop.ctx)
    cl = loop.ctx_len_now.cpu().numpy()
    st = state.cpu().numpy()
    nd = res["n_drafts"][S].cpu().numpy()
    ml = res["match_len"][S].cpu().numpy()
    drafts = host_u32(res["drafts"][S])
    dl = res["draft_len"][S].cpu().numpy()
    cnt = res["count"][S].cpu().numpy()
    SEP = 0xFFFFFFFE
    assert (meta[:, 1] >= 50).any()
    served = np.nonzero(st == 1)[0]
    assert len(served) > 0
    for b in served:
        entries = np.split(words[b, :meta[b, 0]], np.nonzero(words[b, :meta[b, 0]] == SEP)[0] + 1)[:-1]
        entries = [e[:-1] for e in entries]  # drop the separators
        assert len(entries) == meta[b, 1]
        n = int(ml[b])
        suf = ctx[b, cl[b] - n:cl[b]].tolist()
        # every occurrence of the matched suffix followed by a token, and its continuation
        conts = {}
        longer = False
        for e in entries:
            el = e.tolist()
            for p0 in range(n, len(el)):
                if el[p0 - n:p0] == suf:
                    key = tuple(el[p0:p0 + d])
                    conts[key] = conts.get(key, 0) + 1
                    if n < min(16, cl[b]) and p0 > n and el[p0 - n - 1] == ctx[b, cl[b] - n - 1]:
                        longer = True
        assert not longer
        if sum(conts.values()) > 4096:  # past max_occ only the smallest windows count
            continue
        assert nd[b] == min(len(conts), cfg["top_k"])
        for t in range(nd[b]):
            key = tuple(drafts[b, t, :dl[b, t]].tolist())
            assert conts.get(key) == cnt[b, t], (b, t)
        assert list(cnt[b, :nd[b]]) == sorted(cnt[b, :nd[b]], reverse=True)
    # sampled missing-table keys: no occurrence followed by a token in either corpus
    tab = loop.missing.table.cpu().numpy().view(np.uint32)
    slots = tab[4:].reshape(-1, 3)
    keys = slots[slots[:, 0] != 0][:, 1:]
    assert len(keys) > 0
    for k0, k1 in keys[synth.rng_for(94).permutation(len(keys))[:4]]:
        for T in inp["corpora"]:
            hit = (T[:-2] == k0) & (T[1:-1] == k1)
            assert not hit.any()


def test_algorithm1_full_size_pipelined_equals_single(fc):
    """Algorithm 1 through the step executor (4 sub-batches, a missing table
    each) against the single loop over the whole batch (one missing table) on
    the default step loop's store (100M + 5M tokens, 32 sequences, l = 50):
    after every step the same trees and acceptance, and after 100 steps the
    same contexts, lengths and CACHE stores.  A missing table only skips
    searches that would find nothing, so splitting it changes no draft."""
    import bench
    from paper_2502_17139_gb300.step import PipelinedStepLoop, StepLoop
    steps = 100
    inp = bench.make_inputs(1.0, 32, 0, steps + 1)
    cfg, B = inp["cfg"], inp["B"]
    d = cfg["draft_len"]
    sources = [fc.fc_datastore_build(dev(T), synth.VOCAB) for T in inp["corpora"]]
    p = fc.params(cfg["n_max"], cfg["n_min"], cfg["top_k"], d, 4096)
    seq = dict(capacity=8192, min_size=50, chunk=20, ctx_keep=16, missing_capacity=1 << 16, weight=1)
    kv0 = 64
    args = (sources, inp["ctx"], inp["cl"], p, 128, 128, [1, 1], 32, 8, 128, kv0 + (steps + 1) * (d + 1) + 8, kv0,
            synth.VOCAB)
    single = StepLoop(*args, seq_cache=seq)
    piped = PipelinedStepLoop(4, *args, seq_cache=seq)
    kt = torch.zeros((B, 8, 128, 128), dtype=torch.bfloat16, device="cuda")
    zeros = torch.zeros(B, dtype=torch.int32, device="cuda")
    to_dev = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int32)).cuda()
    served = 0
    for s in range(steps):
        ins = (None, kt, kt, zeros, to_dev(inp["plen"][s]), to_dev(inp["rtok"][s]))
        single.step(*ins, attention=False)
        piped.step(*ins, attention=False)
        piped.join()
        for k in ("n_nodes", "tok", "parent"):
            assert torch.equal(single.tree[k], piped.tree[k]), (s, k)
        assert torch.equal(single.acc["acc_len"], piped.acc["acc_len"]), s
        served += int((piped.skip == 1).sum())
    assert served > 0  # the CACHE served queries
    assert torch.equal(single.ctx, piped.ctx)
    assert torch.equal(single.ctx_len_now, piped.ctx_len_now)
    assert torch.equal(single.seq_cache.words, torch.cat([lp.seq_cache.words for lp in piped.loops]))
    assert torch.equal(single.seq_cache.meta, torch.cat([lp.seq_cache.meta for lp in piped.loops]))
    assert fc.fc_get_error() == "FC_OK" and piped.errors() == ["FC_OK"] * 4
