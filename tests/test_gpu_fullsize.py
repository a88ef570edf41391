"""Parity at the full benchmark sizes, where the oracle cannot redo everything.

* Suffix arrays of 100M- and 1B-token corpora: the oracle's certificate (a
  permutation whose adjacent suffixes are strictly increasing), and the bucket
  table against its closed form bucket[v] = #{i : T[i] < v}.
* Retrieval and draft trees for every query on the GPU, compared bit-exactly
  with the oracle on a seeded sample of queries (the oracle scans the whole
  corpus once per query and source).
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
    cfg = synth.CONFIGS[2]
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
    sample = np.sort(synth.rng_for(2, 9).choice(cfg["batch"], 16, replace=False))
    res = []
    for s, T in enumerate(corpora):
        r = orc.retrieve(T, ctx[sample], cl[sample], cfg["n_max"], cfg["n_min"], cfg["top_k"], cfg["draft_len"], 4096)
        compare_rows({k: v[s] for k, v in g.items()}, r, sample)
        res.append(r)
    rt = orc.build_tree(res, [1, 1], root[sample], kvl[sample], cfg["node_budget"], cfg["n_pad"])
    compare_rows(gt, rt, sample)
    # the sample exercises long project-store matches and short general ones
    ml = g["match_len"].cpu().numpy()
    assert (ml[0] == 16).mean() > 0.3 and (ml[1] > 0).mean() > 0.9


def test_one_billion_tokens(fc, orc):
    """Large datastore: 1B tokens (Zipf 1.1, 1% of positions in planted
    16-128-token repeats), 1024 contexts whose last 24 tokens are copied from
    the corpus (half from inside planted repeats), n 24 -> 2, top-64 x 12,
    128-node trees."""
    cfg = synth.CONFIGS[4]
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
    sample = np.sort(synth.rng_for(4, 9).choice(cfg["batch"], 8, replace=False))
    r = orc.retrieve(T, ctx[sample], cl[sample], cfg["n_max"], cfg["n_min"], cfg["top_k"], cfg["draft_len"], 4096)
    compare_rows({k: v[0] for k, v in g.items()}, r, sample)
    rt = orc.build_tree([r], [1], root[sample], kvl[sample], cfg["node_budget"], cfg["n_pad"])
    compare_rows(gt, rt, sample)
    assert (g["match_len"].cpu().numpy() == 24).mean() > 0.9
