"""GPU parity for the all-occurrence trie (Section III-A with Eq. 3's counts
over every retrieved continuation, not a top-k): fc_retrieve_all writes every
distinct continuation in token order, fc_build_tree_all builds the weighted
trie over them.  Both must equal the oracle bit for bit: its retrieval with
no truncation (sorted into token order for the comparison) and its tree
builder over that untruncated list, well past the 256 continuations per source
that the shared-memory builder can take."""
import numpy as np
import pytest
import torch

import paper_2502_17139_gb300.synth as synth

pytestmark = pytest.mark.gpu
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
    return torch.from_numpy(a.copy()).cuda()


def lex_sorted(r, b):
    """The oracle's drafts of query b as (tokens, count) in token order."""
    items = []
    for t in range(int(r["n_drafts"][b])):
        l = int(r["draft_len"][b, t])
        items.append((tuple(int(x) for x in r["drafts"][b, t, :l]), int(r["count"][b, t])))
    return sorted(items)


def check_all(g, r, s, slots, d):
    nd = g["n_drafts"][s].cpu().numpy()
    assert np.array_equal(nd, r["n_drafts"])
    assert np.array_equal(g["match_len"][s].cpu().numpy(), r["match_len"])
    dr = g["drafts"][s].cpu().numpy().view(np.uint32)
    dl = g["draft_len"][s].cpu().numpy()
    ct = g["count"][s].cpu().numpy()
    for b in range(len(nd)):
        got = [(tuple(int(x) for x in dr[b, t, :dl[b, t]]), int(ct[b, t])) for t in range(nd[b])]
        assert got == lex_sorted(r, b), b
        assert (dr[b, nd[b]:] == PAD).all() and (dl[b, nd[b]:] == 0).all() and (ct[b, nd[b]:] == 0).all()
        assert (dr[b, :nd[b]][np.arange(d)[None, :] >= dl[b, :nd[b], None]] == PAD).all()


def compare_tree(g, r):
    for name in ("tok", "parent", "depth", "pos", "n_nodes"):
        gg = g[name].cpu().numpy()
        if r[name].dtype == np.uint32:
            gg = gg.view(np.uint32)
        assert np.array_equal(gg, r[name]), name
    assert np.array_equal(g["mask"].cpu().numpy().view(np.uint64), r["mask"])


@pytest.fixture(scope="module")
def two_sources(fc):
    rng = synth.rng_for(43)
    Tr, _ = synth.make_corpus(rng, 80000, 1.3, 300, n_grams=300, len_range=(8, 40))
    Tc, _ = synth.make_corpus(rng, 400000, 1.05, 300)
    B = 40
    ctx, cl, _ = synth.make_contexts(rng, B, 40, 16, [Tr, Tc, None], [0.4, 0.2, 0.4], 1.1, 300)
    cl[:3] = [0, 1, 2]  # empty and too-short contexts: no match
    srcs = [fc.fc_datastore_build(dev(T), 300) for T in (Tr, Tc)]
    return dict(T=(Tr, Tc), ctx=ctx, cl=cl, srcs=srcs, B=B)


# (max_occ, draft length, n_max, n_min): n_max = 2 forces short matches with
# thousands of occurrences, n_max = 16 the long, rarer ones
CASES = [(4096, 10, 2, 1), (4096, 10, 16, 2), (700, 16, 3, 2), (1, 4, 16, 2)]


@pytest.mark.parametrize("max_occ,d,n_max,n_min", CASES)
def test_retrieve_all(fc, orc, two_sources, max_occ, d, n_max, n_min):
    t = two_sources
    p = fc.params(n_max, n_min, 8, d, max_occ)  # top_k is not used
    g = fc.fc_retrieve_all(t["srcs"], dev(t["ctx"]), dev(t["cl"]), p)
    assert fc.fc_get_error() == "FC_OK"
    widest = 0
    for s, T in enumerate(t["T"]):
        r = orc.retrieve(T, t["ctx"], t["cl"], n_max, n_min, max_occ, d, max_occ)
        check_all(g, r, s, max_occ, d)
        widest = max(widest, int(r["n_drafts"].max()))
    if n_max == 2:
        assert widest > 1000  # far past the shared-memory builder's 256 per source


@pytest.mark.parametrize("w,n_max", [((1, 1), 2), ((3, 1), 2), ((0, 1), 3), ((1, 0), 16)])
def test_trie_all(fc, orc, two_sources, w, n_max):
    t = two_sources
    B, d, max_occ, n_pad = t["B"], 10, 4096, 128
    p = fc.params(n_max, 1, 8, d, max_occ)
    g = fc.fc_retrieve_all(t["srcs"], dev(t["ctx"]), dev(t["cl"]), p)
    root = t["ctx"][np.arange(B), np.maximum(t["cl"] - 1, 0)]
    kvl = np.arange(B, dtype=np.int32) * 7
    wv = np.array(w, np.uint32)
    gt = fc.fc_build_tree_all(g, wv, dev(root), dev(kvl), n_pad, n_pad)
    assert fc.fc_get_error() == "FC_OK"
    res = [orc.retrieve(T, t["ctx"], t["cl"], n_max, 1, max_occ, d, max_occ) for T in t["T"]]
    rt = orc.build_tree(res, wv, root, kvl, n_pad, n_pad)
    compare_tree(gt, rt)
    assert (rt["n_nodes"] == n_pad).mean() > 0.5


@pytest.mark.parametrize("seed", range(6))
def test_trie_all_tiny(fc, orc, seed):
    """Tiny alphabets (deep shared prefixes, drafts cut by the corpus end),
    one to three sources, small budgets and n_pad 64."""
    rng = np.random.default_rng(880 + seed)
    S = 1 + seed % 3
    vocab = int(rng.integers(2, 5))
    Ts = [rng.integers(0, vocab, int(rng.integers(20, 3000))).astype(np.uint32) for _ in range(S)]
    B, stride = 24, 12
    ctx = rng.integers(0, vocab, (B, stride)).astype(np.uint32)
    cl = rng.integers(0, stride + 1, B).astype(np.int32)
    d = int(rng.integers(1, 17))
    max_occ = [4096, 1500, 37, 1][seed % 4]
    n_pad = 64 if seed % 2 else 128
    budget = int(rng.integers(1, n_pad + 1))
    srcs = [fc.fc_datastore_build(dev(T), vocab) for T in Ts]
    p = fc.params(8, 1, 4, d, max_occ)
    g = fc.fc_retrieve_all(srcs, dev(ctx), dev(cl), p)
    res = [orc.retrieve(T, ctx, cl, 8, 1, max_occ, d, max_occ) for T in Ts]
    for s in range(S):
        check_all(g, res[s], s, max_occ, d)
    wv = rng.integers(0, 5, S).astype(np.uint32)
    root = rng.integers(0, vocab, B).astype(np.uint32)
    kvl = rng.integers(0, 100, B).astype(np.int32)
    if S * max_occ <= 8192:
        gt = fc.fc_build_tree_all(g, wv, dev(root), dev(kvl), budget, n_pad)
        compare_tree(gt, orc.build_tree(res, wv, root, kvl, budget, n_pad))
    assert fc.fc_get_error() == "FC_OK"


def test_trie_all_rejects_unsorted(fc):
    d, K = 3, 4
    drafts = np.full((1, 2, K, d), PAD, np.uint32)
    drafts[0, 0, :2] = [[1, 2, 3], [1, 1, 1]]  # query 0: descending
    drafts[0, 1, :2] = [[1, 1, 1], [1, 2, 3]]  # query 1: ascending
    res = dict(drafts=dev(drafts), draft_len=dev(np.full((1, 2, K), 3, np.int32)),
               count=dev(np.ones((1, 2, K), np.int32)), n_drafts=dev(np.array([[2, 2]], np.int32)),
               match_len=dev(np.array([[2, 2]], np.int32)))
    gt = fc.fc_build_tree_all(res, [1], dev(np.array([7, 7], np.uint32)), dev(np.array([5, 5], np.int32)), 64, 64)
    assert fc.fc_get_error() == "FC_ERR_INVALID_ARG"
    nn = gt["n_nodes"].cpu().numpy()
    assert nn[0] == 1 and nn[1] == 6  # 1, 1-1, 1-1-1, 1-2, 1-2-3 under the root
    assert int(gt["tok"][0, 0]) == 7 and int(gt["parent"][0, 1]) == -1
