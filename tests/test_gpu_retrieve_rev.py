"""GPU parity for the reversed-corpus retrieval variant (Section III-A: the
longest context suffix found by one narrowing search in the suffix array of
the reversed corpus): fc_reverse_tokens, the reversed datastore, and
fc_retrieve_rev, whose outputs must equal the oracle's retrieval bit for bit
(and therefore fc_retrieve's)."""
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
    return torch.from_numpy(a.copy()).cuda()


def host_u32(t):
    return t.cpu().numpy().view(np.uint32)


def compare(g, r, s=0, rows=None):
    for name in ("drafts", "draft_len", "count", "n_drafts", "match_len"):
        gg = g[name][s].cpu().numpy()
        if r[name].dtype == np.uint32:
            gg = gg.view(np.uint32)
        if rows is not None:
            gg = gg[rows]
        assert np.array_equal(gg, r[name]), name


@pytest.mark.parametrize("n", [1, 3, 4, 5, 8, 1023, 1 << 20, (1 << 20) + 3])
def test_reverse_tokens(fc, n):
    T = np.random.default_rng(n).integers(0, 1 << 31, n + 1).astype(np.uint32)
    t = dev(T)
    for src in (t[:n], t[1:]):  # 16-byte aligned, then only 4-byte aligned (the scalar path)
        out = fc.fc_reverse_tokens(src)
        assert np.array_equal(host_u32(out), host_u32(src)[::-1])
    assert fc.fc_get_error() == "FC_OK"


@pytest.mark.parametrize("n,vocab,seed", [(1, 3, 0), (2, 2, 1), (97, 2, 2), (5000, 7, 3), (200_000, 32256, 4)])
def test_reversed_datastore(fc, orc, n, vocab, seed):
    T = np.random.default_rng(900 + seed).integers(0, vocab, n).astype(np.uint32)
    ds = fc.fc_datastore_build_reversed(dev(T), vocab)
    R = T[::-1].copy()
    sa = orc.suffix_array(R)
    assert np.array_equal(host_u32(ds.tokens), R)
    assert np.array_equal(host_u32(ds.sa), sa)
    assert np.array_equal(host_u32(ds.bucket), orc.bucket(R, sa, vocab))


@pytest.mark.parametrize("seed", range(10))
def test_retrieve_rev_tiny_sweep(fc, orc, seed):
    """Small alphabets (long nested ranges), contexts copied from the corpus,
    contexts that end exactly at the corpus end (the occurrence without a
    continuation), empty and short contexts, every max_occ regime."""
    rng = np.random.default_rng(700 + seed)
    N = int(rng.integers(2, 4000))
    vocab = int(rng.integers(2, 9))
    T = rng.integers(0, vocab, N).astype(np.uint32)
    B, stride = 48, 24
    ctx = rng.integers(0, vocab, (B, stride)).astype(np.uint32)
    cl = rng.integers(0, stride + 1, B).astype(np.int32)
    for b in range(B):
        L = int(min(cl[b], N))
        if L and b % 3 == 0:
            p0 = int(rng.integers(0, N - L + 1))
            ctx[b, cl[b] - L:cl[b]] = T[p0:p0 + L]
        elif L and b % 3 == 1:
            ctx[b, cl[b] - L:cl[b]] = T[N - L:]
    n_max = int(rng.integers(1, 33))
    n_min = int(rng.integers(1, n_max + 1)) if seed % 2 else min(2, n_max)
    k, d = int(rng.integers(1, 257)), int(rng.integers(1, 17))
    max_occ = [1, 3, 4096, 17][seed % 4]
    t = dev(T)
    ds, rds = fc.fc_datastore_build(t, vocab), fc.fc_datastore_build_reversed(t, vocab)
    p = fc.params(n_max, n_min, k, d, max_occ)
    g = fc.fc_retrieve_rev([ds], [rds], dev(ctx), dev(cl), p)
    r = orc.retrieve(T, ctx, cl, n_max, n_min, k, d, max_occ)
    compare(g, r)
    assert fc.fc_get_error() == "FC_OK"


def test_retrieve_rev_c1(fc, orc):
    """The 1M-token configuration: 32 contexts whose last 16 tokens are copied
    from the corpus, n 16 -> 2, top-16 x 8."""
    cfg = synth.WORKLOADS[1]
    rng = synth.rng_for(1)
    T, _ = synth.build_corpus(rng, cfg["corpus"][0])
    ctx, cl, _ = synth.make_contexts(rng, cfg["batch"], cfg["ctx_len"], cfg["n_copy"], [T], [1.0], 1.1)
    t = dev(T)
    ds, rds = fc.fc_datastore_build(t, synth.VOCAB), fc.fc_datastore_build_reversed(t, synth.VOCAB)
    p = fc.params(cfg["n_max"], cfg["n_min"], cfg["top_k"], cfg["draft_len"], 4096)
    g = fc.fc_retrieve_rev([ds], [rds], dev(ctx), dev(cl), p)
    r = orc.retrieve(T, ctx, cl, cfg["n_max"], cfg["n_min"], cfg["top_k"], cfg["draft_len"], 4096)
    compare(g, r)
    assert (r["match_len"] >= 8).mean() > 0.5


def test_retrieve_rev_two_sources_and_skip(fc, orc):
    rng = synth.rng_for(41)
    Tr, _ = synth.make_corpus(rng, 60000, 1.3, 500, n_grams=300, len_range=(8, 40))
    Tc, _ = synth.make_corpus(rng, 150000, 1.1, 500)
    ctx, cl, _ = synth.make_contexts(rng, 64, 40, 16, [Tr, Tc, None], [0.5, 0.25, 0.25], 1.1, 500)
    srcs = [fc.fc_datastore_build(dev(T), 500) for T in (Tr, Tc)]
    revs = [fc.fc_datastore_build_reversed(dev(T), 500) for T in (Tr, Tc)]
    p = fc.params(16, 2, 64, 10, 4096)
    skip = np.zeros(64, np.int32)
    skip[::5] = 1
    out = fc.retrieve_outputs(2, 64, p)
    for v in out.values():
        v.fill_(-7)
    g = fc.fc_retrieve_rev(srcs, revs, dev(ctx), dev(cl), p, skip=dev(skip), out=out)
    keep = skip == 0
    for s, T in enumerate((Tr, Tc)):
        r = orc.retrieve(T, ctx, cl, 16, 2, 64, 10, 4096)
        for name in r:
            gg = g[name][s].cpu().numpy()
            if r[name].dtype == np.uint32:
                gg = gg.view(np.uint32)
            assert np.array_equal(gg[keep], r[name][keep]), name
            assert (g[name][s].cpu().numpy()[~keep] == -7).all()
    # the same outputs as the forward search, query for query
    f = fc.fc_retrieve(srcs, dev(ctx), dev(cl), p, skip=dev(skip))
    for name in f:
        assert torch.equal(f[name][:, torch.from_numpy(keep).cuda()], g[name][:, torch.from_numpy(keep).cuda()])


def test_retrieve_rev_bad_context_token(fc):
    T = np.arange(100, dtype=np.uint32) % 10
    t = dev(T)
    ds, rds = fc.fc_datastore_build(t, 10), fc.fc_datastore_build_reversed(t, 10)
    ctx = np.array([[1, 2, 3, 4], [1, 2, 99, 4]], np.uint32)
    g = fc.fc_retrieve_rev([ds], [rds], dev(ctx), dev(np.array([4, 4], np.int32)), fc.params(4, 1, 4, 4, 64))
    assert fc.fc_get_error() == "FC_ERR_INVALID_ARG"
    assert int(g["match_len"][0, 0]) == 4 and int(g["match_len"][0, 1]) == 0


def test_retrieve_rev_rejects_mismatched_store(fc):
    T = np.arange(100, dtype=np.uint32) % 10
    ds = fc.fc_datastore_build(dev(T), 10)
    other = fc.fc_datastore_build_reversed(dev(T[:99]), 10)
    with pytest.raises(fc.FastCoderError):
        fc.fc_retrieve_rev([ds], [other], dev(np.zeros((1, 4), np.uint32)), dev(np.array([4], np.int32)),
                           fc.params(4, 1, 4, 4, 64))
