"""GPU tests of the context-keyed replay cache (fc_rcache_*), against its
definition: an insert stores a query's retrieval outputs under its key (the
last min(n_max, ctx_len) context tokens); a lookup of a query that may hit
and whose key is stored copies those outputs back exactly and sets skip = 1,
and otherwise sets skip = 0 and writes nothing.  A tiny table forces probe
chains past occupied slots; a full table reports FC_ERR_CAPACITY."""
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


N_MAX, TOP_K, DLEN, S = 4, 3, 2, 2


def contexts():
    """Six contexts: 0 and 3 share their last four tokens (one key), 1 has a
    two-token context (a two-token key), 4 ends like 1 but is longer (another
    key), 5 is unrelated."""
    stride = 8
    ctx = np.zeros((6, stride), np.int32)
    lens = np.array([6, 2, 5, 7, 8, 4], np.int32)
    rows = [[9, 9, 1, 2, 3, 4], [3, 4], [7, 5, 6, 7, 8], [8, 8, 8, 1, 2, 3, 4], [1, 1, 1, 1, 1, 1, 3, 4],
            [5, 5, 5, 6]]
    for b, r in enumerate(rows):
        ctx[b, :len(r)] = r
    return ctx, lens


def outputs(fc, seed, B, p, equal=((0, 3),)):
    g = torch.Generator().manual_seed(seed)
    o = fc.retrieve_outputs(S, B, p, "cuda")
    host = {k: torch.randint(0, 1000, tuple(v.shape), generator=g, dtype=torch.int32) for k, v in o.items()}
    for a, b in equal:  # queries with one key carry one (deterministic) result
        for k in host:
            host[k][:, b] = host[k][:, a]
    for k in o:
        o[k].copy_(host[k])
    return o, host


def test_rcache_insert_lookup(fc):
    p = fc.params(N_MAX, 1, TOP_K, DLEN, 16)
    ctx_h, lens_h = contexts()
    B = len(lens_h)
    ctx, lens = torch.from_numpy(ctx_h).cuda(), torch.from_numpy(lens_h).cuda()
    cache = fc.RetrievalCache(8, S, p)  # 8 slots for 5 keys: probe chains
    skip = torch.full((B,), 7, dtype=torch.int32, device="cuda")
    probe = fc.retrieve_outputs(S, B, p, "cuda")
    for v in probe.values():
        v.fill_(-5)
    fc.fc_rcache_lookup(cache, ctx, lens, None, skip, probe)  # empty table: every query misses
    torch.cuda.synchronize()
    assert skip.tolist() == [0] * B and all((v == -5).all() for v in probe.values())
    res, host = outputs(fc, 1, B, p)
    fc.fc_rcache_insert(cache, ctx, lens, skip, res)
    assert fc.fc_get_error() == "FC_OK"
    want = torch.tensor([1, 1, 0, 1, 1, 1], dtype=torch.int32, device="cuda")
    got = fc.retrieve_outputs(S, B, p, "cuda")
    for v in got.values():
        v.fill_(-5)
    fc.fc_rcache_lookup(cache, ctx, lens, want, skip, got)
    torch.cuda.synchronize()
    assert skip.tolist() == [1, 1, 0, 1, 1, 1]
    for k in got:
        g = got[k].cpu()
        for b in range(B):
            if b == 2:
                assert (g[:, b] == -5).all(), k  # a query that may not hit is left alone
            else:
                assert torch.equal(g[:, b], host[k][:, b]), (k, b)
    # a context whose key was never stored misses
    other = ctx.clone()
    other[5, 3] = 11
    skip.fill_(7)
    fc.fc_rcache_lookup(cache, other, lens, None, skip, got)
    torch.cuda.synchronize()
    assert skip.tolist() == [1, 1, 1, 1, 1, 0]
    assert fc.fc_get_error() == "FC_OK"


def test_rcache_present_key_not_duplicated_and_full_table(fc):
    p = fc.params(N_MAX, 1, TOP_K, DLEN, 16)
    ctx_h, lens_h = contexts()
    B = len(lens_h)
    ctx, lens = torch.from_numpy(ctx_h).cuda(), torch.from_numpy(lens_h).cuda()
    zero = torch.zeros(B, dtype=torch.int32, device="cuda")
    cache = fc.RetrievalCache(8, S, p)
    res, host = outputs(fc, 2, B, p)
    one = torch.ones(B, dtype=torch.int32, device="cuda")
    one[1] = 0
    fc.fc_rcache_insert(cache, ctx, lens, one, res)  # query 1 alone
    fc.fc_rcache_insert(cache, ctx, lens, one, res)  # again: its key is present, no second entry
    assert fc.fc_get_error() == "FC_OK"
    table = cache.table.view(torch.int32).cpu().numpy().view(np.uint32)
    ew = table.size // 8
    heads = table[::ew][:8]
    assert int((heads != 0xFFFFFFFF).sum()) == 1 and 2 in heads.tolist()
    # four slots for five keys: the table fills and the insert says so
    small = fc.RetrievalCache(4, S, p)
    fc.fc_rcache_insert(small, ctx, lens, zero, res)
    assert fc.fc_get_error() == "FC_ERR_CAPACITY"
    skip = torch.zeros(B, dtype=torch.int32, device="cuda")
    got = fc.retrieve_outputs(S, B, p, "cuda")
    fc.fc_rcache_lookup(small, ctx, lens, None, skip, got)  # what was stored still reads back exactly
    torch.cuda.synchronize()
    hits = skip.cpu().numpy()
    assert 4 <= hits.sum() <= 5
    for k in got:
        g = got[k].cpu()
        for b in np.flatnonzero(hits):
            assert torch.equal(g[:, b], host[k][:, b]), (k, b)
    assert fc.fc_get_error() == "FC_OK"


def test_retrieve_cached_equals_lookup_then_retrieve(fc):
    """fc_retrieve_cached against fc_rcache_lookup followed by fc_retrieve on
    the queries it did not serve: the same outputs and skip flags, for a
    half-filled cache, a want mask, a short context and a context with a token
    outside the vocabulary (recorded only when that query is not served)."""
    import paper_2502_17139_gb300.synth as synth
    rng = synth.rng_for(81)
    vocab = 300
    Ts = [synth.make_corpus(rng, n, 1.1, vocab)[0] for n in (20_000, 5_000)]
    srcs = [fc.fc_datastore_build(torch.from_numpy(T.view(np.int32)).cuda(), vocab) for T in Ts]
    B, stride = 24, 40
    ctx, cl, _ = synth.make_contexts(rng, B, 32, 8, Ts + [None], [0.4, 0.4, 0.2], 1.1, vocab=vocab, ctx_stride=stride)
    cl = cl.copy()
    cl[3] = 2  # shorter than n_max
    ctx[5, cl[5] - 2] = vocab + 7  # a token outside the vocabulary
    ctx_d, cl_d = torch.from_numpy(ctx.view(np.int32)).cuda(), torch.from_numpy(cl).cuda()
    p = fc.params(12, 2, 16, 6, 512)
    cache = fc.RetrievalCache(64, 2, p)
    # fill the cache with the even queries' results
    fill = fc.fc_retrieve(srcs, ctx_d, cl_d, p)
    skip_fill = torch.tensor([b % 2 for b in range(B)], dtype=torch.int32, device="cuda")
    fc.fc_rcache_insert(cache, ctx_d, cl_d, skip_fill, fill)
    fc.fc_get_error()  # the out-of-vocabulary query recorded its error while filling
    for want_h in (None, np.array([1 if b % 3 else 0 for b in range(B)], np.int32)):
        want = None if want_h is None else torch.from_numpy(want_h).cuda()
        ref = fc.retrieve_outputs(2, B, p, "cuda")
        skip_ref = torch.full((B,), 9, dtype=torch.int32, device="cuda")
        fc.fc_rcache_lookup(cache, ctx_d, cl_d, want, skip_ref, ref)
        fc.fc_retrieve(srcs, ctx_d, cl_d, p, skip=skip_ref, out=ref)
        err_ref = fc.fc_get_error()
        got = fc.retrieve_outputs(2, B, p, "cuda")
        skip = torch.full((B,), 9, dtype=torch.int32, device="cuda")
        fc.fc_retrieve_cached(srcs, cache, ctx_d, cl_d, want, skip, p, got)
        err = fc.fc_get_error()
        assert err == err_ref
        assert torch.equal(skip, skip_ref)
        assert int(skip.sum().item()) > 0 and int(skip.sum().item()) < B
        for k in ref:
            assert torch.equal(got[k], ref[k]), k
