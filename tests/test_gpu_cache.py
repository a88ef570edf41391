"""GPU parity for the CACHE and the missing table (Section IV-B; Section
IV-C, Algorithm 1): fc_cache_search, fc_missing_insert, fc_cache_update and
the step loop with Algorithm 1, against oracle/algorithm1.py on the same
seeded inputs.  Everything here is integer work and must be bit-exact.

The stores handed to the GPU are the oracle's entries written out in the
ABI's layout (tokens of each entry followed by FC_SEP_TOKEN); the GPU's
stores are read back the same way and compared entry by entry.
"""
import numpy as np
import pytest
import torch

import paper_2502_17139_gb300.synth as synth

pytestmark = pytest.mark.gpu
PAD = 0xFFFFFFFF
SEP = 0xFFFFFFFE


@pytest.fixture(scope="module")
def fc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2502_17139_gb300 import build
    build.build()
    import paper_2502_17139_gb300.fastcoder as fcm
    return fcm


@pytest.fixture(scope="module")
def a1(orc):
    from oracle import algorithm1
    return algorithm1


def dev(a):
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint32:
        a = a.view(np.int32)
    return torch.from_numpy(a.copy()).cuda()


def host_u32(t):
    return t.cpu().numpy().view(np.uint32)


def write_stores(cache, entries, marks, dropped=None):
    """Fills a SequenceCache with the given entries (test-side layout)."""
    B, cap = cache.words.shape
    words = np.zeros((B, cap), np.uint32)
    meta = np.zeros((B, 4), np.int32)
    for b, es in enumerate(entries):
        w = 0
        for e in es:
            words[b, w:w + len(e)] = e
            words[b, w + len(e)] = SEP
            w += len(e) + 1
        assert w <= cap
        meta[b] = (w, len(es), marks[b], 0 if dropped is None else dropped[b])
    cache.words.copy_(dev(words))
    cache.meta.copy_(dev(meta))


def read_stores(cache):
    words = host_u32(cache.words)
    meta = cache.meta.cpu().numpy()
    out = []
    for b in range(words.shape[0]):
        row = words[b, :meta[b, 0]].tolist()
        es, cur = [], []
        for t in row:
            if t == SEP:
                es.append(cur)
                cur = []
            else:
                cur.append(t)
        assert not cur, "a stored sequence lacks its separator"
        assert len(es) == meta[b, 1]
        out.append(es)
    return out, meta


def read_missing(missing):
    t = missing.table.cpu().numpy().view(np.uint32)
    kl = missing.key_len
    slots = t[4:].reshape(missing.capacity, 1 + kl)
    keys = {tuple(int(x) for x in s[1:]) for s in slots if s[0] != 0}
    return keys, int(t[0]), int(t[1])


def check_state_matches(fc, a1, cache, st):
    got, meta = read_stores(cache)
    for b in range(len(got)):
        assert got[b] == [e.tolist() for e in st.entries[b]], b
        assert meta[b, 0] == st.words[b] and meta[b, 2] == st.out_mark[b] and meta[b, 3] == st.dropped[b], b


# ------------------------------------------------------------------ search
def random_case(rng, B, vocab, max_entries, max_len, stride):
    entries, ctx_rows = [], []
    for b in range(B):
        ne = int(rng.integers(0, max_entries + 1))
        es = [rng.integers(0, vocab, int(rng.integers(1, max_len + 1))).astype(np.uint32) for _ in range(ne)]
        entries.append(es)
        m = int(rng.integers(0, stride + 1))
        row = rng.integers(0, vocab, m).astype(np.uint32)
        if es and m > 4 and rng.random() < 0.7:  # end the context with a stretch of a stored sequence
            e = es[int(rng.integers(0, len(es)))]
            cut = int(rng.integers(1, len(e) + 1))
            take = min(cut, m)
            row[m - take:] = e[cut - take:cut]
        ctx_rows.append(row)
    ctx = np.zeros((B, stride), np.uint32)
    for b, r in enumerate(ctx_rows):
        ctx[b, :len(r)] = r
    return entries, ctx, np.array([len(r) for r in ctx_rows], np.int32)


SEARCH_CASES = [
    # seed, B, vocab, max_entries, max_len, (n_max, n_min, top_k, d, max_occ), min_size
    (0, 40, 4, 12, 20, (4, 1, 8, 4, 4096), 0),
    (1, 40, 3, 60, 40, (16, 2, 64, 10, 4096), 5),
    (2, 33, 30, 200, 30, (16, 2, 64, 10, 4096), 50),
    (3, 17, 2, 30, 60, (32, 3, 256, 16, 7), 1),
    (4, 25, 5, 80, 25, (8, 1, 1, 1, 1), 0),
    (5, 64, 12, 150, 40, (16, 2, 16, 8, 4096), 20),
]


@pytest.mark.parametrize("case", SEARCH_CASES, ids=[f"s{c[0]}" for c in SEARCH_CASES])
def test_cache_search_parity(fc, a1, case):
    seed, B, vocab, max_entries, max_len, pp, min_size = case
    n_max, n_min, top_k, d, max_occ = pp
    rng = np.random.default_rng(5000 + seed)
    stride = 48
    entries, ctx, cl = random_case(rng, B, vocab, max_entries, max_len, stride)
    S = 2
    cache = fc.SequenceCache(B, capacity=16384, min_size=min_size, chunk=20, ctx_keep=16)
    write_stores(cache, entries, cl)
    p = fc.params(n_max, n_min, top_k, d, max_occ)
    out = fc.retrieve_outputs(S + 1, B, p)
    for v in out.values():
        v.fill_(0x5A5A5A5A)
    state = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    fc.fc_cache_search(cache, None, dev(ctx), dev(cl), p, S, out, state)
    assert fc.fc_get_error() == "FC_OK"
    active = [len(es) >= min_size for es in entries]
    want = a1.cache_search([es if act else [] for es, act in zip(entries, active)], ctx, cl, n_max, n_min, top_k,
                           d, max_occ)
    got_state = state.cpu().numpy()
    assert np.array_equal(got_state, np.where(want["n_drafts"] > 0, 1, 0))
    for name in a1.RESULT_FIELDS:
        g = out[name][S].cpu().numpy()
        w = want[name].view(np.int32) if want[name].dtype == np.uint32 else want[name]
        assert np.array_equal(g, w), name
    served = got_state == 1
    for s in range(S):  # cleared where the CACHE served, untouched elsewhere
        assert (out["n_drafts"][s].cpu().numpy()[served] == 0).all()
        assert (host_u32(out["drafts"][s])[served] == PAD).all()
        assert (out["n_drafts"][s].cpu().numpy()[~served] == 0x5A5A5A5A).all()
    assert served.sum() > 0 or min_size > max_entries


@pytest.mark.parametrize("capacity,plant", [(16384, 1.0), (8192, 0.8), (8192, 0.45), (16384, 0.25), (8192, 0.05)])
def test_cache_search_large_store(fc, a1, capacity, plant):
    """Full stores in which one bigram starts a share `plant` of the stored
    sequences: from a few dozen to a few thousand occurrences, so the
    occurrence sort runs by ranking, by bitonic stages over packed rows and,
    past the rows that fit in shared memory, over the store itself; max_occ
    cuts the largest."""
    rng = np.random.default_rng(5100 + int(plant * 100) + capacity)
    B, stride = 6, 40
    entries = []
    for b in range(B):
        es, w = [], 0
        while True:
            L = int(rng.integers(3, 12))
            if w + L + 1 > capacity:
                break
            e = rng.integers(0, 6, L).astype(np.uint32)
            if rng.random() < plant:
                e[:2] = (7, 8)
            es.append(e)
            w += L + 1
        entries.append(es)
    ctx = rng.integers(0, 6, (B, stride)).astype(np.uint32)
    ctx[:, -2:] = (7, 8)
    ctx[1, -3:] = (3, 7, 8)
    cl = np.full(B, stride, np.int32)
    for max_occ, d in ((4096, 16), (100, 4), (1, 1)):
        cache = fc.SequenceCache(B, capacity=capacity, min_size=50, chunk=20, ctx_keep=16)
        write_stores(cache, entries, cl)
        p = fc.params(16, 2, 64, d, max_occ)
        out = fc.retrieve_outputs(2, B, p)
        state = torch.empty(B, dtype=torch.int32, device="cuda")
        fc.fc_cache_search(cache, None, dev(ctx), dev(cl), p, 1, out, state)
        want = a1.cache_search(entries, ctx, cl, 16, 2, 64, d, max_occ)
        for name in a1.RESULT_FIELDS:
            w = want[name].view(np.int32) if want[name].dtype == np.uint32 else want[name]
            assert np.array_equal(out[name][1].cpu().numpy(), w), (name, max_occ)
    assert fc.fc_get_error() == "FC_OK"


# ----------------------------------------------------------- missing table
@pytest.mark.parametrize("capacity,B", [(1024, 2500), (16, 700)])
def test_missing_table_parity(fc, a1, capacity, B):
    rng = np.random.default_rng(5200 + capacity)
    stride, key_len, S = 12, 2, 2
    missing = fc.MissingTable(capacity, key_len)
    st = a1.State(np.zeros(B, np.int32), a1.CacheParams(), key_len, capacity)
    for rnd in range(3):
        ctx = rng.integers(0, 6 + rnd, (B, stride)).astype(np.uint32)  # few distinct keys: many repeats
        cl = rng.integers(0, stride + 1, B).astype(np.int32)
        code = rng.choice([0, 0, 0, 1, 2], B).astype(np.int32)
        n_drafts = (rng.random((S + 1, B)) < 0.3).astype(np.int32) * rng.integers(1, 9, (S + 1, B)).astype(np.int32)
        fc.fc_missing_insert(missing, dev(ctx), dev(cl), dev(code), dev(n_drafts), S)
        a1.missing_update(st, ctx, cl, code, n_drafts[:S])
        keys, stored, dropped = read_missing(missing)
        assert keys == st.missing, rnd
        assert stored == len(st.missing) and dropped == st.missing_dropped, rnd
    assert fc.fc_get_error() == "FC_OK"
    # lookups through the search: with every CACHE below its threshold, a
    # query is skipped exactly when its key is in M
    Bq = 300
    ctx = rng.integers(0, 8, (Bq, stride)).astype(np.uint32)
    cl = rng.integers(0, stride + 1, Bq).astype(np.int32)
    cache = fc.SequenceCache(Bq, capacity=64, min_size=1, chunk=20, ctx_keep=4)
    cache.init(dev(cl))
    p = fc.params(4, key_len, 4, 4, 16)
    out = fc.retrieve_outputs(S + 1, Bq, p)
    state = torch.empty(Bq, dtype=torch.int32, device="cuda")
    fc.fc_cache_search(cache, missing, dev(ctx), dev(cl), p, S, out, state)
    want = np.array([2 if st.key(ctx[b], int(cl[b])) in st.missing else 0 for b in range(Bq)], np.int32)
    assert np.array_equal(state.cpu().numpy(), want)
    assert (want == 2).sum() > 10
    assert (out["n_drafts"][:S].cpu().numpy()[:, want == 2] == 0).all()


# ------------------------------------------------------------------ update
@pytest.mark.parametrize("capacity,ctx_keep,chunk", [(8192, 16, 20), (64, 3, 5), (16, 0, 1)])
def test_cache_update_parity(fc, a1, capacity, ctx_keep, chunk):
    rng = np.random.default_rng(5300 + capacity)
    B, stride, steps = 37, 400, 30
    ctx = rng.integers(0, 1000, (B, stride)).astype(np.uint32)
    prompt = rng.integers(0, 40, B).astype(np.int32)
    cp = a1.CacheParams(min_size=50, chunk=chunk, ctx_keep=ctx_keep, capacity=capacity)
    st = a1.State(prompt, cp, 2, 16)
    cache = fc.SequenceCache(B, capacity=capacity, min_size=50, chunk=chunk, ctx_keep=ctx_keep)
    cache.init(dev(prompt))
    cur = prompt.copy()
    ctx_d = dev(ctx)
    for t in range(steps):
        acc = rng.integers(0, 9, B).astype(np.int32)
        new = np.minimum(cur + acc + 1, stride).astype(np.int32)
        failed = rng.random(B) < 0.1
        new[failed] = cur[failed]  # an append that did not happen
        fc.fc_cache_update(cache, ctx_d, dev(cur), dev(new), dev(acc))
        a1.cache_update(st, ctx, cur, new, acc)
        cur = new
    check_state_matches(fc, a1, cache, st)
    assert fc.fc_get_error() == "FC_OK"
    if capacity == 64:
        assert st.dropped.sum() > 0


# --------------------------------------------------------------- step loop
def _trajectory(fc, a1, orc, seed, B, steps, cq, n_pad=128):
    from paper_2502_17139_gb300.step import StepLoop
    rng = synth.rng_for(seed)
    Tr, _ = synth.make_corpus(rng, 200_000, 1.3, synth.VOCAB, n_grams=500, len_range=(8, 64))
    Tc, _ = synth.make_corpus(rng, 1_000_000, 1.1, synth.VOCAB)
    H, Hkv, D = 8, 2, 128
    stride = 128 + steps * 12
    ctx, cl, _ = synth.make_contexts(rng, B, 128, 16, [Tr, Tc, None], [0.5, 0.25, 0.25], 1.1, ctx_stride=stride)
    plen = np.stack([synth.argmax_draws(rng, B, n_pad)[0] for _ in range(steps)])
    rtok = np.stack([synth.argmax_draws(rng, B, n_pad)[1] for _ in range(steps)])
    p = dict(n_max=16, n_min=2, top_k=64, draft_len=10, max_occ=4096, node_budget=n_pad, n_pad=n_pad)
    cp = a1.CacheParams(min_size=cq["min_size"], chunk=cq["chunk"], ctx_keep=16, capacity=cq["capacity"])
    hist, r_ctx, r_cl, r_kvl, st = a1.step_loop([Tr, Tc], ctx, cl, steps, p, cp, plen, rtok, [1, 1], 1,
                                                synth.VOCAB, cq["missing_capacity"],
                                                kv_len0=np.full(B, 100, np.int32))
    srcs = [fc.fc_datastore_build(dev(Tr), synth.VOCAB), fc.fc_datastore_build(dev(Tc), synth.VOCAB)]
    loop = StepLoop(srcs, ctx, cl, fc.params(16, 2, 64, 10, 4096), n_pad, n_pad, [1, 1], H, Hkv, D,
                    kv_cap=100 + steps * 12, kv_len0=100, vocab=synth.VOCAB, seq_cache=dict(cq, weight=1))
    q = synth.randn_bf16((B, n_pad, H, D), 1, "cuda")
    kt = synth.randn_bf16((B, Hkv, n_pad, D), 2, "cuda")
    vt = synth.randn_bf16((B, Hkv, n_pad, D), 3, "cuda")
    zeros = torch.zeros(B, dtype=torch.int32, device="cuda")
    for t in range(steps):
        loop.step(q, kt, vt, zeros, dev(plen[t]), dev(rtok[t]), attention=(t % 8 == 0))
        assert np.array_equal(loop.skip.cpu().numpy(), hist["code"][t]), t
        assert np.array_equal(loop.res["n_drafts"].cpu().numpy(), hist["n_drafts"][t]), t
        assert np.array_equal(loop.acc["acc_len"].cpu().numpy(), hist["acc_len"][t]), t
        assert np.array_equal(host_u32(loop.acc["bonus"]), hist["bonus"][t]), t
        assert np.array_equal(loop.tree["n_nodes"].cpu().numpy(), hist["n_nodes"][t]), t
    assert fc.fc_get_error() == "FC_OK"
    assert np.array_equal(host_u32(loop.ctx), r_ctx)
    assert np.array_equal(loop.ctx_len_now.cpu().numpy(), r_cl)
    check_state_matches(fc, a1, loop.seq_cache, st)
    keys, stored, dropped = read_missing(loop.missing)
    assert keys == st.missing and dropped == st.missing_dropped
    return np.stack(hist["code"])


def test_algorithm1_step_loop_small_threshold(fc, a1, orc):
    """l = 4 and 8-token output pieces: the CACHE serves from the first few
    steps on, and its searches, the datastore fallbacks, the missing table
    and the updates stay in lockstep with the oracle for 40 steps."""
    codes = _trajectory(fc, a1, orc, 71, 8, 40, dict(capacity=4096, min_size=4, chunk=8, missing_capacity=1 << 12))
    assert (codes == 1).sum() >= 10 and (codes == 0).sum() > 100


def test_algorithm1_step_loop_paper_settings(fc, a1, orc):
    """l = 50 and 20-token pieces (Section V-C): the CACHE switches on part
    way through the trajectory."""
    codes = _trajectory(fc, a1, orc, 72, 12, 90, dict(capacity=8192, min_size=50, chunk=20,
                                                      missing_capacity=1 << 16))
    assert (codes[:30] == 1).sum() == 0 and (codes == 1).sum() > 0
