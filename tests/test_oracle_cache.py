"""Pins for the oracle's CACHE search (O11) and Algorithm 1 with the missing
table (oracle/algorithm1.py).

The CACHE search is checked against brute force over Python lists (searching
suffix lengths from n_max down, unlike the oracle's best-of-scan), against
hand-worked cases in tests/golden/cache_search_handmade.json, and against the
datastore retrieval (O2-O4) in the special case of one stored sequence, where
the two definitions coincide.  Algorithm 1's control flow, the missing table
and the CACHE update are checked on hand-built scenarios whose expected
outcome is written out in the test, and by invariants over a trajectory.
"""
import collections
import json
import os

import numpy as np
import pytest

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
PAD = 0xFFFFFFFF


@pytest.fixture(scope="module")
def a1(orc):
    from oracle import algorithm1
    return algorithm1


def brute_cache_search(entries, c, n_max, n_min, top_k, d, max_occ):
    m = len(c)
    cap = min(n_max, m)
    for n in range(cap, n_min - 1, -1):
        q = list(c[m - n:])
        occ = [(E, p) for E in entries for p in range(n, len(E)) if list(E[p - n:p]) == q]
        if occ:
            break
    else:
        return [], 0
    wins = sorted(occ, key=lambda ep: list(ep[0][ep[1] - n:ep[1] + d]))
    if max_occ:
        wins = wins[:max_occ]
    cnt = collections.Counter(tuple(E[p:p + d]) for E, p in wins)
    ranked = sorted(cnt.items(), key=lambda kv: (-kv[1], list(kv[0])))[:top_k]
    return ranked, n


def check_against(out, b, ranked, n, top_k, d):
    assert out["match_len"][b] == n
    assert out["n_drafts"][b] == len(ranked)
    for t in range(top_k):
        if t < len(ranked):
            seq, c = ranked[t]
            assert out["count"][b, t] == c
            assert out["draft_len"][b, t] == len(seq)
            assert out["drafts"][b, t, :len(seq)].tolist() == list(seq)
            assert all(x == PAD for x in out["drafts"][b, t, len(seq):])
        else:
            assert out["count"][b, t] == 0 and out["draft_len"][b, t] == 0
            assert all(x == PAD for x in out["drafts"][b, t])


def test_cache_search_handmade_golden(a1):
    g = json.load(open(os.path.join(GOLDEN, "cache_search_handmade.json")))
    for case in g["cases"]:
        ctx = np.array([case["ctx"]], np.uint32)
        out = a1.cache_search([[np.array(e, np.uint32) for e in case["entries"]]], ctx, [len(case["ctx"])],
                              case["n_max"], case["n_min"], case["top_k"], case["d"], case["max_occ"])
        assert out["drafts"][0].tolist() == case["drafts"], case["why"]
        assert out["draft_len"][0].tolist() == case["draft_len"], case["why"]
        assert out["count"][0].tolist() == case["count"], case["why"]
        assert out["n_drafts"][0] == case["n_drafts"], case["why"]
        assert out["match_len"][0] == case["match_len"], case["why"]


@pytest.mark.parametrize("seed", range(10))
def test_cache_search_matches_brute_force(a1, seed):
    rng = np.random.default_rng(700 + seed)
    B = 6
    vocab = int(rng.integers(2, 6))
    n_max = int(rng.integers(1, 6))
    n_min = int(rng.integers(1, n_max + 1))
    top_k = int(rng.integers(1, 6))
    d = int(rng.integers(1, 5))
    max_occ = [0, 1, 3, 0, 7][seed % 5]
    entries, ctxs = [], []
    for b in range(B):
        ne = int(rng.integers(0, 9))
        entries.append([rng.integers(0, vocab, int(rng.integers(1, 12))).astype(np.uint32) for _ in range(ne)])
        ctxs.append(rng.integers(0, vocab, int(rng.integers(0, 9))).astype(np.uint32))
    stride = 10
    ctx = np.zeros((B, stride), np.uint32)
    for b, c in enumerate(ctxs):
        ctx[b, :len(c)] = c
    out = a1.cache_search(entries, ctx, [len(c) for c in ctxs], n_max, n_min, top_k, d, max_occ,
                          nthreads=1 + seed % 3)
    for b in range(B):
        ranked, n = brute_cache_search([e.tolist() for e in entries[b]], ctxs[b].tolist(), n_max, n_min, top_k, d,
                                       max_occ)
        check_against(out, b, ranked, n, top_k, d)


@pytest.mark.parametrize("seed", range(4))
def test_one_entry_is_a_datastore(orc, a1, seed):
    # with a single stored sequence, the CACHE search and the datastore
    # retrieval over that sequence as corpus have the same definition
    rng = np.random.default_rng(800 + seed)
    E = rng.integers(0, 4, 300).astype(np.uint32)
    B = 16
    ctx = rng.integers(0, 4, (B, 12)).astype(np.uint32)
    ctx_len = rng.integers(0, 13, B).astype(np.int32)
    args = (6, 2, 5, 4, [0, 2][seed % 2])
    got = a1.cache_search([[E] for _ in range(B)], ctx, ctx_len, *args)
    want = orc.retrieve(E, ctx, ctx_len, *args)
    for name in a1.RESULT_FIELDS:
        assert np.array_equal(got[name], want[name]), name


# ------------------------------------------------------------- Algorithm 1
P = dict(n_max=4, n_min=2, top_k=4, draft_len=3, max_occ=0, node_budget=16, n_pad=16)


def ctx_rows(rows, stride=32):
    ctx = np.zeros((len(rows), stride), np.uint32)
    for b, r in enumerate(rows):
        ctx[b, :len(r)] = r
    return ctx, np.array([len(r) for r in rows], np.int32)


def test_cache_activation_threshold(a1):
    # the CACHE is searched only once it holds l = 2 sequences (Algorithm 1's test)
    T = np.array([1, 2, 3, 4, 5, 6], np.uint32)
    ctx, cl = ctx_rows([[7, 8, 9], [7, 8, 9]])
    st = a1.State(cl, a1.CacheParams(min_size=2), key_len=2, missing_capacity=16)
    st.add_entry(0, [8, 9, 11, 12])
    st.add_entry(1, [8, 9, 11, 12])
    st.add_entry(1, [0, 0])
    res, code = a1.retrieve_step(st, [T], ctx, cl, P)
    assert code.tolist() == [a1.SERVE_DATASTORE, a1.SERVE_CACHE]
    cache_slot = res[-1]
    assert cache_slot["n_drafts"].tolist() == [0, 1]
    assert cache_slot["drafts"][1, 0].tolist() == [11, 12, PAD]
    assert cache_slot["match_len"][1] == 2
    # the datastore is not searched for the sequence the CACHE served
    assert res[0]["n_drafts"][1] == 0
    # [8,9] is not in T either, so sequence 0 found nothing and its key joins M
    assert st.missing == {(8, 9)}


def test_cache_miss_falls_back_to_datastore(a1):
    T = np.array([1, 2, 3, 4, 5, 6], np.uint32)
    ctx, cl = ctx_rows([[9, 2, 3]])
    st = a1.State(cl, a1.CacheParams(min_size=1), key_len=2, missing_capacity=16)
    st.add_entry(0, [5, 5, 5])
    res, code = a1.retrieve_step(st, [T], ctx, cl, P)
    assert code.tolist() == [a1.SERVE_DATASTORE]
    assert res[-1]["n_drafts"][0] == 0
    assert res[0]["n_drafts"][0] == 1 and res[0]["drafts"][0, 0].tolist() == [4, 5, 6]
    assert st.missing == set()


def test_missing_table_skips_and_grows(a1):
    T = np.array([1, 2, 3, 4, 5, 6], np.uint32)
    T2 = np.array([9, 9, 4], np.uint32)
    # seq 0: [6,9] occurs nowhere with a continuation (in T2 it would need 6 first);
    # seq 1: [9,9] occurs in T2 followed by 4; seq 2: shorter than n_min, no key
    ctx, cl = ctx_rows([[1, 6, 9], [3, 9, 9], [5]])
    st = a1.State(cl, a1.CacheParams(min_size=50), key_len=2, missing_capacity=16)
    res, code = a1.retrieve_step(st, [T, T2], ctx, cl, P)
    assert code.tolist() == [0, 0, 0]
    assert res[1]["n_drafts"].tolist() == [0, 1, 0]
    assert st.missing == {(6, 9)}
    # next step: seq 0 is skipped and gets empty results everywhere
    res, code = a1.retrieve_step(st, [T, T2], ctx, cl, P)
    assert code.tolist() == [a1.SKIP_MISSING, 0, 0]
    assert all(r["n_drafts"][0] == 0 for r in res)
    assert st.missing == {(6, 9)}


def test_missing_table_capacity_and_duplicates(a1):
    T = np.array([1, 2, 3], np.uint32)
    # three failing queries: keys (7,7), (7,7) again, (8,8); room for one key
    ctx, cl = ctx_rows([[7, 7], [7, 7], [8, 8]])
    st = a1.State(cl, a1.CacheParams(), key_len=2, missing_capacity=2)
    a1.retrieve_step(st, [T], ctx, cl, P)
    assert st.missing == {(7, 7)}
    assert st.missing_dropped == 1  # (8, 8), counted once


def test_missing_table_not_consulted_when_cache_serves(a1):
    T = np.array([1, 2, 3], np.uint32)
    ctx, cl = ctx_rows([[4, 5]])
    st = a1.State(cl, a1.CacheParams(min_size=1), key_len=2, missing_capacity=16)
    st.missing.add((4, 5))
    st.add_entry(0, [4, 5, 6])
    res, code = a1.retrieve_step(st, [T], ctx, cl, P)
    assert code.tolist() == [a1.SERVE_CACHE]
    assert res[-1]["drafts"][0, 0].tolist() == [6, PAD, PAD]


@pytest.mark.parametrize("seed", range(4))
def test_missing_table_is_sound(orc, a1, seed):
    # every key in M has no occurrence followed by a token in any source, and
    # a skipped query would indeed have retrieved nothing
    rng = np.random.default_rng(900 + seed)
    corpora = [rng.integers(0, 7, int(rng.integers(5, 40))).astype(np.uint32) for _ in range(2)]
    B = 24
    rows = [rng.integers(0, 7, int(rng.integers(0, 6))).tolist() for _ in range(B)]
    ctx, cl = ctx_rows(rows)
    st = a1.State(cl, a1.CacheParams(), key_len=2, missing_capacity=1024)
    for _ in range(2):
        res, code = a1.retrieve_step(st, corpora, ctx, cl, P)
        for key in st.missing:
            for T in corpora:
                assert not any(T[p - 2] == key[0] and T[p - 1] == key[1] for p in range(2, len(T)))
        for b in range(B):
            if code[b] == a1.SKIP_MISSING:
                for T in corpora:
                    r = orc.retrieve(T, ctx[b:b + 1], cl[b:b + 1], P["n_max"], P["n_min"], P["top_k"],
                                     P["draft_len"], 0)
                    assert r["n_drafts"][0] == 0
            if code[b] == a1.SERVE_DATASTORE and cl[b] >= 2 and all(r["n_drafts"][b] == 0 for r in res[:-1]):
                assert tuple(ctx[b, cl[b] - 2:cl[b]].tolist()) in st.missing


def test_cache_update_entries_and_pieces(a1):
    cp = a1.CacheParams(chunk=4, ctx_keep=3)
    ctx = np.arange(100, 132, dtype=np.uint32)[None, :].copy()
    st = a1.State([5], cp, key_len=2, missing_capacity=16)
    # step 1: two accepted draft tokens + bonus -> context 5 -> 8
    a1.cache_update(st, ctx, [5], [8], [2])
    assert [e.tolist() for e in st.entries[0]] == [[102, 103, 104, 105, 106]]
    assert st.out_mark[0] == 5
    # step 2: one accepted + bonus -> 8 -> 10; output 105..109 holds a full piece of 4
    a1.cache_update(st, ctx, [8], [10], [1])
    assert [e.tolist() for e in st.entries[0]][1:] == [[105, 106, 107, 108], [105, 106, 107, 108]]
    assert st.out_mark[0] == 9
    # step 3: nothing accepted (bonus only) -> no verified entry; 9..10 is not a piece yet
    a1.cache_update(st, ctx, [10], [11], [0])
    assert st.n_seq(0) == 3
    # a failed append (length unchanged) stores nothing
    a1.cache_update(st, ctx, [11], [11], [3])
    assert st.n_seq(0) == 3
    assert st.words[0] == sum(len(e) + 1 for e in st.entries[0])


def test_cache_update_capacity(a1):
    cp = a1.CacheParams(chunk=100, ctx_keep=4, capacity=10)
    ctx = np.arange(1, 33, dtype=np.uint32)[None, :].copy()
    st = a1.State([4], cp, key_len=2, missing_capacity=16)
    a1.cache_update(st, ctx, [4], [6], [1])     # entry of 5 tokens: 6 words
    a1.cache_update(st, ctx, [6], [8], [1])     # 5 more tokens: 11 > 10 words, dropped
    assert st.n_seq(0) == 1 and st.dropped[0] == 1 and st.words[0] == 6
    a1.cache_update(st, ctx, [8], [9], [0])     # nothing
    assert st.n_seq(0) == 1


def test_trajectory_invariants(orc, a1):
    import paper_2502_17139_gb300.synth as syn
    rng = np.random.default_rng(1234)
    vocab = 64
    corpora = [syn.zipf_tokens(rng, 4000, 1.1, vocab=vocab).astype(np.uint32),
               syn.zipf_tokens(rng, 2000, 1.1, vocab=vocab).astype(np.uint32)]
    B, steps, stride = 6, 30, 256
    ctx = np.zeros((B, stride), np.uint32)
    ctx[:, :40] = rng.integers(0, vocab, (B, 40))
    cl = np.full(B, 40, np.int32)
    p = dict(n_max=8, n_min=2, top_k=4, draft_len=4, max_occ=64, node_budget=16, n_pad=16)
    plen = rng.integers(0, 5, (steps, B)).astype(np.int32)
    rtok = rng.integers(0, vocab, (steps, B, 16)).astype(np.uint32)
    cp = a1.CacheParams(min_size=4, chunk=5, ctx_keep=8, capacity=4096)
    seen = []

    def on_step(st_i, res, code, tr, am, ac):
        seen.append([state_ref[0].n_seq(b) for b in range(B)])

    state_ref = [a1.State(cl, cp, 2, 256)]
    hist, ctx2, cl2, kv, st = a1.step_loop(corpora, ctx, cl, steps, p, cp, plen, rtok, [1, 1], 1, vocab, 256,
                                           state=state_ref[0], on_step=on_step)
    codes = np.stack(hist["code"])
    assert (codes == a1.SERVE_CACHE).any(), "the CACHE never served: scenario too weak"
    for t in range(steps):
        for b in range(B):
            if codes[t, b] == a1.SERVE_CACHE:
                assert seen[t][b] >= cp.min_size
    for b in range(B):
        assert st.words[b] == sum(len(e) + 1 for e in st.entries[b])
        pieces = (st.out_mark[b] - 40) // cp.chunk
        assert st.out_mark[b] - 40 == pieces * cp.chunk and cl2[b] - st.out_mark[b] < cp.chunk
        # every piece of the output appears among the entries
        stored = {tuple(e.tolist()) for e in st.entries[b]}
        for i in range(pieces):
            s0 = 40 + i * cp.chunk
            assert tuple(ctx2[b, s0:s0 + cp.chunk].tolist()) in stored


def test_missing_table_split_changes_no_draft(orc, a1):
    """A missing table per slice of the sequences (the step executor keeps one
    per sub-batch) instead of one for the batch changes no draft: M only
    skips datastore searches that would find nothing.  The oracle's Algorithm
    1 over the whole batch and over each slice on its own give the same
    trees, acceptance, contexts and CACHE stores; the search states differ
    only where the whole batch's M skipped a query that its slice searched,
    and that search found nothing."""
    import paper_2502_17139_gb300.synth as syn
    rng = np.random.default_rng(4321)
    vocab = 64
    corpora = [syn.zipf_tokens(rng, 400, 1.1, vocab=vocab).astype(np.uint32),
               syn.zipf_tokens(rng, 200, 1.1, vocab=vocab).astype(np.uint32)]
    B, H, steps, stride = 16, 8, 40, 256
    ctx = np.zeros((B, stride), np.uint32)
    ctx[:, :40] = rng.integers(0, vocab, (B, 40))
    cl = np.full(B, 40, np.int32)
    p = dict(n_max=8, n_min=2, top_k=4, draft_len=4, max_occ=64, node_budget=16, n_pad=16)
    plen = rng.integers(0, 3, (steps, B)).astype(np.int32)
    rtok = rng.integers(0, vocab, (steps, B, 16)).astype(np.uint32)
    cp = a1.CacheParams(min_size=50, chunk=5, ctx_keep=8, capacity=4096)  # M at work, the CACHE inactive

    def run(sl):
        return a1.step_loop(corpora, ctx[sl], cl[sl], steps, p, cp, plen[:, sl], rtok[:, sl], [1, 1], 1, vocab, 1024)

    whole = run(slice(0, B))
    parts = [run(slice(0, H)), run(slice(H, B))]
    for k in ("acc_len", "bonus", "n_nodes"):
        got = np.concatenate([np.stack(pt[0][k]) for pt in parts], axis=1)
        assert np.array_equal(np.stack(whole[0][k]), got), k
    assert np.array_equal(whole[1], np.concatenate([pt[1] for pt in parts]))
    assert np.array_equal(whole[2], np.concatenate([pt[2] for pt in parts]))
    st_w = whole[4]
    for h, pt in enumerate(parts):
        for i, e in enumerate(pt[4].entries):
            assert [x.tolist() for x in e] == [x.tolist() for x in st_w.entries[H * h + i]]
    code_w = np.stack(whole[0]["code"])
    code_p = np.concatenate([np.stack(pt[0]["code"]) for pt in parts], axis=1)
    nd_p = np.concatenate([np.stack(pt[0]["n_drafts"]) for pt in parts], axis=2)  # [steps, S + 1, B]
    diff = code_w != code_p
    assert diff.any(), "the whole batch's M never skipped a query its slice searched: scenario too weak"
    assert (code_w[diff] == a1.SKIP_MISSING).all() and (code_p[diff] == a1.SERVE_DATASTORE).all()
    assert (nd_p[:, :2][np.broadcast_to(diff[:, None, :], nd_p[:, :2].shape)] == 0).all()
