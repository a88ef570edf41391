"""Pins for the oracle's suffix array (O1) and retrieval (O2-O4).

The oracle is checked against things other than itself: textbook suffix
arrays, brute-force sorting of Python lists, brute-force substring search on
tiny corpora with small vocabularies (so long repeats and ties occur), and
hand-worked cases in tests/golden/retrieve_handmade.json.
"""
import collections
import json
import os

import numpy as np
import pytest

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
PAD = 0xFFFFFFFF


def brute_sa(T):
    return sorted(range(len(T)), key=lambda i: list(T[i:]))


def test_sa_textbook_banana(orc):
    # "banana" with a=0, b=1, n=2: a, ana, anana, banana, na, nana
    T = np.array([1, 0, 2, 0, 2, 0], np.uint32)
    assert orc.suffix_array(T).tolist() == [5, 3, 1, 0, 4, 2]


def test_sa_constant_string_closed_form(orc):
    # all suffixes of a^n are prefixes of each other: shortest first
    for n in (1, 2, 7, 300):
        T = np.full(n, 4, np.uint32)
        assert orc.suffix_array(T).tolist() == list(range(n - 1, -1, -1))


@pytest.mark.parametrize("seed", range(12))
def test_sa_matches_brute_force(orc, seed):
    rng = np.random.default_rng(seed)
    n = int(rng.integers(1, 1500))
    vocab = int(rng.integers(2, 9))
    T = rng.integers(0, vocab, n).astype(np.uint32)
    if seed % 3 == 0 and n > 40:  # plant a long repeat
        T[n // 2:n // 2 + 20] = T[:20]
    assert orc.suffix_array(T, nthreads=1 + seed % 4).tolist() == brute_sa(T.tolist())


def test_sa_parallel_merge_path(orc):
    rng = np.random.default_rng(5)
    T = rng.integers(0, 3, 200_000).astype(np.uint32)
    sa1 = orc.suffix_array(T, nthreads=1)
    sa8 = orc.suffix_array(T, nthreads=8)
    assert np.array_equal(sa1, sa8)
    assert orc.sa_certificate(T, sa8) == -1


@pytest.mark.parametrize("seed", range(6))
def test_lcp_brute_force(orc, seed):
    rng = np.random.default_rng(40 + seed)
    n = int(rng.integers(1, 800))
    T = rng.integers(0, 1 + seed % 3, n).astype(np.uint32)  # tiny vocabularies: long common prefixes
    sa = orc.suffix_array(T)
    cap = [255, 5, 255, 1, 40, 255][seed]
    got = orc.lcp(T, sa, cap)
    Tl = T.tolist()
    assert got[0] == 0
    for j in range(1, n):
        a, b = Tl[sa[j - 1]:], Tl[sa[j]:]
        l = 0
        while l < min(len(a), len(b)) and a[l] == b[l]:
            l += 1
        assert got[j] == min(l, cap)


def test_sa_certificate_rejects(orc):
    rng = np.random.default_rng(1)
    T = rng.integers(0, 4, 500).astype(np.uint32)
    sa = orc.suffix_array(T)
    assert orc.sa_certificate(T, sa) == -1
    bad = sa.copy()
    bad[10], bad[11] = bad[11], bad[10]
    assert orc.sa_certificate(T, bad) == 10
    dup = sa.copy()
    dup[3] = dup[4]
    assert orc.sa_certificate(T, dup) == len(T)


@pytest.mark.parametrize("seed", range(5))
def test_bucket_brute(orc, seed):
    rng = np.random.default_rng(seed)
    vocab = 9
    T = rng.integers(0, vocab - 2, 400).astype(np.uint32)  # some ids never occur
    sa = orc.suffix_array(T)
    bk = orc.bucket(T, sa, vocab)
    first = [T[i] for i in sa]
    for v in range(vocab + 1):
        exp = next((j for j, t in enumerate(first) if t >= v), len(T))
        assert bk[v] == exp


def _run_case(orc, case):
    T = np.array(case["T"], np.uint32)
    ctx = np.array([case["ctx"]], np.uint32)
    return orc.retrieve(T, ctx, np.array([len(case["ctx"])], np.int32), case["n_max"], case["n_min"],
                        case["top_k"], case["d"], case["max_occ"])


def test_retrieve_handmade_golden(orc):
    with open(os.path.join(GOLDEN, "retrieve_handmade.json")) as f:
        g = json.load(f)
    for case in g["cases"]:
        r = _run_case(orc, case)
        assert r["drafts"][0].tolist() == case["drafts"], case["why"]
        assert r["draft_len"][0].tolist() == case["draft_len"], case["why"]
        assert r["count"][0].tolist() == case["count"], case["why"]
        assert int(r["n_drafts"][0]) == case["n_drafts"], case["why"]
        assert int(r["match_len"][0]) == case["match_len"], case["why"]


def brute_retrieve(T, c, n_max, n_min, k, d, max_occ):
    """Substring search straight from the definition, then Counter ranking."""
    N, m = len(T), len(c)
    for n in range(min(n_max, m), n_min - 1, -1):
        q = c[m - n:]
        occ = [p for p in range(n, N) if T[p - n:p] == q]  # p <= N-1
        if occ:
            break
    else:
        return [], [], 0
    conts = [tuple(T[p:p + d]) for p in occ]
    if max_occ and len(conts) > max_occ:
        conts = sorted(conts)[:max_occ]
    cnt = collections.Counter(conts)
    ranked = sorted(cnt.items(), key=lambda kv: (-kv[1], kv[0]))[:k]
    return [list(s) for s, _ in ranked], [v for _, v in ranked], n


@pytest.mark.parametrize("seed", range(16))
def test_retrieve_matches_brute_force(orc, seed):
    rng = np.random.default_rng(100 + seed)
    N = int(rng.integers(5, 1200))
    vocab = int(rng.integers(2, 7))
    T = rng.integers(0, vocab, N).astype(np.uint32)
    B = 12
    m = 10
    ctx = rng.integers(0, vocab, (B, m)).astype(np.uint32)
    for b in range(B // 2):  # half the contexts end with a corpus substring
        L = int(rng.integers(1, min(m, N) + 1))
        p = int(rng.integers(0, N - L + 1))
        ctx[b, m - L:] = T[p:p + L]
    ctx_len = rng.integers(1, m + 1, B).astype(np.int32)
    for b in range(B):  # ctx_len shorter than the row: keep the copied tail at the end
        ctx[b, :ctx_len[b]] = ctx[b, m - ctx_len[b]:].copy()
    n_max, n_min = int(rng.integers(1, 9)), 1 + seed % 2
    n_min = min(n_min, n_max)
    k, d = int(rng.integers(1, 9)), int(rng.integers(1, 6))
    max_occ = [0, 1, 3, 50][seed % 4]
    r = orc.retrieve(T, ctx, ctx_len, n_max, n_min, k, d, max_occ)
    Tl = T.tolist()
    for b in range(B):
        c = ctx[b, :ctx_len[b]].tolist()
        drafts, counts, n = brute_retrieve(Tl, c, n_max, n_min, k, d, max_occ)
        assert int(r["match_len"][b]) == n
        assert int(r["n_drafts"][b]) == len(drafts)
        for t in range(k):
            if t < len(drafts):
                L = len(drafts[t])
                assert r["draft_len"][b, t] == L
                assert r["drafts"][b, t, :L].tolist() == drafts[t]
                assert (r["drafts"][b, t, L:] == PAD).all()
                assert r["count"][b, t] == counts[t]
            else:
                assert r["draft_len"][b, t] == 0 and r["count"][b, t] == 0
                assert (r["drafts"][b, t] == PAD).all()
        if max_occ:
            assert int(r["count"][b].sum()) <= max_occ


def test_retrieve_drafts_are_corpus_continuations(orc):
    """Every returned draft follows an occurrence of the matched suffix."""
    import paper_2502_17139_gb300.synth as synth
    rng = synth.rng_for(90)
    T, _ = synth.make_corpus(rng, 20000, 1.1, 64, n_grams=40, len_range=(8, 20))
    ctx, cl, _ = synth.make_contexts(rng, 16, 24, 10, [T, None], [0.75, 0.25], 1.1, 64)
    r = orc.retrieve(T, ctx, cl, 8, 2, 6, 5, 64)
    Tb = T.tolist()
    for b in range(16):
        n = int(r["match_len"][b])
        if n == 0:
            continue
        q = ctx[b, cl[b] - n:cl[b]].tolist()
        occ = {p for p in range(n, len(Tb)) if Tb[p - n:p] == q}
        for t in range(int(r["n_drafts"][b])):
            L = int(r["draft_len"][b, t])
            u = r["drafts"][b, t, :L].tolist()
            assert any(Tb[p:p + L] == u and (L == 5 or p + L == len(Tb)) for p in occ)
