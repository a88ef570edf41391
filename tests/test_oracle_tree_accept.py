"""Pins for the oracle's draft tree (O5), tree mask, acceptance (O7), cache
append (O8) and the synthetic target model.

Checks: hand-worked trees (tests/golden/tree_handmade.json), trie invariants
on random draft sets, a brute-force prefix enumeration for the budgeted
selection, acceptance against a token-by-token autoregressive comparison over
every root-to-leaf path, and the cache append as a plain copy.
"""
import itertools
import json
import os

import numpy as np
import pytest

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
PAD = 0xFFFFFFFF


def _src(drafts, lens, counts, k, d):
    B = 1
    out = dict(drafts=np.full((B, k, d), PAD, np.uint32), draft_len=np.zeros((B, k), np.int32),
               count=np.zeros((B, k), np.uint32), n_drafts=np.array([len(drafts)], np.int32),
               match_len=np.array([1], np.int32))
    for t, (u, L, c) in enumerate(zip(drafts, lens, counts)):
        out["drafts"][0, t, :L] = u[:L]
        out["draft_len"][0, t] = L
        out["count"][0, t] = c
    return out


def _mask_bits(row):
    bits = []
    for w, word in enumerate(row.tolist()):
        for j in range(64):
            if (int(word) >> j) & 1:
                bits.append(64 * w + j)
    return bits


def test_tree_handmade_golden(orc):
    with open(os.path.join(GOLDEN, "tree_handmade.json")) as f:
        g = json.load(f)
    r = _src(g["src_r"]["drafts"], [3, 3], g["src_r"]["count"], 4, 3)
    c = _src(g["src_c"]["drafts"], g["src_c"]["len"], g["src_c"]["count"], 4, 3)
    for case in g["cases"]:
        t = orc.build_tree([r, c], case["weights"], [9], [100], case["budget"], 64)
        n = int(t["n_nodes"][0])
        assert n == len(case["tok"]), case["why"]
        assert t["tok"][0, :n].tolist() == case["tok"], case["why"]
        assert t["parent"][0, :n].tolist() == case["parent"], case["why"]
        assert t["depth"][0, :n].tolist() == case["depth"], case["why"]
        assert t["pos"][0, :n].tolist() == [100 + x for x in case["depth"]], case["why"]
        for i in range(n):
            assert _mask_bits(t["mask"][0, i]) == case["mask_rows"][i], case["why"]
        assert (t["tok"][0, n:] == PAD).all() and (t["parent"][0, n:] == -1).all()
        assert (t["mask"][0, n:] == 0).all()


def _random_sources(rng, S, B, k, d, vocab):
    res = []
    for s in range(S):
        o = dict(drafts=np.full((B, k, d), PAD, np.uint32), draft_len=np.zeros((B, k), np.int32),
                 count=np.zeros((B, k), np.uint32), n_drafts=np.zeros(B, np.int32), match_len=np.ones(B, np.int32))
        for b in range(B):
            nd = int(rng.integers(0, k + 1))
            seen = set()
            t = 0
            while t < nd:
                L = int(rng.integers(1, d + 1))
                u = tuple(int(x) for x in rng.integers(0, vocab, L))
                if u in seen:
                    continue
                seen.add(u)
                o["drafts"][b, t, :L] = u
                o["draft_len"][b, t] = L
                o["count"][b, t] = int(rng.integers(1, 20))
                t += 1
            o["n_drafts"][b] = nd
        res.append(o)
    return res


def _paths(tok, parent, n):
    paths = []
    for i in range(n):
        p, v = [], i
        while v > 0:
            p.append(int(tok[v]))
            v = int(parent[v])
        paths.append(tuple(reversed(p)))
    return paths


@pytest.mark.parametrize("seed", range(10))
def test_tree_invariants_and_selection(orc, seed):
    rng = np.random.default_rng(7 + seed)
    S, B, k, d = 1 + seed % 2, 6, 12, 6
    vocab = [2, 3, 50][seed % 3]
    res = _random_sources(rng, S, B, k, d, vocab)
    weights = rng.integers(1, 4, S).astype(np.uint32)
    budget = int(rng.integers(1, 65))
    n_pad = 64 if seed % 2 else 128
    root = rng.integers(0, vocab, B).astype(np.uint32)
    kvl = rng.integers(0, 1000, B).astype(np.int32)
    t = orc.build_tree(res, weights, root, kvl, budget, n_pad)
    for b in range(B):
        n = int(t["n_nodes"][b])
        tok, par, dep = t["tok"][b], t["parent"][b], t["depth"][b]
        # brute force: every distinct prefix with its weight
        w = {}
        for s in range(S):
            for q in range(int(res[s]["n_drafts"][b])):
                L = int(res[s]["draft_len"][b, q])
                u = tuple(res[s]["drafts"][b, q, :L].tolist())
                w[u] = w.get(u, 0) + int(weights[s]) * int(res[s]["count"][b, q])
        W = {}
        for u, x in w.items():
            for l in range(1, len(u) + 1):
                W[u[:l]] = W.get(u[:l], 0) + x
        ranked = sorted(W, key=lambda p: (-W[p], len(p), p))[:budget - 1]
        assert n == 1 + len(ranked) <= budget
        paths = _paths(tok, par, n)
        assert set(paths[1:]) == set(ranked)
        assert paths == sorted(paths)  # preorder == lexicographic order of paths
        assert tok[0] == root[b] and par[0] == -1 and dep[0] == 0
        for i in range(1, n):
            assert 0 <= par[i] < i
            assert dep[i] == dep[par[i]] + 1
            assert t["pos"][b, i] == kvl[b] + dep[i]
        for i in range(n):
            bits = _mask_bits(t["mask"][b, i])
            assert len(bits) == dep[i] + 1
            anc, v = [], i
            while v >= 0:
                anc.append(v)
                v = int(par[v]) if v > 0 else -1
            assert bits == sorted(anc)
        kids = {}
        for i in range(1, n):
            kids.setdefault(int(par[i]), []).append(int(tok[i]))
        for v in kids.values():
            assert len(v) == len(set(v)) and v == sorted(v)
        # every root-to-leaf path is a prefix of some draft
        leaves = [i for i in range(n) if i not in kids]
        for i in leaves:
            if i == 0:
                continue
            assert any(u[:len(paths[i])] == paths[i] for u in w)
        if budget - 1 >= len(W) and not any(a != b2 and b2[:len(a)] == a for a in w for b2 in w):
            assert {paths[i] for i in leaves if i > 0} == set(w)


def test_tree_mask_from_parents(orc):
    import paper_2502_17139_gb300.synth as synth
    rng = synth.rng_for(91)
    B, n_pad = 4, 128
    par = np.full((B, n_pad), -1, np.int32)
    nn = np.array([1, 17, 64, 128], np.int32)
    for b in range(B):
        _, p = synth.random_tree(rng, int(nn[b]), 10, 4, 100)
        par[b, :nn[b]] = p
    m = orc.tree_mask(par, nn, np.array([5, 6, 7, 8], np.int32), n_pad)
    for b in range(B):
        for i in range(nn[b]):
            anc, v = [], i
            while v >= 0:
                anc.append(v)
                v = int(par[b, v]) if v > 0 else -1
            assert _mask_bits(m["mask"][b, i]) == sorted(anc)
            assert m["depth"][b, i] == len(anc) - 1
            assert m["pos"][b, i] == 5 + b + len(anc) - 1
        assert (m["mask"][b, nn[b]:] == 0).all()


def _autoregressive_accept(tok, par, n, argmax):
    """Token-by-token comparison along every root-to-leaf path; the longest
    run of agreements from the root wins."""
    kids = {}
    for i in range(1, n):
        kids.setdefault(int(par[i]), []).append(i)
    best_len, best_path = 0, [0]
    for leaf in range(n):
        if leaf in kids:
            continue
        path, v = [], leaf
        while v >= 0:
            path.append(v)
            v = int(par[v]) if v > 0 else -1
        path.reverse()
        L = 0
        while L + 1 < len(path) and int(tok[path[L + 1]]) == int(argmax[path[L]]):
            L += 1
        if L > best_len:
            best_len, best_path = L, path[:L + 1]
    return best_len, best_path, int(argmax[best_path[-1]])


@pytest.mark.parametrize("seed", range(6))
def test_accept_equals_autoregressive(orc, seed):
    import paper_2502_17139_gb300.synth as synth
    rng = synth.rng_for(92, seed)
    B, n_pad, vocab = 24, 64, [3, 8, 32256][seed % 3]
    tok = np.full((B, n_pad), PAD, np.uint32)
    par = np.full((B, n_pad), -1, np.int32)
    nn = rng.integers(1, n_pad + 1, B).astype(np.int32)
    for b in range(B):
        t, p = synth.random_tree(rng, int(nn[b]), 10, min(4, vocab), vocab)
        tok[b, :nn[b]], par[b, :nn[b]] = t, p
    # predictions: mostly agree with some child, sometimes random
    am = rng.integers(0, vocab, (B, n_pad)).astype(np.uint32)
    for b in range(B):
        for i in range(nn[b]):
            ch = [j for j in range(1, nn[b]) if par[b, j] == i]
            if ch and rng.random() < 0.8:
                am[b, i] = tok[b, ch[int(rng.integers(0, len(ch)))]]
    r = orc.accept(tok, par, nn, am, 12)
    for b in range(B):
        L, path, bonus = _autoregressive_accept(tok[b], par[b], nn[b], am[b])
        assert r["acc_len"][b] == L
        assert r["path"][b, :L + 1].tolist() == path
        assert (r["path"][b, L + 1:] == -1).all()
        assert r["bonus"][b] == bonus


def test_synth_argmax_rule(orc):
    import paper_2502_17139_gb300.synth as synth
    rng = synth.rng_for(93)
    B, n_pad, vocab = 16, 64, 5
    tok = np.full((B, n_pad), PAD, np.uint32)
    par = np.full((B, n_pad), -1, np.int32)
    nn = rng.integers(1, n_pad + 1, B).astype(np.int32)
    for b in range(B):
        t, p = synth.random_tree(rng, int(nn[b]), 10, 4, vocab)
        tok[b, :nn[b]], par[b, :nn[b]] = t, p
    plen, rtok = synth.argmax_draws(rng, B, n_pad, vocab)
    am = orc.synth_argmax(tok, par, nn, plen, rtok, vocab)
    r = orc.accept(tok, par, nn, am, 12)
    for b in range(B):
        chain = [0]
        while True:
            ch = [j for j in range(1, nn[b]) if par[b, j] == chain[-1]]
            if not ch:
                break
            chain.append(min(ch))
        assert r["acc_len"][b] == min(int(plen[b]), len(chain) - 1)
        for i in range(nn[b]):
            ch_tok = {int(tok[b, j]) for j in range(1, nn[b]) if par[b, j] == i}
            on_prefix = i in chain[:int(plen[b])] and chain.index(i) + 1 < len(chain)
            if on_prefix:
                assert am[b, i] == tok[b, chain[chain.index(i) + 1]]
            else:
                assert int(am[b, i]) not in ch_tok


def test_kv_append_is_a_copy(orc):
    rng = np.random.default_rng(3)
    B, n_pad, Hkv, D, cap, stride = 3, 8, 2, 16, 40, 30
    k_tree = rng.integers(0, 65535, (B, Hkv, n_pad, D)).astype(np.uint16)
    v_tree = rng.integers(0, 65535, (B, Hkv, n_pad, D)).astype(np.uint16)
    k_cache = rng.integers(0, 65535, (B, Hkv, cap, D)).astype(np.uint16)
    v_cache = k_cache.copy()
    k0, v0 = k_cache.copy(), v_cache.copy()
    tok = rng.integers(0, 100, (B, n_pad)).astype(np.uint32)
    path = np.array([[0, 2, 5, -1], [0, -1, -1, -1], [0, 1, 3, 7]], np.int32)
    acc = np.array([2, 0, 3], np.int32)
    bonus = np.array([11, 12, 13], np.uint32)
    kvl = np.array([0, 10, 36], np.int32)
    ctx = rng.integers(0, 100, (B, stride)).astype(np.uint32)
    c0 = ctx.copy()
    cl = np.array([5, 6, 26], np.int32)
    kvo, clo, root = orc.kv_append(path, acc, bonus, tok, k_tree, v_tree, k_cache, v_cache, kvl, ctx, cl)
    for b in range(B):
        a = acc[b]
        for t in range(a + 1):
            assert np.array_equal(k_cache[b, :, kvl[b] + t], k_tree[b, :, path[b, t]])
            assert np.array_equal(v_cache[b, :, kvl[b] + t], v_tree[b, :, path[b, t]])
        untouched = [j for j in range(cap) if not kvl[b] <= j <= kvl[b] + a]
        assert np.array_equal(k_cache[b, :, untouched], k0[b, :, untouched])
        assert np.array_equal(v_cache[b, :, untouched], v0[b, :, untouched])
        assert kvo[b] == kvl[b] + a + 1 and clo[b] == cl[b] + a + 1 and root[b] == bonus[b]
        assert ctx[b, cl[b]:cl[b] + a].tolist() == [tok[b, path[b, t + 1]] for t in range(a)]
        assert ctx[b, cl[b] + a] == bonus[b]
        assert np.array_equal(ctx[b, :cl[b]], c0[b, :cl[b]])
