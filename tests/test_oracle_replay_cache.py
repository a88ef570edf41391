"""Pin for the oracle's context-keyed replay cache (O9: ``oracle.cache_key``
and the served-entry logic of ``oracle.step_loop``).

The cache is a reading of the benchmark workload, not a step the paper
defines, so nothing in the paper fixes its values.  What the mathematics
fixes is this: retrieval (Section III-A) reads only the last min(n_max, m)
tokens of a context of m tokens, and the datastores are static.  So a result
the cache serves must equal a fresh retrieval of the context it is served
for, and a trajectory that replays cached results must equal the trajectory
that retrieves every time.  Both are checked here with contexts shorter than
n_max (the key then holds fewer tokens) and a tiny vocabulary, so that keys
recur across sequences and steps and entries are overwritten.

Two planted mistakes, each a plausible slip in the key, must fail the pin:
a key that always slices n_max tokens (so short contexts collide), and a key
shifted one token back (contexts differing in their last token collide).
"""
import numpy as np
import pytest

import paper_2502_17139_gb300.synth as synth

VOCAB = 3
P = dict(n_max=4, n_min=2, top_k=4, draft_len=4, max_occ=0, node_budget=16, n_pad=16)


def workload(seed, B=12, steps=14):
    rng = synth.rng_for(80, seed)
    Tr = rng.integers(0, VOCAB, 3000).astype(np.uint32)
    Tc = rng.integers(0, VOCAB, 7000).astype(np.uint32)
    stride = 5 + (steps + 1) * (P["draft_len"] + 1)
    ctx = np.zeros((B, stride), np.uint32)
    cl = rng.integers(1, 6, B).astype(np.int32)       # 1..5 tokens: most shorter than n_max
    for b in range(B):
        ctx[b, :cl[b]] = rng.integers(0, VOCAB, cl[b])
    hits = synth.cache_hit_pattern(rng, steps, B, 0.7)
    plen = np.stack([synth.argmax_draws(rng, B, P["n_pad"], VOCAB, plen_max=3)[0] for _ in range(steps)])
    rtok = np.stack([synth.argmax_draws(rng, B, P["n_pad"], VOCAB)[1] for _ in range(steps)])
    return [Tr, Tc], ctx, cl, steps, hits, plen, rtok


def run_checked(orc, corpora, ctx, cl, steps, hits, plen, rtok, cache):
    """Runs the oracle's step loop and, at every step, retrieves every
    query's context afresh.  The contexts are followed here independently of
    the loop: each step appends the accepted path's tokens and the bonus.
    Returns (history, final ctx, final ctx_len, number of served results
    that differ from a fresh retrieval, served results from short contexts)."""
    B = ctx.shape[0]
    my_ctx = ctx.copy()
    my_cl = cl.copy()
    bad = [0]
    short_served = [0]
    served_now = {}

    def on_step(st, res, tr, am, ac):
        fresh = [orc.retrieve(T, my_ctx, my_cl, P["n_max"], P["n_min"], P["top_k"], P["draft_len"], P["max_occ"])
                 for T in corpora]
        keys = [orc.cache_key(my_ctx[b], my_cl[b], P["n_max"]) for b in range(B)]
        for b in range(B):
            same = all(np.array_equal(res[s][name][b], fresh[s][name][b]) for s in range(len(corpora))
                       for name in fresh[s])
            if not same:
                bad[0] += 1
            if hits[st, b] and keys[b] in served_now and my_cl[b] < P["n_max"]:
                short_served[0] += 1
        for b in range(B):
            a = int(ac["acc_len"][b])
            for t in range(a):
                my_ctx[b, my_cl[b] + t] = tr["tok"][b, ac["path"][b, t + 1]]
            my_ctx[b, my_cl[b] + a] = ac["bonus"][b]
            my_cl[b] += a + 1

    served_now.update(cache)
    hist, r_ctx, r_cl, _ = orc.step_loop(corpora, ctx, cl, steps, P, hits, plen, rtok, [1, 1], VOCAB,
                                         cache=cache, on_step=on_step)
    assert np.array_equal(r_ctx, my_ctx) and np.array_equal(r_cl, my_cl)
    return hist, r_ctx, r_cl, bad[0], short_served[0]


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_served_results_equal_fresh_retrieval(orc, seed):
    corpora, ctx, cl, steps, hits, plen, rtok = workload(seed)
    no_hits = np.zeros_like(hits)
    cache = {}
    h0, c0, l0, bad0, _ = run_checked(orc, corpora, ctx, cl, steps, no_hits, plen, rtok, cache)  # recording
    assert bad0 == 0
    assert sum(h.sum() for h in h0["hit"]) == 0
    h1, c1, l1, bad1, short = run_checked(orc, corpora, ctx, cl, steps, hits, plen, rtok, cache)  # replay
    assert bad1 == 0
    served = sum(int(h.sum()) for h in h1["hit"])
    assert served > 0.5 * hits.sum()      # the cache served most of the queries that asked for it
    assert short > 0                      # including contexts shorter than n_max
    # replaying cached results changes no outcome
    for name in ("acc_len", "bonus", "n_nodes"):
        for a, b in zip(h0[name], h1[name]):
            assert np.array_equal(a, b), name
    assert np.array_equal(c0, c1) and np.array_equal(l0, l1)
    # the tiny vocabulary makes keys recur: fewer distinct keys than queries
    assert len(cache) < ctx.shape[0] * steps
    assert np.mean([n.mean() for n in h1["n_nodes"]]) > 3


def test_one_pass_hits_on_recurring_keys(orc):
    """Without a recording pass: a query whose key another query of an
    earlier step inserted is served from that entry, and still equals a
    fresh retrieval."""
    corpora, ctx, cl, steps, hits, plen, rtok = workload(5, B=16, steps=12)
    cache = {}
    h, _, _, bad, _ = run_checked(orc, corpora, ctx, cl, steps, np.ones_like(hits), plen, rtok, cache)
    assert bad == 0
    assert sum(int(x.sum()) for x in h["hit"]) > 0


def _key_always_n_max(ctx_row, ctx_len, n_max):
    m = int(ctx_len)
    return bytes(np.int32(n_max).tobytes()) + ctx_row[m - n_max:m].astype(np.uint32).tobytes()


def _key_shifted(ctx_row, ctx_len, n_max):
    m = int(ctx_len)
    k = min(n_max, m)
    return bytes(np.int32(k).tobytes()) + ctx_row[max(0, m - k - 1):m - 1].astype(np.uint32).tobytes()


@pytest.mark.parametrize("wrong_key", [_key_always_n_max, _key_shifted])
def test_planted_key_mistakes_fail_the_pin(orc, monkeypatch, wrong_key):
    monkeypatch.setattr(orc, "cache_key", wrong_key)
    total_bad = 0
    for seed in (0, 1, 2):
        corpora, ctx, cl, steps, hits, plen, rtok = workload(seed)
        cache = {}
        run_checked(orc, corpora, ctx, cl, steps, np.zeros_like(hits), plen, rtok, cache)
        total_bad += run_checked(orc, corpora, ctx, cl, steps, hits, plen, rtok, cache)[3]
    assert total_bad > 0
