"""Algorithm 1 (Section IV-C) with the CACHE of Section IV-B and the missing
table M, stated as plain Python over the oracle's searches.

TEST INFRASTRUCTURE ONLY: imported by tests/ and by the CPU-baseline leg of
bench.py, never by the product package.  It shares no code with the CUDA
path; the stored sequences live here as Python lists of arrays, not in the
GPU's flat layout.

What a step does for every sequence b of a batch (Algorithm 1):
  1. when the CACHE of b holds at least l sequences, search it (O11);
  2. when the CACHE was not searched or found nothing: if the context's key
     is in M, skip retrieval; otherwise search every datastore source (O2-O4);
  3. when nothing was retrieved, add the key to M; otherwise the CACHE is
     updated after verification (step 5);
  4. the draft tree, the target model and acceptance run as in the plain loop;
  5. CACHE update: the verified retrieval (context + accepted draft tokens)
     and every completed 20-token piece of the model's output are stored.

Readings taken where the paper is silent, ambiguous or at odds with itself:
  R1 batch: every sequence has a CACHE of its own (the paper decodes one
     sample at a time and fills the CACHE from that sample's own context and
     output); M is one table for the whole batch (the datastore is static and
     shared, so a suffix that fails for one sequence fails for all).  Inside
     one step every sequence consults M as it was when the step started; the
     step's additions are applied afterwards in sequence order.
  R2 activation: the CACHE is searched when it holds l or more sequences
     (Algorithm 1's test; the prose says "exceeds").  l = 50 (Section V-C).
  R3 the key of M is the last n_min context tokens.  A match of length n
     implies a match of every shorter length at the same position, so
     retrieval from a static datastore returns nothing exactly when those
     n_min tokens never occur followed by a token in any source: the key is
     safe and it is the shortest key that is.  A context shorter than n_min
     has no key: it is never skipped and never added.
  R4 skip tokens are out (they need a tokenizer's notion of line starts), so
     no position is a skip token; the datastore is searched whenever the key
     is not in M (the printed algorithm nests the search under the skip-token
     branch, the prose says retrieval proceeds whenever the strategy allows).
  R5 the verified retrieval stored after a step with acc_len >= 1 accepted
     draft tokens is the last ctx_keep context tokens before the step
     followed by the accepted draft tokens (ctx_keep = n_max by default: no
     retrieval pattern is longer).  The bonus token is the model's own output
     and reaches the CACHE through the output pieces.
  R6 output pieces: the tokens appended to the context after the prompt
     (accepted draft tokens and bonus tokens) are cut into consecutive pieces
     of `chunk` = 20 tokens (Section V-C); a piece is stored once complete.
     In one step the verified retrieval is stored first, then the pieces.
  R7 capacity: a CACHE holds at most `capacity` words, an entry of length L
     costing L + 1 (the GPU layout puts a separator after each entry); an
     entry that does not fit is dropped and counted.  M holds at most
     missing_capacity / 2 keys; a new key that does not fit is dropped and
     counted once per step.
  R8 the tree is built from S + 1 result slots: the datastore sources, then
     the CACHE (weight cache_weight).  When the CACHE serves, the datastore
     slots are empty, and otherwise the CACHE slot is, so the CACHE weight
     never competes with the datastore weights of Eq. 3.
  R9 a step whose append did not happen (the context or the KV cache would
     overflow, so the context length did not change) stores no verified
     retrieval.
"""
from __future__ import annotations

import ctypes as C
import dataclasses

import numpy as np

from . import oracle as O

SERVE_DATASTORE, SERVE_CACHE, SKIP_MISSING = 0, 1, 2
RESULT_FIELDS = ("drafts", "draft_len", "count", "n_drafts", "match_len")


@dataclasses.dataclass
class CacheParams:
    min_size: int = 50     # l, Section V-C
    chunk: int = 20        # output pieces, Section V-C
    ctx_keep: int = 16     # R5
    capacity: int = 8192   # words per sequence, R7


def empty_results(B, top_k, d):
    return dict(drafts=np.full((B, top_k, d), O.PAD, np.uint32), draft_len=np.zeros((B, top_k), np.int32),
                count=np.zeros((B, top_k), np.uint32), n_drafts=np.zeros(B, np.int32),
                match_len=np.zeros(B, np.int32))


def cache_search(entries, ctx, ctx_len, n_max, n_min, top_k, d, max_occ, nthreads: int = 0):
    """O11 for a batch: entries[b] is the list of stored sequences of query b."""
    ctx = O._c(ctx, np.uint32)
    ctx_len = O._c(ctx_len, np.int32)
    B, stride = ctx.shape
    assert len(entries) == B
    flat = [np.asarray(e, np.uint32) for es in entries for e in es]
    eoff = np.zeros(len(flat) + 1, np.int64)
    if flat:
        eoff[1:] = np.cumsum([len(e) for e in flat])
    tok = np.concatenate(flat).astype(np.uint32) if flat and eoff[-1] > 0 else np.zeros(1, np.uint32)
    qent = np.zeros(B + 1, np.int64)
    qent[1:] = np.cumsum([len(es) for es in entries])
    out = empty_results(B, top_k, d)
    rc = O.lib().orc_cache_search(O._p(tok), O._p(eoff), O._p(qent), O._p(ctx), C.c_int(stride), O._p(ctx_len),
                                  C.c_int(B), C.c_int(n_max), C.c_int(n_min), C.c_int(top_k), C.c_int(d),
                                  C.c_uint32(max_occ), O._p(out["drafts"]), O._p(out["draft_len"]),
                                  O._p(out["count"]), O._p(out["n_drafts"]), O._p(out["match_len"]),
                                  C.c_int(nthreads))
    assert rc == 0, rc
    return out


class State:
    """Per-sequence CACHEs plus the batch's missing table M."""

    def __init__(self, prompt_len, cp: CacheParams, key_len: int, missing_capacity: int):
        B = len(prompt_len)
        self.cp = cp
        self.entries = [[] for _ in range(B)]
        self.words = np.zeros(B, np.int64)
        self.out_mark = np.array(prompt_len, np.int64)
        self.dropped = np.zeros(B, np.int64)
        self.key_len = key_len
        self.missing = set()
        self.missing_max = missing_capacity // 2
        self.missing_dropped = 0

    def n_seq(self, b):
        return len(self.entries[b])

    def add_entry(self, b, seq):
        seq = np.asarray(seq, np.uint32)
        cost = len(seq) + 1
        if self.words[b] + cost <= self.cp.capacity:
            self.entries[b].append(seq.copy())
            self.words[b] += cost
        else:
            self.dropped[b] += 1

    def key(self, ctx_row, m):
        return tuple(int(t) for t in ctx_row[m - self.key_len:m]) if m >= self.key_len else None


def retrieve_step(state: State, corpora, ctx, ctx_len, p, nthreads: int = 0):
    """Steps 1-3 of a step.  Returns (results, code): results is a list of
    S + 1 result dicts (the datastore sources, then the CACHE), code[b] is
    SERVE_DATASTORE, SERVE_CACHE or SKIP_MISSING."""
    ctx = np.asarray(ctx, np.uint32)
    ctx_len = np.asarray(ctx_len, np.int32)
    B = ctx.shape[0]
    k, d = p["top_k"], p["draft_len"]
    l = state.cp.min_size
    active = [state.n_seq(b) >= l for b in range(B)]
    rc = cache_search([state.entries[b] if active[b] else [] for b in range(B)], ctx, ctx_len, p["n_max"],
                      p["n_min"], k, d, p["max_occ"], nthreads)
    keys = [state.key(ctx[b], int(ctx_len[b])) for b in range(B)]
    code = np.zeros(B, np.int32)
    for b in range(B):
        if active[b] and rc["n_drafts"][b] > 0:
            code[b] = SERVE_CACHE
        elif keys[b] is not None and keys[b] in state.missing:
            code[b] = SKIP_MISSING
    res = [empty_results(B, k, d) for _ in corpora]
    todo = np.nonzero(code == SERVE_DATASTORE)[0]
    if len(todo):
        for s, T in enumerate(corpora):
            r = O.retrieve(T, ctx[todo], ctx_len[todo], p["n_max"], p["n_min"], k, d, p["max_occ"], nthreads)
            for name in RESULT_FIELDS:
                res[s][name][todo] = r[name]
    missing_update(state, ctx, ctx_len, code, np.stack([r["n_drafts"] for r in res]) if res else np.zeros((0, B)))
    return res + [rc], code


def missing_update(state: State, ctx, ctx_len, code, n_drafts):
    """Step 3: M grows by the keys of the queries whose datastore search
    (code SERVE_DATASTORE) found nothing in any source (n_drafts [S, B]),
    in query order (reading R1), while M has room (R7)."""
    seen = set()
    for b in range(len(code)):
        if code[b] != SERVE_DATASTORE or any(n_drafts[s][b] > 0 for s in range(len(n_drafts))):
            continue
        key = state.key(ctx[b], int(ctx_len[b]))
        if key is None or key in state.missing or key in seen:
            continue
        seen.add(key)
        if len(state.missing) < state.missing_max:
            state.missing.add(key)
        else:
            state.missing_dropped += 1


def cache_update(state: State, ctx, old_len, new_len, acc_len):
    """Step 5 (readings R5, R6, R9)."""
    cp = state.cp
    for b in range(len(old_len)):
        o, n, a = int(old_len[b]), int(new_len[b]), int(acc_len[b])
        if n == o + a + 1 and a >= 1:
            keep = min(cp.ctx_keep, o)
            state.add_entry(b, ctx[b, o - keep:o + a])
        while n - state.out_mark[b] >= cp.chunk:
            mk = int(state.out_mark[b])
            state.add_entry(b, ctx[b, mk:mk + cp.chunk])
            state.out_mark[b] += cp.chunk


def step_loop(corpora, ctx, ctx_len, steps, p, cp: CacheParams, plen, rtok, src_weight, cache_weight, vocab,
              missing_capacity, kv_len0=None, nthreads: int = 0, state: State = None, on_step=None):
    """Integer trajectory of the step loop with Algorithm 1: retrieve_step ->
    tree over S + 1 slots -> synthetic target model -> acceptance -> append ->
    cache_update.  plen[step, b], rtok[step, b, n_pad] are the synthetic target
    model's draws.  Returns (history, ctx, ctx_len, kv_len, state)."""
    ctx = np.array(ctx, dtype=np.uint32, copy=True)
    ctx_len = np.array(ctx_len, dtype=np.int32, copy=True)
    B = ctx.shape[0]
    kv_len = np.zeros(B, np.int32) if kv_len0 is None else np.array(kv_len0, np.int32)
    if state is None:
        state = State(ctx_len, cp, p["n_min"], missing_capacity)
    weights = list(src_weight) + [cache_weight]
    hist = dict(acc_len=[], bonus=[], n_nodes=[], code=[], n_drafts=[])
    for st in range(steps):
        res, code = retrieve_step(state, corpora, ctx, ctx_len, p, nthreads)
        root = np.array([ctx[b, ctx_len[b] - 1] for b in range(B)], np.uint32)
        tr = O.build_tree(res, weights, root, kv_len, p["node_budget"], p["n_pad"], nthreads)
        am = O.synth_argmax(tr["tok"], tr["parent"], tr["n_nodes"], plen[st], rtok[st], vocab)
        ac = O.accept(tr["tok"], tr["parent"], tr["n_nodes"], am, p["draft_len"] + 2)
        if on_step is not None:
            on_step(st, res, code, tr, am, ac)
        old = ctx_len.copy()
        for b in range(B):
            a = int(ac["acc_len"][b])
            for t in range(a):
                ctx[b, ctx_len[b] + t] = tr["tok"][b, ac["path"][b, t + 1]]
            ctx[b, ctx_len[b] + a] = ac["bonus"][b]
            ctx_len[b] += a + 1
            kv_len[b] += a + 1
        cache_update(state, ctx, old, ctx_len, ac["acc_len"])
        hist["acc_len"].append(ac["acc_len"].copy())
        hist["bonus"].append(ac["bonus"].copy())
        hist["n_nodes"].append(tr["n_nodes"].copy())
        hist["code"].append(code)
        hist["n_drafts"].append(np.stack([r["n_drafts"] for r in res]))
    return hist, ctx, ctx_len, kv_len, state
