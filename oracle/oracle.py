"""Python face of the CPU oracle (oracle/fc_oracle.cpp).

TEST INFRASTRUCTURE ONLY: imported by tests/, by __graft_entry__.smoke() and
by the CPU-baseline leg of bench.py, never by the product package.  It shares
no code with the CUDA path.  Arrays are numpy; bf16 tensors travel as their
uint16 bit patterns.

The step-loop driver at the bottom (``step_loop``) follows the decoding loop of
Section II / Section IV-D with the retrieval cache replay described in
``retrieval_cache_step``; parity of that cache with the paper's CACHE
(Section IV-B) is unpinned: it is a context-keyed replay cache, a reading of
the benchmark workload, and its only effect is to skip retrievals whose result
is already known.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "fc_oracle.cpp")
LIB = os.path.join(HERE, "_build", "liboracle.so")
PAD = 0xFFFFFFFF

_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with the host C++ compiler (portable flags only)."""
    os.makedirs(os.path.dirname(LIB), exist_ok=True)
    if force or not os.path.exists(LIB) or os.path.getmtime(LIB) < os.path.getmtime(SRC):
        tmp = LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["g++", "-O2", "-std=c++17", "-shared", "-fPIC", "-pthread", SRC, "-o", tmp])
        os.replace(tmp, LIB)
    return LIB


def lib():
    global _lib
    with _lock:
        if _lib is None:
            build()
            _lib = C.CDLL(LIB)
            _lib.orc_sa_certificate.restype = C.c_int64
    return _lib


def _p(a):
    return C.c_void_p(a.ctypes.data) if a is not None else None


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def hardware_threads() -> int:
    return int(lib().orc_hardware_threads())


# --------------------------------------------------------------------- O1
def suffix_array(T: np.ndarray, nthreads: int = 0) -> np.ndarray:
    T = _c(T, np.uint32)
    sa = np.empty(len(T), dtype=np.uint32)
    rc = lib().orc_suffix_array(_p(T), C.c_uint64(len(T)), _p(sa), C.c_int(nthreads))
    assert rc == 0
    return sa


def bucket(T: np.ndarray, sa: np.ndarray, vocab: int) -> np.ndarray:
    T = _c(T, np.uint32)
    sa = _c(sa, np.uint32)
    out = np.empty(vocab + 1, dtype=np.uint32)
    lib().orc_bucket(_p(T), C.c_uint64(len(T)), _p(sa), C.c_uint32(vocab), _p(out))
    return out


def lcp(T: np.ndarray, sa: np.ndarray, cap: int = 255) -> np.ndarray:
    """lcp[j] = common prefix length of the suffixes at sa[j-1], sa[j] (capped)."""
    T = _c(T, np.uint32)
    sa = _c(sa, np.uint32)
    out = np.empty(len(T), dtype=np.uint8)
    lib().orc_lcp(_p(T), C.c_uint64(len(T)), _p(sa), C.c_uint32(cap), _p(out))
    return out


def sa_certificate(T: np.ndarray, sa: np.ndarray, nthreads: int = 0) -> int:
    """-1 when sa is the suffix array of T, else the first failing index."""
    T = _c(T, np.uint32)
    sa = _c(sa, np.uint32)
    return int(lib().orc_sa_certificate(_p(T), C.c_uint64(len(T)), _p(sa), C.c_int(nthreads)))


# --------------------------------------------------------------- O2 - O4
def retrieve(T, ctx, ctx_len, n_max, n_min, top_k, d, max_occ, nthreads: int = 0):
    """Returns dict(drafts[B,k,d] u32, draft_len[B,k] i32, count[B,k] u32,
    n_drafts[B] i32, match_len[B] i32)."""
    T = _c(T, np.uint32)
    ctx = _c(ctx, np.uint32)
    ctx_len = _c(ctx_len, np.int32)
    B, stride = ctx.shape
    out = dict(drafts=np.empty((B, top_k, d), np.uint32), draft_len=np.empty((B, top_k), np.int32),
               count=np.empty((B, top_k), np.uint32), n_drafts=np.empty(B, np.int32),
               match_len=np.empty(B, np.int32))
    rc = lib().orc_retrieve(_p(T), C.c_uint64(len(T)), _p(ctx), C.c_int(stride), _p(ctx_len), C.c_int(B),
                            C.c_int(n_max), C.c_int(n_min), C.c_int(top_k), C.c_int(d), C.c_uint32(max_occ),
                            _p(out["drafts"]), _p(out["draft_len"]), _p(out["count"]), _p(out["n_drafts"]),
                            _p(out["match_len"]), C.c_int(nthreads))
    assert rc == 0, rc
    return out


# -------------------------------------------------------------------- O5
def build_tree(results, src_weight, root_tok, kv_len, budget, n_pad, nthreads: int = 0):
    """``results``: list over sources of retrieve() dicts (same B, k, d)."""
    S = len(results)
    drafts = _c(np.stack([r["drafts"] for r in results]), np.uint32)
    S_, B, k, d = drafts.shape
    dl = _c(np.stack([r["draft_len"] for r in results]), np.int32)
    ct = _c(np.stack([r["count"] for r in results]), np.uint32)
    nd = _c(np.stack([r["n_drafts"] for r in results]), np.int32)
    w = _c(src_weight, np.uint32)
    root_tok = _c(root_tok, np.uint32)
    kv_len = _c(kv_len, np.int32)
    nw = (n_pad + 63) // 64
    out = dict(tok=np.empty((B, n_pad), np.uint32), parent=np.empty((B, n_pad), np.int32),
               depth=np.empty((B, n_pad), np.int32), pos=np.empty((B, n_pad), np.int32),
               mask=np.empty((B, n_pad, nw), np.uint64), n_nodes=np.empty(B, np.int32))
    rc = lib().orc_build_tree(C.c_int(S), _p(drafts), _p(dl), _p(ct), _p(nd), _p(w), C.c_int(B), C.c_int(k),
                              C.c_int(d), _p(root_tok), _p(kv_len), C.c_int(budget), C.c_int(n_pad),
                              _p(out["tok"]), _p(out["parent"]), _p(out["depth"]), _p(out["pos"]),
                              _p(out["mask"]), _p(out["n_nodes"]), C.c_int(nthreads))
    assert rc == 0, rc
    return out


def tree_mask(parent, n_nodes, kv_len, n_pad):
    parent = _c(parent, np.int32)
    n_nodes = _c(n_nodes, np.int32)
    kv_len = _c(kv_len, np.int32)
    B = parent.shape[0]
    nw = (n_pad + 63) // 64
    out = dict(depth=np.empty((B, n_pad), np.int32), pos=np.empty((B, n_pad), np.int32),
               mask=np.empty((B, n_pad, nw), np.uint64))
    rc = lib().orc_tree_mask(_p(parent), _p(n_nodes), _p(kv_len), C.c_int(B), C.c_int(n_pad),
                             _p(out["depth"]), _p(out["pos"]), _p(out["mask"]))
    assert rc == 0, rc
    return out


# -------------------------------------------------------------------- O6
def rope(x, pos, base=10000.0):
    """O12: rows x[..., D] (float64) rotated by pos[...] (int), rotate-half
    pairing.  Returns float64 of x's shape."""
    x = np.ascontiguousarray(x, np.float64)
    D = x.shape[-1]
    pos = _c(np.broadcast_to(np.asarray(pos, np.int32), x.shape[:-1]), np.int32)
    out = np.empty_like(x)
    rc = lib().orc_rope(_p(x), C.c_int64(x.size // D), C.c_int(D), _p(pos), C.c_double(base), _p(out))
    assert rc == 0, rc
    return out


def tree_attn(q, k_cache, v_cache, kv_len, k_tree, v_tree, mask, n_nodes, scale=None, rows=None,
              nthreads: int = 0, pos=None, rope_base=10000.0):
    """bf16 arrays as uint16 bit patterns: q[B,Np,H,D], caches [B,Hkv,cap,D],
    tree K/V [B,Hkv,Np,D].  Returns fp64 out[B,Np,H,D], or [n_rows, D] for
    ``rows`` = int32[n_rows, 3] of (b, i, h).  With ``pos`` (int32 [B,Np]),
    the queries and the tree keys are rotated by O12 at those positions."""
    q = _c(q, np.uint16)
    k_cache = _c(k_cache, np.uint16)
    v_cache = _c(v_cache, np.uint16)
    k_tree = _c(k_tree, np.uint16)
    v_tree = _c(v_tree, np.uint16)
    mask = _c(mask, np.uint64)
    kv_len = _c(kv_len, np.int32)
    n_nodes = _c(n_nodes, np.int32)
    B, Np, H, D = q.shape
    Hkv, cap = k_cache.shape[1], k_cache.shape[2]
    if scale is None:
        scale = 1.0 / np.sqrt(D)
    if rows is None:
        out = np.empty((B, Np, H, D), np.float64)
        rp, nr = None, 0
    else:
        rows = _c(rows, np.int32).reshape(-1, 3)
        out = np.empty((rows.shape[0], D), np.float64)
        rp, nr = _p(rows), rows.shape[0]
    if pos is None:
        rc = lib().orc_tree_attn(_p(q), _p(k_cache), _p(v_cache), C.c_int(cap), _p(kv_len), _p(k_tree),
                                 _p(v_tree), _p(mask), _p(n_nodes), C.c_int(B), C.c_int(Np), C.c_int(H),
                                 C.c_int(Hkv), C.c_int(D), C.c_double(scale), rp, C.c_int64(nr), _p(out),
                                 C.c_int(nthreads))
    else:
        pos = _c(pos, np.int32)
        assert pos.shape == (B, Np)
        rc = lib().orc_tree_attn_rope(_p(q), _p(k_cache), _p(v_cache), C.c_int(cap), _p(kv_len), _p(k_tree),
                                      _p(v_tree), _p(mask), _p(n_nodes), C.c_int(B), C.c_int(Np), C.c_int(H),
                                      C.c_int(Hkv), C.c_int(D), C.c_double(scale), _p(pos), C.c_double(rope_base),
                                      rp, C.c_int64(nr), _p(out), C.c_int(nthreads))
    assert rc == 0, rc
    return out


# -------------------------------------------------------------------- O7
def accept(tok, parent, n_nodes, argmax, path_cap):
    tok = _c(tok, np.uint32)
    parent = _c(parent, np.int32)
    n_nodes = _c(n_nodes, np.int32)
    argmax = _c(argmax, np.uint32)
    B, Np = tok.shape
    out = dict(acc_len=np.empty(B, np.int32), path=np.empty((B, path_cap), np.int32), bonus=np.empty(B, np.uint32))
    rc = lib().orc_accept(_p(tok), _p(parent), _p(n_nodes), _p(argmax), C.c_int(B), C.c_int(Np),
                          _p(out["acc_len"]), _p(out["path"]), C.c_int(path_cap), _p(out["bonus"]))
    assert rc == 0, rc
    return out


# ------------------------------------------------------------------- O10
def argmax_rows(logits, n_nodes):
    """logits: bf16 bit patterns uint16 [B, Np, V] -> uint32 [B, Np] (rows >= n_nodes are 0)."""
    logits = _c(logits, np.uint16)
    n_nodes = _c(n_nodes, np.int32)
    B, Np, V = logits.shape
    out = np.empty((B, Np), np.uint32)
    rc = lib().orc_argmax_rows(_p(logits), C.c_int(B), C.c_int(Np), C.c_int(V), _p(n_nodes), _p(out))
    assert rc == 0, rc
    return out


# -------------------------------------------------------------------- O8
def kv_append(path, acc_len, bonus, tok, k_tree, v_tree, k_cache, v_cache, kv_len, ctx, ctx_len):
    """In place on k_cache, v_cache, ctx; returns (kv_len_out, ctx_len_out, root_out)."""
    path = _c(path, np.int32)
    acc_len = _c(acc_len, np.int32)
    bonus = _c(bonus, np.uint32)
    tok = _c(tok, np.uint32)
    k_tree = _c(k_tree, np.uint16)
    v_tree = _c(v_tree, np.uint16)
    kv_len = _c(kv_len, np.int32)
    ctx_len = _c(ctx_len, np.int32)
    assert k_cache.dtype == np.uint16 and k_cache.flags.c_contiguous
    assert v_cache.dtype == np.uint16 and v_cache.flags.c_contiguous
    assert ctx.dtype == np.uint32 and ctx.flags.c_contiguous
    B, Np = tok.shape
    Hkv, D = k_tree.shape[1], k_tree.shape[3]
    cap = k_cache.shape[2]
    kv_out = np.empty(B, np.int32)
    cl_out = np.empty(B, np.int32)
    root = np.empty(B, np.uint32)
    rc = lib().orc_kv_append(_p(path), _p(acc_len), _p(bonus), _p(tok), _p(k_tree), _p(v_tree), C.c_int(B),
                             C.c_int(Np), C.c_int(Hkv), C.c_int(D), C.c_int(path.shape[1]), _p(k_cache),
                             _p(v_cache), C.c_int(cap), _p(kv_len), _p(kv_out), _p(ctx), C.c_int(ctx.shape[1]),
                             _p(ctx_len), _p(cl_out), _p(root))
    assert rc == 0, rc
    return kv_out, cl_out, root


def synth_argmax(tok, parent, n_nodes, plen, rtok, vocab):
    tok = _c(tok, np.uint32)
    parent = _c(parent, np.int32)
    n_nodes = _c(n_nodes, np.int32)
    plen = _c(plen, np.int32)
    rtok = _c(rtok, np.uint32)
    B, Np = tok.shape
    out = np.empty((B, Np), np.uint32)
    lib().orc_synth_argmax(_p(tok), _p(parent), _p(n_nodes), C.c_int(B), C.c_int(Np), _p(plen), _p(rtok),
                           C.c_uint32(vocab), _p(out))
    return out


# ------------------------------------------------------------ O9 / loop
def cache_key(ctx_row: np.ndarray, ctx_len: int, n_max: int) -> bytes:
    """The retrieval cache key: the last n_max context tokens (fewer when the
    context is shorter), with their count."""
    m = int(ctx_len)
    k = min(n_max, m)
    return bytes(np.int32(k).tobytes()) + ctx_row[m - k:m].astype(np.uint32).tobytes()


def step_loop(corpora, ctx, ctx_len, steps, p, hits, plen, rtok, src_weight, vocab, kv_len0=None,
              nthreads: int = 0, on_step=None, cache=None):
    """Integer trajectory of the step loop (retrieve -> tree -> accept ->
    append) with the context-keyed replay cache.  Attention does not steer the
    trajectory (acceptance reads the target model's predictions only), so it
    is checked separately on sampled steps.

    p: dict with n_max, n_min, top_k, draft_len, max_occ, node_budget, n_pad.
    hits[step, b]: want-hit flags; plen[step, b], rtok[step, b, n_pad]: the
    synthetic target model's draws.  ``cache`` (a dict) persists the replay
    cache across calls: a first pass records retrieval results, a second pass
    over the same trajectory replays them where hits[step, b] asks for it.
    Returns per-step lists of acc_len and bonus plus the final context."""
    ctx = np.array(ctx, dtype=np.uint32, copy=True)
    ctx_len = np.array(ctx_len, dtype=np.int32, copy=True)
    B = ctx.shape[0]
    kv_len = np.zeros(B, np.int32) if kv_len0 is None else np.array(kv_len0, np.int32)
    cache = {} if cache is None else cache
    hist = dict(acc_len=[], bonus=[], n_nodes=[], hit=[])
    S = len(corpora)
    for st in range(steps):
        res = [dict(drafts=np.full((B, p["top_k"], p["draft_len"]), PAD, np.uint32),
                    draft_len=np.zeros((B, p["top_k"]), np.int32), count=np.zeros((B, p["top_k"]), np.uint32),
                    n_drafts=np.zeros(B, np.int32), match_len=np.zeros(B, np.int32)) for _ in range(S)]
        keys = [cache_key(ctx[b], ctx_len[b], p["n_max"]) for b in range(B)]
        used = np.zeros(B, np.int32)
        for b in range(B):
            if hits[st, b] and keys[b] in cache:
                used[b] = 1
                for s in range(S):
                    for name in res[s]:
                        res[s][name][b] = cache[keys[b]][s][name]
        todo = np.nonzero(used == 0)[0]
        if len(todo):
            for s, T in enumerate(corpora):
                r = retrieve(T, ctx[todo], ctx_len[todo], p["n_max"], p["n_min"], p["top_k"], p["draft_len"],
                             p["max_occ"], nthreads)
                for name in res[s]:
                    res[s][name][todo] = r[name]
            for b in todo:
                cache[keys[b]] = [{name: res[s][name][b].copy() for name in res[s]} for s in range(S)]
        root = np.array([ctx[b, ctx_len[b] - 1] for b in range(B)], np.uint32)
        tr = build_tree(res, src_weight, root, kv_len, p["node_budget"], p["n_pad"], nthreads)
        am = synth_argmax(tr["tok"], tr["parent"], tr["n_nodes"], plen[st], rtok[st], vocab)
        ac = accept(tr["tok"], tr["parent"], tr["n_nodes"], am, p["draft_len"] + 2)
        if on_step is not None:
            on_step(st, res, tr, am, ac)
        for b in range(B):
            a = ac["acc_len"][b]
            for t in range(a):
                ctx[b, ctx_len[b] + t] = tr["tok"][b, ac["path"][b, t + 1]]
            ctx[b, ctx_len[b] + a] = ac["bonus"][b]
            ctx_len[b] += a + 1
            kv_len[b] += a + 1
        hist["acc_len"].append(ac["acc_len"].copy())
        hist["bonus"].append(ac["bonus"].copy())
        hist["n_nodes"].append(tr["n_nodes"].copy())
        hist["hit"].append(used)
    return hist, ctx, ctx_len, kv_len
