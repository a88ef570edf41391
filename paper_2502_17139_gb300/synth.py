"""Seeded synthetic inputs for the retrieve-and-verify step.

This module only draws random inputs: token corpora, query contexts, random
draft trees, attention activations and the random numbers that the synthetic
stand-in for the target model consumes.  It holds none of the method's
arithmetic (no suffix sorting, matching, counting, trie building, masking,
attention or acceptance), so both the CUDA path and the CPU oracle can take
their inputs from here without sharing any of the computation.

The paper evaluates on DevEval, RepoEval and HumanEval with a common datastore
built from The Stack and a per-repository datastore (Section IV-A, Section V-A,
Section V-D).  None of those are available here; the generators below stand in
for them with Zipfian token streams (code token frequencies are heavy-tailed)
plus planted repeated n-grams (the "localness" of code that Section III-B
describes: sequences defined earlier in a file or repository recur later).

Every generator takes an explicit ``numpy.random.Generator`` (PCG64) so that a
configuration is reproducible from ``SEED_BASE + config index``.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional, Sequence

import numpy as np

SEED_BASE = 2502171390
VOCAB = 32256            # DeepSeek-Coder vocabulary size (Section V-A models)
PAD = 0xFFFFFFFF         # draft padding token; never a valid id (ids < vocab)


def rng_for(config_index: int, stream: int = 0) -> np.random.Generator:
    """PCG64 generator for one configuration and one named sub-stream."""
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([SEED_BASE + config_index, stream])))


# --------------------------------------------------------------------------
# token streams
# --------------------------------------------------------------------------
_CDF_CACHE: dict = {}


def zipf_cdf(s: float, vocab: int = VOCAB) -> np.ndarray:
    """Cumulative distribution of a Zipf(s) law over ranks 1..vocab."""
    key = (float(s), int(vocab))
    if key not in _CDF_CACHE:
        w = np.arange(1, vocab + 1, dtype=np.float64) ** (-float(s))
        c = np.cumsum(w)
        c /= c[-1]
        _CDF_CACHE[key] = c
    return _CDF_CACHE[key]


def zipf_tokens(rng: np.random.Generator, n: int, s: float, vocab: int = VOCAB,
                chunk: int = 1 << 24, device=None) -> np.ndarray:
    """``n`` i.i.d. token ids, id = rank - 1 with rank ~ Zipf(s) (inverse CDF).

    With ``device`` (a CUDA device) and a large ``n`` the uniform draws and the
    inverse-CDF lookup run there with a torch generator seeded from ``rng``
    (the same numbers on every run, not the numpy stream); the result still
    comes back as a host array."""
    cdf = zipf_cdf(s, vocab)
    out = np.empty(n, dtype=np.uint32)
    if device is not None and n >= (1 << 26):
        import torch
        g = torch.Generator(device=device)
        g.manual_seed(int(rng.integers(0, 1 << 62)))
        cdf_d = torch.from_numpy(cdf).to(device)
        step = 1 << 27
        for lo in range(0, n, step):
            hi = min(n, lo + step)
            u = torch.rand(hi - lo, generator=g, device=device, dtype=torch.float64)
            r = torch.searchsorted(cdf_d, u, right=True).clamp_(max=vocab - 1)
            out[lo:hi] = r.to(torch.int32).cpu().numpy().view(np.uint32)
        return out
    for lo in range(0, n, chunk):
        hi = min(n, lo + chunk)
        u = rng.random(hi - lo)
        r = np.searchsorted(cdf, u, side="right")
        np.minimum(r, vocab - 1, out=r)
        out[lo:hi] = r.astype(np.uint32)
    return out


def _nonoverlapping_starts(rng: np.random.Generator, n: int, lengths: np.ndarray) -> np.ndarray:
    """Random start offsets for intervals of the given lengths that never
    overlap inside [0, n).  Instances are placed in a random order."""
    total = int(lengths.sum())
    if total > n:
        raise ValueError("planted material longer than the corpus")
    m = len(lengths)
    order = rng.permutation(m)
    gaps = np.sort(rng.integers(0, n - total + 1, size=m))
    lens_in_order = lengths[order]
    before = np.concatenate([[0], np.cumsum(lens_in_order)[:-1]])
    starts = np.empty(m, dtype=np.int64)
    starts[order] = gaps + before
    return starts


@dataclasses.dataclass
class Planted:
    """Where planted repeats were written (instance start, length, gram id)."""
    starts: np.ndarray
    lengths: np.ndarray
    gram: np.ndarray


def plant_repeats(rng: np.random.Generator, corpus: np.ndarray, n_grams: int,
                  len_range: tuple, copies_range: tuple, s: float,
                  vocab: int = VOCAB) -> Planted:
    """Write ``n_grams`` fresh Zipf n-grams, each copied a random number of
    times, at non-overlapping random offsets of ``corpus`` (in place).

    Lengths ~ U[len_range], copies ~ U[copies_range], both inclusive."""
    n = len(corpus)
    if n_grams == 0:
        z = np.zeros(0, dtype=np.int64)
        return Planted(z, z, z)
    glen = rng.integers(len_range[0], len_range[1] + 1, size=n_grams)
    copies = rng.integers(copies_range[0], copies_range[1] + 1, size=n_grams)
    gram_tok = zipf_tokens(rng, int(glen.sum()), s, vocab)
    gram_off = np.concatenate([[0], np.cumsum(glen)[:-1]])
    inst_gram = np.repeat(np.arange(n_grams), copies)
    inst_len = glen[inst_gram]
    starts = _nonoverlapping_starts(rng, n, inst_len)
    # vectorised copy: position k of instance t <- gram token k of its gram
    total = int(inst_len.sum())
    inst_first = np.concatenate([[0], np.cumsum(inst_len)[:-1]])
    t_of = np.repeat(np.arange(len(inst_len)), inst_len)
    k_of = np.arange(total) - inst_first[t_of]
    corpus[starts[t_of] + k_of] = gram_tok[gram_off[inst_gram[t_of]] + k_of]
    return Planted(starts, inst_len, inst_gram)


def grams_for_fraction(n: int, frac: float, len_range: tuple, copies_range: tuple) -> int:
    """Number of planted grams whose copies cover about ``frac`` of ``n``."""
    mean_len = 0.5 * (len_range[0] + len_range[1])
    mean_cp = 0.5 * (copies_range[0] + copies_range[1])
    return max(1, int(round(frac * n / (mean_len * mean_cp))))


def make_corpus(rng: np.random.Generator, n: int, s: float, vocab: int = VOCAB,
                n_grams: int = 0, len_range=(8, 32), copies_range=(2, 8), device=None):
    """Zipf(s) background with planted repeats; returns (uint32 tokens, Planted)."""
    t = zipf_tokens(rng, n, s, vocab, device=device)
    p = plant_repeats(rng, t, n_grams, len_range, copies_range, s, vocab)
    return t, p


# --------------------------------------------------------------------------
# query contexts
# --------------------------------------------------------------------------
def make_contexts(rng: np.random.Generator, batch: int, ctx_len: int, n_copy: int,
                  sources: Sequence[Optional[np.ndarray]], probs: Sequence[float],
                  s: float, vocab: int = VOCAB, ctx_stride: Optional[int] = None,
                  margin: int = 8, planted: Optional[Sequence[Optional[Planted]]] = None,
                  planted_share: float = 0.0):
    """Contexts whose first ``ctx_len - n_copy`` tokens are Zipf draws and
    whose last ``n_copy`` tokens are copied from a random offset of one of the
    ``sources`` (chosen with ``probs``; a ``None`` source leaves the tail as
    pure Zipf draws).  The copy offset p keeps p + n_copy + margin <= len(src)
    so that the copied suffix has a continuation.  With ``planted_share`` > 0,
    that share of the copies start inside a planted repeat of the source.

    Returns (ctx uint32[batch, ctx_stride], ctx_len int32[batch], origin int32[batch])
    where origin is the chosen source index (-1 for pure Zipf)."""
    stride = ctx_stride or ctx_len
    ctx = np.zeros((batch, stride), dtype=np.uint32)
    origin = np.empty(batch, dtype=np.int32)
    head = zipf_tokens(rng, batch * ctx_len, s, vocab).reshape(batch, ctx_len)
    ctx[:, :ctx_len] = head
    choice = rng.choice(len(sources), size=batch, p=np.asarray(probs, dtype=np.float64))
    for b in range(batch):
        src = sources[choice[b]]
        origin[b] = -1 if src is None else choice[b]
        if src is None:
            continue
        hi = len(src) - n_copy - margin
        pl = None if planted is None else planted[choice[b]]
        if pl is not None and len(pl.starts) and rng.random() < planted_share:
            t = int(rng.integers(0, len(pl.starts)))
            p = int(pl.starts[t] + rng.integers(0, max(1, int(pl.lengths[t]))))
            p = min(max(p - n_copy // 2, 0), hi)
        else:
            p = int(rng.integers(0, hi + 1))
        ctx[b, ctx_len - n_copy:ctx_len] = src[p:p + n_copy]
    return ctx, np.full(batch, ctx_len, dtype=np.int32), origin


# --------------------------------------------------------------------------
# random draft trees (for the attention/acceptance-only workload)
# --------------------------------------------------------------------------
def random_tree(rng: np.random.Generator, n_nodes: int, depth_max: int = 10,
                branch_max: int = 4, vocab: int = VOCAB, root_tok: Optional[int] = None):
    """A random rooted tree of exactly ``n_nodes`` nodes, depth <= depth_max,
    at most ``branch_max`` children per node, sibling tokens distinct.

    Nodes are returned in depth-first preorder with children visited in
    ascending token order (the tree layout the draft-tree builder emits), as
    (tok uint32[n_nodes], parent int32[n_nodes]); parent[0] = -1."""
    par = [-1]
    dep = [0]
    tok = [int(rng.integers(0, vocab)) if root_tok is None else int(root_tok)]
    kids = [set()]
    while len(par) < n_nodes:
        open_nodes = [i for i in range(len(par))
                      if dep[i] < depth_max and len(kids[i]) < min(branch_max, vocab)]
        v = open_nodes[int(rng.integers(0, len(open_nodes)))]
        while True:
            t = int(rng.integers(0, vocab))
            if t not in kids[v]:
                break
        kids[v].add(t)
        par.append(v)
        dep.append(dep[v] + 1)
        tok.append(t)
        kids.append(set())
    children = [[] for _ in par]
    for i in range(1, len(par)):
        children[par[i]].append(i)
    order = []
    stack = [0]
    while stack:
        v = stack.pop()
        order.append(v)
        for c in sorted(children[v], key=lambda c: tok[c], reverse=True):
            stack.append(c)
    new_id = {old: new for new, old in enumerate(order)}
    out_tok = np.array([tok[o] for o in order], dtype=np.uint32)
    out_par = np.array([-1 if par[o] < 0 else new_id[par[o]] for o in order], dtype=np.int32)
    return out_tok, out_par


# --------------------------------------------------------------------------
# random numbers consumed by the synthetic target model
# --------------------------------------------------------------------------
def argmax_draws(rng: np.random.Generator, batch: int, n_pad: int, vocab: int = VOCAB,
                 plen_max: int = 8, s: float = 1.1):
    """Per sequence: an agreeing-prefix length ~ U{0..plen_max} and one random
    token per tree slot, drawn from the corpus' Zipf(s) law (the target model
    emits code-like tokens, so the next context suffix can match the
    datastore again).  The synthetic target model follows the tree's first
    branch for that many steps and otherwise predicts the slot's random token
    (moved past any child token of the node)."""
    plen = rng.integers(0, plen_max + 1, size=batch).astype(np.int32)
    rtok = zipf_tokens(rng, batch * n_pad, s, vocab).reshape(batch, n_pad)
    return plen, rtok


def cache_hit_pattern(rng: np.random.Generator, steps: int, batch: int, p: float = 0.5) -> np.ndarray:
    """Seeded Bernoulli(p) 'want a cache hit' flags, int32[steps, batch]."""
    return (rng.random((steps, batch)) < p).astype(np.int32)


def randn_bf16(shape, seed: int, device="cpu"):
    """bf16 N(0,1) activations from a seeded torch generator on ``device``."""
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(int(seed) & ((1 << 63) - 1))
    return torch.randn(*shape, generator=g, device=device, dtype=torch.float32).to(torch.bfloat16)


# --------------------------------------------------------------------------
# the five workloads (sizes follow the benchmark configurations)
# --------------------------------------------------------------------------
WORKLOADS = {
    1: dict(name="c1 single-source 1M", corpus=[dict(n=1_000_000, s=1.1, n_grams=2000, len_range=(8, 32), copies_range=(2, 8))],
            batch=32, ctx_len=64, n_copy=16, probs=[1.0], n_max=16, n_min=2, top_k=16, draft_len=8,
            node_budget=64, n_pad=64, H=32, Hkv=32, D=128, kv_len=512),
    2: dict(name="c2 two-source 100M+5M", corpus=[dict(n=5_000_000, s=1.3, n_grams=20000, len_range=(8, 64), copies_range=(2, 8)),
                                                  dict(n=100_000_000, s=1.1, n_grams=0)],
            batch=256, ctx_len=128, n_copy=16, probs=[0.5, 0.25, 0.25], n_max=16, n_min=2, top_k=64, draft_len=10,
            node_budget=64, n_pad=64),
    3: dict(name="c3 tree attention 7B shape", batch=16, H=32, Hkv=32, D=128, kv_len=4096, n_pad=64,
            n_nodes=64, depth_max=10, branch_max=4),
    4: dict(name="c4 1B-token retrieval", corpus=[dict(n=1_000_000_000, s=1.1, frac=0.01, len_range=(16, 128), copies_range=(2, 8))],
            batch=1024, ctx_len=64, n_copy=24, probs=[1.0], planted_share=0.5, n_max=24, n_min=2, top_k=64, draft_len=12,
            node_budget=128, n_pad=128),
    5: dict(name="c5 step loop two-source GQA", batch=32, ctx_len=128, n_copy=16, probs=[0.5, 0.25, 0.25],
            n_max=16, n_min=2, top_k=64, draft_len=10, node_budget=128, n_pad=128,
            H=32, Hkv=8, D=128, kv_len=16384, steps=256, hit_p=0.5),
}


def scaled_corpus_spec(spec: dict, scale: float) -> dict:
    """A corpus spec shrunk by ``scale`` (planted material shrinks with it)."""
    out = dict(spec)
    out["n"] = max(1000, int(spec["n"] * scale))
    if spec.get("n_grams"):
        out["n_grams"] = max(1, int(spec["n_grams"] * scale))
    return out


def build_corpus(rng: np.random.Generator, spec: dict, vocab: int = VOCAB, device=None):
    """Corpus from a spec dict (see WORKLOADS); ``device`` as for zipf_tokens."""
    n = spec["n"]
    lr = spec.get("len_range", (8, 32))
    cr = spec.get("copies_range", (2, 8))
    grams = spec.get("n_grams", 0)
    if spec.get("frac"):
        grams = grams_for_fraction(n, spec["frac"], lr, cr)
    return make_corpus(rng, n, spec["s"], vocab, grams, lr, cr, device=device)


def decoder_weights(hidden: int, layers: int, H: int, Hkv: int, D: int, inter: int, vocab: int, seed: int,
                    device="cpu"):
    """Seeded random-init weights of a LLaMA-family decoder (the paper's
    target models are DeepSeek-Coder and CodeLlama; no trained weights are
    available), as bf16 torch tensors on ``device``: every projection
    N(0, 1/fan_in), the embedding N(0, 1), norm weights 1 + N(0, 0.1^2).
    Layout: per layer attn_norm [hidden], wq [hidden][H*D], wkv
    [hidden][2*Hkv*D] (K columns, then V), wo [H*D][hidden], mlp_norm
    [hidden], wgu [hidden][2*inter] (gate, then up), wd [inter][hidden];
    embed [vocab][hidden], final_norm [hidden], lm_head [hidden][vocab]."""
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(int(seed) & ((1 << 63) - 1))

    def mat(k, n, scale=None):
        s = (1.0 / math.sqrt(k)) if scale is None else scale
        return (torch.randn((k, n), generator=g, device=device, dtype=torch.float32) * s).to(torch.bfloat16)

    def norm(n):
        return (1.0 + 0.1 * torch.randn((n,), generator=g, device=device, dtype=torch.float32)).to(torch.bfloat16)

    W = {"embed": mat(vocab, hidden, 1.0), "layers": []}
    for _ in range(layers):
        W["layers"].append({"attn_norm": norm(hidden), "wq": mat(hidden, H * D), "wkv": mat(hidden, 2 * Hkv * D),
                            "wo": mat(H * D, hidden), "mlp_norm": norm(hidden), "wgu": mat(hidden, 2 * inter),
                            "wd": mat(inter, hidden)})
    W["final_norm"] = norm(hidden)
    W["lm_head"] = mat(hidden, vocab)
    return W
