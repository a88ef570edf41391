"""The two retrieval variants' rules, restated on the CPU and checked against
the oracle and plain sorting (no GPU, no kernel code):

* reversed corpus: read backwards, the context suffixes of lengths 1, 2, ...
  are prefixes of one another, so their ranges in the suffix array of the
  reversed corpus are nested; narrowing one token at a time (the occurrence
  at reversed position 0, the corpus ending with the pattern, has no
  continuation) finds the oracle's longest match n*;
* all-occurrence trie: merging sorted, duplicate-free draft lists by rank (own
  index plus, per other list, the drafts that precede it, an equal draft of an
  earlier list first) is a stable sort of their concatenation."""
import numpy as np
import pytest


def narrow(sa, R, T, ctx_tail, n_min):
    """Longest n in [n_min, len(ctx_tail)] found by nested narrowing (bisect on
    the token at depth n within the current range), 0 if none."""
    N = len(T)
    cap = len(ctx_tail)

    def key(j, n):  # token at depth n of reversed suffix sa[j], -1 past its end
        at = int(sa[j]) + n
        return -1 if at >= N else int(R[at])

    def bound(lo, hi, n, c, upper):
        while lo < hi:
            mid = (lo + hi) // 2
            k = key(mid, n)
            if (k > c) if upper else (k >= c):
                hi = mid
            else:
                lo = mid + 1
        return lo

    best, lo, hi = 0, 0, N
    ends = True
    for n in range(1, cap + 1):
        c = int(ctx_tail[cap - n])
        lo, hi = bound(lo, hi, n - 1, c, False), bound(lo, hi, n - 1, c, True)
        ends = ends and int(T[N - n]) == c if n <= N else False
        if hi - lo - (1 if ends else 0) <= 0:
            break
        if n >= n_min:
            best = n
    return best


@pytest.mark.parametrize("seed", range(6))
def test_reversed_narrowing_finds_the_oracle_match(orc, seed):
    rng = np.random.default_rng(4100 + seed)
    vocab = int(rng.integers(2, 6))
    N = int(rng.integers(30, 1500))
    T = rng.integers(0, vocab, N).astype(np.uint32)
    R = T[::-1].copy()
    sa = orc.suffix_array(R)
    B, stride = 40, 14
    ctx = rng.integers(0, vocab, (B, stride)).astype(np.uint32)
    cl = rng.integers(0, stride + 1, B).astype(np.int32)
    for b in range(B):
        L = int(min(cl[b], N))
        if L and b % 3 == 0:
            p0 = int(rng.integers(0, N - L + 1))
            ctx[b, cl[b] - L:cl[b]] = T[p0:p0 + L]
        elif L and b % 3 == 1:  # ends exactly at the corpus end
            ctx[b, cl[b] - L:cl[b]] = T[N - L:]
    n_max, n_min = 12, 2
    want = orc.retrieve(T, ctx, cl, n_max, n_min, 4, 3, 4096)["match_len"]
    for b in range(B):
        m = int(cl[b])
        cap = min(n_max, m)
        got = narrow(sa, R, T, ctx[b, m - cap:m], n_min) if cap >= n_min else 0
        assert got == int(want[b]), (b, got, int(want[b]))


def merge_by_rank(lists):
    """Merged position of every draft: its index in its own list plus, per
    other list, the count of drafts before it there (an equal draft of an
    earlier list counts as before)."""
    out = [None] * sum(len(x) for x in lists)
    for s, L in enumerate(lists):
        for t, d in enumerate(L):
            rank = t
            for s2, L2 in enumerate(lists):
                if s2 == s:
                    continue
                rank += sum(1 for e in L2 if e < d or (e == d and s2 < s))
            assert out[rank] is None
            out[rank] = (d, s)
    return out


@pytest.mark.parametrize("seed", range(5))
def test_rank_merge_is_a_stable_sort(seed):
    rng = np.random.default_rng(4200 + seed)
    lists = []
    for _ in range(int(rng.integers(1, 4))):
        drafts = {tuple(int(x) for x in rng.integers(0, 3, int(rng.integers(1, 5)))) for _ in range(int(rng.integers(0, 40)))}
        lists.append(sorted(drafts))  # ascending, a prefix before its extensions, no duplicates
    merged = merge_by_rank(lists)
    stable = sorted(((d, s) for s, L in enumerate(lists) for d in L), key=lambda x: (x[0], x[1]))
    assert merged == stable
    # equal drafts (from different lists) end up adjacent
    for i in range(1, len(merged)):
        if merged[i][0] == merged[i - 1][0]:
            assert merged[i][1] > merged[i - 1][1]


def runs_by_depth(drafts, w):
    """For sorted unique drafts with weights w: every trie node (u, l) (the
    length-l prefix of draft u, new at u when l > lcp(u-1, u)) with its weight
    and parent, found by numbering, for each depth l, the run starts (lcp < l)."""
    U = len(drafts)
    lcp = [0] * U
    for u in range(1, U):
        a, b = drafts[u - 1], drafts[u]
        k = 0
        while k < min(len(a), len(b)) and a[k] == b[k]:
            k += 1
        lcp[u] = k
    ps = np.concatenate([[0], np.cumsum(w)])
    nodes = {}
    prev_rid = prev_rpos = None
    for l in range(1, max(len(d) for d in drafts) + 1):
        start = [u == 0 or lcp[u] < l for u in range(U)]
        rid = list(np.cumsum(start) - 1)      # the run each draft belongs to
        rpos = [u for u in range(U) if start[u]] + [U]
        for u in range(U):
            if lcp[u] < l <= len(drafts[u]):
                W = ps[rpos[rid[u] + 1]] - ps[u]
                parent = drafts[prev_rpos[prev_rid[u]]][:l - 1] if l > 1 else ()
                nodes[drafts[u][:l]] = (int(W), parent)
        prev_rid, prev_rpos = rid, rpos
    return nodes


@pytest.mark.parametrize("seed", range(5))
def test_run_numbering_gives_trie_weights_and_parents(seed):
    rng = np.random.default_rng(4300 + seed)
    drafts = sorted({tuple(int(x) for x in rng.integers(0, 3, int(rng.integers(1, 7)))) for _ in range(60)})
    w = [int(x) for x in rng.integers(1, 9, len(drafts))]
    got = runs_by_depth(drafts, w)
    # brute force: a prefix weighs the drafts that start with it; its parent drops one token
    want = {}
    for d in drafts:
        for l in range(1, len(d) + 1):
            p = d[:l]
            want[p] = (sum(wi for di, wi in zip(drafts, w) if di[:l] == p), p[:-1])
    assert got == want
