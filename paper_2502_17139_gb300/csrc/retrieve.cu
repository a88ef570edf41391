// fc_retrieve: batched suffix-match draft retrieval (Section III-A; Section
// IV-C, Algorithm 1 par_search over D_r and D_c; Section V-C n_max = 16),
// and the context-keyed replay cache used by the step loop.
//
// One CTA per (query, source).  Design:
//   * search: every suffix length n gets a warp, its two half-warps find the
//     lower and the upper bound of the pattern's suffix-array range at once,
//     so all lengths n_max..n_min are searched together and the longest
//     non-empty range is picked afterwards (a match of length n implies
//     matches of every shorter length, so the longest non-empty range is the
//     answer).  The first-token bucket table narrows each search to the
//     suffixes that start with the pattern's first token.  Each round of a
//     search probes 16 pivots, one per lane (a 17-ary search: ~6 rounds for
//     ten million suffixes instead of ~24 binary steps), and a probe reads its
//     suffix's tokens as aligned 16-byte vectors, all loads in flight at once.
//   * the suffix that is exactly the pattern at the corpus end (no
//     continuation) is the smallest suffix of its range when present; it is
//     dropped.
//   * counting: in SA order the occurrences' continuations are sorted, so
//     equal continuations are adjacent, and two neighbours carry the same
//     continuation exactly when their common prefix (the datastore's LCP
//     array) covers the match plus the draft length.  Runs come from one
//     coalesced byte read per occurrence and a block scan (no hash table and
//     no token reads).
//   * top-k: a histogram of run counts finds the k-th largest count; the runs
//     above it and the first runs equal to it (in token order) are kept and
//     ranked by (count descending, token order ascending).
//   * reversed-corpus variant (fc_retrieve_rev): with the suffix array of the
//     reversed corpus, the context suffixes of lengths 1, 2, ... read
//     backwards are prefixes of one another, so their ranges are nested and
//     one narrowing search (a warp, one more token per step, 16 pivots a
//     round, two loads a probe) finds n* without trying every length; the
//     forward suffix array is then searched for n* alone, and everything
//     after it is shared with fc_retrieve, so the outputs are the same.
//   * all-continuations variant (fc_retrieve_all): no top-k; every run is
//     written, in SA order, which is ascending token order (the input of the
//     all-occurrence trie).
#include <algorithm>

#include "fc_common.cuh"
#include "fc_topk.cuh"

FC_DEFINE_ERROR_WORD(ret)

namespace {

constexpr int RT_THREADS = 512;
constexpr int CMP_GROUPS = FC_MAX_NMAX / 4 + 1;    // 16-byte groups covering a pattern at any alignment

struct DsView {
  const uint32_t* T;
  const uint32_t* sa;
  const uint32_t* bucket;
  const uint8_t* lcp;
  uint64_t n;
  uint32_t vocab;
  const uint4* keys;  // suffix keys (two uint4 per SA entry) or nullptr
};
struct DsArgs {
  DsView ds[FC_MAX_SOURCES];
};

struct RetOut {
  uint32_t* drafts;
  int32_t* draft_len;
  uint32_t* count;
  int32_t* n_drafts;
  int32_t* match_len;
  unsigned int* err;  // the launch's error word (NULL: this file's own)
};

// Sign of the suffix T[i..N) cut to n tokens against pat[0..n), knowing
// T[i] == pat[0] (1 <= n <= FC_MAX_NMAX).  The tokens come in aligned 16-byte
// groups (the corpus is 16-byte aligned), all loads issued before any
// comparison; a group that would cross the corpus end is read token by token.
__device__ __forceinline__ int cmp_suffix_vec(const uint32_t* __restrict__ T, uint64_t N, uint64_t i,
                                              const uint32_t* pat, int n) {
  const uint64_t base = i & ~(uint64_t)3;
  const int off = (int)(i - base);
  const int ngrp = (off + n + 3) >> 2;
  uint32_t w[4 * CMP_GROUPS];
#pragma unroll
  for (int g = 0; g < CMP_GROUPS; ++g) {
    const uint64_t q = base + 4 * (uint64_t)g;
    if (g < ngrp && q + 4 <= N) {
      const uint4 v = __ldg(reinterpret_cast<const uint4*>(T + q));
      w[4 * g] = v.x;
      w[4 * g + 1] = v.y;
      w[4 * g + 2] = v.z;
      w[4 * g + 3] = v.w;
    } else {
#pragma unroll
      for (int e = 0; e < 4; ++e) w[4 * g + e] = (g < ngrp && q + e < N) ? __ldg(T + q + e) : 0u;
    }
  }
  const uint64_t avail = N - i;  // tokens of the suffix
  int res = 0;
#pragma unroll
  for (int k = 1; k < FC_MAX_NMAX; ++k) {
    // token i + k sits at w[off + k]; select on the alignment so every index is static
    const uint32_t t = off == 0 ? w[k] : off == 1 ? w[k + 1] : off == 2 ? w[k + 2] : w[k + 3];
    if (k < n && res == 0) {
      if ((uint64_t)k >= avail) {
        res = -1;
      } else {
        const uint32_t b = pat[k];
        if (t != b) res = t < b ? -1 : 1;
      }
    }
  }
  return res;
}

// The same sign for the suffix at SA index piv, from its key entry: the
// suffix start and tokens 1..7 in one 32-byte read (FC_PAD_TOKEN past the
// corpus end, where the suffix ended and sorts first).  Tokens from 8 on
// come from the corpus, and only when the first eight tie.
__device__ __forceinline__ int cmp_suffix_key(const uint4* __restrict__ keys, const uint32_t* __restrict__ T,
                                              uint64_t N, uint32_t piv, const uint32_t* pat, int n, uint32_t* at) {
  const uint4 a = __ldg(keys + 2 * (size_t)piv), c = __ldg(keys + 2 * (size_t)piv + 1);
  *at = a.x;
  const uint32_t t[8] = {a.x, a.y, a.z, a.w, c.x, c.y, c.z, c.w};
  int res = 0;
#pragma unroll
  for (int k = 1; k < 8; ++k) {
    if (k < n && res == 0) {
      const uint32_t v = t[k], q = pat[k];
      if (v == FC_PAD_TOKEN)
        res = -1;
      else if (v != q)
        res = v < q ? -1 : 1;
    }
  }
  if (res != 0 || n <= 8) return res;
  // token 7 is known equal: compare tokens 8 .. n-1
  return cmp_suffix_vec(T, N, (uint64_t)a.x + 7, pat + 7, n - 7);
}

struct RetSmem {
  uint32_t runs[FC_MAX_OCC + 1];   // run starts (occurrence index), runs[R] = nocc
  uint32_t work[FC_MAX_OCC];       // head flags, then the count histogram
  uint32_t sel[FC_MAX_TOPK];       // kept runs
  uint32_t order[FC_MAX_TOPK];     // kept runs by (count desc, run asc)
  uint32_t ctx[FC_MAX_NMAX];
  uint32_t lo[FC_MAX_NMAX + 1];
  uint32_t hi[FC_MAX_NMAX + 1];
  uint32_t endhit[FC_MAX_NMAX + 1];
  uint32_t wsum[RT_THREADS / 32];
  RunsScratch rs;
  uint32_t n_star, first, cnt, bad, n_rev;
  int32_t rc_slot;
};

// The replay-cache lookup folded into retrieval (fc_retrieve_cached): table
// NULL means none.
struct RcFused {
  const uint32_t* table;
  int capacity;
  const int32_t* want;  // NULL: every query may be served
  int32_t* skip;        // out: 1 = served from the cache
};

// n* through the reversed corpus R (R[i] = T[N-1-i]), by one warp.  The
// context read backwards, rp = ctx[m-1], ctx[m-2], ..., has range(n) = the
// reversed-SA range of suffixes that start with rp[0..n); range(n+1) is the
// part of range(n) whose token at depth n is rp[n] (a suffix of exactly n
// tokens sorts before the rest).  An occurrence at R position r ends the
// forward window just before T position N - r, so the one at r = 0 (the
// corpus ends with the pattern) has no continuation and does not count.  The
// counts only fall as n grows, so the narrowing stops at the first empty
// one.  Returns the longest n in [n_min, cap] with a count, or 0.
__device__ int rev_match_len(const DsView& rv, const uint32_t* __restrict__ T, uint64_t N, const uint32_t* ctx,
                             int cap, int n_min) {
  const int lane = threadIdx.x & 31, hl = lane & 15;
  const bool upper = lane >= 16;
  const unsigned half_mask = upper ? 0xFFFF0000u : 0x0000FFFFu;
  const uint32_t* __restrict__ R = rv.T;
  int best = 0;
  uint32_t c = ctx[cap - 1];
  uint32_t lo = __ldg(rv.bucket + c), hi = __ldg(rv.bucket + c + 1);
  bool ends = __ldg(T + N - 1) == c;  // T[N-n .. N) equals the pattern (R suffix 0 in the range)
  for (int n = 1;; ++n) {
    if (hi - lo <= (ends ? 1u : 0u)) break;
    if (n >= n_min) best = n;
    if (n == cap) break;
    c = ctx[cap - 1 - n];
    // bound search in [lo, hi): lower half-warp the first suffix whose token at
    // depth n is >= c, upper half-warp the first one > c
    uint32_t blo = lo, bhi = hi;
    while (__any_sync(0xFFFFFFFFu, blo < bhi)) {
      const bool active = blo < bhi;
      const uint32_t piv = blo + (uint32_t)(((uint64_t)(hl + 1) * (bhi - blo)) / 17u);
      bool pred = true;  // the suffix at piv is past the bound
      if (active) {
        const uint64_t at = (uint64_t)__ldg(rv.sa + piv) + (uint64_t)n;
        if (at >= N) {
          pred = false;  // exactly n tokens: before every suffix that has a token at depth n
        } else {
          const uint32_t t = __ldg(R + at);
          pred = upper ? (t > c) : (t >= c);
        }
      }
      const unsigned bal = __ballot_sync(0xFFFFFFFFu, !pred) & half_mask;
      const int t = __popc(bal);
      const int base_lane = upper ? 16 : 0;
      const uint32_t p_before = __shfl_sync(0xFFFFFFFFu, piv, base_lane + max(t - 1, 0));
      const uint32_t p_at = __shfl_sync(0xFFFFFFFFu, piv, base_lane + min(t, 15));
      if (active) {
        if (t > 0) blo = p_before + 1;
        if (t < 16) bhi = p_at;
      }
    }
    lo = __shfl_sync(0xFFFFFFFFu, blo, 0);
    hi = __shfl_sync(0xFFFFFFFFu, blo, 16);
    ends = ends && (uint64_t)n < N && __ldg(T + N - 1 - n) == c;
  }
  return best;
}

// ---------------------------------------------------------------------------
// Replay cache.  Entry layout (32-bit words): [0] key length or EMPTY /
// CLAIMED, [1 .. 1+n_max) key tokens, then per source: drafts[k*d],
// draft_len[k], count[k], n_drafts, match_len.
// ---------------------------------------------------------------------------
constexpr uint32_t RC_EMPTY = 0xFFFFFFFFu;
constexpr uint32_t RC_CLAIMED = 0xFFFFFFFEu;

__host__ __device__ inline size_t rc_src_words(const fc_retrieve_params& p) {
  return (size_t)p.top_k * p.draft_len + 2 * (size_t)p.top_k + 2;
}
__host__ __device__ inline size_t rc_entry_words(int S, const fc_retrieve_params& p) {
  size_t w = 1 + (size_t)p.n_max + (size_t)S * rc_src_words(p);
  return (w + 3) & ~(size_t)3;
}

__device__ uint64_t rc_hash(const uint32_t* key, int len) {
  uint64_t h = 1469598103934665603ull ^ (uint64_t)len;
  for (int i = 0; i < len; ++i) {
    h ^= key[i];
    h *= 1099511628211ull;
  }
  h ^= h >> 29;
  return h;
}

struct RcSmem {
  uint32_t key[FC_MAX_NMAX];
  int klen;
  int slot;
};

__device__ void rc_load_key(RcSmem& sm, const uint32_t* ctx, int stride, const int32_t* ctx_len, int b, int n_max) {
  int m = max(0, min((int)ctx_len[b], stride));
  int kl = min(n_max, m);
  if (threadIdx.x < kl) sm.key[threadIdx.x] = ctx[(size_t)b * stride + (m - kl) + threadIdx.x];
  if (threadIdx.x == 0) sm.klen = kl;
  __syncthreads();
}

// Warp 0 compares the entry's key with sm.key: lane i reads key word i, so
// the words arrive in one round trip (n_max <= 32).  `head` is the entry's
// first word, already read.  Warp-uniform result.
__device__ bool rc_key_equal_warp(const uint32_t* entry, uint32_t head, const uint32_t* key, int klen, int lane) {
  const bool len_ok = head == (uint32_t)klen;
  const uint32_t w = (len_ok && lane < klen) ? entry[1 + lane] : 0u;
  return __all_sync(0xFFFFFFFFu, len_ok && (lane >= klen || w == key[lane]));
}

// Warp 0's probe for `key`: the slot of an entry holding it, or -1 (an empty
// slot ends the chain).  Every lane returns the same slot.
__device__ int rc_find_warp(const uint32_t* table, int capacity, size_t ew, const uint32_t* key, int klen, int lane) {
  const uint64_t h = rc_hash(key, klen);
  for (int probe = 0; probe < capacity; ++probe) {
    const size_t e = (h + probe) & (uint64_t)(capacity - 1);
    const uint32_t* ent = table + e * ew;
    const uint32_t st = ent[0];
    if (st == RC_EMPTY) break;
    if (st != RC_CLAIMED && rc_key_equal_warp(ent, st, key, klen, lane)) return (int)e;
  }
  return -1;
}

// A query's outputs and a cache entry's result area, word by word: flat
// index i over S * rc_src_words(p) words (source s, then drafts, draft
// lengths, counts, n_drafts, match_len) names one word of the entry
// (entry[i]) and one output word (*rc_out_word(...)).
__device__ __forceinline__ uint32_t* rc_out_word(const RetOut& o, int i, int per, int k, int d, int B, int b) {
  const int s = i / per, r = i - s * per;
  const size_t sb = (size_t)s * B + b;
  if (r < k * d) return o.drafts + sb * k * d + r;
  if (r < k * d + k) return reinterpret_cast<uint32_t*>(o.draft_len) + sb * k + (r - k * d);
  if (r < k * d + 2 * k) return o.count + sb * k + (r - k * d - k);
  return r == k * d + 2 * k ? reinterpret_cast<uint32_t*>(o.n_drafts) + sb : reinterpret_cast<uint32_t*>(o.match_len) + sb;
}

// Copies a query's whole result between a cache entry and the outputs with
// the CTA's threads, sixteen loads in flight per thread before their stores
// (a lookup or an insert is a few such round trips, not one per array).
template <bool TO_OUT>
__device__ __forceinline__ void rc_copy(uint32_t* entry, const RetOut& o, int S, const fc_retrieve_params& p, int B,
                                        int b, int s_first = 0, int s_count = -1) {
  constexpr int U = 16;
  const int k = p.top_k, d = p.draft_len, per = (int)rc_src_words(p);
  const int n = (s_first + (s_count < 0 ? S - s_first : s_count)) * per;  // sources [s_first, s_first + count)
  for (int i0 = s_first * per + threadIdx.x; i0 < n; i0 += U * blockDim.x) {
    uint32_t v[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int i = i0 + u * blockDim.x;
      v[u] = i < n ? (TO_OUT ? entry[i] : *rc_out_word(o, i, per, k, d, B, b)) : 0u;
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int i = i0 + u * blockDim.x;
      if (i < n) {
        if (TO_OUT)
          *rc_out_word(o, i, per, k, d, B, b) = v[u];
        else
          entry[i] = v[u];
      }
    }
  }
}

template <bool REV, bool ALL>
__global__ void __launch_bounds__(RT_THREADS) k_retrieve(DsArgs args, DsArgs rev, const uint32_t* __restrict__ ctx,
                                                         int stride, const int32_t* __restrict__ ctx_len, int B,
                                                         const int32_t* __restrict__ skip, fc_retrieve_params p,
                                                         RetOut o, RcFused rc) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  RetSmem& sm = *reinterpret_cast<RetSmem*>(smem_raw);
  const int b = blockIdx.x, s = blockIdx.y, tid = threadIdx.x;
  if (skip && skip[b]) return;
  const DsView ds = args.ds[s];
  const uint32_t* __restrict__ T = ds.T;
  const uint64_t N = ds.n;
  const int k = ALL ? (int)p.max_occ : p.top_k, d = p.draft_len;  // output slots per query and source
  const size_t sb = (size_t)s * B + b;

  int m = ctx_len[b];
  m = max(0, min(m, stride));
  const int cap = min(p.n_max, m);
  if (tid == 0) sm.bad = 0;
  __syncthreads();
  if (tid < cap) {
    uint32_t t = ctx[(size_t)b * stride + (m - cap) + tid];
    sm.ctx[tid] = t;
    if (t >= ds.vocab) sm.bad = 1;
  }
  __syncthreads();
  if constexpr (!REV && !ALL) {
    // Replay cache first: the key is the context's last min(n_max, ctx_len)
    // tokens, the ones just loaded.  A served query copies this source's
    // stored result and is done (as fc_rcache_lookup, then a skipped
    // retrieval: a served query records no token error).
    if (rc.table) {
      if (tid < 32) {
        const size_t ew = rc_entry_words((int)gridDim.y, p);
        const int slot = (!rc.want || rc.want[b]) ? rc_find_warp(rc.table, rc.capacity, ew, sm.ctx, cap, tid) : -1;
        if (tid == 0) sm.rc_slot = slot;
      }
      __syncthreads();
      const int slot = sm.rc_slot;
      if (s == 0 && tid == 0) rc.skip[b] = slot >= 0 ? 1 : 0;
      if (slot >= 0) {
        const size_t ew = rc_entry_words((int)gridDim.y, p);
        rc_copy<true>(const_cast<uint32_t*>(rc.table) + (size_t)slot * ew + 1 + p.n_max, o, (int)gridDim.y, p, B, b,
                      s, 1);
        return;
      }
    }
  }
  if (sm.bad && tid == 0) fc_flag(FC_ERR_WORD(o.err), FC_EBIT_INVALID);

  // ---- search: one warp per n, one half-warp per bound, 16 pivots a round
  // (lengths n_top down to n_top - n_count + 1; with the reversed corpus only n*)
  int n_top = cap, n_count = (cap >= p.n_min && !sm.bad) ? cap - p.n_min + 1 : 0;
  if constexpr (REV) {
    if (tid < 32) {
      const int r = n_count ? rev_match_len(rev.ds[s], T, N, sm.ctx, cap, p.n_min) : 0;
      if (tid == 0) sm.n_rev = (uint32_t)r;
    }
    __syncthreads();
    n_top = (int)sm.n_rev;
    n_count = n_top ? 1 : 0;
  }
  const int npairs = 2 * n_count;
  {
    const int warp = tid >> 5, lane = tid & 31, hl = lane & 15;
    const bool upper = lane >= 16;
    const unsigned half_mask = upper ? 0xFFFF0000u : 0x0000FFFFu;
    for (int w = warp; w < n_count; w += RT_THREADS / 32) {
      const int n = n_top - w;
      const uint32_t* pat = sm.ctx + (cap - n);
      const uint32_t t0 = pat[0];
      uint32_t lo = __ldg(ds.bucket + t0), hi = __ldg(ds.bucket + t0 + 1);
      // invariant: the bound (first index whose suffix is >= the pattern, or >
      // it for the upper bound) lies in [lo, hi], hi meaning "none below hi"
      while (__any_sync(0xFFFFFFFFu, lo < hi)) {
        const bool active = lo < hi;
        const uint32_t piv = lo + (uint32_t)(((uint64_t)(hl + 1) * (hi - lo)) / 17u);
        bool pred = true;  // suffix at piv is past the bound's side
        if (active) {
          uint32_t at = 0;
          const int c = ds.keys ? cmp_suffix_key(ds.keys, T, N, piv, pat, n, &at)
                                : cmp_suffix_vec(T, N, (at = __ldg(ds.sa + piv)), pat, n);
          FC_DEBUG_CHECK(at < N);
          pred = upper ? (c > 0) : (c >= 0);
        }
        const unsigned bal = __ballot_sync(0xFFFFFFFFu, !pred) & half_mask;
        const int t = __popc(bal);  // pivots before the bound (a prefix of the half-warp)
        const int base_lane = upper ? 16 : 0;
        const uint32_t p_before = __shfl_sync(0xFFFFFFFFu, piv, base_lane + max(t - 1, 0));
        const uint32_t p_at = __shfl_sync(0xFFFFFFFFu, piv, base_lane + min(t, 15));
        if (active) {
          if (t > 0) lo = p_before + 1;
          if (t < 16) hi = p_at;
        }
      }
      if (hl == 0) {
        if (upper) {
          sm.hi[n] = lo;
        } else {
          sm.lo[n] = lo;
          // the suffix that is exactly the pattern at the corpus end sorts first in its range
          sm.endhit[n] = (lo < N && (uint64_t)__ldg(ds.sa + lo) + n == N) ? 1u : 0u;
        }
      }
    }
  }
  __syncthreads();
  if (tid == 0) {
    uint32_t ns = 0, first = 0, cnt = 0;
    if (npairs) {
      for (int n = n_top; n > n_top - n_count; --n) {
        uint32_t l = sm.lo[n], h = sm.hi[n];
        if (l < h && sm.endhit[n]) ++l;
        if (l < h) {
          ns = n;
          first = l;
          cnt = h - l;
          break;
        }
      }
    }
    sm.n_star = ns;
    sm.first = first;
    sm.cnt = min(cnt, p.max_occ);
  }
  __syncthreads();
  const int ns = (int)sm.n_star;
  uint32_t* dr = o.drafts + sb * k * d;
  int32_t* dl = o.draft_len + sb * k;
  uint32_t* ct = o.count + sb * k;
  if (ns == 0) {
    for (int e = tid; e < k * d; e += RT_THREADS) dr[e] = FC_PAD_TOKEN;
    for (int e = tid; e < k; e += RT_THREADS) {
      dl[e] = 0;
      ct[e] = 0;
    }
    if (tid == 0) {
      o.n_drafts[sb] = 0;
      o.match_len[sb] = 0;
    }
    return;
  }
  const uint32_t nocc = sm.cnt, first = sm.first;

  // ---- runs of equal continuations -------------------------------------
  // neighbours j-1, j share their continuation iff lcp[j] >= n* + d
  const uint32_t need = (uint32_t)ns + (uint32_t)d;
  for (uint32_t e = tid; e < nocc; e += RT_THREADS)
    sm.work[e] = (e == 0 || (uint32_t)__ldg(ds.lcp + first + e) < need) ? 1u : 0u;
  __syncthreads();
  uint32_t nd_sel;
  if constexpr (ALL)
    nd_sel = runs_from_heads<RT_THREADS>(nocc, sm.runs, sm.work, sm.wsum, sm.rs);
  else
    nd_sel = rank_runs<RT_THREADS>(nocc, k, sm.runs, sm.work, sm.sel, sm.order, sm.wsum, sm.rs);
  auto run_count = [&](uint32_t r) { return sm.runs[r + 1] - sm.runs[r]; };
  auto run_at = [&](int t) -> uint32_t { return ALL ? (uint32_t)t : sm.order[t]; };  // the run in output slot t
  // ---- outputs ---------------------------------------------------------
  const int nd = (int)nd_sel;
  for (int e = tid; e < k * d; e += RT_THREADS) {
    int t = e / d, x = e - t * d;
    uint32_t v = FC_PAD_TOKEN;
    if (t < nd) {
      const uint64_t pp = (uint64_t)__ldg(ds.sa + first + sm.runs[run_at(t)]) + (uint64_t)ns;
      if (FC_DEBUG_CHECK(pp < N)) {
        const uint64_t len = min((uint64_t)d, N - pp);
        if ((uint64_t)x < len) v = __ldg(T + pp + x);
      }
    }
    dr[e] = v;
  }
  for (int t = tid; t < k; t += RT_THREADS) {
    if (t < nd) {
      const uint32_t r = run_at(t);
      const uint64_t pp = (uint64_t)__ldg(ds.sa + first + sm.runs[r]) + (uint64_t)ns;
      dl[t] = pp < N ? (int32_t)min((uint64_t)d, N - pp) : 0;
      ct[t] = run_count(r);
    } else {
      dl[t] = 0;
      ct[t] = 0;
    }
  }
  if (tid == 0) {
    o.n_drafts[sb] = nd;
    o.match_len[sb] = ns;
  }
}

bool params_ok(const fc_retrieve_params& p) { return fc_retrieve_params_ok(p); }

__global__ void k_rc_init(uint32_t* table, int capacity, size_t entry_words) {
  for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < (size_t)capacity;
       e += (size_t)gridDim.x * blockDim.x)
    table[e * entry_words] = RC_EMPTY;
}

__global__ void k_rc_lookup(const uint32_t* __restrict__ table, int capacity, int S, fc_retrieve_params p,
                            const uint32_t* __restrict__ ctx, int stride, const int32_t* __restrict__ ctx_len,
                            int B, const int32_t* __restrict__ want, int32_t* __restrict__ skip, RetOut o) {
  __shared__ RcSmem sm;
  const int b = blockIdx.x;
  rc_load_key(sm, ctx, stride, ctx_len, b, p.n_max);
  const size_t ew = rc_entry_words(S, p);
  if (threadIdx.x < 32) {  // warp 0 probes; every lane takes the same path
    const int lane = threadIdx.x;
    const int slot = (!want || want[b]) ? rc_find_warp(table, capacity, ew, sm.key, sm.klen, lane) : -1;
    if (lane == 0) {
      sm.slot = slot;
      skip[b] = slot >= 0 ? 1 : 0;
    }
  }
  __syncthreads();
  if (sm.slot < 0) return;
  rc_copy<true>(const_cast<uint32_t*>(table) + (size_t)sm.slot * ew + 1 + p.n_max, o, S, p, B, b);
}

__global__ void k_rc_insert(uint32_t* table, int capacity, int S, fc_retrieve_params p,
                            const uint32_t* __restrict__ ctx, int stride, const int32_t* __restrict__ ctx_len, int B,
                            const int32_t* __restrict__ skip, RetOut o) {
  __shared__ RcSmem sm;
  const int b = blockIdx.x;
  if (skip && skip[b]) return;
  rc_load_key(sm, ctx, stride, ctx_len, b, p.n_max);
  const size_t ew = rc_entry_words(S, p);
  if (threadIdx.x < 32) {  // warp 0 probes: lane 0 claims, the warp compares keys
    const int lane = threadIdx.x;
    int slot = -1;
    bool present = false;
    const uint64_t h = rc_hash(sm.key, sm.klen);
    for (int probe = 0; probe < capacity && slot < 0 && !present; ++probe) {
      const size_t e = (h + probe) & (uint64_t)(capacity - 1);
      uint32_t* ent = table + e * ew;
      uint32_t st = 0;
      if (lane == 0) st = atomicCAS(ent, RC_EMPTY, RC_CLAIMED);
      st = __shfl_sync(0xFFFFFFFFu, st, 0);
      if (st == RC_EMPTY) {
        slot = (int)e;
      } else if (st != RC_CLAIMED && rc_key_equal_warp(ent, st, sm.key, sm.klen, lane)) {
        present = true;  // an equal key holds the same (deterministic) result
      }
    }
    if (lane == 0) {
      if (slot < 0 && !present) fc_flag(FC_ERR_WORD(o.err), FC_EBIT_CAPACITY);
      sm.slot = slot;
    }
  }
  __syncthreads();
  if (sm.slot < 0) return;
  uint32_t* ent = table + (size_t)sm.slot * ew;
  for (int i = threadIdx.x; i < sm.klen; i += blockDim.x) ent[1 + i] = sm.key[i];
  rc_copy<false>(ent + 1 + p.n_max, o, S, p, B, b);
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) atomicExch(ent, (uint32_t)sm.klen);
}

}  // namespace

static fc_status launch_retrieve(bool all, const fc_datastore* sources, const fc_datastore* rev_sources, int n_sources,
                                 const uint32_t* d_ctx, int ctx_stride, const int32_t* d_ctx_len, int batch,
                                 const int32_t* d_skip, fc_retrieve_params p, uint32_t* d_drafts,
                                 int32_t* d_draft_len, uint32_t* d_count, int32_t* d_n_drafts, int32_t* d_match_len,
                                 fc_stream stream, RcFused rc = RcFused{nullptr, 0, nullptr, nullptr}) {
  if (!sources || n_sources < 1 || n_sources > FC_MAX_SOURCES || batch < 0 || ctx_stride < 1 ||
      batch > 65535 * 16)
    return FC_ERR_INVALID_ARG;
  if (!params_ok(p)) return (p.n_max > 0 && p.top_k > 0 && p.draft_len > 0) ? FC_ERR_UNSUPPORTED : FC_ERR_INVALID_ARG;
  if (batch == 0) return FC_OK;
  if (!d_ctx || !d_ctx_len || !d_drafts || !d_draft_len || !d_count || !d_n_drafts || !d_match_len)
    return FC_ERR_INVALID_ARG;
  DsArgs a{};
  for (int s = 0; s < n_sources; ++s) {
    const fc_datastore& ds = sources[s];
    if (!ds.tokens || !ds.sa || !ds.bucket || !ds.lcp || ds.n_tokens == 0 || ds.n_tokens >= 0xFFFFFFFFull ||
        ds.vocab == 0)
      return FC_ERR_INVALID_ARG;
    if (reinterpret_cast<uintptr_t>(ds.tokens) % 16) return FC_ERR_INVALID_ARG;  // read as 16-byte vectors
    if (reinterpret_cast<uintptr_t>(ds.keys) % 32) return FC_ERR_INVALID_ARG;
    a.ds[s] = DsView{ds.tokens, ds.sa, ds.bucket, ds.lcp, ds.n_tokens, ds.vocab,
                     reinterpret_cast<const uint4*>(ds.keys)};
  }
  DsArgs r{};
  if (rev_sources) {
    for (int s = 0; s < n_sources; ++s) {
      const fc_datastore& rv = rev_sources[s];
      if (!rv.tokens || !rv.sa || !rv.bucket || rv.n_tokens != sources[s].n_tokens || rv.vocab != sources[s].vocab)
        return FC_ERR_INVALID_ARG;
      r.ds[s] = DsView{rv.tokens, rv.sa, rv.bucket, rv.lcp, rv.n_tokens, rv.vocab, nullptr};
    }
  }
  const int variant = all ? 2 : (rev_sources ? 1 : 0);
  auto kern = all ? k_retrieve<false, true> : (rev_sources ? k_retrieve<true, false> : k_retrieve<false, false>);
  static std::atomic<unsigned long long> attr_done[3];
  const fc_status st = fc_once_per_device(attr_done[variant], [&](int) {
    return fc_cuda_status(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sizeof(RetSmem)));
  });
  if (st != FC_OK) return st;
  RetOut o{d_drafts, d_draft_len, d_count, d_n_drafts, d_match_len, fc_error_slot()};
  dim3 grid((unsigned)batch, (unsigned)n_sources);
  kern<<<grid, RT_THREADS, sizeof(RetSmem), static_cast<cudaStream_t>(stream)>>>(a, r, d_ctx, ctx_stride, d_ctx_len,
                                                                                 batch, d_skip, p, o, rc);
  return FC_CHECK_LAUNCH();
}

extern "C" fc_status fc_retrieve(const fc_datastore* sources, int n_sources, const uint32_t* d_ctx, int ctx_stride,
                                 const int32_t* d_ctx_len, int batch, const int32_t* d_skip, fc_retrieve_params p,
                                 uint32_t* d_drafts, int32_t* d_draft_len, uint32_t* d_count, int32_t* d_n_drafts,
                                 int32_t* d_match_len, fc_stream stream) {
  FC_NVTX_RANGE();
  return launch_retrieve(false, sources, nullptr, n_sources, d_ctx, ctx_stride, d_ctx_len, batch, d_skip, p, d_drafts,
                         d_draft_len, d_count, d_n_drafts, d_match_len, stream);
}

extern "C" fc_status fc_retrieve_all(const fc_datastore* sources, int n_sources, const uint32_t* d_ctx,
                                     int ctx_stride, const int32_t* d_ctx_len, int batch, const int32_t* d_skip,
                                     fc_retrieve_params p, uint32_t* d_drafts, int32_t* d_draft_len,
                                     uint32_t* d_count, int32_t* d_n_drafts, int32_t* d_match_len, fc_stream stream) {
  FC_NVTX_RANGE();
  return launch_retrieve(true, sources, nullptr, n_sources, d_ctx, ctx_stride, d_ctx_len, batch, d_skip, p, d_drafts,
                         d_draft_len, d_count, d_n_drafts, d_match_len, stream);
}

extern "C" fc_status fc_retrieve_rev(const fc_datastore* sources, const fc_datastore* rev_sources, int n_sources,
                                     const uint32_t* d_ctx, int ctx_stride, const int32_t* d_ctx_len, int batch,
                                     const int32_t* d_skip, fc_retrieve_params p, uint32_t* d_drafts,
                                     int32_t* d_draft_len, uint32_t* d_count, int32_t* d_n_drafts,
                                     int32_t* d_match_len, fc_stream stream) {
  FC_NVTX_RANGE();
  if (!rev_sources) return FC_ERR_INVALID_ARG;
  return launch_retrieve(false, sources, rev_sources, n_sources, d_ctx, ctx_stride, d_ctx_len, batch, d_skip, p, d_drafts,
                         d_draft_len, d_count, d_n_drafts, d_match_len, stream);
}

extern "C" size_t fc_rcache_bytes(int capacity, int n_sources, fc_retrieve_params p) {
  if (capacity < 1 || n_sources < 1 || n_sources > FC_MAX_SOURCES || !params_ok(p)) return 0;
  return (size_t)capacity * rc_entry_words(n_sources, p) * 4;
}

static bool rc_args_ok(int capacity, int n_sources, const fc_retrieve_params& p) {
  return capacity >= 1 && capacity <= (1 << 24) && (capacity & (capacity - 1)) == 0 && n_sources >= 1 &&
         n_sources <= FC_MAX_SOURCES && params_ok(p);
}

extern "C" fc_status fc_rcache_init(void* d_table, size_t bytes, int capacity, int n_sources, fc_retrieve_params p,
                                    fc_stream stream) {
  FC_NVTX_RANGE();
  if (!d_table || !rc_args_ok(capacity, n_sources, p)) return FC_ERR_INVALID_ARG;
  if (bytes < fc_rcache_bytes(capacity, n_sources, p)) return FC_ERR_WORKSPACE;
  unsigned g = (unsigned)std::min<size_t>((capacity + 255) / 256, 4096);
  k_rc_init<<<g, 256, 0, static_cast<cudaStream_t>(stream)>>>(static_cast<uint32_t*>(d_table), capacity,
                                                              rc_entry_words(n_sources, p));
  return FC_CHECK_LAUNCH();
}

extern "C" fc_status fc_rcache_lookup(const void* d_table, int capacity, int n_sources, fc_retrieve_params p,
                                      const uint32_t* d_ctx, int ctx_stride, const int32_t* d_ctx_len, int batch,
                                      const int32_t* d_want_hit, int32_t* d_skip, uint32_t* d_drafts,
                                      int32_t* d_draft_len, uint32_t* d_count, int32_t* d_n_drafts,
                                      int32_t* d_match_len, fc_stream stream) {
  FC_NVTX_RANGE();
  if (!d_table || !rc_args_ok(capacity, n_sources, p) || batch < 0 || ctx_stride < 1) return FC_ERR_INVALID_ARG;
  if (batch == 0) return FC_OK;
  if (!d_ctx || !d_ctx_len || !d_skip || !d_drafts || !d_draft_len || !d_count || !d_n_drafts || !d_match_len)
    return FC_ERR_INVALID_ARG;
  RetOut o{d_drafts, d_draft_len, d_count, d_n_drafts, d_match_len, fc_error_slot()};
  k_rc_lookup<<<batch, 128, 0, static_cast<cudaStream_t>(stream)>>>(static_cast<const uint32_t*>(d_table), capacity,
                                                                     n_sources, p, d_ctx, ctx_stride, d_ctx_len, batch,
                                                                     d_want_hit, d_skip, o);
  return FC_CHECK_LAUNCH();
}

extern "C" fc_status fc_retrieve_cached(const fc_datastore* sources, int n_sources, const uint32_t* d_ctx,
                                        int ctx_stride, const int32_t* d_ctx_len, int batch, const void* d_table,
                                        int capacity, const int32_t* d_want_hit, int32_t* d_skip,
                                        fc_retrieve_params p, uint32_t* d_drafts, int32_t* d_draft_len,
                                        uint32_t* d_count, int32_t* d_n_drafts, int32_t* d_match_len,
                                        fc_stream stream) {
  FC_NVTX_RANGE();
  if (!d_table || !rc_args_ok(capacity, n_sources, p) || (batch > 0 && !d_skip)) return FC_ERR_INVALID_ARG;
  return launch_retrieve(false, sources, nullptr, n_sources, d_ctx, ctx_stride, d_ctx_len, batch, nullptr, p, d_drafts,
                         d_draft_len, d_count, d_n_drafts, d_match_len, stream,
                         RcFused{static_cast<const uint32_t*>(d_table), capacity, d_want_hit, d_skip});
}

extern "C" fc_status fc_rcache_insert(void* d_table, int capacity, int n_sources, fc_retrieve_params p,
                                      const uint32_t* d_ctx, int ctx_stride, const int32_t* d_ctx_len, int batch,
                                      const int32_t* d_skip, const uint32_t* d_drafts, const int32_t* d_draft_len,
                                      const uint32_t* d_count, const int32_t* d_n_drafts, const int32_t* d_match_len,
                                      fc_stream stream) {
  FC_NVTX_RANGE();
  if (!d_table || !rc_args_ok(capacity, n_sources, p) || batch < 0 || ctx_stride < 1) return FC_ERR_INVALID_ARG;
  if (batch == 0) return FC_OK;
  if (!d_ctx || !d_ctx_len || !d_drafts || !d_draft_len || !d_count || !d_n_drafts || !d_match_len)
    return FC_ERR_INVALID_ARG;
  RetOut o{const_cast<uint32_t*>(d_drafts), const_cast<int32_t*>(d_draft_len), const_cast<uint32_t*>(d_count),
           const_cast<int32_t*>(d_n_drafts), const_cast<int32_t*>(d_match_len), fc_error_slot()};
  k_rc_insert<<<batch, 128, 0, static_cast<cudaStream_t>(stream)>>>(static_cast<uint32_t*>(d_table), capacity,
                                                                     n_sources, p, d_ctx, ctx_stride, d_ctx_len, batch,
                                                                     d_skip, o);
  return FC_CHECK_LAUNCH();
}
