// CPU oracle for the FastCoder retrieve-and-verify step (arXiv 2502.17139).
//
// TEST INFRASTRUCTURE ONLY.  This file is the slow, plain, obviously-correct
// statement of what the step computes.  It is used by the test suite, by
// __graft_entry__.smoke() and by the CPU-baseline leg of bench.py, and by
// nothing else.  It shares no code, header, table or helper with the CUDA
// path under paper_2502_17139_gb300/, and it does not include anything from
// there.
//
// Each function cites the passage of the paper it follows.  Where the paper
// is silent the function states the reading it takes.  Every function is
// pinned by the tests in tests/test_oracle_*.py against brute force,
// closed forms, invariants or library routines.
//
// Conventions shared with the public C ABI (these are interface facts, not
// code): token ids are uint32 < vocab; PAD = 0xFFFFFFFF pads draft slots;
// bf16 values are passed as their raw uint16 bit patterns.

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <map>
#include <thread>
#include <vector>

namespace {

const uint32_t kPad = 0xFFFFFFFFu;

int resolve_threads(int nthreads) {
  if (nthreads > 0) return nthreads;
  unsigned h = std::thread::hardware_concurrency();
  return h ? (int)h : 1;
}

// Run f(i) for i in [0, n) on up to nthreads threads (static interleave).
template <class F>
void parallel_for(int64_t n, int nthreads, F f) {
  nthreads = resolve_threads(nthreads);
  if (nthreads <= 1 || n <= 1) {
    for (int64_t i = 0; i < n; ++i) f(i);
    return;
  }
  std::vector<std::thread> pool;
  std::atomic<int64_t> next(0);
  for (int t = 0; t < nthreads; ++t) {
    pool.emplace_back([&]() {
      for (;;) {
        int64_t i = next.fetch_add(1);
        if (i >= n) break;
        f(i);
      }
    });
  }
  for (auto& th : pool) th.join();
}

// Lexicographic comparison of the suffixes T[a..N) and T[b..N) as uint32
// strings.  A suffix that is a proper prefix of the other is the smaller one
// (the end of the corpus sorts before every token).
bool suffix_less(const uint32_t* T, uint64_t N, uint64_t a, uint64_t b) {
  if (a == b) return false;
  uint64_t i = a, j = b;
  while (i < N && j < N) {
    if (T[i] != T[j]) return T[i] < T[j];
    ++i;
    ++j;
  }
  return i == N && j < N;  // a ran out first -> a is a proper prefix of b
}

double bf16_to_double(uint16_t h) {
  uint32_t bits = (uint32_t)h << 16;
  float f;
  std::memcpy(&f, &bits, sizeof f);
  return (double)f;
}

}  // namespace

extern "C" {

// ---------------------------------------------------------------------------
// O1. Suffix array (Section III-A: retrieval is a suffix match over a
// datastore of context/continuation pairs; Section IV-A, Eq. 1-2: every
// position of every file splits into a context and a continuation, organised
// as in REST, i.e. a suffix array over the token corpus).
//
// sa = the permutation of [0, N) that sorts the suffixes T[i..N).  Method: a
// plain comparison sort with the suffix comparator above, split over threads
// and merged.
// ---------------------------------------------------------------------------
int orc_suffix_array(const uint32_t* T, uint64_t N, uint32_t* sa, int nthreads) {
  std::vector<uint32_t> idx(N);
  for (uint64_t i = 0; i < N; ++i) idx[i] = (uint32_t)i;
  auto less = [&](uint32_t a, uint32_t b) { return suffix_less(T, N, a, b); };
  int nt = resolve_threads(nthreads);
  if (N < 100000 || nt == 1) {
    std::sort(idx.begin(), idx.end(), less);
  } else {
    int parts = 1;
    while (parts * 2 <= nt) parts *= 2;
    std::vector<uint64_t> cut(parts + 1);
    for (int p = 0; p <= parts; ++p) cut[p] = N * (uint64_t)p / (uint64_t)parts;
    parallel_for(parts, parts, [&](int64_t p) {
      std::sort(idx.begin() + cut[p], idx.begin() + cut[p + 1], less);
    });
    for (int width = 1; width < parts; width *= 2) {
      int pairs = parts / (2 * width);
      parallel_for(pairs, pairs, [&](int64_t q) {
        uint64_t lo = cut[2 * width * q], mid = cut[2 * width * q + width], hi = cut[2 * width * (q + 1)];
        std::inplace_merge(idx.begin() + lo, idx.begin() + mid, idx.begin() + hi, less);
      });
    }
  }
  std::memcpy(sa, idx.data(), N * sizeof(uint32_t));
  return 0;
}

// First-token bucket table: bucket[v] = the first SA index whose suffix starts
// with a token >= v, bucket[vocab] = N.  (An index over the SA, not a step of
// the paper; it narrows the suffix search by the pattern's first token.)
int orc_bucket(const uint32_t* T, uint64_t N, const uint32_t* sa, uint32_t vocab, uint32_t* bucket) {
  uint64_t j = 0;
  for (uint64_t v = 0; v <= vocab; ++v) {
    while (j < N && T[sa[j]] < v) ++j;
    bucket[v] = (uint32_t)(v == vocab ? N : j);
  }
  return 0;
}

// Longest common prefix of each suffix with its predecessor in SA order,
// capped: lcp[j] = LCP(T[sa[j-1]..N), T[sa[j]..N)) limited to cap, lcp[0] = 0.
// (An index over the SA that lets equal continuations be grouped without
// reading them; its values follow from the definition directly.)
int orc_lcp(const uint32_t* T, uint64_t N, const uint32_t* sa, uint32_t cap, uint8_t* lcp) {
  if (N == 0) return 0;
  lcp[0] = 0;
  for (uint64_t j = 1; j < N; ++j) {
    uint64_t a = sa[j - 1], b = sa[j], l = 0;
    while (l < cap && a + l < N && b + l < N && T[a + l] == T[b + l]) ++l;
    lcp[j] = (uint8_t)l;
  }
  return 0;
}

// Certificate that sa is the suffix array of T, usable at any size:
// sa is a permutation of [0, N) and suffix(sa[j]) < suffix(sa[j+1]) for all j.
// Returns -1 when valid; otherwise the first offending SA index (or N when
// sa is not a permutation).
int64_t orc_sa_certificate(const uint32_t* T, uint64_t N, const uint32_t* sa, int nthreads) {
  std::vector<uint8_t> seen(N, 0);
  for (uint64_t j = 0; j < N; ++j) {
    if (sa[j] >= N || seen[sa[j]]) return (int64_t)N;
    seen[sa[j]] = 1;
  }
  if (N < 2) return -1;
  int nt = resolve_threads(nthreads);
  std::vector<int64_t> bad(nt, -1);
  int64_t chunks = nt * 8;
  std::vector<int64_t> first_bad(chunks, -1);
  parallel_for(chunks, nt, [&](int64_t c) {
    uint64_t lo = (N - 1) * (uint64_t)c / (uint64_t)chunks;
    uint64_t hi = (N - 1) * (uint64_t)(c + 1) / (uint64_t)chunks;
    for (uint64_t j = lo; j < hi; ++j) {
      if (!suffix_less(T, N, sa[j], sa[j + 1])) {
        first_bad[c] = (int64_t)j;
        return;
      }
    }
  });
  for (int64_t c = 0; c < chunks; ++c)
    if (first_bad[c] >= 0) return first_bad[c];
  return -1;
}

// ---------------------------------------------------------------------------
// O2-O4. Retrieval (Section III-A; Section IV-C, Algorithm 1 par_search;
// Section V-C: n_max = 16).
//
// For a context c of length m, try suffix lengths n from min(n_max, m) down to
// n_min: the pattern q is the last n tokens of c; the datastore has a match
// when q occurs in the corpus immediately before some position p with
// p <= N-1 (so that at least one continuation token follows).  The first n
// (the longest) with a match is n*.  Readings where the paper is silent:
//   * n stops at n_min (the paper only says "decreased by one");
//   * an occurrence that ends at the corpus end has no continuation and does
//     not count;
//   * when the match has more than max_occ occurrences, the max_occ whose
//     windows T[p-n*, min(p+d, N)) are lexicographically smallest are kept
//     (max_occ = 0 keeps all);
//   * the "top-k high-frequency" candidates are the distinct continuations
//     u(p) = T[p, min(p+d, N)) (length is part of identity), ranked by count
//     descending, then by token ids ascending (a prefix before its
//     extensions).
//
// Method: one linear scan of the corpus per context computing, at every p,
// the length of the common suffix of T[0..p) and c (capped at n_max), then a
// second scan collecting the occurrences of n*, then std::map counting.
//
// Outputs per query b: drafts[b][k][d] (PAD beyond a draft's length and for
// absent drafts), draft_len[b][k], count[b][k] (0 for absent drafts),
// n_drafts[b], match_len[b] (= n*, 0 for no match).
// ---------------------------------------------------------------------------
int orc_retrieve(const uint32_t* T, uint64_t N, const uint32_t* ctx, int ctx_stride,
                 const int32_t* ctx_len, int B, int n_max, int n_min, int top_k, int d,
                 uint32_t max_occ, uint32_t* drafts, int32_t* draft_len, uint32_t* count,
                 int32_t* n_drafts, int32_t* match_len, int nthreads) {
  if (n_min < 1 || n_max < n_min || top_k < 1 || d < 1) return 1;
  parallel_for(B, nthreads, [&](int64_t b) {
    const uint32_t* c = ctx + (size_t)b * ctx_stride;
    int m = ctx_len[b];
    uint32_t* dr = drafts + (size_t)b * top_k * d;
    int32_t* dl = draft_len + (size_t)b * top_k;
    uint32_t* ct = count + (size_t)b * top_k;
    for (int i = 0; i < top_k * d; ++i) dr[i] = kPad;
    for (int i = 0; i < top_k; ++i) { dl[i] = 0; ct[i] = 0; }
    n_drafts[b] = 0;
    match_len[b] = 0;
    int cap = std::min(n_max, m);
    if (cap < n_min || N < 2) return;
    // Scan 1: the longest common suffix ending right before p, p in [1, N-1].
    int best = 0;
    for (uint64_t p = 1; p + 1 <= N; ++p) {
      int k = 0;
      while (k < cap && (uint64_t)k < p && T[p - 1 - k] == c[m - 1 - k]) ++k;
      if (k > best) best = k;
    }
    if (best < n_min) return;
    int ns = best;
    // Scan 2: every occurrence of the n*-token pattern with a continuation.
    std::vector<uint64_t> occ;
    for (uint64_t p = (uint64_t)ns; p + 1 <= N; ++p) {
      bool eq = true;
      for (int k = 0; k < ns && eq; ++k) eq = (T[p - ns + k] == c[m - ns + k]);
      if (eq) occ.push_back(p);
    }
    auto cont = [&](uint64_t p) {
      uint64_t e = std::min<uint64_t>(p + (uint64_t)d, N);
      return std::vector<uint32_t>(T + p, T + e);
    };
    if (max_occ > 0 && occ.size() > max_occ) {
      // All windows share their first n* tokens, so ordering the windows is
      // ordering the continuations (shorter-is-smaller).
      std::stable_sort(occ.begin(), occ.end(), [&](uint64_t a, uint64_t b2) { return cont(a) < cont(b2); });
      occ.resize(max_occ);
    }
    std::map<std::vector<uint32_t>, uint32_t> freq;
    for (uint64_t p : occ) freq[cont(p)] += 1;
    std::vector<std::pair<uint32_t, std::vector<uint32_t>>> ranked;
    for (auto& kv : freq) ranked.push_back({kv.second, kv.first});
    std::stable_sort(ranked.begin(), ranked.end(), [](const auto& x, const auto& y) {
      if (x.first != y.first) return x.first > y.first;
      return x.second < y.second;
    });
    int nd = (int)std::min<size_t>(ranked.size(), (size_t)top_k);
    for (int t = 0; t < nd; ++t) {
      const auto& seq = ranked[t].second;
      for (size_t i = 0; i < seq.size(); ++i) dr[(size_t)t * d + i] = seq[i];
      dl[t] = (int32_t)seq.size();
      ct[t] = ranked[t].first;
    }
    n_drafts[b] = nd;
    match_len[b] = ns;
  });
  return 0;
}

// ---------------------------------------------------------------------------
// O5. Draft tree (Section IV-D, Eq. 3 node weight alpha*t_r + beta*t_c; the
// tree mask of Eq. 4; position ids by depth; Section V-C: alpha = beta = 1 and
// at most 64 draft tokens).
//
// The drafts of all S sources are merged: a draft u found in source s with
// count c_s(u) gets weight w(u) = sum_s weight[s] * c_s(u) (integer weights).
// A pointer trie rooted at root_tok (the last context token, whose K/V is not
// yet cached) receives every draft; a node's weight W is the sum of w(u) over
// the drafts passing through it.  Readings where the paper is silent:
//   * the budget counts the root; the root plus the (budget - 1) non-root
//     nodes ranked by (W descending, depth ascending, token path ascending)
//     are kept (a prefix-closed set because W(parent) >= W(child));
//   * nodes are emitted in depth-first preorder with children in ascending
//     token order, so parent[i] < i;
//   * mask row i has bit j set iff j is an ancestor of i or i itself (a
//     chain then reduces to causal attention);
//   * pos[i] = kv_len + depth[i].
// Padding rows (i >= n_nodes): tok = PAD, parent = -1, depth = -1, pos = -1,
// mask = 0.
// ---------------------------------------------------------------------------
namespace {
struct TrieNode {
  uint32_t tok = 0;
  int depth = 0;
  int parent = -1;
  uint64_t W = 0;
  std::vector<uint32_t> path;          // tokens from the root's child down to this node
  std::map<uint32_t, int> children;    // token -> node index (ascending)
  bool keep = false;
};
}  // namespace

int orc_build_tree(int S, const uint32_t* drafts, const int32_t* draft_len, const uint32_t* count,
                   const int32_t* n_drafts, const uint32_t* src_weight, int B, int top_k, int d,
                   const uint32_t* root_tok, const int32_t* kv_len, int budget, int n_pad,
                   uint32_t* tok, int32_t* parent, int32_t* depth, int32_t* pos, uint64_t* mask,
                   int32_t* n_nodes, int nthreads) {
  if (budget < 1 || budget > n_pad) return 1;
  int nw = (n_pad + 63) / 64;
  parallel_for(B, nthreads, [&](int64_t b) {
    std::map<std::vector<uint32_t>, uint64_t> w;
    for (int s = 0; s < S; ++s) {
      size_t sb = (size_t)s * B + b;
      for (int t = 0; t < n_drafts[sb]; ++t) {
        int len = draft_len[sb * top_k + t];
        if (len <= 0) continue;
        const uint32_t* u = drafts + (sb * top_k + t) * d;
        w[std::vector<uint32_t>(u, u + len)] += (uint64_t)src_weight[s] * count[sb * top_k + t];
      }
    }
    std::vector<TrieNode> nodes(1);
    nodes[0].tok = root_tok[b];
    for (auto& kv : w) {
      int cur = 0;
      nodes[0].W += kv.second;
      for (uint32_t x : kv.first) {
        auto it = nodes[cur].children.find(x);
        int nxt;
        if (it == nodes[cur].children.end()) {
          TrieNode nn;
          nn.tok = x;
          nn.depth = nodes[cur].depth + 1;
          nn.parent = cur;
          nn.path = nodes[cur].path;
          nn.path.push_back(x);
          nxt = (int)nodes.size();
          nodes[cur].children[x] = nxt;
          nodes.push_back(nn);
        } else {
          nxt = it->second;
        }
        nodes[nxt].W += kv.second;
        cur = nxt;
      }
    }
    std::vector<int> cand;
    for (int i = 1; i < (int)nodes.size(); ++i) cand.push_back(i);
    std::sort(cand.begin(), cand.end(), [&](int x, int y) {
      if (nodes[x].W != nodes[y].W) return nodes[x].W > nodes[y].W;
      if (nodes[x].depth != nodes[y].depth) return nodes[x].depth < nodes[y].depth;
      return nodes[x].path < nodes[y].path;
    });
    nodes[0].keep = true;
    for (int r = 0; r < (int)cand.size() && r < budget - 1; ++r) nodes[cand[r]].keep = true;
    // Depth-first preorder over kept nodes, children ascending by token.
    std::vector<int> order;
    std::vector<int> stack{0};
    while (!stack.empty()) {
      int v = stack.back();
      stack.pop_back();
      order.push_back(v);
      for (auto it = nodes[v].children.rbegin(); it != nodes[v].children.rend(); ++it)
        if (nodes[it->second].keep) stack.push_back(it->second);
    }
    std::vector<int> out_id(nodes.size(), -1);
    for (int i = 0; i < (int)order.size(); ++i) out_id[order[i]] = i;
    size_t base = (size_t)b * n_pad;
    for (int i = 0; i < n_pad; ++i) {
      tok[base + i] = kPad;
      parent[base + i] = -1;
      depth[base + i] = -1;
      pos[base + i] = -1;
      for (int q = 0; q < nw; ++q) mask[(base + i) * nw + q] = 0;
    }
    for (int i = 0; i < (int)order.size(); ++i) {
      const TrieNode& nd = nodes[order[i]];
      tok[base + i] = nd.tok;
      parent[base + i] = nd.parent < 0 ? -1 : out_id[nd.parent];
      depth[base + i] = nd.depth;
      pos[base + i] = kv_len[b] + nd.depth;
      // ancestors-or-self, walking up the pointer trie
      for (int a = order[i]; a >= 0; a = nodes[a].parent) {
        int j = out_id[a];
        mask[(base + i) * nw + j / 64] |= (uint64_t)1 << (j % 64);
      }
    }
    n_nodes[b] = (int32_t)order.size();
  });
  return 0;
}

// Tree mask, depth and position ids from parent pointers alone (Eq. 4 and the
// position adjustment of Section IV-D), for trees given as (parent[], n_nodes)
// in the layout above.  Returns 1 if some parent[i] is not in [0, i).
int orc_tree_mask(const int32_t* parent, const int32_t* n_nodes, const int32_t* kv_len, int B,
                  int n_pad, int32_t* depth, int32_t* pos, uint64_t* mask) {
  int nw = (n_pad + 63) / 64;
  for (int b = 0; b < B; ++b) {
    size_t base = (size_t)b * n_pad;
    for (int i = 0; i < n_pad; ++i) {
      depth[base + i] = -1;
      pos[base + i] = -1;
      for (int q = 0; q < nw; ++q) mask[(base + i) * nw + q] = 0;
    }
    for (int i = 0; i < n_nodes[b]; ++i) {
      int dd = 0;
      for (int a = i; a >= 0; a = (a == 0 ? -1 : parent[base + a])) {
        if (a > 0 && (parent[base + a] < 0 || parent[base + a] >= a)) return 1;
        mask[(base + i) * nw + a / 64] |= (uint64_t)1 << (a % 64);
        if (a != i) ++dd;
      }
      depth[base + i] = dd;
      pos[base + i] = kv_len[b] + dd;
    }
  }
  return 0;
}

// ---------------------------------------------------------------------------
// O6. Tree attention (Section IV-D, Eq. 4).  For sequence b, query head h and
// tree node i < n_nodes[b], with kv head g = h / (H / Hkv):
//   keys  = every cached key K_cache[b, g, 0..kv_len) and every tree key
//           K_tree[b, g, j] with mask[i] bit j set;
//   s     = scale * (q . k) in double precision from the exact bf16 values;
//   out   = sum softmax(s) * v.
// Rows i >= n_nodes[b] are zero.  Q and K are taken as already rotated by the
// caller (position encoding is outside this operation); orc_tree_attn_rope
// below is the same attention with the rotation of O12 applied to the
// queries and the tree keys.
//
// rows == nullptr: every (b, i, h) is computed into out[B][n_pad][H][D].
// Otherwise rows holds n_rows triples (b, i, h) and out is [n_rows][D].
// ---------------------------------------------------------------------------
}  // extern "C"

namespace {

// O12. Rotary position embedding (Su et al., "RoFormer", 2021): dimension
// pairs are rotated by pos * f_i with f_i = base^(-2i/D).  The pairing is the
// rotate-half one of the LLaMA family that the paper's models (DeepSeek-Coder,
// CodeLlama) belong to: dimension i pairs with i + D/2, for i < D/2.  The
// position of a tree node is kv_len + depth (Section IV-D adjusts the
// positional indices of the tree's tokens).
void rope_row(double* x, int D, double pos, double base) {
  const int h = D / 2;
  for (int i = 0; i < h; ++i) {
    const double a = pos * std::pow(base, -2.0 * i / D);
    const double c = std::cos(a), sn = std::sin(a);
    const double x0 = x[i], x1 = x[i + h];
    x[i] = x0 * c - x1 * sn;
    x[i + h] = x1 * c + x0 * sn;
  }
}

int tree_attn_impl(const uint16_t* q, const uint16_t* k_cache, const uint16_t* v_cache, int kv_cap,
                   const int32_t* kv_len, const uint16_t* k_tree, const uint16_t* v_tree, const uint64_t* mask,
                   const int32_t* n_nodes, int B, int n_pad, int H, int Hkv, int D, double scale,
                   const int32_t* pos, double base, const int32_t* rows, int64_t n_rows, double* out,
                   int nthreads) {
  if (Hkv < 1 || H % Hkv != 0 || (pos && D % 2)) return 1;
  int G = H / Hkv;
  int nw = (n_pad + 63) / 64;
  int64_t total = rows ? n_rows : (int64_t)B * n_pad * H;
  parallel_for(total, nthreads, [&](int64_t r) {
    int b, i, h;
    double* o;
    if (rows) {
      b = rows[3 * r];
      i = rows[3 * r + 1];
      h = rows[3 * r + 2];
      o = out + (size_t)r * D;
    } else {
      h = (int)(r % H);
      i = (int)((r / H) % n_pad);
      b = (int)(r / ((int64_t)H * n_pad));
      o = out + (size_t)r * D;
    }
    for (int x = 0; x < D; ++x) o[x] = 0.0;
    if (i >= n_nodes[b]) return;
    int g = h / G;
    const uint16_t* qv = q + (((size_t)b * n_pad + i) * H + h) * D;
    std::vector<double> qd(D), kd(D);
    for (int x = 0; x < D; ++x) qd[x] = bf16_to_double(qv[x]);
    if (pos) rope_row(qd.data(), D, pos[(size_t)b * n_pad + i], base);
    std::vector<double> s;
    std::vector<const uint16_t*> vrow;
    int L = kv_len[b];
    for (int j = 0; j < L; ++j) {
      const uint16_t* kr = k_cache + (((size_t)b * Hkv + g) * kv_cap + j) * D;
      double acc = 0.0;
      for (int x = 0; x < D; ++x) acc += qd[x] * bf16_to_double(kr[x]);
      s.push_back(acc * scale);
      vrow.push_back(v_cache + (((size_t)b * Hkv + g) * kv_cap + j) * D);
    }
    const uint64_t* mrow = mask + ((size_t)b * n_pad + i) * nw;
    for (int j = 0; j < n_pad; ++j) {
      if (!((mrow[j / 64] >> (j % 64)) & 1)) continue;
      const uint16_t* kr = k_tree + (((size_t)b * Hkv + g) * n_pad + j) * D;
      for (int x = 0; x < D; ++x) kd[x] = bf16_to_double(kr[x]);
      if (pos) rope_row(kd.data(), D, pos[(size_t)b * n_pad + j], base);
      double acc = 0.0;
      for (int x = 0; x < D; ++x) acc += qd[x] * kd[x];
      s.push_back(acc * scale);
      vrow.push_back(v_tree + (((size_t)b * Hkv + g) * n_pad + j) * D);
    }
    if (s.empty()) return;
    double mx = s[0];
    for (double v : s) mx = std::max(mx, v);
    double sum = 0.0;
    for (double& v : s) {
      v = std::exp(v - mx);
      sum += v;
    }
    for (size_t j = 0; j < s.size(); ++j) {
      double pj = s[j] / sum;
      for (int x = 0; x < D; ++x) o[x] += pj * bf16_to_double(vrow[j][x]);
    }
  });
  return 0;
}

}  // namespace

extern "C" {

int orc_tree_attn(const uint16_t* q, const uint16_t* k_cache, const uint16_t* v_cache, int kv_cap,
                  const int32_t* kv_len, const uint16_t* k_tree, const uint16_t* v_tree,
                  const uint64_t* mask, const int32_t* n_nodes, int B, int n_pad, int H, int Hkv,
                  int D, double scale, const int32_t* rows, int64_t n_rows, double* out,
                  int nthreads) {
  return tree_attn_impl(q, k_cache, v_cache, kv_cap, kv_len, k_tree, v_tree, mask, n_nodes, B, n_pad, H, Hkv, D,
                        scale, nullptr, 0.0, rows, n_rows, out, nthreads);
}

// The same attention with the queries of node i and the tree keys of node j
// rotated (O12) by pos[b][i] and pos[b][j]; the cached keys are taken as
// rotated already (they were rotated at their own positions when appended).
int orc_tree_attn_rope(const uint16_t* q, const uint16_t* k_cache, const uint16_t* v_cache, int kv_cap,
                       const int32_t* kv_len, const uint16_t* k_tree, const uint16_t* v_tree,
                       const uint64_t* mask, const int32_t* n_nodes, int B, int n_pad, int H, int Hkv,
                       int D, double scale, const int32_t* pos, double base, const int32_t* rows,
                       int64_t n_rows, double* out, int nthreads) {
  return tree_attn_impl(q, k_cache, v_cache, kv_cap, kv_len, k_tree, v_tree, mask, n_nodes, B, n_pad, H, Hkv, D,
                        scale, pos, base, rows, n_rows, out, nthreads);
}

// O12 on its own: rows x[n][D] (double) rotated by pos[n].
int orc_rope(const double* x, int64_t n, int D, const int32_t* pos, double base, double* out) {
  if (D < 2 || D % 2) return 1;
  for (int64_t r = 0; r < n; ++r) {
    for (int c = 0; c < D; ++c) out[r * D + c] = x[r * D + c];
    rope_row(out + r * D, D, pos[r], base);
  }
  return 0;
}

// ---------------------------------------------------------------------------
// O7. Greedy acceptance (Section IV-D: every correct token from the start is
// accepted and everything after the first error is rejected; Eq. 7 counts the
// tokens produced per forward).
//
// Walk from the root: at node cur, the target model's prediction argmax[cur]
// is accepted when some child of cur carries that token (siblings are
// distinct, so at most one does); then continue from that child.  acc_len =
// the number of draft tokens accepted, path[0..acc_len] the node ids (path[0]
// = 0, the rest -1), bonus = argmax at the last accepted node (the token the
// target model contributes on its own).  Returns 1 if a path exceeds path_cap.
// ---------------------------------------------------------------------------
int orc_accept(const uint32_t* tok, const int32_t* parent, const int32_t* n_nodes,
               const uint32_t* argmax, int B, int n_pad, int32_t* acc_len, int32_t* path,
               int path_cap, uint32_t* bonus) {
  for (int b = 0; b < B; ++b) {
    size_t base = (size_t)b * n_pad;
    for (int t = 0; t < path_cap; ++t) path[(size_t)b * path_cap + t] = -1;
    int cur = 0, len = 0;
    path[(size_t)b * path_cap] = 0;
    for (;;) {
      int next = -1;
      for (int j = 1; j < n_nodes[b]; ++j)
        if (parent[base + j] == cur && tok[base + j] == argmax[base + cur]) next = j;
      if (next < 0) break;
      ++len;
      if (len >= path_cap) return 1;
      path[(size_t)b * path_cap + len] = next;
      cur = next;
    }
    acc_len[b] = len;
    bonus[b] = argmax[base + cur];
  }
  return 0;
}

// ---------------------------------------------------------------------------
// O10. The target model's greedy prediction at every tree node (Section IV-D:
// verification compares each draft token with the model's most likely next
// token): argmax over the vocabulary of the node's logits row.  bf16 values
// are compared exactly as real numbers (-0 equals +0); the first index of the
// maximum wins; a NaN counts as larger than every number and the first NaN
// wins (the convention of torch.argmax and numpy.argmax).  Rows >= n_nodes[b]
// get 0.
int orc_argmax_rows(const uint16_t* logits, int B, int n_pad, int vocab, const int32_t* n_nodes,
                    uint32_t* argmax) {
  for (int b = 0; b < B; ++b) {
    for (int i = 0; i < n_pad; ++i) {
      uint32_t best = 0;
      if (i < n_nodes[b]) {
        const uint16_t* row = logits + ((size_t)b * n_pad + i) * (size_t)vocab;
        double bv = bf16_to_double(row[0]);
        bool bnan = std::isnan(bv);
        for (int v = 1; v < vocab && !bnan; ++v) {
          const double x = bf16_to_double(row[v]);
          if (std::isnan(x)) {
            best = (uint32_t)v;
            bnan = true;
          } else if (x > bv) {
            best = (uint32_t)v;
            bv = x;
          }
        }
      }
      argmax[(size_t)b * n_pad + i] = best;
    }
  }
  return 0;
}

// ---------------------------------------------------------------------------
// O8. Cache update after acceptance (implied by the decoding loop of
// Section II and Section IV-D): the K/V rows of the accepted path (root
// included) move into the cache at kv_len..kv_len+acc_len, kv_len grows by
// acc_len + 1, the accepted draft tokens and the bonus token are appended to
// the context, and the bonus token becomes the next root.  Returns 1 when a
// cache or context would overflow its capacity.
// ---------------------------------------------------------------------------
int orc_kv_append(const int32_t* path, const int32_t* acc_len, const uint32_t* bonus,
                  const uint32_t* tok, const uint16_t* k_tree, const uint16_t* v_tree, int B,
                  int n_pad, int Hkv, int D, int path_cap, uint16_t* k_cache, uint16_t* v_cache,
                  int kv_cap, const int32_t* kv_len_in, int32_t* kv_len_out, uint32_t* ctx,
                  int ctx_stride, const int32_t* ctx_len_in, int32_t* ctx_len_out,
                  uint32_t* root_out) {
  for (int b = 0; b < B; ++b) {
    int a = acc_len[b];
    if (kv_len_in[b] + a + 1 > kv_cap || ctx_len_in[b] + a + 1 > ctx_stride || a + 1 > path_cap)
      return 1;
    for (int t = 0; t <= a; ++t) {
      int node = path[(size_t)b * path_cap + t];
      for (int g = 0; g < Hkv; ++g) {
        size_t src = (((size_t)b * Hkv + g) * n_pad + node) * D;
        size_t dst = (((size_t)b * Hkv + g) * kv_cap + kv_len_in[b] + t) * D;
        std::memcpy(k_cache + dst, k_tree + src, D * sizeof(uint16_t));
        std::memcpy(v_cache + dst, v_tree + src, D * sizeof(uint16_t));
      }
    }
    kv_len_out[b] = kv_len_in[b] + a + 1;
    uint32_t* c = ctx + (size_t)b * ctx_stride;
    for (int t = 0; t < a; ++t) c[ctx_len_in[b] + t] = tok[(size_t)b * n_pad + path[(size_t)b * path_cap + t + 1]];
    c[ctx_len_in[b] + a] = bonus[b];
    ctx_len_out[b] = ctx_len_in[b] + a + 1;
    root_out[b] = bonus[b];
  }
  return 0;
}

// ---------------------------------------------------------------------------
// Synthetic stand-in for the target model's greedy predictions (workload
// scaffolding, not part of the method: the paper's target model is an LLM).
// Along the tree's first branch (root, its first child, that node's first
// child, ...) the model agrees with the tree for the first plen[b] steps;
// every other prediction is the node's random token rtok[b][i], moved up by
// one (mod vocab) while it equals a token of one of the node's children, at
// most n_pad times (when the children cover the whole vocabulary the last
// candidate stands).
// ---------------------------------------------------------------------------
int orc_synth_argmax(const uint32_t* tok, const int32_t* parent, const int32_t* n_nodes, int B,
                     int n_pad, const int32_t* plen, const uint32_t* rtok, uint32_t vocab,
                     uint32_t* argmax) {
  for (int b = 0; b < B; ++b) {
    size_t base = (size_t)b * n_pad;
    int n = n_nodes[b];
    for (int i = 0; i < n_pad; ++i) argmax[base + i] = 0;
    std::vector<int> agree_child(n, -1);
    int cur = 0;
    for (int t = 0; t < plen[b]; ++t) {
      int first = -1;
      for (int j = 1; j < n && first < 0; ++j)
        if (parent[base + j] == cur) first = j;
      if (first < 0) break;
      agree_child[cur] = first;
      cur = first;
    }
    for (int i = 0; i < n; ++i) {
      if (agree_child[i] >= 0) {
        argmax[base + i] = tok[base + agree_child[i]];
        continue;
      }
      uint32_t x = rtok[base + i] % vocab;
      for (int tries = 0; tries < n_pad; ++tries) {
        bool clash = false;
        for (int j = 1; j < n; ++j)
          if (parent[base + j] == i && tok[base + j] == x) clash = true;
        if (!clash) break;
        x = (x + 1) % vocab;
      }
      argmax[base + i] = x;
    }
  }
  return 0;
}

// ---------------------------------------------------------------------------
// O11. CACHE search (Section IV-B: the CACHE stores token sequences, each a
// verified retrieval "context + accepted draft" or a piece of the model's
// output; Section IV-C, Algorithm 1: search(CACHE) retrieves from it the same
// way the datastore is searched).
//
// Query b owns the entries e in [qent[b], qent[b+1]); entry e is the token
// sequence tok[eoff[e] .. eoff[e+1]).  The search is O2-O4 with the entries
// as the corpus, under the reading that a stored sequence is a unit of its
// own: a match lies inside one entry, and a continuation stops at the end of
// its entry.  So for a context c of length m and cap = min(n_max, m):
//   * n* is the largest n in [n_min, cap] for which some entry E of length L
//     has E[p-n .. p) = c[m-n .. m) with n <= p <= L-1 (one continuation
//     token or more);
//   * the occurrences are all such (e, p) for n*; with more than max_occ of
//     them, the max_occ whose windows E[p-n* .. min(p+d, L)) are
//     lexicographically smallest are kept (max_occ = 0 keeps all);
//   * continuations u = E[p .. min(p+d, L)) are counted as distinct
//     sequences and ranked by count descending, then token ids ascending.
// Method: for every entry and position, the common suffix length by direct
// comparison; then the occurrences of n*; then std::map counting.  Outputs as
// orc_retrieve.
// ---------------------------------------------------------------------------
int orc_cache_search(const uint32_t* tok, const int64_t* eoff, const int64_t* qent, const uint32_t* ctx,
                     int ctx_stride, const int32_t* ctx_len, int B, int n_max, int n_min, int top_k, int d,
                     uint32_t max_occ, uint32_t* drafts, int32_t* draft_len, uint32_t* count,
                     int32_t* n_drafts, int32_t* match_len, int nthreads) {
  if (n_min < 1 || n_max < n_min || top_k < 1 || d < 1) return 1;
  parallel_for(B, nthreads, [&](int64_t b) {
    const uint32_t* c = ctx + (size_t)b * ctx_stride;
    const int m = ctx_len[b];
    uint32_t* dr = drafts + (size_t)b * top_k * d;
    int32_t* dl = draft_len + (size_t)b * top_k;
    uint32_t* ct = count + (size_t)b * top_k;
    for (int i = 0; i < top_k * d; ++i) dr[i] = kPad;
    for (int i = 0; i < top_k; ++i) { dl[i] = 0; ct[i] = 0; }
    n_drafts[b] = 0;
    match_len[b] = 0;
    const int cap = std::min(n_max, m);
    if (cap < n_min) return;
    // common suffix length of E[0..p) and c, at most cap
    auto common = [&](const uint32_t* E, int64_t p) {
      int k = 0;
      while (k < cap && k < p && E[p - 1 - k] == c[m - 1 - k]) ++k;
      return k;
    };
    int best = 0;
    for (int64_t e = qent[b]; e < qent[b + 1]; ++e) {
      const uint32_t* E = tok + eoff[e];
      const int64_t L = eoff[e + 1] - eoff[e];
      for (int64_t p = 1; p <= L - 1; ++p) best = std::max(best, common(E, p));
    }
    if (best < n_min) return;
    const int ns = best;
    struct Occ {
      std::vector<uint32_t> window, cont;
    };
    std::vector<Occ> occ;
    for (int64_t e = qent[b]; e < qent[b + 1]; ++e) {
      const uint32_t* E = tok + eoff[e];
      const int64_t L = eoff[e + 1] - eoff[e];
      for (int64_t p = ns; p <= L - 1; ++p) {
        if (common(E, p) < ns) continue;
        const int64_t end = std::min<int64_t>(p + d, L);
        occ.push_back({std::vector<uint32_t>(E + p - ns, E + end), std::vector<uint32_t>(E + p, E + end)});
      }
    }
    if (max_occ > 0 && occ.size() > max_occ) {
      std::stable_sort(occ.begin(), occ.end(), [](const Occ& x, const Occ& y) { return x.window < y.window; });
      occ.resize(max_occ);
    }
    std::map<std::vector<uint32_t>, uint32_t> freq;
    for (const Occ& o : occ) freq[o.cont] += 1;
    std::vector<std::pair<uint32_t, std::vector<uint32_t>>> ranked;
    for (auto& kv : freq) ranked.push_back({kv.second, kv.first});
    std::stable_sort(ranked.begin(), ranked.end(), [](const auto& x, const auto& y) {
      if (x.first != y.first) return x.first > y.first;
      return x.second < y.second;
    });
    const int nd = (int)std::min<size_t>(ranked.size(), (size_t)top_k);
    for (int t = 0; t < nd; ++t) {
      const auto& seq = ranked[t].second;
      for (size_t i = 0; i < seq.size(); ++i) dr[(size_t)t * d + i] = seq[i];
      dl[t] = (int32_t)seq.size();
      ct[t] = ranked[t].first;
    }
    n_drafts[b] = nd;
    match_len[b] = ns;
  });
  return 0;
}

int orc_hardware_threads(void) { return resolve_threads(0); }

}  // extern "C"
