// fc_build_tree / fc_tree_mask: draft-tree construction (Section IV-D: trie
// over the retrieved drafts, node weight alpha*t_r + beta*t_c of Eq. 3, the
// top-weighted nodes as the draft tree; the tree mask of Eq. 4; position ids
// by depth; Section V-C: alpha = beta = 1, at most 64 draft tokens).
//
// One CTA per query, everything in shared memory, no pointer trie:
//   1. gather the drafts of all sources with weight w = src_weight * count;
//   2. sort them lexicographically (threads rank drafts against all others,
//      comparing zero-padded pairs of tokens packed in 64-bit words, then
//      lengths) and merge duplicates across sources (weights add);
//   3. with neighbour LCPs, every trie node is a pair (u, l): the prefix of
//      length l of sorted unique draft u, new at u when l > lcp(u-1, u).
//      Its weight is the weight sum of the contiguous run of drafts that
//      share that prefix (prefix sums over the sorted drafts);
//   4. a radix select on the distinct (W, 31 - l, 8191 - u) keys finds the
//      heaviest budget - 1 nodes (ties: shallower, then smaller path); a
//      parent's key always exceeds its child's, so the kept set is a tree;
//   5. (u, l) order is depth-first preorder with children in ascending
//      token order: a scan over a kept-flag table [u][l] numbers the nodes
//      and maps a parent (the run start of prefix l - 1) to its index;
//      masks are ancestor walks.
#include <algorithm>

#include "fc_common.cuh"

FC_DEFINE_ERROR_WORD(tree)

namespace {

constexpr int BT_THREADS = 512;
constexpr int BT_MAX_DRAFTS = 512;
constexpr int PK_WORDS = FC_MAX_DRAFT_LEN / 2;  // 64-bit words per packed draft

struct TreeIn {
  const uint32_t* drafts;
  const int32_t* draft_len;
  const uint32_t* count;
  const int32_t* n_drafts;
  uint32_t w[FC_MAX_SOURCES];
};
struct TreeOut {
  uint32_t* tok;
  int32_t* parent;
  int32_t* depth;
  int32_t* pos;
  uint64_t* mask;
  int32_t* n_nodes;
  unsigned int* err;  // the launch's error word (NULL: this file's own)
};

struct BtLayout {
  size_t tok, len, w, order, uniq, wu, ps, lcp, coff, flag, ckey, pk, tab, total;
};

__host__ __device__ inline BtLayout bt_layout(int M, int d) {
  BtLayout L;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    size_t o = off;
    off = (off + bytes + 15) & ~(size_t)15;
    return o;
  };
  L.tok = take((size_t)M * d * 4);
  L.len = take((size_t)M * 4);
  L.w = take((size_t)M * 8);
  L.order = take((size_t)M * 4);
  L.uniq = take((size_t)M * 4);
  L.wu = take((size_t)M * 8);
  L.ps = take((size_t)(M + 1) * 8);
  L.lcp = take((size_t)(M + 1) * 4);
  L.coff = take((size_t)(M + 1) * 4);
  L.flag = take((size_t)(M + 1) * 4);
  L.ckey = take((size_t)M * d * 8);
  L.pk = take((size_t)M * PK_WORDS * 8);  // each draft as zero-padded token pairs
  L.tab = take((size_t)M * d * 4);  // kept flags [u][l - 1], then their preorder ranks
  L.total = off;
  return L;
}

// Exclusive scan of a[0..n) in place (n <= 8192); returns the total.
__device__ uint32_t block_scan_array(uint32_t* a, int n, uint32_t* wsum) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int chunk = (n + BT_THREADS - 1) / BT_THREADS;
  const int lo = min(n, tid * chunk), hi = min(n, lo + chunk);
  uint32_t s = 0;
  for (int i = lo; i < hi; ++i) s += a[i];
  uint32_t inc = s;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    uint32_t y = __shfl_up_sync(0xFFFFFFFFu, inc, o);
    if (lane >= o) inc += y;
  }
  if (lane == 31) wsum[warp] = inc;
  __syncthreads();
  if (tid == 0) {
    uint32_t run = 0;
    for (int w = 0; w < BT_THREADS / 32; ++w) {
      uint32_t c = wsum[w];
      wsum[w] = run;
      run += c;
    }
    wsum[BT_THREADS / 32] = run;
  }
  __syncthreads();
  uint32_t pre = wsum[warp] + inc - s;
  for (int i = lo; i < hi; ++i) {
    uint32_t v = a[i];
    a[i] = pre;
    pre += v;
  }
  uint32_t total = wsum[BT_THREADS / 32];
  __syncthreads();
  return total;
}

// Warp 0 (all 32 lanes): out[i] = sum of a[0..i) for i <= n (64-bit).  The
// caller synchronises the block before reading out.
__device__ void warp_scan_u64(const uint64_t* a, uint64_t* out, uint32_t n) {
  const uint32_t lane = threadIdx.x & 31;
  const uint32_t chunk = (n + 31) / 32;
  const uint32_t lo = min(n, lane * chunk), hi = min(n, lo + chunk);
  uint64_t s = 0;
  for (uint32_t i = lo; i < hi; ++i) s += a[i];
  uint64_t inc = s;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint64_t y = __shfl_up_sync(0xFFFFFFFFu, inc, o);
    if ((int)lane >= o) inc += y;
  }
  uint64_t pre = inc - s;
  for (uint32_t i = lo; i < hi; ++i) {
    out[i] = pre;
    pre += a[i];
  }
  if (lane == 31) out[n] = inc;
}

// The k-th largest (1 <= k <= n) of n distinct 64-bit keys, by radix select
// over bytes from the most significant: each pass histograms the byte of
// the keys that match the bytes fixed so far and fixes the byte whose bin
// holds the k-th largest.  Called by the whole block.
__device__ uint64_t radix_select_desc(const uint64_t* key, uint32_t n, uint32_t k, uint32_t* hist) {
  __shared__ uint64_t s_pre, s_or, s_and;
  __shared__ uint32_t s_k;
  const int tid = threadIdx.x;
  // bytes on which all keys agree need no pass: start below them
  if (tid == 0) {
    s_or = 0;
    s_and = ~0ull;
  }
  __syncthreads();
  {
    uint64_t o = 0, a = ~0ull;
    for (uint32_t i = tid; i < n; i += BT_THREADS) {
      o |= key[i];
      a &= key[i];
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      o |= __shfl_xor_sync(0xFFFFFFFFu, o, off);
      a &= __shfl_xor_sync(0xFFFFFFFFu, a, off);
    }
    if ((tid & 31) == 0) {
      atomicOr(reinterpret_cast<unsigned long long*>(&s_or), o);
      atomicAnd(reinterpret_cast<unsigned long long*>(&s_and), a);
    }
  }
  __syncthreads();
  const uint64_t diff = s_or ^ s_and;  // bits that vary among the keys
  if (diff == 0) return s_or;          // n == 1
  const int top = 63 - __clzll((long long)diff);
  uint64_t pmask = (top >= 63) ? 0ull : ~((2ull << top) - 1ull);  // agreed bits above `top`
  uint64_t pre = s_or & pmask;
  for (int shift = top & ~7; shift >= 0; shift -= 8) {
    for (int i = tid; i < 256; i += BT_THREADS) hist[i] = 0;
    if (tid == 0) {
      s_pre = pre;
      s_k = k;
    }
    __syncthreads();
    for (uint32_t i = tid; i < n; i += BT_THREADS) {
      const uint64_t x = key[i];
      if ((x & pmask) == pre) atomicAdd(&hist[(x >> shift) & 255u], 1u);
    }
    __syncthreads();
    if (tid < 32) {  // lane L owns bins [8L, 8L + 8); suffix sums from the top bin
      uint32_t c[8], tot = 0;
#pragma unroll
      for (int q = 0; q < 8; ++q) tot += (c[q] = hist[8 * tid + q]);
      uint32_t suf = tot;  // inclusive suffix over lanes >= tid
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_down_sync(0xFFFFFFFFu, suf, o);
        if (tid + o < 32) suf += y;
      }
      const uint32_t above = suf - tot;  // keys in higher lanes' bins
      if (above < k && suf >= k) {       // the k-th largest lies in this lane's bins
        uint32_t acc = above, k_rem = 0;
        int chosen = -1;
#pragma unroll
        for (int q = 7; q >= 0; --q) {
          if (chosen < 0) {
            if (acc + c[q] >= k) {
              chosen = q;
              k_rem = k - acc;
            } else {
              acc += c[q];
            }
          }
        }
        s_pre = pre | ((uint64_t)(8 * tid + chosen) << shift);
        s_k = k_rem;
      }
    }
    __syncthreads();
    pre = s_pre;
    k = s_k;
    pmask |= (uint64_t)0xFF << shift;
    __syncthreads();
  }
  return pre;
}

// -1 / 0 / 1 lexicographic comparison of two drafts (a prefix sorts first).
__device__ __forceinline__ int cmp_draft(const uint32_t* a, int la, const uint32_t* b, int lb) {
  int l = min(la, lb);
  for (int i = 0; i < l; ++i)
    if (a[i] != b[i]) return a[i] < b[i] ? -1 : 1;
  return la < lb ? -1 : (la > lb ? 1 : 0);
}

__global__ void __launch_bounds__(BT_THREADS) k_build_tree(TreeIn in, int S, int B, int k, int d,
                                                           const uint32_t* __restrict__ root_tok,
                                                           const int32_t* __restrict__ kv_len, int budget, int n_pad,
                                                           TreeOut out) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  __shared__ uint32_t wsum[BT_THREADS / 32 + 1];
  __shared__ int32_t sel_u[FC_MAX_NODES], sel_l[FC_MAX_NODES], par_s[FC_MAX_NODES];
  const int M0 = S * k;
  const BtLayout L = bt_layout(M0, d);
  uint32_t* tok = reinterpret_cast<uint32_t*>(smem_raw + L.tok);
  int32_t* len = reinterpret_cast<int32_t*>(smem_raw + L.len);
  uint64_t* w = reinterpret_cast<uint64_t*>(smem_raw + L.w);
  uint32_t* order = reinterpret_cast<uint32_t*>(smem_raw + L.order);
  uint32_t* uniq = reinterpret_cast<uint32_t*>(smem_raw + L.uniq);
  uint64_t* wu = reinterpret_cast<uint64_t*>(smem_raw + L.wu);
  uint64_t* ps = reinterpret_cast<uint64_t*>(smem_raw + L.ps);
  uint32_t* lcp = reinterpret_cast<uint32_t*>(smem_raw + L.lcp);
  uint32_t* coff = reinterpret_cast<uint32_t*>(smem_raw + L.coff);
  uint32_t* flag = reinterpret_cast<uint32_t*>(smem_raw + L.flag);
  uint64_t* ckey = reinterpret_cast<uint64_t*>(smem_raw + L.ckey);
  uint64_t* pk = reinterpret_cast<uint64_t*>(smem_raw + L.pk);
  uint32_t* tab = reinterpret_cast<uint32_t*>(smem_raw + L.tab);
  __shared__ uint32_t hist[256];
  const int b = blockIdx.x, tid = threadIdx.x;

  // 1. valid drafts, compacted in (source, slot) order
  for (int i = tid; i < M0; i += BT_THREADS) {
    int s = i / k, t = i - s * k;
    size_t sb = (size_t)s * B + b;
    int nd = min(max((int)in.n_drafts[sb], 0), k);
    int l = (t < nd) ? in.draft_len[sb * k + t] : 0;
    flag[i] = (l > 0 && l <= d) ? 1u : 0u;
  }
  __syncthreads();
  // keep the flags: scan a copy in coff
  for (int i = tid; i < M0; i += BT_THREADS) coff[i] = flag[i];
  __syncthreads();
  uint32_t M = block_scan_array(coff, M0, wsum);
  for (int i = tid; i < M0; i += BT_THREADS) {
    if (!flag[i]) continue;
    int s = i / k, t = i - s * k;
    size_t sb = (size_t)s * B + b;
    uint32_t j = coff[i];
    int l = in.draft_len[sb * k + t];
    len[j] = l;
    uint32_t cnt = in.count[sb * k + t];
    if (cnt > (1u << 20)) {  // weights are packed into 46-bit sort keys
      fc_flag(FC_ERR_WORD(out.err), FC_EBIT_INVALID);
      cnt = 1u << 20;
    }
    w[j] = (uint64_t)in.w[s] * cnt;
    for (int x = 0; x < d; ++x) tok[j * d + x] = (x < l) ? in.drafts[(sb * k + t) * d + x] : 0u;
  }
  __syncthreads();

  // 2. rank sort of the drafts by token sequence; equal drafts keep
  //    (source, slot) order through the index tie-break.  Drafts compare as
  //    their token pairs packed in 64-bit words, zero-padded, then by
  //    length: a difference in the padded words always has the lexicographic
  //    sign (a zero pad only ever ties with a real token), and padded words
  //    that agree mean one draft is a prefix of the other.
  for (uint32_t x = tid; x < M * (uint32_t)PK_WORDS; x += BT_THREADS) {
    const uint32_t i = x / PK_WORDS, q = x - i * PK_WORDS;
    const int l = len[i];
    const uint32_t t0 = (2 * (int)q < l) ? tok[i * d + 2 * q] : 0u;
    const uint32_t t1 = (2 * (int)q + 1 < l) ? tok[i * d + 2 * q + 1] : 0u;
    pk[x] = ((uint64_t)t0 << 32) | t1;
  }
  for (uint32_t i = tid; i < M; i += BT_THREADS) order[i] = 0;
  __syncthreads();
  {
    // several threads per draft when they fit (slices of the j range)
    const uint32_t split = M > 0 ? umax(1u, umin(8u, (uint32_t)BT_THREADS / M)) : 1u;
    for (uint32_t x = tid; x < M * split; x += BT_THREADS) {
      const uint32_t i = x / split, h = x - i * split;
      const ulonglong2* pv = reinterpret_cast<const ulonglong2*>(pk);
      uint64_t a[PK_WORDS];
#pragma unroll
      for (int q = 0; q < PK_WORDS / 2; ++q) {
        const ulonglong2 v = pv[i * (PK_WORDS / 2) + q];
        a[2 * q] = v.x;
        a[2 * q + 1] = v.y;
      }
      const int la = len[i];
      const uint32_t j0 = h * M / split, j1 = (h + 1) * M / split;
      uint32_t rank = 0;
      for (uint32_t j = j0; j < j1; ++j) {
        int res = 0;  // sign of draft j vs draft i
#pragma unroll
        for (int q = 0; q < PK_WORDS / 2; ++q) {
          const ulonglong2 v = pv[j * (PK_WORDS / 2) + q];
          if (res == 0 && v.x != a[2 * q]) res = (v.x < a[2 * q]) ? -1 : 1;
          if (res == 0 && v.y != a[2 * q + 1]) res = (v.y < a[2 * q + 1]) ? -1 : 1;
        }
        if (res == 0) res = (len[j] < la) ? -1 : (len[j] > la ? 1 : 0);
        rank += (res < 0 || (res == 0 && j < i)) ? 1u : 0u;
      }
      atomicAdd(&order[i], rank);  // order[] holds ranks here
    }
  }
  __syncthreads();
  for (uint32_t i = tid; i < M; i += BT_THREADS) flag[i] = order[i];  // rank of draft i
  __syncthreads();
  for (uint32_t i = tid; i < M; i += BT_THREADS) order[flag[i]] = i;
  __syncthreads();
  for (uint32_t r = tid; r < M; r += BT_THREADS) {
    uint32_t i = order[r];
    flag[r] = (r == 0 || cmp_draft(tok + order[r - 1] * d, len[order[r - 1]], tok + i * d, len[i]) != 0) ? 1u : 0u;
    coff[r] = flag[r];
  }
  __syncthreads();
  uint32_t U = block_scan_array(coff, (int)M, wsum);  // coff[r] = unique index of run start
  for (uint32_t u = tid; u < U; u += BT_THREADS) wu[u] = 0;
  __syncthreads();
  for (uint32_t r = tid; r < M; r += BT_THREADS) {
    uint32_t u = coff[r] + flag[r] - 1u;  // unique index of the run containing r
    if (flag[r]) uniq[u] = order[r];
    atomicAdd(reinterpret_cast<unsigned long long*>(&wu[u]), (unsigned long long)w[order[r]]);
  }
  __syncthreads();

  // 3. neighbour LCPs, prefix sums of weights, candidate counts
  for (uint32_t u = tid; u < U; u += BT_THREADS) {
    uint32_t l = 0;
    if (u > 0) {
      const uint32_t* a = tok + uniq[u - 1] * d;
      const uint32_t* c = tok + uniq[u] * d;
      int lim = min(len[uniq[u - 1]], len[uniq[u]]);
      while ((int)l < lim && a[l] == c[l]) ++l;
    }
    lcp[u] = l;
    coff[u] = (uint32_t)len[uniq[u]] - l;
  }
  __syncthreads();
  if (tid < 32) warp_scan_u64(wu, ps, U);  // ps[u] = sum of wu[0..u), ps[U] = total
  uint32_t C = block_scan_array(coff, (int)U, wsum);
  for (uint32_t u = tid; u < U; u += BT_THREADS) {
    // deepest first: the run of (u, l) ends at the first e > u with lcp[e] < l,
    // which only moves right as l falls, so one scan serves every depth
    const int lu = len[uniq[u]];
    uint32_t e = u + 1;
    for (int l = lu; l > (int)lcp[u]; --l) {
      while (e < U && (int)lcp[e] >= l) ++e;
      const uint64_t W = ps[e] - ps[u];
      ckey[coff[u] + (l - lcp[u] - 1)] = (W << 18) | ((uint64_t)(31 - l) << 13) | (uint64_t)(8191u - u);
    }
  }
  for (uint32_t x = tid; x < U * (uint32_t)d; x += BT_THREADS) tab[x] = 0;
  __syncthreads();

  // 4. the nsel largest keys (all distinct): radix select of the threshold,
  //    8 bits at a time from the top
  const int nsel = (int)umin((uint32_t)(budget - 1), C);
  uint64_t thr = 0;
  if (nsel > 0 && (uint32_t)nsel < C) thr = radix_select_desc(ckey, C, (uint32_t)nsel, hist);
  // 5. kept flags in the (u, l) table, scanned into preorder ranks
  for (uint32_t c = tid; c < C; c += BT_THREADS) {
    const uint64_t key = ckey[c];
    if (nsel > 0 && key >= thr) {
      const int u = 8191 - (int)(key & 8191u), l = 31 - (int)((key >> 13) & 31u);
      tab[u * d + l - 1] = 1u;
    }
  }
  __syncthreads();
  const uint32_t nkept = block_scan_array(tab, (int)(U * (uint32_t)d), wsum);
  if (nkept != (uint32_t)nsel && tid == 0) fc_flag(FC_ERR_WORD(out.err), FC_EBIT_INTERNAL);
  for (uint32_t c = tid; c < C; c += BT_THREADS) {
    const uint64_t key = ckey[c];
    if (nsel > 0 && key >= thr) {
      const int u = 8191 - (int)(key & 8191u), l = 31 - (int)((key >> 13) & 31u);
      const int idx = 1 + (int)tab[u * d + l - 1];
      if (idx < FC_MAX_NODES) {
        sel_u[idx] = u;
        sel_l[idx] = l;
      }
    }
  }
  __syncthreads();
  const int n = 1 + min(nsel, FC_MAX_NODES - 1);
  for (int i = 1 + tid; i < n; i += BT_THREADS) {
    const int u = sel_u[i], l = sel_l[i];
    int pidx = 0;
    if (l > 1) {  // the parent is the prefix l - 1, first seen at the start of its run
      int up = u;
      while (up > 0 && (int)lcp[up] >= l - 1) --up;
      pidx = 1 + (int)tab[up * d + l - 2];
    }
    par_s[i] = pidx;
  }
  if (tid == 0) par_s[0] = -1;
  __syncthreads();
  const int nw = n_pad / 64;
  const size_t base = (size_t)b * n_pad;
  const int kvl = kv_len[b];
  for (int i = tid; i < n_pad; i += BT_THREADS) {
    uint32_t tk = FC_PAD_TOKEN;
    int pa = -1, de = -1, po = -1;
    uint64_t m0 = 0, m1 = 0;
    if (i < n) {
      tk = (i == 0) ? root_tok[b] : tok[uniq[sel_u[i]] * d + sel_l[i] - 1];
      de = (i == 0) ? 0 : sel_l[i];
      pa = par_s[i];
      po = kvl + de;
      for (int a = i; a >= 0; a = par_s[a]) {
        if (a < 64) m0 |= 1ull << a;
        else m1 |= 1ull << (a - 64);
      }
    }
    out.tok[base + i] = tk;
    out.parent[base + i] = pa;
    out.depth[base + i] = de;
    out.pos[base + i] = po;
    out.mask[(base + i) * nw] = m0;
    if (nw > 1) out.mask[(base + i) * nw + 1] = m1;
  }
  if (tid == 0) out.n_nodes[b] = n;
}

// ---------------------------------------------------------------------------
// fc_build_tree_all: the same tree (Eq. 3 weights, the heaviest budget - 1
// nodes, preorder, Eq. 4 masks) over every distinct continuation of every
// source, the all-occurrence reading of Section III-A: up to 8192 drafts per
// query, so the per-query arrays live in a global workspace.  Each source's
// drafts arrive in ascending token order (fc_retrieve_all's output), so
//   * the merged order needs no sort: a draft's merged position is its index
//     in its own list plus, for every other source, how many of that
//     source's drafts precede it (a binary search; an equal draft of an
//     earlier source precedes it), and equal drafts end up adjacent;
//   * a node (u, l) is again the length-l prefix of unique draft u, new at u
//     when l > lcp(u-1, u); the drafts under it form the run of u at depth
//     l, the maximal range whose inner neighbour LCPs are >= l.  For each
//     depth, run starts (lcp < l) are numbered by a block scan, which gives
//     every node's run end (its weight is a prefix-sum difference) and its
//     parent (the run of depth l - 1 that contains u).
// ---------------------------------------------------------------------------
constexpr int BTA_MAX_DRAFTS = 8192;  // 13 bits of draft index in the selection key

struct AllLayout {
  size_t tok, len, w, pk, order, flag, coff, uniq, wu, ps, lcp, rid, rpos, rid_p, rpos_p, ckey, cpar, tab, total;
};

__host__ __device__ inline AllLayout all_layout(int M, int d) {
  AllLayout L;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    size_t o = off;
    off = (off + bytes + 255) & ~(size_t)255;
    return o;
  };
  L.tok = take((size_t)M * d * 4);
  L.len = take((size_t)M * 4);
  L.w = take((size_t)M * 8);
  L.pk = take((size_t)M * PK_WORDS * 8);
  L.order = take((size_t)M * 4);
  L.flag = take((size_t)(M + 1) * 4);
  L.coff = take((size_t)(M + 1) * 4);
  L.uniq = take((size_t)M * 4);
  L.wu = take((size_t)M * 8);
  L.ps = take((size_t)(M + 1) * 8);
  L.lcp = take((size_t)(M + 1) * 4);
  L.rid = take((size_t)(M + 1) * 4);     // run number of u at the current depth
  L.rpos = take((size_t)(M + 2) * 4);    // start of each run at the current depth, then U
  L.rid_p = take((size_t)(M + 1) * 4);   // the same at the previous depth
  L.rpos_p = take((size_t)(M + 2) * 4);
  L.ckey = take((size_t)M * d * 8);
  L.cpar = take((size_t)M * d * 4);      // a candidate's parent draft (the run start one level up)
  L.tab = take((size_t)M * d * 4);
  L.total = off;
  return L;
}

// Sign of packed draft a against packed draft b (zero-padded token pairs,
// then the lengths: the order of cmp_draft).
__device__ __forceinline__ int cmp_packed(const uint64_t* a, int la, const uint64_t* b, int lb) {
#pragma unroll
  for (int q = 0; q < PK_WORDS; ++q)
    if (a[q] != b[q]) return a[q] < b[q] ? -1 : 1;
  return la < lb ? -1 : (la > lb ? 1 : 0);
}

__global__ void __launch_bounds__(BT_THREADS, 1) k_build_tree_all(TreeIn in, int S, int B, int k, int d,
                                                               const uint32_t* __restrict__ root_tok,
                                                               const int32_t* __restrict__ kv_len, int budget,
                                                               int n_pad, unsigned char* ws, size_t ws_per_query,
                                                               TreeOut out) {
  __shared__ uint32_t wsum[BT_THREADS / 32 + 1];
  __shared__ int32_t sel_u[FC_MAX_NODES], sel_l[FC_MAX_NODES], par_s[FC_MAX_NODES];
  __shared__ uint32_t hist[256];
  __shared__ uint32_t s_off[FC_MAX_SOURCES + 1];
  __shared__ int s_bad;
  const int M0 = S * k;
  const AllLayout L = all_layout(M0, d);
  unsigned char* base = ws + (size_t)blockIdx.x * ws_per_query;
  uint32_t* tok = reinterpret_cast<uint32_t*>(base + L.tok);
  int32_t* len = reinterpret_cast<int32_t*>(base + L.len);
  uint64_t* w = reinterpret_cast<uint64_t*>(base + L.w);
  uint64_t* pk = reinterpret_cast<uint64_t*>(base + L.pk);
  uint32_t* order = reinterpret_cast<uint32_t*>(base + L.order);
  uint32_t* flag = reinterpret_cast<uint32_t*>(base + L.flag);
  uint32_t* coff = reinterpret_cast<uint32_t*>(base + L.coff);
  uint32_t* uniq = reinterpret_cast<uint32_t*>(base + L.uniq);
  uint64_t* wu = reinterpret_cast<uint64_t*>(base + L.wu);
  uint64_t* ps = reinterpret_cast<uint64_t*>(base + L.ps);
  uint32_t* lcp = reinterpret_cast<uint32_t*>(base + L.lcp);
  uint32_t* rid = reinterpret_cast<uint32_t*>(base + L.rid);
  uint32_t* rpos = reinterpret_cast<uint32_t*>(base + L.rpos);
  uint32_t* rid_p = reinterpret_cast<uint32_t*>(base + L.rid_p);
  uint32_t* rpos_p = reinterpret_cast<uint32_t*>(base + L.rpos_p);
  uint64_t* ckey = reinterpret_cast<uint64_t*>(base + L.ckey);
  uint32_t* cpar = reinterpret_cast<uint32_t*>(base + L.cpar);
  uint32_t* tab = reinterpret_cast<uint32_t*>(base + L.tab);
  const int b = blockIdx.x, tid = threadIdx.x;

  // 1. valid drafts compacted in (source, slot) order; s_off[s] = source s's first
  for (int i = tid; i < M0; i += BT_THREADS) {
    const int s = i / k, t = i - s * k;
    const size_t sb = (size_t)s * B + b;
    const int nd = min(max((int)in.n_drafts[sb], 0), k);
    const int l = (t < nd) ? in.draft_len[sb * k + t] : 0;
    flag[i] = (l > 0 && l <= d) ? 1u : 0u;
    coff[i] = flag[i];
  }
  if (tid == 0) s_bad = 0;
  __syncthreads();
  const uint32_t M = block_scan_array(coff, M0, wsum);
  if (tid <= S) s_off[tid] = (tid < S) ? coff[tid * k] : M;
  for (int i = tid; i < M0; i += BT_THREADS) {
    if (!flag[i]) continue;
    const int s = i / k, t = i - s * k;
    const size_t sb = (size_t)s * B + b;
    const uint32_t j = coff[i];
    const int l = in.draft_len[sb * k + t];
    len[j] = l;
    uint32_t cnt = in.count[sb * k + t];
    if (cnt > (1u << 17)) {  // weights are packed into 46-bit selection keys
      fc_flag(FC_ERR_WORD(out.err), FC_EBIT_INVALID);
      cnt = 1u << 17;
    }
    w[j] = (uint64_t)in.w[s] * cnt;
    for (int x = 0; x < d; ++x) tok[j * d + x] = (x < l) ? in.drafts[(sb * k + t) * d + x] : 0u;
  }
  __syncthreads();
  for (uint32_t x = tid; x < M * (uint32_t)PK_WORDS; x += BT_THREADS) {
    const uint32_t i = x / PK_WORDS, q = x - i * PK_WORDS;
    const int l = len[i];
    const uint32_t t0 = (2 * (int)q < l) ? tok[i * d + 2 * q] : 0u;
    const uint32_t t1 = (2 * (int)q + 1 < l) ? tok[i * d + 2 * q + 1] : 0u;
    pk[x] = ((uint64_t)t0 << 32) | t1;
  }
  __syncthreads();
  auto src_of = [&](uint32_t j) {
    int s = 0;
    while (s + 1 < S && j >= s_off[s + 1]) ++s;
    return s;
  };
  // every source's list strictly ascending, or the merge below is undefined
  for (uint32_t j = tid; j < M; j += BT_THREADS) {
    const int s = src_of(j);
    if (j > s_off[s] && cmp_packed(pk + (j - 1) * PK_WORDS, len[j - 1], pk + j * PK_WORDS, len[j]) >= 0) s_bad = 1;
  }
  __syncthreads();
  const int nw = n_pad / 64;
  const size_t obase = (size_t)b * n_pad;
  if (s_bad) {  // reject the query: a root-only tree
    if (tid == 0) fc_flag(FC_ERR_WORD(out.err), FC_EBIT_INVALID);
    for (int i = tid; i < n_pad; i += BT_THREADS) {
      out.tok[obase + i] = (i == 0) ? root_tok[b] : FC_PAD_TOKEN;
      out.parent[obase + i] = -1;
      out.depth[obase + i] = (i == 0) ? 0 : -1;
      out.pos[obase + i] = (i == 0) ? kv_len[b] : -1;
      out.mask[(obase + i) * nw] = (i == 0) ? 1ull : 0ull;
      if (nw > 1) out.mask[(obase + i) * nw + 1] = 0;
    }
    if (tid == 0) out.n_nodes[b] = 1;
    return;
  }

  // 2. merged order: own index plus, per other source, the drafts before it
  for (uint32_t j = tid; j < M; j += BT_THREADS) {
    const int s = src_of(j);
    const uint64_t* a = pk + j * PK_WORDS;
    const int la = len[j];
    uint32_t rank = j - s_off[s];
    for (int s2 = 0; s2 < S; ++s2) {
      if (s2 == s) continue;
      uint32_t lo = s_off[s2], hi = s_off[s2 + 1];  // first draft of s2 not before j
      while (lo < hi) {
        const uint32_t mid = (lo + hi) >> 1;
        const int c = cmp_packed(pk + mid * PK_WORDS, len[mid], a, la);
        if (c < 0 || (c == 0 && s2 < s)) lo = mid + 1;
        else hi = mid;
      }
      rank += lo - s_off[s2];
    }
    order[rank] = j;
  }
  __syncthreads();
  // 3. unique drafts (equal ones, from different sources, are adjacent) and their weights
  for (uint32_t r = tid; r < M; r += BT_THREADS) {
    flag[r] = (r == 0 || cmp_packed(pk + order[r - 1] * PK_WORDS, len[order[r - 1]], pk + order[r] * PK_WORDS,
                                    len[order[r]]) != 0) ? 1u : 0u;
    coff[r] = flag[r];
  }
  __syncthreads();
  const uint32_t U = block_scan_array(coff, (int)M, wsum);
  for (uint32_t u = tid; u < U; u += BT_THREADS) wu[u] = 0;
  __syncthreads();
  for (uint32_t r = tid; r < M; r += BT_THREADS) {
    const uint32_t u = coff[r] + flag[r] - 1u;
    if (flag[r]) uniq[u] = order[r];
    atomicAdd(reinterpret_cast<unsigned long long*>(&wu[u]), (unsigned long long)w[order[r]]);
  }
  __syncthreads();
  // 4. neighbour LCPs, weight prefix sums, candidate offsets
  for (uint32_t u = tid; u < U; u += BT_THREADS) {
    uint32_t l = 0;
    if (u > 0) {
      const uint32_t* a = tok + uniq[u - 1] * d;
      const uint32_t* c = tok + uniq[u] * d;
      const int lim = min(len[uniq[u - 1]], len[uniq[u]]);
      while ((int)l < lim && a[l] == c[l]) ++l;
    }
    lcp[u] = l;
    coff[u] = (uint32_t)len[uniq[u]] - l;
  }
  __syncthreads();
  if (tid < 32) warp_scan_u64(wu, ps, U);
  const uint32_t C = block_scan_array(coff, (int)U, wsum);
  for (uint32_t x = tid; x < U * (uint32_t)d; x += BT_THREADS) tab[x] = 0;
  // 5. per depth: number the runs (starts: lcp < l), then every node (u, l)
  //    gets its weight from its run and its parent from the run one level up
  for (int l = 1; l <= d; ++l) {
    for (uint32_t u = tid; u < U; u += BT_THREADS) rid[u] = (u == 0 || (int)lcp[u] < l) ? 1u : 0u;
    __syncthreads();
    const uint32_t R = block_scan_array(rid, (int)U, wsum);  // rid[u] = starts before u
    for (uint32_t u = tid; u < U; u += BT_THREADS) {
      if (u == 0 || (int)lcp[u] < l) {
        rpos[rid[u]] = u;
      } else {
        rid[u] -= 1u;  // the run u belongs to
      }
    }
    if (tid == 0) rpos[R] = U;
    __syncthreads();
    for (uint32_t u = tid; u < U; u += BT_THREADS) {
      if ((int)lcp[u] < l && l <= len[uniq[u]]) {  // node (u, l) is new at u, which starts its run
        const uint32_t e = rpos[rid[u] + 1];
        const uint64_t W = ps[e] - ps[u];
        const uint32_t c = coff[u] + (uint32_t)(l - (int)lcp[u] - 1);
        ckey[c] = (W << 18) | ((uint64_t)(31 - l) << 13) | (uint64_t)(8191u - u);
        cpar[c] = (l > 1) ? rpos_p[rid_p[u]] : 0u;
      }
    }
    __syncthreads();
    uint32_t* t0 = rid_p;
    rid_p = rid;
    rid = t0;
    t0 = rpos_p;
    rpos_p = rpos;
    rpos = t0;
  }
  // 6. the nsel largest keys, kept flags, preorder ranks (as k_build_tree)
  const int nsel = (int)umin((uint32_t)(budget - 1), C);
  uint64_t thr = 0;
  if (nsel > 0 && (uint32_t)nsel < C) thr = radix_select_desc(ckey, C, (uint32_t)nsel, hist);
  for (uint32_t c = tid; c < C; c += BT_THREADS) {
    const uint64_t key = ckey[c];
    if (nsel > 0 && key >= thr) {
      const int u = 8191 - (int)(key & 8191u), l = 31 - (int)((key >> 13) & 31u);
      tab[u * d + l - 1] = 1u;
    }
  }
  __syncthreads();
  const uint32_t nkept = block_scan_array(tab, (int)(U * (uint32_t)d), wsum);
  if (nkept != (uint32_t)nsel && tid == 0) fc_flag(FC_ERR_WORD(out.err), FC_EBIT_INTERNAL);
  for (uint32_t c = tid; c < C; c += BT_THREADS) {
    const uint64_t key = ckey[c];
    if (nsel > 0 && key >= thr) {
      const int u = 8191 - (int)(key & 8191u), l = 31 - (int)((key >> 13) & 31u);
      const int idx = 1 + (int)tab[u * d + l - 1];
      if (idx < FC_MAX_NODES) {
        sel_u[idx] = u;
        sel_l[idx] = l;
        par_s[idx] = (l > 1) ? 1 + (int)tab[cpar[c] * d + l - 2] : 0;
      }
    }
  }
  if (tid == 0) par_s[0] = -1;
  __syncthreads();
  const int n = 1 + min(nsel, FC_MAX_NODES - 1);
  const int kvl = kv_len[b];
  for (int i = tid; i < n_pad; i += BT_THREADS) {
    uint32_t tk = FC_PAD_TOKEN;
    int pa = -1, de = -1, po = -1;
    uint64_t m0 = 0, m1 = 0;
    if (i < n) {
      tk = (i == 0) ? root_tok[b] : tok[uniq[sel_u[i]] * d + sel_l[i] - 1];
      de = (i == 0) ? 0 : sel_l[i];
      pa = par_s[i];
      po = kvl + de;
      for (int a = i; a >= 0; a = par_s[a]) {
        if (a < 64) m0 |= 1ull << a;
        else m1 |= 1ull << (a - 64);
      }
    }
    out.tok[obase + i] = tk;
    out.parent[obase + i] = pa;
    out.depth[obase + i] = de;
    out.pos[obase + i] = po;
    out.mask[(obase + i) * nw] = m0;
    if (nw > 1) out.mask[(obase + i) * nw + 1] = m1;
  }
  if (tid == 0) out.n_nodes[b] = n;
}

// Mask, depth, position ids from parent pointers: one warp per tree.
__global__ void k_tree_mask(const int32_t* __restrict__ parent, const int32_t* __restrict__ n_nodes,
                            const int32_t* __restrict__ kv_len, int B, int n_pad, int32_t* __restrict__ depth,
                            int32_t* __restrict__ pos, uint64_t* __restrict__ mask, unsigned int* err) {
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (warp >= B) return;
  const int b = warp, nw = n_pad / 64;
  const size_t base = (size_t)b * n_pad;
  const int n = n_nodes[b];
  bool bad = (n < 1 || n > n_pad);
  for (int i = lane; i < n_pad && !bad; i += 32)
    if (i < n && i > 0 && (parent[base + i] < 0 || parent[base + i] >= i)) bad = true;
  bad = __any_sync(0xFFFFFFFFu, bad);
  if (bad && lane == 0) fc_flag(FC_ERR_WORD(err), FC_EBIT_INVALID);
  for (int i = lane; i < n_pad; i += 32) {
    uint64_t m0 = 0, m1 = 0;
    int de = -1, po = -1;
    if (!bad && i < n) {
      de = 0;
      for (int a = i; a >= 0; a = (a == 0) ? -1 : parent[base + a]) {
        if (a < 64) m0 |= 1ull << a;
        else m1 |= 1ull << (a - 64);
        if (a != i) ++de;
      }
      po = kv_len[b] + de;
    }
    depth[base + i] = de;
    pos[base + i] = po;
    mask[(base + i) * nw] = m0;
    if (nw > 1) mask[(base + i) * nw + 1] = m1;
  }
}

}  // namespace

extern "C" fc_status fc_build_tree(int n_sources, const uint32_t* d_drafts, const int32_t* d_draft_len,
                                   const uint32_t* d_count, const int32_t* d_n_drafts, const uint32_t* src_weight,
                                   int top_k, int draft_len, const uint32_t* d_root_tok, const int32_t* d_kv_len,
                                   int batch, int node_budget, int n_pad, uint32_t* d_tok, int32_t* d_parent,
                                   int32_t* d_depth, int32_t* d_pos, uint64_t* d_mask, int32_t* d_n_nodes,
                                   fc_stream stream) {
  FC_NVTX_RANGE();
  if (n_sources < 1 || n_sources > FC_MAX_SOURCES || top_k < 1 || draft_len < 1 || batch < 0 || !src_weight)
    return FC_ERR_INVALID_ARG;
  if (n_pad != 64 && n_pad != 128) return FC_ERR_UNSUPPORTED;
  if (node_budget < 1 || node_budget > n_pad) return FC_ERR_INVALID_ARG;
  if (n_sources * top_k > BT_MAX_DRAFTS || draft_len > FC_MAX_DRAFT_LEN || top_k > FC_MAX_TOPK)
    return FC_ERR_UNSUPPORTED;
  for (int s = 0; s < n_sources; ++s)
    if (src_weight[s] > 65535u) return FC_ERR_UNSUPPORTED;
  if (batch == 0) return FC_OK;
  if (!d_drafts || !d_draft_len || !d_count || !d_n_drafts || !d_root_tok || !d_kv_len || !d_tok || !d_parent ||
      !d_depth || !d_pos || !d_mask || !d_n_nodes)
    return FC_ERR_INVALID_ARG;
  TreeIn in{d_drafts, d_draft_len, d_count, d_n_drafts, {0, 0, 0, 0}};
  for (int s = 0; s < n_sources; ++s) in.w[s] = src_weight[s];
  TreeOut out{d_tok, d_parent, d_depth, d_pos, d_mask, d_n_nodes, fc_error_slot()};
  const size_t smem = bt_layout(n_sources * top_k, draft_len).total;
  if (cudaFuncSetAttribute(k_build_tree, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
    return FC_ERR_CUDA;
  k_build_tree<<<batch, BT_THREADS, smem, static_cast<cudaStream_t>(stream)>>>(
      in, n_sources, batch, top_k, draft_len, d_root_tok, d_kv_len, node_budget, n_pad, out);
  return FC_CHECK_LAUNCH();
}

extern "C" fc_status fc_tree_mask(const int32_t* d_parent, const int32_t* d_n_nodes, const int32_t* d_kv_len,
                                  int batch, int n_pad, int32_t* d_depth, int32_t* d_pos, uint64_t* d_mask,
                                  fc_stream stream) {
  FC_NVTX_RANGE();
  if (batch < 0) return FC_ERR_INVALID_ARG;
  if (n_pad != 64 && n_pad != 128) return FC_ERR_UNSUPPORTED;
  if (batch == 0) return FC_OK;
  if (!d_parent || !d_n_nodes || !d_kv_len || !d_depth || !d_pos || !d_mask) return FC_ERR_INVALID_ARG;
  const int threads = 128;
  const unsigned blocks = (unsigned)((batch * 32 + threads - 1) / threads);
  k_tree_mask<<<blocks, threads, 0, static_cast<cudaStream_t>(stream)>>>(d_parent, d_n_nodes, d_kv_len, batch, n_pad,
                                                                         d_depth, d_pos, d_mask, fc_error_slot());
  return FC_CHECK_LAUNCH();
}

static size_t bta_per_query(int n_sources, int slots, int draft_len) {
  return (all_layout(n_sources * slots, draft_len).total + 255) & ~(size_t)255;
}

extern "C" size_t fc_build_tree_all_workspace(int n_sources, int slots, int draft_len, int batch) {
  if (n_sources < 1 || n_sources > FC_MAX_SOURCES || slots < 1 || draft_len < 1 || draft_len > FC_MAX_DRAFT_LEN ||
      batch < 1 || n_sources * slots > BTA_MAX_DRAFTS)
    return 0;
  return bta_per_query(n_sources, slots, draft_len) * (size_t)batch;
}

extern "C" fc_status fc_build_tree_all(int n_sources, const uint32_t* d_drafts, const int32_t* d_draft_len,
                                       const uint32_t* d_count, const int32_t* d_n_drafts,
                                       const uint32_t* src_weight, int slots, int draft_len,
                                       const uint32_t* d_root_tok, const int32_t* d_kv_len, int batch,
                                       int node_budget, int n_pad, void* d_ws, size_t ws_bytes, uint32_t* d_tok,
                                       int32_t* d_parent, int32_t* d_depth, int32_t* d_pos, uint64_t* d_mask,
                                       int32_t* d_n_nodes, fc_stream stream) {
  FC_NVTX_RANGE();
  if (n_sources < 1 || n_sources > FC_MAX_SOURCES || slots < 1 || draft_len < 1 || batch < 0 || !src_weight)
    return FC_ERR_INVALID_ARG;
  if (n_pad != 64 && n_pad != 128) return FC_ERR_UNSUPPORTED;
  if (node_budget < 1 || node_budget > n_pad) return FC_ERR_INVALID_ARG;
  if (n_sources * slots > BTA_MAX_DRAFTS || draft_len > FC_MAX_DRAFT_LEN) return FC_ERR_UNSUPPORTED;
  for (int s = 0; s < n_sources; ++s)
    if (src_weight[s] > 65535u) return FC_ERR_UNSUPPORTED;
  if (batch == 0) return FC_OK;
  if (!d_drafts || !d_draft_len || !d_count || !d_n_drafts || !d_root_tok || !d_kv_len || !d_tok || !d_parent ||
      !d_depth || !d_pos || !d_mask || !d_n_nodes)
    return FC_ERR_INVALID_ARG;
  const size_t per = bta_per_query(n_sources, slots, draft_len);
  if (!d_ws || ws_bytes < per * (size_t)batch) return FC_ERR_WORKSPACE;
  if (reinterpret_cast<uintptr_t>(d_ws) % 256) return FC_ERR_INVALID_ARG;
  TreeIn in{d_drafts, d_draft_len, d_count, d_n_drafts, {0, 0, 0, 0}};
  for (int s = 0; s < n_sources; ++s) in.w[s] = src_weight[s];
  TreeOut out{d_tok, d_parent, d_depth, d_pos, d_mask, d_n_nodes, fc_error_slot()};
  k_build_tree_all<<<batch, BT_THREADS, 0, static_cast<cudaStream_t>(stream)>>>(
      in, n_sources, batch, slots, draft_len, d_root_tok, d_kv_len, node_budget, n_pad,
      static_cast<unsigned char*>(d_ws), per, out);
  return FC_CHECK_LAUNCH();
}
