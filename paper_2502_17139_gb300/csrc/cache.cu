// The CACHE and the missing table of Algorithm 1 (Section IV-B; Section
// IV-C, Algorithm 1; Section V-C: l = 50, output pieces of 20 tokens).
//
// k_cache_search, one CTA per query.  A CACHE holds at most
// FC_CACHE_MAX_WORDS words, so the CTA copies it into shared memory and scans
// every position; no suffix array is kept, because the store changes every
// step.
//   * pass 1: at every position p whose word is not a separator, the length
//     of the common suffix of the words before p and the context (at most
//     min(n_max, m)), kept as one byte per position.  A separator never
//     equals a context token, so a match stays inside its stored sequence.
//     The block maximum is n*.
//   * pass 2: the positions whose length reaches n* are the occurrences.
//   * the stores repeat text (each verified retrieval keeps the context
//     suffix, so consecutive entries overlap), so many occurrences carry the
//     same continuation.  Each occurrence becomes a packed row (its
//     continuation, cut at d tokens or at the separator); a shared-memory
//     hash table with exact comparison collapses equal rows into one
//     distinct row with a count.
//   * the distinct rows are sorted in token order: a few by ranking (every
//     row counts the rows before it), more by a bitonic sort with one element
//     (first 16-byte chunk and row) per thread, partners closer than a warp
//     trading through shuffles.  The first chunk decides most comparisons in
//     registers, and a tie reads the next chunks one by one.  All windows share the n*
//     matched tokens, so the first max_occ occurrences in this order are the
//     ones with the smallest windows: the cap shortens the run it cuts.
//   * topk_runs keeps the top-k runs by (count desc, token order).
//   * more occurrences than rows (a store of one repeated n-gram): a bitonic
//     sort of the positions that compares continuations in the store.
//   * a query the CACHE does not serve probes the missing table M.
// k_missing_insert, one CTA for the batch: dedups the new keys (against M and
// against earlier queries of the batch), admits them in query order while M
// has room, and claims slots with atomicCAS.  The keys it inserts are
// distinct and absent, so no thread ever waits on another's slot.
// k_cache_update, one warp per query: appends the verified retrieval and the
// completed output pieces.
#include <algorithm>

#include "fc_common.cuh"
#include "fc_topk.cuh"

FC_DEFINE_ERROR_WORD(cache)

namespace {

constexpr int CS_THREADS = 512;
constexpr int MI_THREADS = 1024;
constexpr int CU_WARPS = 8;
constexpr uint32_t NO_POS = 0xFFFFFFFFu;  // bitonic padding, sorts last
constexpr int M_HEADER = 4;               // words before the slots of M
constexpr uint32_t RANK_SORT_MAX = 128;   // distinct rows sorted by ranking rather than bitonic stages
constexpr uint32_t ROWS_MIN = 512;        // rows always available
constexpr uint32_t ROWS_MAX = 1024;       // most occurrences sorted over packed rows
constexpr uint32_t NO_IDX = 0xFFFFFFFFu;

struct CacheView {
  uint32_t* words;
  int32_t* meta;
  int capacity, min_size, chunk, ctx_keep;
  unsigned int* err;  // the launch's error word (NULL: this file's own)
};

struct ResOut {
  uint32_t* drafts;
  int32_t* draft_len;
  uint32_t* count;
  int32_t* n_drafts;
  int32_t* match_len;
};

// ------------------------------------------------------------ missing table
// key token i comes from at(i), i < len
template <class At>
__device__ __forceinline__ uint64_t key_hash(At at, int len) {
  uint64_t h = 0x9E3779B97F4A7C15ull ^ (uint64_t)len;
  for (int i = 0; i < len; ++i) {
    h = (h ^ at(i)) * 0xBF58476D1CE4E5B9ull;
    h ^= h >> 31;
  }
  return h;
}
__device__ __forceinline__ uint32_t key_tag(uint64_t h) { return (uint32_t)(h >> 32) | 1u; }

// true when the key is in M.  M never holds more than capacity / 2 keys, so a
// probe sequence always reaches an empty slot.
template <class At>
__device__ bool missing_contains(const uint32_t* table, int capacity, int key_len, At at) {
  const uint64_t h = key_hash(at, key_len);
  const uint32_t tag = key_tag(h);
  const uint32_t mask = (uint32_t)capacity - 1u;
  const size_t sw = 1 + (size_t)key_len;
  for (uint32_t probe = 0; probe < (uint32_t)capacity; ++probe) {
    const uint32_t* slot = table + M_HEADER + (size_t)(((uint32_t)h + probe) & mask) * sw;
    const uint32_t t = slot[0];
    if (t == 0) return false;
    if (t == tag) {
      bool eq = true;
      for (int i = 0; i < key_len && eq; ++i) eq = slot[1 + i] == at(i);
      if (eq) return true;
    }
  }
  return false;
}

// ------------------------------------------------------------- CACHE search
// Order of the continuations at positions a and b of a store T[0..n_tok): a
// continuation ends after d tokens or at its separator, and a shorter one
// sorts before its extensions.  Both sides' FC_MAX_DRAFT_LEN tokens are
// loaded first (independent loads, clamped inside the store) and compared in
// registers, instead of a chain of dependent loads.  n_tok >= 1.
__device__ __forceinline__ int cont_cmp16(const uint32_t* T, uint32_t n_tok, uint32_t a, uint32_t b, int d) {
  uint32_t ta[FC_MAX_DRAFT_LEN], tb[FC_MAX_DRAFT_LEN];
#pragma unroll
  for (int i = 0; i < FC_MAX_DRAFT_LEN; ++i) {
    const uint32_t ia = a + i, ib = b + i;
    ta[i] = T[min(ia, n_tok - 1)];
    tb[i] = T[min(ib, n_tok - 1)];
    if (ia >= n_tok || i >= d) ta[i] = FC_SEP_TOKEN;
    if (ib >= n_tok || i >= d) tb[i] = FC_SEP_TOKEN;
  }
  int res = 0;
  bool done = false;
#pragma unroll
  for (int i = 0; i < FC_MAX_DRAFT_LEN; ++i) {
    const bool ea = ta[i] == FC_SEP_TOKEN, eb = tb[i] == FC_SEP_TOKEN;
    if (!done && (ea || eb || ta[i] != tb[i])) {
      done = true;
      res = (ea && eb) ? 0 : ea ? -1 : eb ? 1 : (ta[i] < tb[i] ? -1 : 1);
    }
  }
  return res;
}

struct CsSmem {
  uint32_t work[FC_MAX_OCC];  // first: 16-byte aligned, also the distinct rows' sort elements
  uint32_t runs[FC_MAX_OCC + 1];
  uint32_t sel[FC_MAX_TOPK];
  uint32_t order[FC_MAX_TOPK];
  uint32_t rctx[FC_MAX_NMAX];                        // the context suffix, last token first
  uint32_t wsum[CS_THREADS / 32];
  RunsScratch rs;
  uint32_t best, nocc, bad, n_rep;
  int state;
};

__host__ __device__ inline uint32_t pow2_ceil(uint32_t x) {
  uint32_t p = 1;
  while (p < x) p <<= 1;
  return p;
}

// dynamic shared memory: the fixed part, the staged store (capacity words),
// the occurrence list (the next power of two), the match lengths (bytes),
// then rows_cap packed rows (64 bytes each)
__host__ __device__ inline size_t cs_fixed_bytes() { return (sizeof(CsSmem) + 15) & ~(size_t)15; }
size_t cs_base_bytes(int capacity) {
  return cs_fixed_bytes() + 4 * (size_t)capacity + 4 * (size_t)pow2_ceil((uint32_t)capacity) +
         (((size_t)capacity + 15) & ~(size_t)15);
}
// the largest power of two <= ROWS_MAX whose rows fit next to the rest
uint32_t cs_rows_cap(int capacity, size_t smem_limit) {
  const size_t base = cs_base_bytes(capacity);
  uint32_t rc = ROWS_MAX;
  while (rc > ROWS_MIN && base + 64 * (size_t)rc > smem_limit) rc >>= 1;
  return rc;
}
size_t cs_smem_bytes(int capacity, uint32_t rows_cap) { return cs_base_bytes(capacity) + 64 * (size_t)rows_cap; }

// Row of a continuation: token t as t + 1, the end (after d
// tokens or at the separator) and everything past it as 0, so that comparing
// rows word by word is comparing continuations (a shorter one first).  Row x
// keeps its 16-byte chunk q at slot q ^ (x & 3): rows read at random indices
// then spread over all 32 banks instead of 8.
__device__ __forceinline__ void pack_row(const uint32_t* T, uint32_t n_tok, uint32_t pos, int d, uint4* row,
                                         uint32_t sw) {
  uint32_t w[FC_MAX_DRAFT_LEN];
  bool ended = false;
#pragma unroll
  for (int i = 0; i < FC_MAX_DRAFT_LEN; ++i) {
    const uint32_t t = (pos + i < n_tok) ? T[pos + i] : FC_SEP_TOKEN;
    ended = ended || i >= d || t == FC_SEP_TOKEN;
    w[i] = ended ? 0u : t + 1u;
  }
#pragma unroll
  for (int q = 0; q < FC_MAX_DRAFT_LEN / 4; ++q)
    row[q ^ sw] = make_uint4(w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]);
}

__device__ __forceinline__ bool rows_equal(const uint4 (*rows)[FC_MAX_DRAFT_LEN / 4], uint32_t ix, uint32_t iy) {
  bool eq = true;
#pragma unroll
  for (int q = 0; q < FC_MAX_DRAFT_LEN / 4; ++q) {
    const uint4 u = rows[ix][q ^ (ix & 3)], v = rows[iy][q ^ (iy & 3)];
    eq = eq && u.x == v.x && u.y == v.y && u.z == v.z && u.w == v.w;
  }
  return eq;
}

__device__ __forceinline__ uint32_t row_hash(const uint4 (*rows)[FC_MAX_DRAFT_LEN / 4], uint32_t ix) {
  uint64_t h = 0x9E3779B97F4A7C15ull;
#pragma unroll
  for (int q = 0; q < FC_MAX_DRAFT_LEN / 4; ++q) {
    const uint4 u = rows[ix][q ^ (ix & 3)];
    h = (h ^ u.x) * 0xBF58476D1CE4E5B9ull;
    h = (h ^ u.y) * 0x94D049BB133111EBull;
    h = (h ^ u.z) * 0xBF58476D1CE4E5B9ull;
    h = (h ^ u.w) * 0x94D049BB133111EBull;
  }
  return (uint32_t)(h ^ (h >> 32));
}

__global__ void __launch_bounds__(CS_THREADS, 1) k_cache_search(CacheView c, const uint32_t* __restrict__ table,
                                                             int table_cap, const uint32_t* __restrict__ ctx,
                                                             int stride, const int32_t* __restrict__ ctx_len, int B,
                                                             fc_retrieve_params p, int S, ResOut o,
                                                             int32_t* __restrict__ state, uint32_t rows_cap) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  CsSmem& sm = *reinterpret_cast<CsSmem*>(smem_raw);
  uint32_t* T = reinterpret_cast<uint32_t*>(smem_raw + cs_fixed_bytes());
  uint32_t* occ = T + c.capacity;
  uint8_t* mlen = reinterpret_cast<uint8_t*>(occ + pow2_ceil((uint32_t)c.capacity));
  uint4(*rows)[FC_MAX_DRAFT_LEN / 4] =
      reinterpret_cast<uint4(*)[FC_MAX_DRAFT_LEN / 4]>(mlen + ((c.capacity + 15) & ~15));
  const int b = blockIdx.x, tid = threadIdx.x;
  const int k = p.top_k, d = p.draft_len;

  // ---- prologue: the context suffix and the store, behind one barrier
  int m = ctx_len[b];
  m = max(0, min(m, stride));
  const int cap = min(p.n_max, m);
  const int32_t* meta = c.meta + 4 * (size_t)b;
  const int nt_raw = meta[0];
  const uint32_t n_tok = (nt_raw >= 0 && nt_raw <= c.capacity) ? (uint32_t)nt_raw : 0u;
  const bool searched = meta[1] >= c.min_size && cap >= p.n_min && n_tok >= 2;
  if (tid == 0) {
    sm.bad = 0;
    sm.best = 0;
    sm.nocc = 0;
    if (nt_raw < 0 || nt_raw > c.capacity) fc_flag(FC_ERR_WORD(c.err), FC_EBIT_INTERNAL);
  }
  __syncthreads();
  if (tid < cap) {
    const uint32_t t = ctx[(size_t)b * stride + (m - 1 - tid)];
    sm.rctx[tid] = t;
    if (t >= FC_SEP_TOKEN) sm.bad = 1;
  }
  if (searched) {  // 16-byte rows; the capacity is a multiple of 4 words
    const uint4* src = reinterpret_cast<const uint4*>(c.words + (size_t)b * c.capacity);
    uint4* dst = reinterpret_cast<uint4*>(T);
    for (uint32_t i = tid; i < (n_tok + 3) / 4; i += CS_THREADS) dst[i] = src[i];
  }
  __syncthreads();
  const bool bad = sm.bad != 0;
  if (bad && tid == 0) fc_flag(FC_ERR_WORD(c.err), FC_EBIT_INVALID);
  const bool active = searched && !bad;

  // ---- pass 1: at every position with a continuation, the length of the
  // common suffix of the words before it and the context (at most cap)
  if (active) {
    const uint32_t last = sm.rctx[0];
    uint32_t best = 0;
    for (uint32_t q0 = tid; q0 < n_tok; q0 += 4 * CS_THREADS) {
      uint32_t tq[4], tp[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const uint32_t q = q0 + u * CS_THREADS;
        tq[u] = (q < n_tok) ? T[q] : FC_SEP_TOKEN;
        tp[u] = (q >= 1 && q < n_tok) ? T[q - 1] : FC_SEP_TOKEN;
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const uint32_t q = q0 + u * CS_THREADS;
        uint32_t len = 0;
        if (tq[u] != FC_SEP_TOKEN && tp[u] == last) {
          len = 1;
          while (len < (uint32_t)cap && len < q && T[q - 1 - len] == sm.rctx[len]) ++len;
        }
        if (q < n_tok) mlen[q] = (uint8_t)len;
        best = max(best, len);
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) best = max(best, __shfl_xor_sync(0xFFFFFFFFu, best, off));
    if ((tid & 31) == 0 && best > 0) atomicMax(&sm.best, best);
    __syncthreads();
  }
  const uint32_t ns = active && sm.best >= (uint32_t)p.n_min ? sm.best : 0u;

  auto cont_cmp = [=](uint32_t a, uint32_t bpos) -> int { return cont_cmp16(T, n_tok, a, bpos, d); };
  // (continuation, position): a total order on the occurrences
  auto occ_before = [=](uint32_t a, uint32_t bpos) -> bool {
    if (a == NO_POS || bpos == NO_POS) return bpos == NO_POS && a != NO_POS;
    const int cr = cont_cmp(a, bpos);
    return cr < 0 || (cr == 0 && a < bpos);
  };

  uint32_t nd = 0;
  if (ns > 0) {
    // ---- pass 2: the occurrences are the positions whose length reaches n*
    for (uint32_t c16 = tid; c16 * 16 < n_tok; c16 += CS_THREADS) {
      const uint4 v = reinterpret_cast<const uint4*>(mlen)[c16];
      const uint32_t wv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
      for (int e = 0; e < 16; ++e) {
        const uint32_t q = c16 * 16 + e;
        if (q < n_tok && ((wv[e >> 2] >> (8 * (e & 3))) & 0xFFu) >= ns) occ[atomicAdd(&sm.nocc, 1u)] = q;
      }
    }
    __syncthreads();
    const uint32_t nocc = sm.nocc;
    const uint32_t kept = min(nocc, p.max_occ);
    if (nocc <= rows_cap) {
      // ---- equal continuations collapse first: each occurrence becomes a
      // packed row; a hash table over the rows (exact comparison on a hash
      // match) maps it to the first row with its content, which counts it
      uint32_t* ht = sm.runs;                  // HT slots: row + 1, 0 = empty
      uint32_t* cnt = sm.runs + 2 * ROWS_MAX;  // per row: its occurrences
      uint32_t* rpos = sm.runs + 3 * ROWS_MAX; // per row: its position
      uint4* sk = reinterpret_cast<uint4*>(sm.work);  // sort elements: first chunk ...
      uint32_t* sr = sm.runs;                          // ... and row (after the table)
      const uint32_t HT = 2 * pow2_ceil(nocc);
      for (uint32_t i = tid; i < nocc; i += CS_THREADS) {
        pack_row(T, n_tok, occ[i], d, rows[i], i & 3);
        cnt[i] = 0;
        rpos[i] = occ[i];
      }
      for (uint32_t i = tid; i < HT; i += CS_THREADS) ht[i] = 0;
      if (tid == 0) sm.n_rep = 0;
      __syncthreads();
      uint32_t my_rep[2] = {NO_IDX, NO_IDX};  // distinct rows this thread found
#pragma unroll
      for (int it = 0; it < 2; ++it) {
        const uint32_t i = tid + it * CS_THREADS;
        if (i >= nocc) continue;
        const uint32_t h = row_hash(rows, i);
        uint32_t rep = i;
        for (uint32_t probe = 0; probe < HT; ++probe) {
          const uint32_t v = atomicCAS(&ht[(h + probe) & (HT - 1)], 0u, i + 1);
          if (v == 0) break;
          if (rows_equal(rows, v - 1, i)) {
            rep = v - 1;
            break;
          }
        }
        atomicAdd(&cnt[rep], 1u);
        if (rep == i) my_rep[it] = i;
      }
      __syncthreads();  // the table is done with: its words now hold rows
#pragma unroll
      for (int it = 0; it < 2; ++it) {
        if (my_rep[it] == NO_IDX) continue;
        const uint32_t i = my_rep[it], slot = atomicAdd(&sm.n_rep, 1u);
        sk[slot] = rows[i][i & 3];
        sr[slot] = i;
      }
      __syncthreads();
      // ---- sort the R distinct rows in token order.  An element is its
      // first chunk and its row; the first chunk decides most comparisons in
      // registers, and a tie reads the next chunks one at a time.
      const uint32_t R = sm.n_rep;
      const uint32_t n2 = pow2_ceil(R);
      const int nchunks = (d + 3) / 4;
      const uint4 top = make_uint4(0xFFFFFFFFu, 0xFFFFFFFFu, 0xFFFFFFFFu, 0xFFFFFFFFu);  // above every real chunk
      for (uint32_t i = R + tid; i < n2; i += CS_THREADS) {
        sk[i] = top;
        sr[i] = NO_IDX;
      }
      auto cmp4 = [](const uint4& x, const uint4& y) -> int {
        return x.x != y.x ? (x.x < y.x ? -1 : 1)
             : x.y != y.y ? (x.y < y.y ? -1 : 1)
             : x.z != y.z ? (x.z < y.z ? -1 : 1)
             : x.w != y.w ? (x.w < y.w ? -1 : 1) : 0;
      };
      // -1 / 0 / 1; padding elements are equal to each other
      auto el_cmp = [&](const uint4& xk, uint32_t xr, const uint4& yk, uint32_t yr) -> int {
        int c = cmp4(xk, yk);
        if (c != 0 || xr == NO_IDX || yr == NO_IDX) return c;
        for (int q = 1; q < nchunks && c == 0; ++q) c = cmp4(rows[xr][q ^ (xr & 3)], rows[yr][q ^ (yr & 3)]);
        return c;
      };
      __syncthreads();
      if (n2 <= RANK_SORT_MAX) {
        // few rows: ranking.  A group of tpe threads counts the rows ordered
        // before one row; every comparison is independent, so many warps
        // share the work even for a handful of rows.
        const uint32_t tpe = min(32u, CS_THREADS / n2);
        const uint32_t i = tid / tpe, part = tid % tpe;
        uint4 mk = top;
        uint32_t mr = NO_IDX, rank = 0;
        if (i < R) {
          mk = sk[i];
          mr = sr[i];
          for (uint32_t j = part; j < R; j += tpe)
            if (j != i) rank += el_cmp(sk[j], sr[j], mk, mr) < 0 ? 1u : 0u;
        }
        for (uint32_t off = 1; off < tpe; off <<= 1) rank += __shfl_xor_sync(0xFFFFFFFFu, rank, off);
        __syncthreads();
        if (i < R && part == 0) {
          sk[rank] = mk;
          sr[rank] = mr;
        }
        __syncthreads();
      } else if (n2 <= CS_THREADS) {
        // bitonic sort with one element per thread: partners closer than a
        // warp trade through shuffles, farther ones through shared memory
        uint4 xk = tid < n2 ? sk[tid] : top;
        uint32_t xr = tid < n2 ? sr[tid] : NO_IDX;
        for (uint32_t kk = 2; kk <= n2; kk <<= 1) {
          for (uint32_t j = kk >> 1; j > 0; j >>= 1) {
            uint4 yk;
            uint32_t yr;
            if (j >= 32) {
              __syncthreads();
              if (tid < n2) {
                sk[tid] = xk;
                sr[tid] = xr;
              }
              __syncthreads();
              yk = tid < n2 ? sk[tid ^ j] : xk;
              yr = tid < n2 ? sr[tid ^ j] : xr;
            } else {
              yk.x = __shfl_xor_sync(0xFFFFFFFFu, xk.x, j);
              yk.y = __shfl_xor_sync(0xFFFFFFFFu, xk.y, j);
              yk.z = __shfl_xor_sync(0xFFFFFFFFu, xk.z, j);
              yk.w = __shfl_xor_sync(0xFFFFFFFFu, xk.w, j);
              yr = __shfl_xor_sync(0xFFFFFFFFu, xr, j);
            }
            if (tid < n2) {
              const bool want_min = ((tid & j) == 0) == ((tid & kk) == 0);
              const int c = el_cmp(yk, yr, xk, xr);
              if (want_min ? c < 0 : c > 0) {
                xk = yk;
                xr = yr;
              }
            }
          }
        }
        __syncthreads();
        if (tid < n2) {
          sk[tid] = xk;
          sr[tid] = xr;
        }
        __syncthreads();
      } else {
        // bitonic sort in shared memory
        for (uint32_t kk = 2; kk <= n2; kk <<= 1) {
          for (uint32_t j = kk >> 1; j > 0; j >>= 1) {
            for (uint32_t i = tid; i < n2; i += CS_THREADS) {
              const uint32_t ixj = i ^ j;
              if (ixj > i) {
                const uint4 xk = sk[i], yk = sk[ixj];
                const uint32_t xr = sr[i], yr = sr[ixj];
                const int c = el_cmp(xk, xr, yk, yr);
                if ((i & kk) == 0 ? c > 0 : c < 0) {
                  sk[i] = yk;
                  sk[ixj] = xk;
                  sr[i] = yr;
                  sr[ixj] = xr;
                }
              }
            }
            __syncthreads();
          }
        }
      }
      // ---- runs in token order; the first `kept` occurrences survive the
      // max_occ cap, so the run holding the cut is shortened and later ones
      // drop out.  Run r's continuation sits at position occ[r].
      constexpr int RI = ROWS_MAX / CS_THREADS;
      uint32_t c_it[RI], p_it[RI], local = 0;
#pragma unroll
      for (int it = 0; it < RI; ++it) {
        const uint32_t r = tid * RI + it;
        c_it[it] = r < R ? cnt[sr[r]] : 0u;
        p_it[it] = r < R ? rpos[sr[r]] : 0u;
        local += c_it[it];
      }
      // (the scan's barriers separate these reads of sr from the writes of
      // runs, which share its words)
      uint32_t before = block_excl_scan<CS_THREADS>(local, &sm.rs.total, sm.wsum);
#pragma unroll
      for (int it = 0; it < RI; ++it) {
        const uint32_t r = tid * RI + it;
        if (r < R && before < kept) {
          sm.runs[r] = before;
          occ[r] = p_it[it];
          if (before + c_it[it] >= kept) {  // the last run that survives
            sm.runs[r + 1] = kept;
            sm.rs.n_runs = r + 1;
          }
        }
        before += c_it[it];
      }
      __syncthreads();
      nd = topk_runs<CS_THREADS>(sm.rs.n_runs, k, sm.runs, sm.work, sm.sel, sm.order, sm.wsum, sm.rs);
    } else {
      // more occurrences than rows: bitonic sort of the positions, comparing
      // continuations in the store; runs from neighbour comparisons
      const uint32_t n2 = pow2_ceil(nocc);
      for (uint32_t i = nocc + tid; i < n2; i += CS_THREADS) occ[i] = NO_POS;
      __syncthreads();
      for (uint32_t kk = 2; kk <= n2; kk <<= 1) {
        for (uint32_t j = kk >> 1; j > 0; j >>= 1) {
          for (uint32_t i = tid; i < n2; i += CS_THREADS) {
            const uint32_t ixj = i ^ j;
            if (ixj > i) {
              const uint32_t a = occ[i], bb = occ[ixj];
              const bool asc = (i & kk) == 0;
              if (a != bb && (asc ? occ_before(bb, a) : occ_before(a, bb))) {
                occ[i] = bb;
                occ[ixj] = a;
              }
            }
          }
          __syncthreads();
        }
      }
      for (uint32_t e = tid; e < kept; e += CS_THREADS)
        sm.work[e] = (e == 0 || cont_cmp(occ[e - 1], occ[e]) != 0) ? 1u : 0u;
      __syncthreads();
      const uint32_t R = runs_from_heads<CS_THREADS>(kept, sm.runs, sm.work, sm.wsum, sm.rs);
      // run r's continuation: its first occurrence
      uint32_t pos_it[FC_MAX_OCC / CS_THREADS];
#pragma unroll
      for (int it = 0; it < FC_MAX_OCC / CS_THREADS; ++it) {
        const uint32_t r = tid + it * CS_THREADS;
        pos_it[it] = r < R ? occ[sm.runs[r]] : 0u;
      }
      __syncthreads();
#pragma unroll
      for (int it = 0; it < FC_MAX_OCC / CS_THREADS; ++it) {
        const uint32_t r = tid + it * CS_THREADS;
        if (r < R) occ[r] = pos_it[it];
      }
      __syncthreads();
      nd = topk_runs<CS_THREADS>(R, k, sm.runs, sm.work, sm.sel, sm.order, sm.wsum, sm.rs);
    }

  }

  // ---- the CACHE slot (slot S) -----------------------------------------
  const size_t sb = (size_t)S * B + b;
  uint32_t* dr = o.drafts + sb * k * d;
  int32_t* dl = o.draft_len + sb * k;
  uint32_t* ct = o.count + sb * k;
  auto cont_len = [=](uint32_t pos) {
    int len = 0;
    while (len < d && pos + len < n_tok && T[pos + len] != FC_SEP_TOKEN) ++len;
    return len;
  };
  for (int e = tid; e < k * d; e += CS_THREADS) {
    const int t = e / d, x = e - t * d;
    uint32_t v = FC_PAD_TOKEN;
    if (t < (int)nd) {
      const uint32_t pos = occ[sm.order[t]];
      if (x < cont_len(pos)) v = T[pos + x];
    }
    dr[e] = v;
  }
  for (int t = tid; t < k; t += CS_THREADS) {
    if (t < (int)nd) {
      const uint32_t r = sm.order[t];
      dl[t] = cont_len(occ[r]);
      ct[t] = sm.runs[r + 1] - sm.runs[r];
    } else {
      dl[t] = 0;
      ct[t] = 0;
    }
  }
  if (tid == 0) {
    o.n_drafts[sb] = (int32_t)nd;
    o.match_len[sb] = nd ? (int32_t)ns : 0;
    int st = FC_SERVE_DATASTORE;
    if (nd > 0) {
      st = FC_SERVE_CACHE;
    } else if (table && !bad && m >= p.n_min) {
      // the key is the last n_min tokens, in reading order
      const uint32_t* rc = sm.rctx;
      const int kl = p.n_min;
      if (missing_contains(table, table_cap, kl, [=](int i) { return rc[kl - 1 - i]; })) st = FC_SKIP_MISSING;
    }
    state[b] = st;
    sm.state = st;
  }
  __syncthreads();
  if (sm.state == FC_SERVE_DATASTORE) return;
  // the datastore slots stay empty for a query that skips the datastore
  for (int s = 0; s < S; ++s) {
    const size_t q = (size_t)s * B + b;
    for (int e = tid; e < k * d; e += CS_THREADS) o.drafts[q * k * d + e] = FC_PAD_TOKEN;
    for (int e = tid; e < k; e += CS_THREADS) {
      o.draft_len[q * k + e] = 0;
      o.count[q * k + e] = 0;
    }
    if (tid == 0) {
      o.n_drafts[q] = 0;
      o.match_len[q] = 0;
    }
  }
}

// --------------------------------------------------------- missing insert
__global__ void __launch_bounds__(MI_THREADS) k_missing_insert(uint32_t* table, int capacity, int key_len,
                                                               const uint32_t* __restrict__ ctx, int stride,
                                                               const int32_t* __restrict__ ctx_len, int B,
                                                               const int32_t* __restrict__ state,
                                                               const int32_t* __restrict__ n_drafts, int S) {
  __shared__ uint32_t tags[MI_THREADS];
  __shared__ uint32_t wsum[MI_THREADS / 32];
  __shared__ uint32_t total;
  const int tid = threadIdx.x;
  const uint32_t limit = (uint32_t)capacity / 2;
  const uint32_t mask = (uint32_t)capacity - 1u;
  const size_t sw = 1 + (size_t)key_len;
  auto key_of = [&](int q) {
    const int mq = max(0, min((int)ctx_len[q], stride));
    return ctx + (size_t)q * stride + (mq - key_len);
  };
  for (int base = 0; base < B; base += MI_THREADS) {
    const int b = base + tid;
    bool pend = false;
    uint64_t h = 0;
    uint32_t tag = 0;
    const uint32_t* key = nullptr;
    if (b < B && state[b] == FC_SERVE_DATASTORE && min((int)ctx_len[b], stride) >= key_len) {
      bool empty = true;
      for (int s = 0; s < S; ++s) empty &= n_drafts[(size_t)s * B + b] == 0;
      if (empty) {
        key = key_of(b);
        const uint32_t* kp = key;
        auto at = [=](int i) { return kp[i]; };
        pend = !missing_contains(table, capacity, key_len, at);
        h = key_hash(at, key_len);
        tag = key_tag(h);
      }
    }
    tags[tid] = pend ? tag : 0u;
    __syncthreads();
    // a key repeated in the batch is inserted by its first query only
    if (pend) {
      for (int j = 0; j < tid && pend; ++j) {
        if (tags[j] != tag) continue;
        const uint32_t* other = key_of(base + j);
        bool eq = true;
        for (int i = 0; i < key_len && eq; ++i) eq = other[i] == key[i];
        if (eq) pend = false;
      }
    }
    const uint32_t rank = block_excl_scan<MI_THREADS>(pend ? 1u : 0u, &total, wsum);
    const uint32_t fill = table[0];
    if (pend && fill + rank < limit) {
      for (uint32_t probe = 0; probe < (uint32_t)capacity; ++probe) {
        uint32_t* slot = table + M_HEADER + (size_t)(((uint32_t)h + probe) & mask) * sw;
        if (atomicCAS(slot, 0u, tag) == 0u) {
          for (int i = 0; i < key_len; ++i) slot[1 + i] = key[i];
          break;
        }
      }
    }
    __syncthreads();
    if (tid == 0) {
      const uint32_t room = fill < limit ? limit - fill : 0u;
      const uint32_t admitted = min(total, room);
      table[0] = fill + admitted;
      table[1] += total - admitted;
    }
    __syncthreads();
  }
}

// ------------------------------------------------------------ CACHE update
__global__ void __launch_bounds__(CU_WARPS * 32) k_cache_update(CacheView c, const uint32_t* __restrict__ ctx,
                                                                int stride, const int32_t* __restrict__ len_old,
                                                                const int32_t* __restrict__ len_new,
                                                                const int32_t* __restrict__ acc_len, int B) {
  const int lane = threadIdx.x & 31;
  const int b = blockIdx.x * CU_WARPS + (threadIdx.x >> 5);
  if (b >= B) return;
  const int o = len_old[b], n = len_new[b], a = acc_len[b];
  int32_t* meta = c.meta + 4 * (size_t)b;
  int w = meta[0], ns = meta[1], mark = meta[2], dropped = meta[3];
  if (o < 0 || n < o || n > stride || mark < 0 || w < 0 || w > c.capacity) {
    if (lane == 0) fc_flag(FC_ERR_WORD(c.err), FC_EBIT_INVALID);
    return;
  }
  const uint32_t* row = ctx + (size_t)b * stride;
  uint32_t* words = c.words + (size_t)b * c.capacity;
  auto store = [&](int s0, int L) {
    bool bad = false;
    for (int i = lane; i < L; i += 32) bad |= row[s0 + i] >= FC_SEP_TOKEN;
    if (__any_sync(0xFFFFFFFFu, bad)) {
      if (lane == 0) fc_flag(FC_ERR_WORD(c.err), FC_EBIT_INVALID);
      return;
    }
    if (w + L + 1 <= c.capacity) {
      for (int i = lane; i < L; i += 32) words[w + i] = row[s0 + i];
      if (lane == 0) words[w + L] = FC_SEP_TOKEN;
      w += L + 1;
      ++ns;
    } else {
      ++dropped;
    }
  };
  if (n == o + a + 1 && a >= 1) {
    const int keep = min(c.ctx_keep, o);
    store(o - keep, keep + a);
  }
  while (n - mark >= c.chunk) {
    store(mark, c.chunk);
    mark += c.chunk;
  }
  __syncwarp();
  if (lane == 0) {
    meta[0] = w;
    meta[1] = ns;
    meta[2] = mark;
    meta[3] = dropped;
  }
}

__global__ void k_cache_init(int32_t* meta, const int32_t* __restrict__ prompt_len, int B) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  meta[4 * (size_t)b + 0] = 0;
  meta[4 * (size_t)b + 1] = 0;
  meta[4 * (size_t)b + 2] = prompt_len[b];
  meta[4 * (size_t)b + 3] = 0;
}

bool cache_ok(const fc_cache* c) {
  return c && c->d_words && c->d_meta && c->capacity >= 16 && c->capacity <= FC_CACHE_MAX_WORDS &&
         c->capacity % 4 == 0 && c->min_size >= 0 && c->chunk >= 1 && c->ctx_keep >= 0 &&
         c->ctx_keep <= FC_MAX_NMAX && reinterpret_cast<uintptr_t>(c->d_words) % 16 == 0;
}

bool missing_cap_ok(int capacity) {
  return capacity >= 2 && capacity <= (1 << 24) && (capacity & (capacity - 1)) == 0;
}

CacheView view_of(const fc_cache* c) {
  return CacheView{c->d_words, c->d_meta, c->capacity, c->min_size, c->chunk, c->ctx_keep, fc_error_slot()};
}

}  // namespace

extern "C" fc_status fc_cache_init(const fc_cache* cache, int batch, const int32_t* d_prompt_len, fc_stream stream) {
  FC_NVTX_RANGE();
  if (!cache_ok(cache) || batch < 0) return FC_ERR_INVALID_ARG;
  if (batch == 0) return FC_OK;
  if (!d_prompt_len) return FC_ERR_INVALID_ARG;
  k_cache_init<<<(batch + 255) / 256, 256, 0, static_cast<cudaStream_t>(stream)>>>(cache->d_meta, d_prompt_len,
                                                                                  batch);
  return FC_CHECK_LAUNCH();
}

extern "C" size_t fc_missing_bytes(int capacity, int key_len) {
  if (!missing_cap_ok(capacity) || key_len < 1 || key_len > FC_MAX_NMAX) return 0;
  return 4 * ((size_t)M_HEADER + (size_t)capacity * (1 + (size_t)key_len));
}

extern "C" fc_status fc_missing_init(void* d_table, size_t bytes, int capacity, int key_len, fc_stream stream) {
  FC_NVTX_RANGE();
  const size_t need = fc_missing_bytes(capacity, key_len);
  if (!d_table || need == 0) return FC_ERR_INVALID_ARG;
  if (bytes < need) return FC_ERR_WORKSPACE;
  return fc_cuda_status(cudaMemsetAsync(d_table, 0, need, static_cast<cudaStream_t>(stream)));
}

extern "C" fc_status fc_cache_search(const fc_cache* cache, const void* d_missing, int missing_capacity,
                                     const uint32_t* d_ctx, int ctx_stride, const int32_t* d_ctx_len, int batch,
                                     fc_retrieve_params p, int n_sources, uint32_t* d_drafts, int32_t* d_draft_len,
                                     uint32_t* d_count, int32_t* d_n_drafts, int32_t* d_match_len, int32_t* d_state,
                                     fc_stream stream) {
  FC_NVTX_RANGE();
  if (!cache_ok(cache) || batch < 0 || ctx_stride < 1 || n_sources < 0 || n_sources >= FC_MAX_SOURCES ||
      batch > 65535 * 16)
    return FC_ERR_INVALID_ARG;
  if (d_missing && !missing_cap_ok(missing_capacity)) return FC_ERR_INVALID_ARG;
  if (!fc_retrieve_params_ok(p))
    return (p.n_max > 0 && p.top_k > 0 && p.draft_len > 0) ? FC_ERR_UNSUPPORTED : FC_ERR_INVALID_ARG;
  if (batch == 0) return FC_OK;
  if (!d_ctx || !d_ctx_len || !d_drafts || !d_draft_len || !d_count || !d_n_drafts || !d_match_len || !d_state)
    return FC_ERR_INVALID_ARG;
  // the device's opt-in shared memory per block, set as the kernel's limit once per device
  static std::atomic<unsigned long long> attr_done;
  static std::atomic<size_t> dev_limit[64];
  size_t smem_limit = 0;
  const fc_status st = fc_once_per_device(attr_done, [&](int dev) {
    int optin = 0;
    if (cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess) return FC_ERR_CUDA;
    const size_t limit = (size_t)optin;
    if (cs_smem_bytes(FC_CACHE_MAX_WORDS, cs_rows_cap(FC_CACHE_MAX_WORDS, limit)) > limit) return FC_ERR_INTERNAL;
    if (cudaFuncSetAttribute(k_cache_search, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)limit) != cudaSuccess)
      return FC_ERR_CUDA;
    if (dev < 64) dev_limit[dev].store(limit);
    smem_limit = limit;
    return FC_OK;
  });
  if (st != FC_OK) return st;
  if (!smem_limit) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev >= 64) return FC_ERR_CUDA;
    smem_limit = dev_limit[dev].load();
  }
  const uint32_t rows_cap = cs_rows_cap(cache->capacity, smem_limit);
  ResOut o{d_drafts, d_draft_len, d_count, d_n_drafts, d_match_len};
  k_cache_search<<<batch, CS_THREADS, cs_smem_bytes(cache->capacity, rows_cap),
                   static_cast<cudaStream_t>(stream)>>>(view_of(cache), static_cast<const uint32_t*>(d_missing),
                                                        missing_capacity, d_ctx, ctx_stride, d_ctx_len, batch, p,
                                                        n_sources, o, d_state, rows_cap);
  return FC_CHECK_LAUNCH();
}

extern "C" fc_status fc_missing_insert(void* d_missing, int missing_capacity, int key_len, const uint32_t* d_ctx,
                                       int ctx_stride, const int32_t* d_ctx_len, int batch, const int32_t* d_state,
                                       const int32_t* d_n_drafts, int n_sources, fc_stream stream) {
  FC_NVTX_RANGE();
  if (!d_missing || !missing_cap_ok(missing_capacity) || key_len < 1 || key_len > FC_MAX_NMAX || batch < 0 ||
      ctx_stride < 1 || n_sources < 0 || n_sources > FC_MAX_SOURCES)
    return FC_ERR_INVALID_ARG;
  if (batch == 0) return FC_OK;
  if (!d_ctx || !d_ctx_len || !d_state || (n_sources > 0 && !d_n_drafts)) return FC_ERR_INVALID_ARG;
  k_missing_insert<<<1, MI_THREADS, 0, static_cast<cudaStream_t>(stream)>>>(
      static_cast<uint32_t*>(d_missing), missing_capacity, key_len, d_ctx, ctx_stride, d_ctx_len, batch, d_state,
      d_n_drafts, n_sources);
  return FC_CHECK_LAUNCH();
}

extern "C" fc_status fc_cache_update(const fc_cache* cache, const uint32_t* d_ctx, int ctx_stride,
                                     const int32_t* d_ctx_len_old, const int32_t* d_ctx_len_new,
                                     const int32_t* d_acc_len, int batch, fc_stream stream) {
  FC_NVTX_RANGE();
  if (!cache_ok(cache) || batch < 0 || ctx_stride < 1) return FC_ERR_INVALID_ARG;
  if (batch == 0) return FC_OK;
  if (!d_ctx || !d_ctx_len_old || !d_ctx_len_new || !d_acc_len) return FC_ERR_INVALID_ARG;
  k_cache_update<<<(batch + CU_WARPS - 1) / CU_WARPS, CU_WARPS * 32, 0, static_cast<cudaStream_t>(stream)>>>(
      view_of(cache), d_ctx, ctx_stride, d_ctx_len_old, d_ctx_len_new, d_acc_len, batch);
  return FC_CHECK_LAUNCH();
}
