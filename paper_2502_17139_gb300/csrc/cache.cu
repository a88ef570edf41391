// The CACHE and the missing table of Algorithm 1 (Section IV-B; Section
// IV-C, Algorithm 1; Section V-C: l = 50, output pieces of 20 tokens).
//
// k_cache_search, one CTA per query.  A CACHE holds at most
// FC_CACHE_MAX_WORDS words, so the CTA copies it into shared memory and scans
// every position; no suffix array is kept, because the store changes every
// step.
//   * pass 1: at every position p whose word is not a separator, the length
//     of the common suffix of the words before p and the context (at most
//     min(n_max, m)).  A separator never equals a context token, so a match
//     stays inside its stored sequence.  The block maximum is n*.
//   * pass 2: the positions whose common suffix reaches n* are the
//     occurrences; they are bitonic-sorted by (continuation, position), a
//     continuation ending after d tokens or at its separator, a shorter one
//     before its extensions.  All windows share the n* matched tokens, so
//     the first max_occ occurrences are those with the smallest windows.
//   * equal neighbours form runs; rank_runs keeps the top-k by
//     (count desc, token order).
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

struct CacheView {
  uint32_t* words;
  int32_t* meta;
  int capacity, min_size, chunk, ctx_keep;
};

struct ResOut {
  uint32_t* drafts;
  int32_t* draft_len;
  uint32_t* count;
  int32_t* n_drafts;
  int32_t* match_len;
};

// ------------------------------------------------------------ missing table
__device__ __forceinline__ uint64_t key_hash(const uint32_t* key, int len) {
  uint64_t h = 0x9E3779B97F4A7C15ull ^ (uint64_t)len;
  for (int i = 0; i < len; ++i) {
    h = (h ^ key[i]) * 0xBF58476D1CE4E5B9ull;
    h ^= h >> 31;
  }
  return h;
}
__device__ __forceinline__ uint32_t key_tag(uint64_t h) { return (uint32_t)(h >> 32) | 1u; }

// true when `key` is in M.  M never holds more than capacity / 2 keys, so a
// probe sequence always reaches an empty slot.
__device__ bool missing_contains(const uint32_t* table, int capacity, int key_len, const uint32_t* key) {
  const uint64_t h = key_hash(key, key_len);
  const uint32_t tag = key_tag(h);
  const uint32_t mask = (uint32_t)capacity - 1u;
  const size_t sw = 1 + (size_t)key_len;
  for (uint32_t probe = 0; probe < (uint32_t)capacity; ++probe) {
    const uint32_t* slot = table + M_HEADER + (size_t)(((uint32_t)h + probe) & mask) * sw;
    const uint32_t t = slot[0];
    if (t == 0) return false;
    if (t == tag) {
      bool eq = true;
      for (int i = 0; i < key_len && eq; ++i) eq = slot[1 + i] == key[i];
      if (eq) return true;
    }
  }
  return false;
}

// ------------------------------------------------------------- CACHE search
struct CsSmem {
  uint32_t runs[FC_MAX_OCC + 1];
  uint32_t work[FC_MAX_OCC];
  uint32_t sel[FC_MAX_TOPK];
  uint32_t order[FC_MAX_TOPK];
  uint32_t ctx[FC_MAX_NMAX];
  uint32_t wsum[CS_THREADS / 32];
  RunsScratch rs;
  uint32_t best, nocc, bad, n_tok;
};

__host__ __device__ inline uint32_t pow2_ceil(uint32_t x) {
  uint32_t p = 1;
  while (p < x) p <<= 1;
  return p;
}

size_t cs_smem_bytes(int capacity) {
  return ((sizeof(CsSmem) + 15) & ~(size_t)15) + 4 * (size_t)capacity + 4 * (size_t)pow2_ceil((uint32_t)capacity);
}

__global__ void __launch_bounds__(CS_THREADS) k_cache_search(CacheView c, const uint32_t* __restrict__ table,
                                                             int table_cap, const uint32_t* __restrict__ ctx,
                                                             int stride, const int32_t* __restrict__ ctx_len, int B,
                                                             fc_retrieve_params p, int S, ResOut o,
                                                             int32_t* __restrict__ state) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  CsSmem& sm = *reinterpret_cast<CsSmem*>(smem_raw);
  uint32_t* T = reinterpret_cast<uint32_t*>(smem_raw + ((sizeof(CsSmem) + 15) & ~(size_t)15));
  uint32_t* occ = T + c.capacity;
  const int b = blockIdx.x, tid = threadIdx.x;
  const int k = p.top_k, d = p.draft_len;

  int m = ctx_len[b];
  m = max(0, min(m, stride));
  const int cap = min(p.n_max, m);
  const int32_t* meta = c.meta + 4 * (size_t)b;
  if (tid == 0) {
    sm.bad = 0;
    sm.best = 0;
    sm.nocc = 0;
    const int nt = meta[0];
    sm.n_tok = (nt >= 0 && nt <= c.capacity) ? (uint32_t)nt : 0u;
    if (nt < 0 || nt > c.capacity) fc_flag(&g_fc_err, FC_EBIT_INTERNAL);
  }
  __syncthreads();
  if (tid < cap) {
    const uint32_t t = ctx[(size_t)b * stride + (m - cap) + tid];
    sm.ctx[tid] = t;
    if (t >= FC_SEP_TOKEN) sm.bad = 1;
  }
  __syncthreads();
  if (sm.bad && tid == 0) fc_flag(&g_fc_err, FC_EBIT_INVALID);
  const uint32_t n_tok = sm.n_tok;
  const bool active = !sm.bad && meta[1] >= c.min_size && cap >= p.n_min && n_tok >= 2;

  if (active) {
    // stage the store (16-byte rows; the capacity is a multiple of 4 words)
    const uint4* src = reinterpret_cast<const uint4*>(c.words + (size_t)b * c.capacity);
    uint4* dst = reinterpret_cast<uint4*>(T);
    for (uint32_t i = tid; i < (n_tok + 3) / 4; i += CS_THREADS) dst[i] = src[i];
    __syncthreads();
    // pass 1: the longest common suffix over all positions with a continuation
    uint32_t best = 0;
    for (uint32_t q = tid + 1; q < n_tok; q += CS_THREADS) {
      if (T[q] == FC_SEP_TOKEN) continue;
      uint32_t len = 0;
      while (len < (uint32_t)cap && len < q && T[q - 1 - len] == sm.ctx[cap - 1 - len]) ++len;
      best = max(best, len);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) best = max(best, __shfl_xor_sync(0xFFFFFFFFu, best, off));
    if ((tid & 31) == 0 && best > 0) atomicMax(&sm.best, best);
    __syncthreads();
  }
  const uint32_t ns = active && sm.best >= (uint32_t)p.n_min ? sm.best : 0u;

  // continuation order: ends at d tokens or at the separator; shorter first
  auto cont_cmp = [=](uint32_t a, uint32_t bpos) -> int {
    for (int i = 0; i < d; ++i) {
      const uint32_t ta = (a + i < n_tok) ? T[a + i] : FC_SEP_TOKEN;
      const uint32_t tb = (bpos + i < n_tok) ? T[bpos + i] : FC_SEP_TOKEN;
      const bool ea = ta == FC_SEP_TOKEN, eb = tb == FC_SEP_TOKEN;
      if (ea || eb) return (ea && eb) ? 0 : (ea ? -1 : 1);
      if (ta != tb) return ta < tb ? -1 : 1;
    }
    return 0;
  };

  uint32_t nd = 0;
  if (ns > 0) {
    // pass 2: the occurrences of the n*-token suffix
    for (uint32_t q = tid + ns; q < n_tok; q += CS_THREADS) {
      if (T[q] == FC_SEP_TOKEN) continue;
      bool hit = true;
      for (uint32_t j = 0; j < ns && hit; ++j) hit = T[q - 1 - j] == sm.ctx[cap - 1 - j];
      if (hit) occ[atomicAdd(&sm.nocc, 1u)] = q;
    }
    __syncthreads();
    const uint32_t nocc = sm.nocc;
    const uint32_t n2 = pow2_ceil(nocc);
    for (uint32_t i = nocc + tid; i < n2; i += CS_THREADS) occ[i] = NO_POS;
    __syncthreads();
    // bitonic sort by (continuation, position)
    for (uint32_t kk = 2; kk <= n2; kk <<= 1) {
      for (uint32_t j = kk >> 1; j > 0; j >>= 1) {
        for (uint32_t i = tid; i < n2; i += CS_THREADS) {
          const uint32_t ixj = i ^ j;
          if (ixj > i) {
            const uint32_t a = occ[i], bb = occ[ixj];
            bool a_first;  // a sorts before bb
            if (a == NO_POS || bb == NO_POS) {
              a_first = bb == NO_POS && a != NO_POS;
            } else {
              const int cr = cont_cmp(a, bb);
              a_first = cr < 0 || (cr == 0 && a < bb);
            }
            const bool asc = (i & kk) == 0;
            if (a != bb && (asc ? !a_first : a_first)) {
              occ[i] = bb;
              occ[ixj] = a;
            }
          }
        }
        __syncthreads();
      }
    }
    const uint32_t kept = min(nocc, p.max_occ);
    for (uint32_t e = tid; e < kept; e += CS_THREADS) sm.work[e] = (e == 0 || cont_cmp(occ[e - 1], occ[e]) != 0);
    __syncthreads();
    nd = rank_runs<CS_THREADS>(kept, k, sm.runs, sm.work, sm.sel, sm.order, sm.wsum, sm.rs);
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
      const uint32_t pos = occ[sm.runs[sm.order[t]]];
      if (x < cont_len(pos)) v = T[pos + x];
    }
    dr[e] = v;
  }
  for (int t = tid; t < k; t += CS_THREADS) {
    if (t < (int)nd) {
      const uint32_t r = sm.order[t];
      dl[t] = cont_len(occ[sm.runs[r]]);
      ct[t] = sm.runs[r + 1] - sm.runs[r];
    } else {
      dl[t] = 0;
      ct[t] = 0;
    }
  }
  __shared__ int st_sh;
  if (tid == 0) {
    o.n_drafts[sb] = (int32_t)nd;
    o.match_len[sb] = nd ? (int32_t)ns : 0;
    int st = FC_SERVE_DATASTORE;
    if (nd > 0) {
      st = FC_SERVE_CACHE;
    } else if (table && !sm.bad && m >= p.n_min &&
               missing_contains(table, table_cap, p.n_min, sm.ctx + (cap - p.n_min))) {
      st = FC_SKIP_MISSING;
    }
    state[b] = st;
    st_sh = st;
  }
  __syncthreads();
  if (st_sh == FC_SERVE_DATASTORE) return;
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
        pend = !missing_contains(table, capacity, key_len, key);
        h = key_hash(key, key_len);
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
    if (lane == 0) fc_flag(&g_fc_err, FC_EBIT_INVALID);
    return;
  }
  const uint32_t* row = ctx + (size_t)b * stride;
  uint32_t* words = c.words + (size_t)b * c.capacity;
  auto store = [&](int s0, int L) {
    bool bad = false;
    for (int i = lane; i < L; i += 32) bad |= row[s0 + i] >= FC_SEP_TOKEN;
    if (__any_sync(0xFFFFFFFFu, bad)) {
      if (lane == 0) fc_flag(&g_fc_err, FC_EBIT_INVALID);
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
  return CacheView{c->d_words, c->d_meta, c->capacity, c->min_size, c->chunk, c->ctx_keep};
}

}  // namespace

extern "C" fc_status fc_cache_init(const fc_cache* cache, int batch, const int32_t* d_prompt_len, fc_stream stream) {
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
  if (!cache_ok(cache) || batch < 0 || ctx_stride < 1 || n_sources < 0 || n_sources >= FC_MAX_SOURCES ||
      batch > 65535 * 16)
    return FC_ERR_INVALID_ARG;
  if (d_missing && !missing_cap_ok(missing_capacity)) return FC_ERR_INVALID_ARG;
  if (!fc_retrieve_params_ok(p))
    return (p.n_max > 0 && p.top_k > 0 && p.draft_len > 0) ? FC_ERR_UNSUPPORTED : FC_ERR_INVALID_ARG;
  if (batch == 0) return FC_OK;
  if (!d_ctx || !d_ctx_len || !d_drafts || !d_draft_len || !d_count || !d_n_drafts || !d_match_len || !d_state)
    return FC_ERR_INVALID_ARG;
  static bool attr_done = false;
  if (!attr_done) {
    if (cudaFuncSetAttribute(k_cache_search, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)cs_smem_bytes(FC_CACHE_MAX_WORDS)) != cudaSuccess)
      return FC_ERR_CUDA;
    attr_done = true;
  }
  ResOut o{d_drafts, d_draft_len, d_count, d_n_drafts, d_match_len};
  k_cache_search<<<batch, CS_THREADS, cs_smem_bytes(cache->capacity), static_cast<cudaStream_t>(stream)>>>(
      view_of(cache), static_cast<const uint32_t*>(d_missing), missing_capacity, d_ctx, ctx_stride, d_ctx_len, batch,
      p, n_sources, o, d_state);
  return FC_CHECK_LAUNCH();
}

extern "C" fc_status fc_missing_insert(void* d_missing, int missing_capacity, int key_len, const uint32_t* d_ctx,
                                       int ctx_stride, const int32_t* d_ctx_len, int batch, const int32_t* d_state,
                                       const int32_t* d_n_drafts, int n_sources, fc_stream stream) {
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
  if (!cache_ok(cache) || batch < 0 || ctx_stride < 1) return FC_ERR_INVALID_ARG;
  if (batch == 0) return FC_OK;
  if (!d_ctx || !d_ctx_len_old || !d_ctx_len_new || !d_acc_len) return FC_ERR_INVALID_ARG;
  k_cache_update<<<(batch + CU_WARPS - 1) / CU_WARPS, CU_WARPS * 32, 0, static_cast<cudaStream_t>(stream)>>>(
      view_of(cache), d_ctx, ctx_stride, d_ctx_len_old, d_ctx_len_new, d_acc_len, batch);
  return FC_CHECK_LAUNCH();
}
