// fc_datastore_build: suffix array + first-token bucket table of a uint32
// token corpus (the datastore organisation of Section IV-A, Eq. 1-2, which
// follows REST's suffix-array index).
//
// Method (GPU prefix doubling): after round r every position i carries the
// dense rank of its first 2^r tokens.  A round sorts the positions by the
// pair (rank[i], rank[i + h] + 1) (0 when i + h runs past the end, so a
// shorter suffix sorts first), with a stable LSD radix sort written here
// (8-bit digits, per-block histograms, a global exclusive scan and a stable
// scatter that ranks equal digits inside a warp with __match_any_sync), then
// re-ranks by scanning "key differs from its predecessor" flags.  The loop
// stops when every rank is distinct.  All passes stream the arrays once
// (HBM-bound); only the rank gather rank[i + h] is random.

#include "fc_common.cuh"

FC_DEFINE_ERROR_WORD(sa)

namespace {

constexpr int RS_THREADS = 256;
constexpr int RS_ITEMS = 16;
constexpr int RS_TILE = RS_THREADS * RS_ITEMS;  // 4096 keys per block
constexpr int RS_WARPS = RS_THREADS / 32;
constexpr int RS_WARP_CHUNK = 32 * RS_ITEMS;    // 512 consecutive keys per warp

constexpr int SCAN_THREADS = 1024;
constexpr int SCAN_ITEMS = 4;
constexpr int SCAN_TILE = SCAN_THREADS * SCAN_ITEMS;

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }
inline size_t cdiv(size_t a, size_t b) { return (a + b - 1) / b; }

struct Layout {
  size_t key_a, key_b, val_b, rank, head, hist, scan_tmp, ctl, total;
  size_t nb;          // radix blocks
  size_t scan_len;    // longest array the scan sees
};

size_t scan_tmp_elems(size_t len) {
  size_t t = 0;
  while (len > (size_t)SCAN_TILE) {
    len = cdiv(len, SCAN_TILE);
    t += len;
  }
  return t + 16;
}

Layout layout_for(uint64_t n) {
  Layout L;
  L.nb = cdiv(n, RS_TILE);
  L.scan_len = n > 256 * L.nb ? n : 256 * L.nb;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    size_t o = off;
    off = align_up(off + bytes, 256);
    return o;
  };
  L.key_a = take(n * 8);
  L.key_b = take(n * 8);
  L.val_b = take(n * 4);
  L.rank = take(n * 4);
  L.head = take(n * 4);
  L.hist = take(256 * L.nb * 4);
  L.scan_tmp = take(scan_tmp_elems(L.scan_len) * 4);
  L.ctl = take(64);
  L.total = off;
  return L;
}

__global__ void k_check_tokens(const uint32_t* __restrict__ T, uint64_t n, uint32_t vocab, uint32_t* ctl) {
  for (uint64_t i = blockIdx.x * (uint64_t)blockDim.x + threadIdx.x; i < n; i += (uint64_t)gridDim.x * blockDim.x)
    if (T[i] >= vocab) {
      atomicOr(ctl, 1u);
      return;
    }
}

// First round: key = (T[i], T[i+1] + 1 or 0), val = i.
__global__ void k_keys_first(const uint32_t* __restrict__ T, uint64_t n, uint64_t* __restrict__ key,
                             uint32_t* __restrict__ val) {
  for (uint64_t i = blockIdx.x * (uint64_t)blockDim.x + threadIdx.x; i < n; i += (uint64_t)gridDim.x * blockDim.x) {
    uint64_t lo = (i + 1 < n) ? (uint64_t)T[i + 1] + 1 : 0;
    key[i] = ((uint64_t)T[i] << 32) | lo;
    val[i] = (uint32_t)i;
  }
}

// Later rounds: positions in current SA order; key = (rank[i], rank[i+h] + 1 or 0).
// val may alias sa (each element rewrites its own value).
__global__ void k_keys_round(const uint32_t* sa, const uint32_t* __restrict__ rank, uint64_t n, uint64_t h,
                             uint64_t* __restrict__ key, uint32_t* val) {
  for (uint64_t j = blockIdx.x * (uint64_t)blockDim.x + threadIdx.x; j < n; j += (uint64_t)gridDim.x * blockDim.x) {
    uint32_t i = sa[j];
    uint64_t lo = ((uint64_t)i + h < n) ? (uint64_t)rank[i + h] + 1 : 0;
    key[j] = ((uint64_t)rank[i] << 32) | lo;
    val[j] = i;
  }
}

__global__ void __launch_bounds__(RS_THREADS) k_radix_hist(const uint64_t* __restrict__ key, uint64_t n, int shift,
                                                           uint32_t* __restrict__ hist, uint64_t nb) {
  __shared__ uint32_t h[256];
  h[threadIdx.x] = 0;
  __syncthreads();
  uint64_t base = blockIdx.x * (uint64_t)RS_TILE;
#pragma unroll 4
  for (int k = 0; k < RS_ITEMS; ++k) {
    uint64_t idx = base + (uint64_t)k * RS_THREADS + threadIdx.x;
    if (idx < n) atomicAdd(&h[(uint32_t)(key[idx] >> shift) & 255u], 1u);
  }
  __syncthreads();
  hist[(uint64_t)threadIdx.x * nb + blockIdx.x] = h[threadIdx.x];
}

// Stable scatter of one 8-bit digit.  offs[d * nb + block] is the exclusive
// scan of the digit-major histogram: where this block's digit-d keys start.
// The block first ranks its keys (per warp with __match_any_sync, then across
// warps and digits), places them in shared memory in digit order, and then
// writes them out in that order: consecutive threads write consecutive
// addresses of a digit's run, so the stores coalesce instead of spraying
// 8- and 4-byte writes over 256 runs.
constexpr uint32_t RS_SMEM = RS_TILE * (8 + 4);  // keys and values of one tile

__global__ void __launch_bounds__(RS_THREADS) k_radix_scatter(const uint64_t* __restrict__ kin,
                                                              const uint32_t* __restrict__ vin,
                                                              uint64_t* __restrict__ kout,
                                                              uint32_t* __restrict__ vout, uint64_t n, int shift,
                                                              const uint32_t* __restrict__ offs, uint64_t nb) {
  extern __shared__ __align__(16) unsigned char rs_smem[];
  uint64_t* skey = reinterpret_cast<uint64_t*>(rs_smem);
  uint32_t* sval = reinterpret_cast<uint32_t*>(rs_smem + RS_TILE * 8);
  __shared__ uint32_t wbin[RS_WARPS][256];
  __shared__ uint32_t base_s[256];
  __shared__ uint32_t doff[256];   // where digit d starts in the block's digit order
  __shared__ uint32_t wsum[RS_THREADS / 32];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  for (int d = tid; d < RS_WARPS * 256; d += RS_THREADS) (&wbin[0][0])[d] = 0;
  base_s[tid] = offs[(uint64_t)tid * nb + blockIdx.x];
  __syncthreads();
  const uint64_t b0 = blockIdx.x * (uint64_t)RS_TILE;
  const uint32_t count = (uint32_t)min((uint64_t)RS_TILE, n - b0);
  const uint64_t w0 = b0 + (uint64_t)warp * RS_WARP_CHUNK;
  const uint32_t lt = (1u << lane) - 1u;
  uint64_t key[RS_ITEMS];
  uint32_t val[RS_ITEMS];
  uint32_t lr[RS_ITEMS];
#pragma unroll
  for (int it = 0; it < RS_ITEMS; ++it) {
    uint64_t idx = w0 + (uint64_t)it * 32 + lane;
    bool ok = idx < n;
    key[it] = ok ? kin[idx] : 0ull;
    val[it] = ok ? vin[idx] : 0u;
    uint32_t d = ok ? ((uint32_t)(key[it] >> shift) & 255u) : 256u;
    uint32_t peers = __match_any_sync(0xFFFFFFFFu, d);
    uint32_t cnt = (d < 256u) ? wbin[warp][d] : 0u;
    lr[it] = cnt + __popc(peers & lt);
    __syncwarp();
    if (d < 256u && lane == __ffs(peers) - 1) wbin[warp][d] = cnt + __popc(peers);
    __syncwarp();
  }
  __syncthreads();
  // per digit (thread tid = digit): warp prefix, then the digit's block total
  uint32_t run = 0;
#pragma unroll
  for (int w = 0; w < RS_WARPS; ++w) {
    uint32_t c = wbin[w][tid];
    wbin[w][tid] = run;
    run += c;
  }
  // exclusive scan of the digit totals over the 256 digits
  uint32_t inc = run;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(0xFFFFFFFFu, inc, o);
    if (lane >= o) inc += y;
  }
  if (lane == 31) wsum[warp] = inc;
  __syncthreads();
  uint32_t before = 0;
  for (int w = 0; w < warp; ++w) before += wsum[w];
  doff[tid] = before + inc - run;
  __syncthreads();
#pragma unroll
  for (int it = 0; it < RS_ITEMS; ++it) {
    uint64_t idx = w0 + (uint64_t)it * 32 + lane;
    if (idx < n) {
      const uint32_t d = (uint32_t)(key[it] >> shift) & 255u;
      const uint32_t at = doff[d] + wbin[warp][d] + lr[it];
      skey[at] = key[it];
      sval[at] = val[it];
    }
  }
  __syncthreads();
  for (uint32_t j = tid; j < count; j += RS_THREADS) {
    const uint64_t k = skey[j];
    const uint32_t d = (uint32_t)(k >> shift) & 255u;
    const uint64_t pos = (uint64_t)base_s[d] + (j - doff[d]);
    kout[pos] = k;
    vout[pos] = sval[j];
  }
}

// ---- exclusive sum scan of uint32 (three-phase, recursive on the host) ----
__device__ __forceinline__ uint32_t block_exclusive_scan(uint32_t x, uint32_t* total) {
  __shared__ uint32_t warp_sums[SCAN_THREADS / 32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t inc = x;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    uint32_t y = __shfl_up_sync(0xFFFFFFFFu, inc, o);
    if (lane >= o) inc += y;
  }
  if (lane == 31) warp_sums[warp] = inc;
  __syncthreads();
  if (warp == 0) {
    uint32_t v = (lane < (int)(blockDim.x >> 5)) ? warp_sums[lane] : 0u;
    uint32_t vi = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      uint32_t y = __shfl_up_sync(0xFFFFFFFFu, vi, o);
      if (lane >= o) vi += y;
    }
    warp_sums[lane] = vi - v;
    if (lane == 31) *total = vi;
  }
  __syncthreads();
  uint32_t r = warp_sums[warp] + inc - x;
  __syncthreads();
  return r;
}

__global__ void __launch_bounds__(SCAN_THREADS) k_scan_reduce(const uint32_t* __restrict__ in, uint64_t n,
                                                              uint32_t* __restrict__ partial) {
  __shared__ uint32_t tot;
  uint64_t base = blockIdx.x * (uint64_t)SCAN_TILE + (uint64_t)threadIdx.x * SCAN_ITEMS;
  uint32_t s = 0;
#pragma unroll
  for (int k = 0; k < SCAN_ITEMS; ++k)
    if (base + k < n) s += in[base + k];
  block_exclusive_scan(s, &tot);
  if (threadIdx.x == 0) partial[blockIdx.x] = tot;
}

__global__ void __launch_bounds__(SCAN_THREADS) k_scan_apply(uint32_t* __restrict__ data, uint64_t n,
                                                             const uint32_t* __restrict__ partial) {
  __shared__ uint32_t tot;
  uint64_t base = blockIdx.x * (uint64_t)SCAN_TILE + (uint64_t)threadIdx.x * SCAN_ITEMS;
  uint32_t v[SCAN_ITEMS];
  uint32_t s = 0;
#pragma unroll
  for (int k = 0; k < SCAN_ITEMS; ++k) {
    v[k] = (base + k < n) ? data[base + k] : 0u;
    s += v[k];
  }
  uint32_t pre = block_exclusive_scan(s, &tot) + (partial ? partial[blockIdx.x] : 0u);
#pragma unroll
  for (int k = 0; k < SCAN_ITEMS; ++k) {
    if (base + k < n) data[base + k] = pre;
    pre += v[k];
  }
}

cudaError_t exclusive_scan(uint32_t* data, uint64_t n, uint32_t* tmp, cudaStream_t s) {
  if (n == 0) return cudaSuccess;
  uint64_t nt = cdiv(n, SCAN_TILE);
  if (nt == 1) {
    k_scan_apply<<<1, SCAN_THREADS, 0, s>>>(data, n, nullptr);
    return cudaGetLastError();
  }
  k_scan_reduce<<<(unsigned)nt, SCAN_THREADS, 0, s>>>(data, n, tmp);
  cudaError_t e = exclusive_scan(tmp, nt, tmp + nt, s);
  if (e != cudaSuccess) return e;
  k_scan_apply<<<(unsigned)nt, SCAN_THREADS, 0, s>>>(data, n, tmp);
  return cudaGetLastError();
}

// rank[val[j]] = number of distinct keys before position j (dense rank);
// sa[j] = val[j]; ctl[1] = number of distinct keys.
__global__ void k_ranks(const uint64_t* __restrict__ key, const uint32_t* val, const uint32_t* __restrict__ excl,
                        uint64_t n, uint32_t* __restrict__ rank, uint32_t* sa, uint32_t* ctl) {
  for (uint64_t j = blockIdx.x * (uint64_t)blockDim.x + threadIdx.x; j < n; j += (uint64_t)gridDim.x * blockDim.x) {
    uint32_t h = (j == 0 || key[j] != key[j - 1]) ? 1u : 0u;
    uint32_t v = val[j];
    rank[v] = excl[j] + h - 1u;
    sa[j] = v;
    if (j == n - 1) ctl[1] = excl[j] + h;
  }
}

__global__ void k_heads(const uint64_t* __restrict__ key, uint64_t n, uint32_t* __restrict__ head) {
  for (uint64_t j = blockIdx.x * (uint64_t)blockDim.x + threadIdx.x; j < n; j += (uint64_t)gridDim.x * blockDim.x)
    head[j] = (j == 0 || key[j] != key[j - 1]) ? 1u : 0u;
}

// bucket[v] = first j with T[sa[j]] >= v (binary search), bucket[vocab] = n.
__global__ void k_bucket(const uint32_t* __restrict__ T, const uint32_t* __restrict__ sa, uint64_t n,
                         uint32_t vocab, uint32_t* __restrict__ bucket) {
  for (uint64_t v = blockIdx.x * (uint64_t)blockDim.x + threadIdx.x; v <= vocab; v += (uint64_t)gridDim.x * blockDim.x) {
    uint64_t lo = 0, hi = n;
    while (lo < hi) {
      uint64_t mid = (lo + hi) >> 1;
      if (T[sa[mid]] < v) lo = mid + 1;
      else hi = mid;
    }
    bucket[v] = (uint32_t)lo;
  }
}

// lcp[j] = common prefix length of the suffixes at sa[j-1] and sa[j], capped.
// rank is the inverse suffix array; each thread takes one text position i
// (so each suffix is compared with its predecessor in SA order once).
__global__ void k_lcp(const uint32_t* __restrict__ T, const uint32_t* __restrict__ sa,
                      const uint32_t* __restrict__ rank, uint64_t n, uint8_t* __restrict__ lcp) {
  for (uint64_t i = blockIdx.x * (uint64_t)blockDim.x + threadIdx.x; i < n; i += (uint64_t)gridDim.x * blockDim.x) {
    const uint32_t j = rank[i];
    uint32_t l = 0;
    if (j > 0) {
      const uint64_t pr = sa[j - 1];
      while (l < FC_LCP_CAP && i + l < n && pr + l < n && T[i + l] == T[pr + l]) ++l;
    }
    lcp[j] = (uint8_t)l;
  }
}

inline int bits_for(uint64_t x) {
  int b = 0;
  while (x) {
    ++b;
    x >>= 1;
  }
  return b;
}

inline unsigned grid_for(uint64_t n, int threads) {
  uint64_t g = cdiv(n, threads);
  if (g > 152ull * 64) g = 152ull * 64;
  return (unsigned)(g ? g : 1);
}

}  // namespace

extern "C" size_t fc_datastore_build_workspace(uint64_t n_tokens, uint32_t vocab) {
  (void)vocab;
  if (n_tokens == 0) return 0;
  return layout_for(n_tokens).total;
}

extern "C" fc_status fc_datastore_build(const uint32_t* d_tokens, uint64_t n, uint32_t vocab, uint32_t* d_sa,
                                        uint32_t* d_bucket, uint8_t* d_lcp, void* d_ws, size_t ws_bytes,
                                        fc_stream stream, fc_datastore* out) {
  FC_NVTX_RANGE();
  if (!d_tokens || !d_sa || !d_bucket || !d_lcp || n == 0 || n >= 0xFFFFFFFFull || vocab == 0 ||
      vocab >= 0x80000000u)
    return FC_ERR_INVALID_ARG;
  Layout L = layout_for(n);
  if (!d_ws || ws_bytes < L.total) return FC_ERR_WORKSPACE;
  if (reinterpret_cast<uintptr_t>(d_ws) % 256) return FC_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  char* ws = static_cast<char*>(d_ws);
  uint64_t* key_a = reinterpret_cast<uint64_t*>(ws + L.key_a);
  uint64_t* key_b = reinterpret_cast<uint64_t*>(ws + L.key_b);
  uint32_t* val_b = reinterpret_cast<uint32_t*>(ws + L.val_b);
  uint32_t* rank = reinterpret_cast<uint32_t*>(ws + L.rank);
  uint32_t* head = reinterpret_cast<uint32_t*>(ws + L.head);
  uint32_t* hist = reinterpret_cast<uint32_t*>(ws + L.hist);
  uint32_t* stmp = reinterpret_cast<uint32_t*>(ws + L.scan_tmp);
  uint32_t* ctl = reinterpret_cast<uint32_t*>(ws + L.ctl);
  const unsigned g = grid_for(n, 256);
  uint32_t hctl[2] = {0, 0};

  if (cudaFuncSetAttribute(k_radix_scatter, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)RS_SMEM) != cudaSuccess)
    return FC_ERR_CUDA;
  if (cudaMemsetAsync(ctl, 0, 64, s) != cudaSuccess) return FC_ERR_CUDA;
  k_check_tokens<<<g, 256, 0, s>>>(d_tokens, n, vocab, ctl);
  if (cudaMemcpyAsync(hctl, ctl, 8, cudaMemcpyDeviceToHost, s) != cudaSuccess) return FC_ERR_CUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return FC_ERR_CUDA;
  if (hctl[0]) return FC_ERR_INVALID_ARG;

  k_keys_first<<<g, 256, 0, s>>>(d_tokens, n, key_a, d_sa);
  uint64_t max_hi = vocab - 1, max_lo = vocab;
  uint64_t h = 1;
  for (int round = 0;; ++round) {
    if (round > 40) return FC_ERR_INTERNAL;
    // LSD passes over the populated bits of the low then the high word.
    uint64_t* kin = key_a;
    uint32_t* vin = d_sa;
    uint64_t* kout = key_b;
    uint32_t* vout = val_b;
    int shifts[16];
    int np = 0;
    for (int b = 0; b < bits_for(max_lo); b += 8) shifts[np++] = b;
    for (int b = 0; b < bits_for(max_hi); b += 8) shifts[np++] = 32 + b;
    for (int p = 0; p < np; ++p) {
      k_radix_hist<<<(unsigned)L.nb, RS_THREADS, 0, s>>>(kin, n, shifts[p], hist, L.nb);
      if (exclusive_scan(hist, 256 * L.nb, stmp, s) != cudaSuccess) return FC_ERR_CUDA;
      k_radix_scatter<<<(unsigned)L.nb, RS_THREADS, RS_SMEM, s>>>(kin, vin, kout, vout, n, shifts[p], hist, L.nb);
      std::swap(kin, kout);
      std::swap(vin, vout);
    }
    // kin/vin now hold the sorted keys and positions.
    k_heads<<<g, 256, 0, s>>>(kin, n, head);
    if (exclusive_scan(head, n, stmp, s) != cudaSuccess) return FC_ERR_CUDA;
    k_ranks<<<g, 256, 0, s>>>(kin, vin, head, n, rank, d_sa, ctl);
    if (cudaMemcpyAsync(hctl, ctl, 8, cudaMemcpyDeviceToHost, s) != cudaSuccess) return FC_ERR_CUDA;
    if (cudaStreamSynchronize(s) != cudaSuccess) return FC_ERR_CUDA;
    uint64_t groups = hctl[1];
    if (groups == n) break;
    if (groups == 0 || groups > n) return FC_ERR_INTERNAL;
    h = (round == 0) ? 2 : h * 2;
    if (h >= 2 * n + 2) return FC_ERR_INTERNAL;
    k_keys_round<<<g, 256, 0, s>>>(d_sa, rank, n, h, key_a, d_sa);
    max_hi = groups - 1;
    max_lo = groups;
  }
  k_bucket<<<grid_for((uint64_t)vocab + 1, 256), 256, 0, s>>>(d_tokens, d_sa, n, vocab, d_bucket);
  // every group is a single suffix now, so rank is the inverse suffix array
  k_lcp<<<g, 256, 0, s>>>(d_tokens, d_sa, rank, n, d_lcp);
  if (cudaGetLastError() != cudaSuccess) return FC_ERR_CUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return FC_ERR_CUDA;
  if (out) {
    out->tokens = d_tokens;
    out->sa = d_sa;
    out->bucket = d_bucket;
    out->lcp = d_lcp;
    out->n_tokens = n;
    out->vocab = vocab;
    out->keys = nullptr;
  }
  return FC_OK;
}

// ---------------------------------------------------------------------------
// Datastore build without any allocation: the scratch space lives in a
// fixed array compiled into this library instead of caller memory.
//
// Some callers cannot call cudaMalloc: a serving process whose memory manager
// reserves all free device memory for its KV cache up front (a later
// cudaMalloc fails, or fragments that reservation), or a plugin inside a host
// application that owns every device allocation.  They can still build a
// small datastore (a repository's own project store) here.
//
// The array is a file-scope __device__ variable.  A GPU holds it from the
// moment this file's device code is loaded there until the process exits.
// Under CUDA's default lazy module loading that moment is the first datastore
// build (this entry point or fc_datastore_build) made on the device, not the
// library's load: the first call itself places the 30 MiB.  A caller that
// reserves all free device memory must therefore make one call (a small
// corpus is enough) before reserving it.
//
// Host code cannot pass the variable's name to a kernel (on the host it is
// only a stand-in, not a device address): every call looks up the device
// address on the current device with cudaGetSymbolAddress.  The lookup is
// not cached, so the address stays right after a device reset reloads the
// module elsewhere.  The first call on a device loads the module, so it
// should come before any stream capture.  Every call shares the one array
// and leaves its contents behind; the build clears what must start at zero
// itself.  Calls whose work overlaps on the GPU (two streams, two host
// threads) race on the array and must not be made.
// ---------------------------------------------------------------------------
namespace {
constexpr size_t kNoAllocScratchBytes = (size_t)30 << 20;  // 30 MiB
static __device__ __align__(256) unsigned char g_sa_scratch[kNoAllocScratchBytes];

fc_status scratch_for_current_device(void** out) {
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_sa_scratch) != cudaSuccess || !p) return FC_ERR_CUDA;
  *out = p;
  return FC_OK;
}
}  // namespace

extern "C" fc_status fc_datastore_build_noalloc(const uint32_t* d_tokens, uint64_t n_tokens, uint32_t vocab,
                                                uint32_t* d_sa, uint32_t* d_bucket, uint8_t* d_lcp,
                                                fc_stream stream, fc_datastore* out) {
  FC_NVTX_RANGE();
  if (n_tokens > FC_NOALLOC_MAX_TOKENS) return FC_ERR_CAPACITY;
  if (n_tokens > 0 && fc_datastore_build_workspace(n_tokens, vocab) > kNoAllocScratchBytes) return FC_ERR_CAPACITY;
  void* ws = nullptr;
  fc_status st = scratch_for_current_device(&ws);
  if (st != FC_OK) return st;
  return fc_datastore_build(d_tokens, n_tokens, vocab, d_sa, d_bucket, d_lcp, ws, kNoAllocScratchBytes, stream, out);
}

// ---------------------------------------------------------------------------
// Suffix keys: entry j = (sa[j], T[sa[j] + 1 .. sa[j] + 7]), FC_PAD_TOKEN past
// the corpus end; 32 bytes, written as two 16-byte stores.
// ---------------------------------------------------------------------------
namespace {
__global__ void k_suffix_keys(const uint32_t* __restrict__ T, const uint32_t* __restrict__ sa, uint64_t n,
                              uint4* __restrict__ keys) {
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  for (uint64_t j = blockIdx.x * (uint64_t)blockDim.x + threadIdx.x; j < n; j += stride) {
    const uint64_t i = __ldg(sa + j);
    uint32_t t[8];
    t[0] = (uint32_t)i;
#pragma unroll
    for (int k = 1; k < 8; ++k) t[k] = (i + k < n) ? __ldg(T + i + k) : FC_PAD_TOKEN;
    keys[2 * j] = make_uint4(t[0], t[1], t[2], t[3]);
    keys[2 * j + 1] = make_uint4(t[4], t[5], t[6], t[7]);
  }
}
}  // namespace

extern "C" fc_status fc_datastore_keys(const fc_datastore* ds, uint32_t* d_keys, fc_stream stream) {
  FC_NVTX_RANGE();
  if (!ds || !ds->tokens || !ds->sa || !d_keys || ds->n_tokens == 0 || ds->n_tokens >= 0xFFFFFFFFull)
    return FC_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(d_keys) % 32) return FC_ERR_INVALID_ARG;
  const uint64_t n = ds->n_tokens;
  k_suffix_keys<<<grid_for(n, 256), 256, 0, static_cast<cudaStream_t>(stream)>>>(ds->tokens, ds->sa, n,
                                                                                 reinterpret_cast<uint4*>(d_keys));
  return FC_CHECK_LAUNCH();
}

// ---------------------------------------------------------------------------
// The reversed corpus R[i] = T[n-1-i], whose suffix array serves
// fc_retrieve_rev.  Aligned 16-byte groups where both sides allow it: output
// group q (tokens 4q .. 4q+3) reads input tokens n-4-4q .. n-1-4q, which are
// 16-byte aligned exactly when n is a multiple of 4.
// ---------------------------------------------------------------------------
namespace {
__global__ void k_reverse(const uint32_t* __restrict__ in, uint64_t n, uint32_t* __restrict__ out) {
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  const uint64_t t0 = blockIdx.x * (uint64_t)blockDim.x + threadIdx.x;
  const bool vec = (n % 4 == 0) && (reinterpret_cast<uintptr_t>(in) % 16 == 0) &&
                   (reinterpret_cast<uintptr_t>(out) % 16 == 0);
  if (vec) {
    const uint64_t groups = n / 4;
    for (uint64_t q = t0; q < groups; q += stride) {
      const uint4 v = __ldg(reinterpret_cast<const uint4*>(in) + (groups - 1 - q));
      reinterpret_cast<uint4*>(out)[q] = make_uint4(v.w, v.z, v.y, v.x);
    }
  } else {
    for (uint64_t i = t0; i < n; i += stride) out[i] = __ldg(in + (n - 1 - i));
  }
}
}  // namespace

extern "C" fc_status fc_reverse_tokens(const uint32_t* d_tokens, uint64_t n_tokens, uint32_t* d_out,
                                       fc_stream stream) {
  FC_NVTX_RANGE();
  if (n_tokens == 0) return FC_OK;
  if (!d_tokens || !d_out || d_tokens == d_out || n_tokens >= 0xFFFFFFFFull) return FC_ERR_INVALID_ARG;
  const uint64_t a = reinterpret_cast<uintptr_t>(d_tokens), b = reinterpret_cast<uintptr_t>(d_out);
  if (a < b + 4 * n_tokens && b < a + 4 * n_tokens) return FC_ERR_INVALID_ARG;  // overlapping buffers
  k_reverse<<<grid_for(cdiv(n_tokens, 4), 256), 256, 0, static_cast<cudaStream_t>(stream)>>>(d_tokens, n_tokens,
                                                                                            d_out);
  return FC_CHECK_LAUNCH();
}
