// fc_accept, fc_argmax_accept, fc_kv_append and fc_synth_argmax: the end of a
// decoding step.
//
// Acceptance follows Section IV-D (every correct token from the start is
// accepted, everything after the first error rejected); the cache append
// closes the decoding loop (accepted tokens' K/V join the cache, the target
// model's own next token becomes the next root).  fc_synth_argmax is the
// workload's stand-in for the target model's greedy predictions.
#include "fc_common.cuh"

FC_DEFINE_ERROR_WORD(step)

namespace {

// One warp per sequence.  The tree (parents, tokens, predictions) is staged in
// shared memory with one coalesced read; children of `cur` sit after it in
// preorder, so the warp scans node ids cur+1 .. n-1 in chunks of 32 with one
// ballot each.
constexpr int ACC_WARPS = 4;  // sequences per CTA
__global__ void __launch_bounds__(ACC_WARPS * 32) k_accept(const uint32_t* __restrict__ tok,
                                                           const int32_t* __restrict__ parent,
                                                           const int32_t* __restrict__ n_nodes,
                                                           const uint32_t* __restrict__ argmax, int B, int n_pad,
                                                           int32_t* __restrict__ acc_len, int32_t* __restrict__ path,
                                                           int path_cap, uint32_t* __restrict__ bonus,
                                                           unsigned int* err) {
  extern __shared__ uint32_t acc_smem[];  // [ACC_WARPS][3][n_pad]
  // Launched as a programmatic dependent of the row argmax (fc_argmax_accept):
  // wait here until that grid's results are visible.  A no-op otherwise.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int b = blockIdx.x * ACC_WARPS + w;
  if (b >= B) return;
  uint32_t* s_tok = acc_smem + (size_t)w * 3 * n_pad;
  int32_t* s_par = reinterpret_cast<int32_t*>(s_tok + n_pad);
  uint32_t* s_am = s_tok + 2 * n_pad;
  const size_t base = (size_t)b * n_pad;
  const int n = min(max((int)n_nodes[b], 1), n_pad);
  for (int j = lane; j < n; j += 32) {
    s_tok[j] = tok[base + j];
    s_par[j] = parent[base + j];
    s_am[j] = argmax[base + j];
  }
  int32_t* pth = path + (size_t)b * path_cap;
  for (int t = lane; t < path_cap; t += 32) pth[t] = -1;
  __syncwarp();
  int cur = 0, len = 0;
  bool overflow = false;
  for (;;) {
    const uint32_t want = s_am[cur];
    int next = -1;
    for (int j0 = cur + 1; j0 < n && next < 0; j0 += 32) {
      const int j = j0 + lane;
      const bool hit = j < n && s_par[j] == cur && s_tok[j] == want;
      const uint32_t m = __ballot_sync(0xFFFFFFFFu, hit);
      if (m) next = j0 + __ffs(m) - 1;
    }
    if (next < 0) break;
    if (len + 1 >= path_cap) {
      overflow = true;
      break;
    }
    ++len;
    if (lane == 0) pth[len] = next;
    cur = next;
  }
  if (lane == 0) {
    pth[0] = 0;
    acc_len[b] = len;
    bonus[b] = s_am[cur];
    if (overflow) fc_flag(FC_ERR_WORD(err), FC_EBIT_CAPACITY);
  }
}

// One CTA per sequence: copy (acc_len + 1) rows x Hkv heads of K and V
// (16-byte vectors), then update lengths, context and root.
__global__ void k_kv_append(const int32_t* __restrict__ path, const int32_t* __restrict__ acc_len,
                            const uint32_t* __restrict__ bonus, const uint32_t* __restrict__ tok,
                            const uint4* __restrict__ k_tree, const uint4* __restrict__ v_tree, int n_pad, int Hkv,
                            int D, int path_cap, uint4* __restrict__ k_cache, uint4* __restrict__ v_cache, int kv_cap,
                            const int32_t* __restrict__ kv_len_in, int32_t* __restrict__ kv_len_out,
                            uint32_t* __restrict__ ctx, int ctx_stride, const int32_t* __restrict__ ctx_len_in,
                            int32_t* __restrict__ ctx_len_out, uint32_t* __restrict__ root_out,
                            unsigned int* err) {
  const int b = blockIdx.x;
  const int a = acc_len[b];
  const int kvl = kv_len_in[b], cl = ctx_len_in[b];
  const bool ok = a >= 0 && a + 1 <= path_cap && kvl >= 0 && kvl + a + 1 <= kv_cap && cl >= 0 &&
                  cl + a + 1 <= ctx_stride;
  if (!ok) {
    if (threadIdx.x == 0) {
      fc_flag(FC_ERR_WORD(err), FC_EBIT_CAPACITY);
      kv_len_out[b] = kvl;
      ctx_len_out[b] = cl;
      root_out[b] = (cl > 0 && cl <= ctx_stride) ? ctx[(size_t)b * ctx_stride + cl - 1] : 0u;
    }
    return;
  }
  const int vec = D / 8;  // uint4 per row
  const int rows = (a + 1) * Hkv;
  const int32_t* pth = path + (size_t)b * path_cap;
  for (int e = threadIdx.x; e < rows * vec; e += blockDim.x) {
    int r = e / vec, x = e - r * vec;
    int t = r / Hkv, g = r - t * Hkv;
    int node = pth[t];
    if (node < 0 || node >= n_pad) {
      fc_flag(FC_ERR_WORD(err), FC_EBIT_INVALID);
      continue;
    }
    size_t src = (((size_t)b * Hkv + g) * n_pad + node) * vec + x;
    size_t dst = (((size_t)b * Hkv + g) * kv_cap + kvl + t) * vec + x;
    k_cache[dst] = k_tree[src];
    v_cache[dst] = v_tree[src];
  }
  uint32_t* c = ctx + (size_t)b * ctx_stride;
  for (int t = threadIdx.x; t < a; t += blockDim.x) {
    int node = pth[t + 1];
    c[cl + t] = (node >= 0 && node < n_pad) ? tok[(size_t)b * n_pad + node] : FC_PAD_TOKEN;
  }
  if (threadIdx.x == 0) {
    c[cl + a] = bonus[b];
    kv_len_out[b] = kvl + a + 1;
    ctx_len_out[b] = cl + a + 1;
    root_out[b] = bonus[b];
  }
}

// ---- greedy predictions from logits: one warp per tree node's row ----
// Ordering of (value, index) candidates: a NaN beats every number (the first
// NaN wins), otherwise the larger value, ties to the smaller index (-0 == +0).
__device__ __forceinline__ bool am_better(float a, int ia, float b, int ib) {
  const bool na = a != a, nb = b != b;
  if (na || nb) return na && (!nb || ia < ib);
  return a > b || (a == b && ia < ib);
}

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

constexpr int AM_WARPS = 8;  // rows per CTA

// NaN-propagating maximum of two bf16 pairs.
__device__ __forceinline__ uint32_t max_nan_bf16x2(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("max.NaN.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}

// Rows (b, i) with i < n_nodes[b]: argmax over the vocabulary.  The row is read
// once: a scalar head up to a 16-byte boundary, then 16-byte chunks (8 bf16)
// with eight loads in flight per lane, then a scalar tail.  Per chunk a lane
// only takes the NaN-propagating maximum (three max.bf16x2) and keeps the
// first chunk holding its best value (or its first NaN); afterwards it rereads
// that one chunk for the first element equal to it.  The warp reduction then
// orders candidates by (value, index).
__global__ void __launch_bounds__(AM_WARPS * 32) k_argmax_rows(const uint16_t* __restrict__ logits, int vocab,
                                                                const int32_t* __restrict__ n_nodes, int n_pad,
                                                                uint32_t* __restrict__ argmax) {
  // the acceptance walk may be scheduled now; it waits for this grid's results
  asm volatile("griddepcontrol.launch_dependents;");
  const int b = blockIdx.y, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int i = blockIdx.x * AM_WARPS + warp;
  if (i >= n_pad) return;
  const int n = min(max((int)n_nodes[b], 0), n_pad);
  const size_t row = (size_t)b * n_pad + i;
  if (i >= n) {
    if (lane == 0) argmax[row] = 0u;
    return;
  }
  const uint16_t* p = logits + row * (size_t)vocab;
  float bv = -INFINITY;
  int bi = 0x7FFFFFFF;
  // head: elements before the first 16-byte boundary
  const int head = min(vocab, (int)(((16u - (uint32_t)(reinterpret_cast<uintptr_t>(p) & 15u)) & 15u) >> 1));
  if (lane < head) {
    bv = __uint_as_float((uint32_t)__ldg(p + lane) << 16);
    bi = lane;
  }
  const int nvec = (vocab - head) >> 3;  // whole 8-element chunks
  const uint4* pv = reinterpret_cast<const uint4*>(p + head);
  float cv = -INFINITY;  // this lane's best chunk maximum
  int cc = -1;           // and its chunk
  auto take = [&](uint4 v, int c) {
    const uint32_t m = max_nan_bf16x2(max_nan_bf16x2(v.x, v.y), max_nan_bf16x2(v.z, v.w));
    const float lo = bf16_lo(m), hi = bf16_hi(m);
    const float mc = (lo != lo || hi != hi) ? __int_as_float(0x7FC00000) : fmaxf(lo, hi);
    if (cv == cv && (mc != mc || mc > cv || cc < 0)) {  // a NaN sticks; otherwise a strictly larger one
      cv = mc;
      cc = c;
    }
  };
  int c = lane;
  for (; c + 7 * 32 < nvec; c += 8 * 32) {  // eight 16-byte loads in flight per lane
    uint4 v[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) v[u] = __ldg(pv + c + 32 * u);
#pragma unroll
    for (int u = 0; u < 8; ++u) take(v[u], c + 32 * u);
  }
  for (; c < nvec; c += 32) take(__ldg(pv + c), c);
  if (cc >= 0) {  // the first element of the best chunk that attains its maximum
    const uint4 v = __ldg(pv + cc);
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
    int e = 7;
#pragma unroll
    for (int q = 3; q >= 0; --q) {
      const float hi = bf16_hi(w[q]), lo = bf16_lo(w[q]);
      if (hi == cv || (cv != cv && hi != hi)) e = 2 * q + 1;
      if (lo == cv || (cv != cv && lo != lo)) e = 2 * q;
    }
    const int idx = head + 8 * cc + e;
    if (am_better(cv, idx, bv, bi)) {
      bv = cv;
      bi = idx;
    }
  }
  // tail: the last (vocab - head) % 8 elements
  const int t0 = head + 8 * nvec;
  if (t0 + lane < vocab) {
    const float x = __uint_as_float((uint32_t)__ldg(p + t0 + lane) << 16);
    if (am_better(x, t0 + lane, bv, bi)) {
      bv = x;
      bi = t0 + lane;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(0xFFFFFFFFu, bv, o);
    const int oi = __shfl_xor_sync(0xFFFFFFFFu, bi, o);
    if (am_better(ov, oi, bv, bi)) {
      bv = ov;
      bi = oi;
    }
  }
  if (lane == 0) argmax[row] = (uint32_t)bi;
}

// One CTA per sequence, one thread per node.
__global__ void k_synth_argmax(const uint32_t* __restrict__ tok, const int32_t* __restrict__ parent,
                               const int32_t* __restrict__ n_nodes, int n_pad, const int32_t* __restrict__ plen,
                               const uint32_t* __restrict__ rtok, uint32_t vocab, uint32_t* __restrict__ argmax) {
  __shared__ int agree[FC_MAX_NODES];
  __shared__ int par_s[FC_MAX_NODES];
  __shared__ int first_child[FC_MAX_NODES];
  __shared__ uint32_t tok_s[FC_MAX_NODES];
  const int b = blockIdx.x;
  const size_t base = (size_t)b * n_pad;
  const int n = min(max((int)n_nodes[b], 1), n_pad);
  for (int i = threadIdx.x; i < n_pad; i += blockDim.x) {  // the tree, staged once (coalesced)
    agree[i] = -1;
    first_child[i] = n_pad;
    par_s[i] = parent[base + i];
    tok_s[i] = tok[base + i];
  }
  __syncthreads();
  for (int j = 1 + threadIdx.x; j < n; j += blockDim.x) {  // first child: the smallest later node below
    const int p = par_s[j];
    if (p >= 0 && p < j) atomicMin(&first_child[p], j);
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int cur = 0;
    for (int t = 0; t < plen[b]; ++t) {
      const int first = first_child[cur];
      if (first >= n) break;
      agree[cur] = first;
      cur = first;
    }
  }
  __syncthreads();
  for (int i = threadIdx.x; i < n_pad; i += blockDim.x) {
    uint32_t x = 0;
    if (i < n) {
      if (agree[i] >= 0) {
        x = tok_s[agree[i]];
      } else {
        x = rtok[base + i] % vocab;
        for (int tries = 0; tries < n_pad; ++tries) {  // bounded: children may cover a tiny vocabulary
          bool clash = false;
          for (int j = i + 1; j < n; ++j)
            if (par_s[j] == i && tok_s[j] == x) clash = true;
          if (!clash) break;
          x = (x + 1u) % vocab;
        }
      }
    }
    argmax[base + i] = x;
  }
}

}  // namespace

extern "C" fc_status fc_accept(const uint32_t* d_tok, const int32_t* d_parent, const int32_t* d_n_nodes,
                               const uint32_t* d_argmax, int batch, int n_pad, int32_t* d_acc_len, int32_t* d_path,
                               int path_cap, uint32_t* d_bonus, fc_stream stream) {
  FC_NVTX_RANGE();
  if (batch < 0 || n_pad < 1 || n_pad > 1024 || path_cap < 1) return FC_ERR_INVALID_ARG;
  if (batch == 0) return FC_OK;
  if (!d_tok || !d_parent || !d_n_nodes || !d_argmax || !d_acc_len || !d_path || !d_bonus) return FC_ERR_INVALID_ARG;
  const unsigned blocks = (unsigned)((batch + ACC_WARPS - 1) / ACC_WARPS);
  const size_t smem = (size_t)ACC_WARPS * 3 * n_pad * sizeof(uint32_t);  // <= 48 KB for n_pad <= 1024
  k_accept<<<blocks, ACC_WARPS * 32, smem, static_cast<cudaStream_t>(stream)>>>(
      d_tok, d_parent, d_n_nodes, d_argmax, batch, n_pad, d_acc_len, d_path, path_cap, d_bonus, fc_error_slot());
  return FC_CHECK_LAUNCH();
}

extern "C" fc_status fc_argmax_accept(const void* d_logits, int vocab, const uint32_t* d_tok,
                                      const int32_t* d_parent, const int32_t* d_n_nodes, int batch, int n_pad,
                                      uint32_t* d_argmax, int32_t* d_acc_len, int32_t* d_path, int path_cap,
                                      uint32_t* d_bonus, fc_stream stream) {
  FC_NVTX_RANGE();
  if (batch < 0 || n_pad < 1 || n_pad > 1024 || path_cap < 1 || vocab < 1) return FC_ERR_INVALID_ARG;
  if (batch > 65535) return FC_ERR_UNSUPPORTED;
  if (batch == 0) return FC_OK;
  if (!d_logits || !d_tok || !d_parent || !d_n_nodes || !d_argmax || !d_acc_len || !d_path || !d_bonus)
    return FC_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(d_logits) % 2) return FC_ERR_INVALID_ARG;
  const dim3 grid((unsigned)((n_pad + AM_WARPS - 1) / AM_WARPS), (unsigned)batch);
  k_argmax_rows<<<grid, AM_WARPS * 32, 0, static_cast<cudaStream_t>(stream)>>>(
      static_cast<const uint16_t*>(d_logits), vocab, d_n_nodes, n_pad, d_argmax);
  const fc_status st = FC_CHECK_LAUNCH();
  if (st != FC_OK) return st;
  // the walk as a programmatic dependent launch: it is scheduled while the
  // argmax grid runs and waits (griddepcontrol.wait) for its completion
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)((batch + ACC_WARPS - 1) / ACC_WARPS));
  cfg.blockDim = dim3(ACC_WARPS * 32);
  cfg.dynamicSmemBytes = (size_t)ACC_WARPS * 3 * n_pad * sizeof(uint32_t);
  cfg.stream = static_cast<cudaStream_t>(stream);
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr.val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  if (cudaLaunchKernelEx(&cfg, k_accept, d_tok, d_parent, d_n_nodes, (const uint32_t*)d_argmax, batch, n_pad,
                         d_acc_len, d_path, path_cap, d_bonus, fc_error_slot()) != cudaSuccess)
    return FC_ERR_CUDA;
  return FC_CHECK_LAUNCH();
}

extern "C" fc_status fc_kv_append(const int32_t* d_path, const int32_t* d_acc_len, const uint32_t* d_bonus,
                                  const uint32_t* d_tok, const void* d_k_tree, const void* d_v_tree, int batch,
                                  int n_pad, int Hkv, int D, int path_cap, void* d_k_cache, void* d_v_cache, int kv_cap,
                                  const int32_t* d_kv_len_in, int32_t* d_kv_len_out, uint32_t* d_ctx, int ctx_stride,
                                  const int32_t* d_ctx_len_in, int32_t* d_ctx_len_out, uint32_t* d_root_out,
                                  fc_stream stream) {
  FC_NVTX_RANGE();
  if (batch < 0 || n_pad < 1 || Hkv < 1 || D < 8 || D % 8 || path_cap < 1 || kv_cap < 1 || ctx_stride < 1)
    return FC_ERR_INVALID_ARG;
  if (batch == 0) return FC_OK;
  if (!d_path || !d_acc_len || !d_bonus || !d_tok || !d_k_tree || !d_v_tree || !d_k_cache || !d_v_cache ||
      !d_kv_len_in || !d_kv_len_out || !d_ctx || !d_ctx_len_in || !d_ctx_len_out || !d_root_out)
    return FC_ERR_INVALID_ARG;
  if (d_kv_len_in == d_kv_len_out || d_ctx_len_in == d_ctx_len_out) return FC_ERR_INVALID_ARG;
  const uintptr_t al = reinterpret_cast<uintptr_t>(d_k_tree) | reinterpret_cast<uintptr_t>(d_v_tree) |
                       reinterpret_cast<uintptr_t>(d_k_cache) | reinterpret_cast<uintptr_t>(d_v_cache);
  if (al % 16) return FC_ERR_INVALID_ARG;
  k_kv_append<<<batch, 256, 0, static_cast<cudaStream_t>(stream)>>>(
      d_path, d_acc_len, d_bonus, d_tok, static_cast<const uint4*>(d_k_tree), static_cast<const uint4*>(d_v_tree), n_pad,
      Hkv, D, path_cap, static_cast<uint4*>(d_k_cache), static_cast<uint4*>(d_v_cache), kv_cap, d_kv_len_in,
      d_kv_len_out, d_ctx, ctx_stride, d_ctx_len_in, d_ctx_len_out, d_root_out, fc_error_slot());
  return FC_CHECK_LAUNCH();
}

extern "C" fc_status fc_synth_argmax(const uint32_t* d_tok, const int32_t* d_parent, const int32_t* d_n_nodes,
                                     int batch, int n_pad, const int32_t* d_plen, const uint32_t* d_rtok,
                                     uint32_t vocab, uint32_t* d_argmax, fc_stream stream) {
  FC_NVTX_RANGE();
  if (batch < 0 || n_pad < 1 || n_pad > FC_MAX_NODES || vocab < 2) return FC_ERR_INVALID_ARG;
  if (batch == 0) return FC_OK;
  if (!d_tok || !d_parent || !d_n_nodes || !d_plen || !d_rtok || !d_argmax) return FC_ERR_INVALID_ARG;
  k_synth_argmax<<<batch, 128, 0, static_cast<cudaStream_t>(stream)>>>(d_tok, d_parent, d_n_nodes, n_pad, d_plen,
                                                                       d_rtok, vocab, d_argmax);
  return FC_CHECK_LAUNCH();
}

// ---------------------------------------------------------------------------
// Self-test of the bounded waits (no counterpart in the paper): one CTA waits
// on an mbarrier phase with the kernels' own bounded wait.  With arrive != 0
// the phase completes first and the wait succeeds; with arrive == 0 nothing
// ever arrives, the wait gives up after limit_cycles and the kernel records
// FC_ERR_TIMEOUT and returns: the path a stuck pipeline takes, exercised
// without faulting or hanging anything.
// ---------------------------------------------------------------------------
namespace {
__global__ void k_selftest_wait(int arrive, unsigned long long limit_cycles, unsigned int* err) {
  __shared__ __align__(8) uint64_t bar_word;
  __shared__ int abort_flag;
  const uint32_t bar = smem_u32(&bar_word);
  if (threadIdx.x == 0) {
    abort_flag = 0;
    mbar_init(bar, 1);
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    if (arrive) mbar_arrive(bar);
    if (!mbar_wait_bounded(bar, 0, &abort_flag, limit_cycles)) fc_flag(FC_ERR_WORD(err), FC_EBIT_TIMEOUT);
  }
}
}  // namespace

extern "C" fc_status fc_selftest_wait(int arrive, unsigned long long limit_cycles, fc_stream stream) {
  FC_NVTX_RANGE();
  if (limit_cycles == 0 || limit_cycles > 4000000000ull) return FC_ERR_INVALID_ARG;
  k_selftest_wait<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(arrive, limit_cycles, fc_error_slot());
  return FC_CHECK_LAUNCH();
}
