// fc_accept, fc_kv_append and fc_synth_argmax: the end of a decoding step.
//
// Acceptance follows Section IV-D (every correct token from the start is
// accepted, everything after the first error rejected); the cache append
// closes the decoding loop (accepted tokens' K/V join the cache, the target
// model's own next token becomes the next root).  fc_synth_argmax is the
// workload's stand-in for the target model's greedy predictions.
#include "fc_common.cuh"

FC_DEFINE_ERROR_WORD(step)

namespace {

// One warp per sequence.  Children of `cur` sit after it in preorder, so the
// warp scans node ids cur+1 .. n-1 in chunks of 32 with one ballot each.
__global__ void k_accept(const uint32_t* __restrict__ tok, const int32_t* __restrict__ parent,
                         const int32_t* __restrict__ n_nodes, const uint32_t* __restrict__ argmax, int B, int n_pad,
                         int32_t* __restrict__ acc_len, int32_t* __restrict__ path, int path_cap,
                         uint32_t* __restrict__ bonus) {
  const int b = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (b >= B) return;
  const size_t base = (size_t)b * n_pad;
  const int n = min(max((int)n_nodes[b], 1), n_pad);
  int32_t* pth = path + (size_t)b * path_cap;
  for (int t = lane; t < path_cap; t += 32) pth[t] = -1;
  __syncwarp();
  int cur = 0, len = 0;
  bool overflow = false;
  for (;;) {
    const uint32_t want = argmax[base + cur];
    int next = -1;
    for (int j0 = cur + 1; j0 < n && next < 0; j0 += 32) {
      int j = j0 + lane;
      bool hit = j < n && parent[base + j] == cur && tok[base + j] == want;
      uint32_t m = __ballot_sync(0xFFFFFFFFu, hit);
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
    bonus[b] = argmax[base + cur];
    if (overflow) fc_flag(&g_fc_err, FC_EBIT_CAPACITY);
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
                            int32_t* __restrict__ ctx_len_out, uint32_t* __restrict__ root_out) {
  const int b = blockIdx.x;
  const int a = acc_len[b];
  const int kvl = kv_len_in[b], cl = ctx_len_in[b];
  const bool ok = a >= 0 && a + 1 <= path_cap && kvl >= 0 && kvl + a + 1 <= kv_cap && cl >= 0 &&
                  cl + a + 1 <= ctx_stride;
  if (!ok) {
    if (threadIdx.x == 0) {
      fc_flag(&g_fc_err, FC_EBIT_CAPACITY);
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
      fc_flag(&g_fc_err, FC_EBIT_INVALID);
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

// One CTA per sequence, one thread per node.
__global__ void k_synth_argmax(const uint32_t* __restrict__ tok, const int32_t* __restrict__ parent,
                               const int32_t* __restrict__ n_nodes, int n_pad, const int32_t* __restrict__ plen,
                               const uint32_t* __restrict__ rtok, uint32_t vocab, uint32_t* __restrict__ argmax) {
  __shared__ int agree[FC_MAX_NODES];
  __shared__ int par_s[FC_MAX_NODES];
  __shared__ uint32_t tok_s[FC_MAX_NODES];
  const int b = blockIdx.x;
  const size_t base = (size_t)b * n_pad;
  const int n = min(max((int)n_nodes[b], 1), n_pad);
  for (int i = threadIdx.x; i < n_pad; i += blockDim.x) {  // the tree, staged once (coalesced)
    agree[i] = -1;
    par_s[i] = parent[base + i];
    tok_s[i] = tok[base + i];
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int cur = 0;
    for (int t = 0; t < plen[b]; ++t) {
      int first = -1;
      for (int j = cur + 1; j < n && first < 0; ++j)
        if (par_s[j] == cur) first = j;
      if (first < 0) break;
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
  if (batch < 0 || n_pad < 1 || n_pad > 1024 || path_cap < 1) return FC_ERR_INVALID_ARG;
  if (batch == 0) return FC_OK;
  if (!d_tok || !d_parent || !d_n_nodes || !d_argmax || !d_acc_len || !d_path || !d_bonus) return FC_ERR_INVALID_ARG;
  const int threads = 128;
  const unsigned blocks = (unsigned)((batch * 32 + threads - 1) / threads);
  k_accept<<<blocks, threads, 0, static_cast<cudaStream_t>(stream)>>>(d_tok, d_parent, d_n_nodes, d_argmax, batch,
                                                                      n_pad, d_acc_len, d_path, path_cap, d_bonus);
  return FC_CHECK_LAUNCH();
}

extern "C" fc_status fc_kv_append(const int32_t* d_path, const int32_t* d_acc_len, const uint32_t* d_bonus,
                                  const uint32_t* d_tok, const void* d_k_tree, const void* d_v_tree, int batch,
                                  int n_pad, int Hkv, int D, int path_cap, void* d_k_cache, void* d_v_cache, int kv_cap,
                                  const int32_t* d_kv_len_in, int32_t* d_kv_len_out, uint32_t* d_ctx, int ctx_stride,
                                  const int32_t* d_ctx_len_in, int32_t* d_ctx_len_out, uint32_t* d_root_out,
                                  fc_stream stream) {
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
      d_kv_len_out, d_ctx, ctx_stride, d_ctx_len_in, d_ctx_len_out, d_root_out);
  return FC_CHECK_LAUNCH();
}

extern "C" fc_status fc_synth_argmax(const uint32_t* d_tok, const int32_t* d_parent, const int32_t* d_n_nodes,
                                     int batch, int n_pad, const int32_t* d_plen, const uint32_t* d_rtok,
                                     uint32_t vocab, uint32_t* d_argmax, fc_stream stream) {
  if (batch < 0 || n_pad < 1 || n_pad > FC_MAX_NODES || vocab < 2) return FC_ERR_INVALID_ARG;
  if (batch == 0) return FC_OK;
  if (!d_tok || !d_parent || !d_n_nodes || !d_plen || !d_rtok || !d_argmax) return FC_ERR_INVALID_ARG;
  k_synth_argmax<<<batch, 128, 0, static_cast<cudaStream_t>(stream)>>>(d_tok, d_parent, d_n_nodes, n_pad, d_plen,
                                                                       d_rtok, vocab, d_argmax);
  return FC_CHECK_LAUNCH();
}
