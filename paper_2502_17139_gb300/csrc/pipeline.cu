// Native step executor: one call enqueues a whole decoding step (Section
// IV-C and IV-D: retrieval -> draft tree -> tree attention -> verification
// -> cache append) for every sub-batch of a batch, each sub-batch on CUDA
// streams of its own.
//
// The sequences of a batch are independent, so sub-batch h may run step
// s + 1 while sub-batch h' is still in step s.  Per sub-batch the executor
// owns two streams: a high-priority one for the latency-bound chain
// (replay-cache lookup with retrieval and insert, or Algorithm 1's CACHE
// search, retrieval and missing-table insert; tree build, predictions,
// acceptance, append and, with the CACHE, its update) and a low-priority one for the attention launch,
// ordered by an event pair.  When SMs free up, the block scheduler then
// starts another sub-batch's chain ahead of this sub-batch's remaining
// attention CTAs.  The executor holds no device memory: every buffer
// belongs to the caller, and every launch goes through this library's own
// entry points.  Issuing a step costs the host one call instead of one call
// per kernel, so several sub-batches can be kept in flight.
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdint>
#include <new>
#include <vector>

#include "../../include/fastcoder.h"
#include "fc_common.cuh"

struct fc_pipeline {
  fc_pipeline_desc d;
  std::vector<fc_pipeline_part> parts;
  std::vector<fc_datastore> sources;
  std::vector<uint32_t> weight;
  std::vector<cudaStream_t> chain, attn;
  std::vector<cudaEvent_t> ev_pre, ev_post, ev_done, ev_fork;
  cudaEvent_t ev_start = nullptr;
  int p_chain = 0, p_attn = 0;                    // the two streams' priorities
  std::vector<cudaGraphNode_t>* capture_attn = nullptr;  // while capturing: the attention nodes
};

// A sub-batch's steps captured into a CUDA graph whose kernel nodes keep the
// priorities of the streams they were captured on.
struct fc_pipeline_graph {
  cudaGraph_t graph = nullptr;
  cudaGraphExec_t exec = nullptr;
  int p_chain = 0, p_attn = 0;
};

namespace {

void destroy_handles(fc_pipeline* pl) {
  for (cudaStream_t s : pl->chain)
    if (s) cudaStreamDestroy(s);
  for (cudaStream_t s : pl->attn)
    if (s) cudaStreamDestroy(s);
  for (auto* v : {&pl->ev_pre, &pl->ev_post, &pl->ev_done, &pl->ev_fork})
    for (cudaEvent_t e : *v)
      if (e) cudaEventDestroy(e);
  if (pl->ev_start) cudaEventDestroy(pl->ev_start);
}

bool part_ok(const fc_pipeline_desc& d, const fc_pipeline_part& p) {
  if (p.batch < 1 || p.first < 0 || p.ctx_stride < 1) return false;
  const void* need[] = {p.ctx, p.ctx_len[0], p.ctx_len[1], p.kv_len[0], p.kv_len[1], p.root, p.skip, p.drafts,
                        p.draft_len, p.count, p.n_drafts, p.match_len, p.tok, p.parent, p.depth, p.pos, p.mask,
                        p.n_nodes, p.k_cache, p.v_cache, p.attn_out, p.argmax, p.acc_len, p.path, p.bonus};
  for (const void* q : need)
    if (!q) return false;
  if (p.ctx_len[0] == p.ctx_len[1] || p.kv_len[0] == p.kv_len[1]) return false;
  if (p.rcache && p.rcache_capacity < 1) return false;
  if (d.rope_base > 0.f && !p.k_tree_rot) return false;
  const fc_cache& q = p.seq_cache;
  if (q.d_words) {  // Algorithm 1: the CACHE replaces the replay cache
    if (p.rcache || !q.d_meta || q.capacity < 16 || q.capacity % 4 || q.capacity > FC_CACHE_MAX_WORDS ||
        q.min_size < 0 || q.chunk < 1 || q.ctx_keep < 0 || q.ctx_keep > FC_MAX_NMAX ||
        reinterpret_cast<uintptr_t>(q.d_words) % 16)
      return false;
    // M: a power-of-two capacity from 2 to 2^24 slots
    if (p.missing && (p.missing_capacity < 2 || p.missing_capacity > (1 << 24) ||
                      (p.missing_capacity & (p.missing_capacity - 1))))
      return false;
  } else if (p.missing) {
    return false;
  }
  return true;
}

// Stage events of part h: [4 stages][start, end]; null entries are skipped.
void stage_event(void* const* ev, int h, int stage, int end, cudaStream_t s) {
  if (!ev) return;
  cudaEvent_t e = static_cast<cudaEvent_t>(ev[h * 8 + stage * 2 + end]);
  if (e) cudaEventRecord(e, s);
}

#define FC_TRY(call)                  \
  do {                                \
    const fc_status st_ = (call);     \
    if (st_ != FC_OK) return st_;     \
  } while (0)

}  // namespace

extern "C" fc_status fc_pipeline_create(const fc_pipeline_desc* d, fc_pipeline** out) {
  FC_NVTX_RANGE();
  if (!d || !out) return FC_ERR_INVALID_ARG;
  *out = nullptr;
  if (d->n_parts < 1 || !d->parts || d->n_sources < 1 || !d->sources || !d->src_weight) return FC_ERR_INVALID_ARG;
  if (d->node_budget < 1 || d->n_pad < 1 || d->H < 1 || d->Hkv < 1 || d->D < 1 || d->kv_cap < 1 ||
      d->path_cap < 1 || d->vocab < 1 || !(d->scale > 0.f) || d->rope_base < 0.f)
    return FC_ERR_INVALID_ARG;
  for (int h = 0; h < d->n_parts; ++h)
    if (!part_ok(*d, d->parts[h])) return FC_ERR_INVALID_ARG;
  fc_pipeline* pl = new (std::nothrow) fc_pipeline();
  if (!pl) return FC_ERR_CAPACITY;
  pl->d = *d;
  pl->parts.assign(d->parts, d->parts + d->n_parts);
  pl->sources.assign(d->sources, d->sources + d->n_sources);
  pl->weight.assign(d->src_weight, d->src_weight + d->n_sources);
  pl->weight.push_back(d->cache_weight);  // slot n_sources: the CACHE's result (Algorithm 1 parts)
  pl->d.parts = nullptr;  // the copies above are the ones used
  pl->d.sources = nullptr;
  pl->d.src_weight = nullptr;
  int lo = 0, hi = 0;  // least and greatest priority (greatest is the most negative)
  bool ok = cudaDeviceGetStreamPriorityRange(&lo, &hi) == cudaSuccess;
  const int p_chain = std::max(hi, -1), p_attn = lo;
  pl->p_chain = p_chain;
  pl->p_attn = p_attn;
  const int n = d->n_parts;
  pl->chain.assign(n, nullptr);
  pl->attn.assign(n, nullptr);
  pl->ev_pre.assign(n, nullptr);
  pl->ev_post.assign(n, nullptr);
  pl->ev_done.assign(n, nullptr);
  pl->ev_fork.assign(n, nullptr);
  ok = ok && cudaEventCreateWithFlags(&pl->ev_start, cudaEventDisableTiming) == cudaSuccess;
  for (int h = 0; ok && h < n; ++h) {
    ok = cudaStreamCreateWithPriority(&pl->chain[h], cudaStreamNonBlocking, p_chain) == cudaSuccess &&
         cudaStreamCreateWithPriority(&pl->attn[h], cudaStreamNonBlocking, p_attn) == cudaSuccess &&
         cudaEventCreateWithFlags(&pl->ev_pre[h], cudaEventDisableTiming) == cudaSuccess &&
         cudaEventCreateWithFlags(&pl->ev_post[h], cudaEventDisableTiming) == cudaSuccess &&
         cudaEventCreateWithFlags(&pl->ev_done[h], cudaEventDisableTiming) == cudaSuccess &&
         cudaEventCreateWithFlags(&pl->ev_fork[h], cudaEventDisableTiming) == cudaSuccess;
  }
  if (!ok) {
    destroy_handles(pl);
    delete pl;
    return FC_ERR_CUDA;
  }
  *out = pl;
  return FC_OK;
}

extern "C" void fc_pipeline_destroy(fc_pipeline* pl) {
  if (!pl) return;
  for (cudaStream_t s : pl->chain)
    if (s) cudaStreamSynchronize(s);
  for (cudaStream_t s : pl->attn)
    if (s) cudaStreamSynchronize(s);
  destroy_handles(pl);
  delete pl;
}

namespace {

// One sub-batch's step on its streams (the chain stream already waits for
// whatever the step must follow).
fc_status enqueue_part(fc_pipeline* pl, int h, int c, bool attention, const void* d_q, const void* d_k_tree,
                       const void* d_v_tree, const int32_t* d_want_hit, const int32_t* d_plen,
                       const uint32_t* d_rtok, void* const* stage_events) {
  const fc_pipeline_desc& d = pl->d;
  const int nx = 1 - c, S = d.n_sources, Np = d.n_pad;
  const bool rope = d.rope_base > 0.f;
  const size_t q_row = (size_t)Np * d.H * d.D * 2, kt_row = (size_t)d.Hkv * Np * d.D * 2;  // bytes per sequence
  const fc_pipeline_part& P = pl->parts[h];
  cudaStream_t s = pl->chain[h], sa = pl->attn[h];
  const int B = P.batch;
  const void* q = attention ? static_cast<const char*>(d_q) + (size_t)P.first * q_row : nullptr;
  const void* kt = static_cast<const char*>(d_k_tree) + (size_t)P.first * kt_row;
  const void* vt = static_cast<const char*>(d_v_tree) + (size_t)P.first * kt_row;
  const int32_t* want = d_want_hit ? d_want_hit + P.first : nullptr;
  FcErrorScope scope(P.err);  // the sub-batch's kernels record errors in its own word

  const bool seq = P.seq_cache.d_words != nullptr;
  stage_event(stage_events, h, 0, 0, s);
  if (seq) {  // Algorithm 1: the CACHE and M first, the datastores for the queries they leave
    FC_TRY(fc_cache_search(&P.seq_cache, P.missing, P.missing_capacity, P.ctx, P.ctx_stride, P.ctx_len[c], B, d.p,
                           S, P.drafts, P.draft_len, P.count, P.n_drafts, P.match_len, P.skip, s));
    FC_TRY(fc_retrieve(pl->sources.data(), S, P.ctx, P.ctx_stride, P.ctx_len[c], B, P.skip, d.p, P.drafts,
                       P.draft_len, P.count, P.n_drafts, P.match_len, s));
    if (P.missing)
      FC_TRY(fc_missing_insert(P.missing, P.missing_capacity, d.p.n_min, P.ctx, P.ctx_stride, P.ctx_len[c], B,
                               P.skip, P.n_drafts, S, s));
  } else if (P.rcache) {  // replay-cache lookup and retrieval of the queries it did not serve, one launch
    FC_TRY(fc_retrieve_cached(pl->sources.data(), S, P.ctx, P.ctx_stride, P.ctx_len[c], B, P.rcache,
                              P.rcache_capacity, want, P.skip, d.p, P.drafts, P.draft_len, P.count, P.n_drafts,
                              P.match_len, s));
    FC_TRY(fc_rcache_insert(P.rcache, P.rcache_capacity, S, d.p, P.ctx, P.ctx_stride, P.ctx_len[c], B, P.skip,
                            P.drafts, P.draft_len, P.count, P.n_drafts, P.match_len, s));
  } else {
    FC_TRY(fc_retrieve(pl->sources.data(), S, P.ctx, P.ctx_stride, P.ctx_len[c], B, nullptr, d.p, P.drafts,
                       P.draft_len, P.count, P.n_drafts, P.match_len, s));
  }
  stage_event(stage_events, h, 0, 1, s);
  stage_event(stage_events, h, 1, 0, s);
  FC_TRY(fc_build_tree(seq ? S + 1 : S, P.drafts, P.draft_len, P.count, P.n_drafts, pl->weight.data(), d.p.top_k,
                       d.p.draft_len, P.root, P.kv_len[c], B, d.node_budget, Np, P.tok, P.parent, P.depth, P.pos,
                       P.mask, P.n_nodes, s));
  stage_event(stage_events, h, 1, 1, s);
  if (rope) {
    FC_TRY(fc_rope(kt, P.k_tree_rot, B, Np, d.Hkv, d.D, 1, P.pos, d.rope_base, s));
    kt = P.k_tree_rot;
  }
  if (attention) {  // on its own stream, ordered by an event pair
    if (cudaEventRecord(pl->ev_pre[h], s) != cudaSuccess || cudaStreamWaitEvent(sa, pl->ev_pre[h], 0) != cudaSuccess)
      return FC_ERR_CUDA;
    stage_event(stage_events, h, 2, 0, sa);
    if (rope)
      FC_TRY(fc_tree_attn_rope(q, P.k_cache, P.v_cache, d.kv_cap, P.kv_len[c], kt, vt, P.mask, P.n_nodes, B, Np,
                               d.H, d.Hkv, d.D, d.scale, P.pos, d.rope_base, P.attn_out, P.attn_ws,
                               P.attn_ws_bytes, sa));
    else
      FC_TRY(fc_tree_attn(q, P.k_cache, P.v_cache, d.kv_cap, P.kv_len[c], kt, vt, P.mask, P.n_nodes, B, Np, d.H,
                          d.Hkv, d.D, d.scale, P.attn_out, P.attn_ws, P.attn_ws_bytes, sa));
    stage_event(stage_events, h, 2, 1, sa);
    if (pl->capture_attn) {  // capturing: the attention launch is the node the attention stream ends on
      cudaStreamCaptureStatus cs;
      const cudaGraphNode_t* deps = nullptr;
      size_t nd = 0;
      if (cudaStreamGetCaptureInfo(sa, &cs, nullptr, nullptr, &deps, nullptr, &nd) != cudaSuccess ||
          cs != cudaStreamCaptureStatusActive)
        return FC_ERR_CUDA;
      pl->capture_attn->insert(pl->capture_attn->end(), deps, deps + nd);
    }
    if (cudaEventRecord(pl->ev_post[h], sa) != cudaSuccess ||
        cudaStreamWaitEvent(s, pl->ev_post[h], 0) != cudaSuccess)
      return FC_ERR_CUDA;
  }
  stage_event(stage_events, h, 3, 0, s);
  FC_TRY(fc_synth_argmax(P.tok, P.parent, P.n_nodes, B, Np, d_plen + P.first, d_rtok + (size_t)P.first * Np,
                         d.vocab, P.argmax, s));
  FC_TRY(fc_accept(P.tok, P.parent, P.n_nodes, P.argmax, B, Np, P.acc_len, P.path, d.path_cap, P.bonus, s));
  FC_TRY(fc_kv_append(P.path, P.acc_len, P.bonus, P.tok, kt, vt, B, Np, d.Hkv, d.D, d.path_cap, P.k_cache,
                      P.v_cache, d.kv_cap, P.kv_len[c], P.kv_len[nx], P.ctx, P.ctx_stride, P.ctx_len[c],
                      P.ctx_len[nx], P.root, s));
  if (seq)  // the verified retrieval and the completed output pieces go to the CACHE
    FC_TRY(fc_cache_update(&P.seq_cache, P.ctx, P.ctx_stride, P.ctx_len[c], P.ctx_len[nx], P.acc_len, B, s));
  stage_event(stage_events, h, 3, 1, s);
  return FC_OK;
}

bool step_args_ok(const fc_pipeline* pl, int phase, int flags, const void* d_q, const void* d_k_tree,
                  const void* d_v_tree, const int32_t* d_plen, const uint32_t* d_rtok) {
  const bool attention = !(flags & FC_PIPELINE_NO_ATTENTION);
  return pl && (phase == 0 || phase == 1) && !(flags & ~FC_PIPELINE_NO_ATTENTION) && (!attention || d_q) &&
         d_k_tree && d_v_tree && d_plen && d_rtok;
}

}  // namespace

extern "C" fc_status fc_pipeline_step(fc_pipeline* pl, int phase, int flags, const void* d_q, const void* d_k_tree,
                                      const void* d_v_tree, const int32_t* d_want_hit, const int32_t* d_plen,
                                      const uint32_t* d_rtok, fc_stream caller, void* const* stage_events) {
  FC_NVTX_RANGE();
  if (!step_args_ok(pl, phase, flags, d_q, d_k_tree, d_v_tree, d_plen, d_rtok)) return FC_ERR_INVALID_ARG;
  const bool attention = !(flags & FC_PIPELINE_NO_ATTENTION);
  if (cudaEventRecord(pl->ev_start, static_cast<cudaStream_t>(caller)) != cudaSuccess) return FC_ERR_CUDA;
  for (int h = 0; h < pl->d.n_parts; ++h) {
    if (cudaStreamWaitEvent(pl->chain[h], pl->ev_start, 0) != cudaSuccess) return FC_ERR_CUDA;
    FC_TRY(enqueue_part(pl, h, phase, attention, d_q, d_k_tree, d_v_tree, d_want_hit, d_plen, d_rtok, stage_events));
  }
  return FC_OK;
}

extern "C" fc_status fc_pipeline_step_part(fc_pipeline* pl, int part, int phase, int flags, const void* d_q,
                                           const void* d_k_tree, const void* d_v_tree, const int32_t* d_want_hit,
                                           const int32_t* d_plen, const uint32_t* d_rtok, fc_stream caller,
                                           void* const* stage_events) {
  FC_NVTX_RANGE();
  if (!step_args_ok(pl, phase, flags, d_q, d_k_tree, d_v_tree, d_plen, d_rtok) || part < 0 ||
      part >= pl->d.n_parts)
    return FC_ERR_INVALID_ARG;
  if (cudaEventRecord(pl->ev_fork[part], static_cast<cudaStream_t>(caller)) != cudaSuccess ||
      cudaStreamWaitEvent(pl->chain[part], pl->ev_fork[part], 0) != cudaSuccess)
    return FC_ERR_CUDA;
  return enqueue_part(pl, part, phase, !(flags & FC_PIPELINE_NO_ATTENTION), d_q, d_k_tree, d_v_tree, d_want_hit,
                      d_plen, d_rtok, stage_events);
}

extern "C" fc_status fc_pipeline_error(fc_pipeline* pl, int part) {
  FC_NVTX_RANGE();
  if (!pl || part < 0 || part >= (int)pl->parts.size() || !pl->parts[part].err) return FC_ERR_INVALID_ARG;
  cudaStream_t s = pl->chain[part];
  unsigned int* w = pl->parts[part].err;
  unsigned int h = 0;
  // the chain stream already follows the attention stream of every step
  if (cudaMemcpyAsync(&h, w, sizeof h, cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaMemsetAsync(w, 0, sizeof h, s) != cudaSuccess || cudaStreamSynchronize(s) != cudaSuccess)
    return FC_ERR_CUDA;
  return fc_status_of_bits(h);
}

extern "C" fc_stream fc_pipeline_stream(const fc_pipeline* pl, int part) {
  if (!pl || part < 0 || part >= (int)pl->chain.size()) return nullptr;
  return pl->chain[part];
}

extern "C" fc_status fc_pipeline_join_part(fc_pipeline* pl, int part, fc_stream caller) {
  if (!pl || part < 0 || part >= (int)pl->chain.size()) return FC_ERR_INVALID_ARG;
  if (cudaEventRecord(pl->ev_done[part], pl->chain[part]) != cudaSuccess ||
      cudaStreamWaitEvent(static_cast<cudaStream_t>(caller), pl->ev_done[part], 0) != cudaSuccess)
    return FC_ERR_CUDA;
  return FC_OK;
}

extern "C" fc_status fc_pipeline_join(fc_pipeline* pl, fc_stream caller) {
  if (!pl) return FC_ERR_INVALID_ARG;
  cudaStream_t cs = static_cast<cudaStream_t>(caller);
  for (size_t h = 0; h < pl->chain.size(); ++h)
    if (cudaEventRecord(pl->ev_done[h], pl->chain[h]) != cudaSuccess ||
        cudaStreamWaitEvent(cs, pl->ev_done[h], 0) != cudaSuccess)
      return FC_ERR_CUDA;
  return FC_OK;
}

namespace {

void graph_free(fc_pipeline_graph* g) {
  if (!g) return;
  if (g->exec) cudaGraphExecDestroy(g->exec);
  if (g->graph) cudaGraphDestroy(g->graph);
  delete g;
}

// The graph's kernel nodes, with their type checked.
fc_status kernel_nodes(cudaGraph_t graph, std::vector<cudaGraphNode_t>* out) {
  size_t n = 0;
  if (cudaGraphGetNodes(graph, nullptr, &n) != cudaSuccess) return FC_ERR_CUDA;
  std::vector<cudaGraphNode_t> nodes(n);
  if (n && cudaGraphGetNodes(graph, nodes.data(), &n) != cudaSuccess) return FC_ERR_CUDA;
  out->clear();
  for (cudaGraphNode_t v : nodes) {
    cudaGraphNodeType t;
    if (cudaGraphNodeGetType(v, &t) != cudaSuccess) return FC_ERR_CUDA;
    if (t == cudaGraphNodeTypeKernel) out->push_back(v);
  }
  return FC_OK;
}

}  // namespace

extern "C" fc_status fc_pipeline_capture_part(fc_pipeline* pl, int part, int n_steps, int phase0, int flags,
                                              const void* const* d_q, const void* const* d_k_tree,
                                              const void* const* d_v_tree, const int32_t* const* d_want_hit,
                                              const int32_t* const* d_plen, const uint32_t* const* d_rtok,
                                              fc_pipeline_graph** out) {
  FC_NVTX_RANGE();
  if (!out) return FC_ERR_INVALID_ARG;
  *out = nullptr;
  if (!pl || part < 0 || part >= pl->d.n_parts || n_steps < 1 || (phase0 != 0 && phase0 != 1) || !d_k_tree ||
      !d_v_tree || !d_plen || !d_rtok || (!(flags & FC_PIPELINE_NO_ATTENTION) && !d_q))
    return FC_ERR_INVALID_ARG;
  for (int t = 0; t < n_steps; ++t)
    if (!step_args_ok(pl, (phase0 + t) & 1, flags, d_q ? d_q[t] : nullptr, d_k_tree[t], d_v_tree[t], d_plen[t],
                      d_rtok[t]))
      return FC_ERR_INVALID_ARG;
  const bool attention = !(flags & FC_PIPELINE_NO_ATTENTION);
  fc_pipeline_graph* g = new (std::nothrow) fc_pipeline_graph();
  if (!g) return FC_ERR_CAPACITY;
  g->p_chain = pl->p_chain;
  g->p_attn = pl->p_attn;
  std::vector<cudaGraphNode_t> attn_nodes;
  cudaStream_t s = pl->chain[part];
  if (cudaStreamBeginCapture(s, cudaStreamCaptureModeThreadLocal) != cudaSuccess) {
    graph_free(g);
    return FC_ERR_CUDA;
  }
  pl->capture_attn = &attn_nodes;
  fc_status st = FC_OK;
  for (int t = 0; t < n_steps && st == FC_OK; ++t)
    st = enqueue_part(pl, part, (phase0 + t) & 1, attention, d_q ? d_q[t] : nullptr, d_k_tree[t], d_v_tree[t],
                      d_want_hit ? d_want_hit[t] : nullptr, d_plen[t], d_rtok[t], nullptr);
  pl->capture_attn = nullptr;
  const cudaError_t ce = cudaStreamEndCapture(s, &g->graph);  // ends the capture on every path
  if (st == FC_OK && ce != cudaSuccess) st = FC_ERR_CUDA;
  // every kernel at its stream's priority: the chain's above the attention's
  std::vector<cudaGraphNode_t> kn;
  if (st == FC_OK) st = kernel_nodes(g->graph, &kn);
  for (size_t i = 0; st == FC_OK && i < kn.size(); ++i) {
    cudaLaunchAttributeValue v{};
    v.priority = std::find(attn_nodes.begin(), attn_nodes.end(), kn[i]) != attn_nodes.end() ? g->p_attn : g->p_chain;
    if (cudaGraphKernelNodeSetAttribute(kn[i], cudaLaunchAttributePriority, &v) != cudaSuccess) st = FC_ERR_CUDA;
  }
  if (st == FC_OK &&
      cudaGraphInstantiateWithFlags(&g->exec, g->graph, cudaGraphInstantiateFlagUseNodePriority) != cudaSuccess)
    st = FC_ERR_CUDA;
  // the executable graph's device-side setup now, not at its first launch
  if (st == FC_OK && cudaGraphUpload(g->exec, s) != cudaSuccess) st = FC_ERR_CUDA;
  if (st != FC_OK) {
    graph_free(g);
    return st;
  }
  *out = g;
  return FC_OK;
}

extern "C" fc_status fc_pipeline_graph_launch(fc_pipeline_graph* g, fc_stream s) {
  if (!g || !g->exec) return FC_ERR_INVALID_ARG;
  return cudaGraphLaunch(g->exec, static_cast<cudaStream_t>(s)) == cudaSuccess ? FC_OK : FC_ERR_CUDA;
}

extern "C" fc_status fc_pipeline_graph_kernels(const fc_pipeline_graph* g, int* n_chain, int* n_attn) {
  if (!g || !g->graph || !n_chain || !n_attn) return FC_ERR_INVALID_ARG;
  std::vector<cudaGraphNode_t> kn;
  const fc_status st = kernel_nodes(g->graph, &kn);
  if (st != FC_OK) return st;
  *n_chain = *n_attn = 0;
  for (cudaGraphNode_t v : kn) {
    cudaLaunchAttributeValue a{};
    if (cudaGraphKernelNodeGetAttribute(v, cudaLaunchAttributePriority, &a) != cudaSuccess) return FC_ERR_CUDA;
    if (a.priority == g->p_attn && g->p_attn != g->p_chain)
      ++*n_attn;
    else if (a.priority == g->p_chain)
      ++*n_chain;
    else
      return FC_ERR_INTERNAL;
  }
  return FC_OK;
}

extern "C" void fc_pipeline_graph_destroy(fc_pipeline_graph* g) { graph_free(g); }
