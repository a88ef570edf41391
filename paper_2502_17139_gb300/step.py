"""One retrieve-and-verify decoding step, composed from the C-ABI calls.

A step (Section IV-C Algorithm 1 and Section IV-D) for a batch of sequences:
  retrieval -> fc_build_tree -> fc_tree_attn -> target-model predictions (the
  synthetic stand-in) -> fc_accept -> fc_kv_append (cache rows, context,
  lengths and next root).

Retrieval takes one of two forms:
  * with ``seq_cache`` (Algorithm 1 with the CACHE of Section IV-B and the
    missing table): fc_cache_search -> fc_retrieve on the datastore sources
    for the queries the CACHE did not serve and M did not skip ->
    fc_missing_insert; after the append, fc_cache_update stores the verified
    retrieval and the completed output pieces.  The tree merges S + 1 result
    slots, the CACHE's last.
  * otherwise the context-keyed replay cache: lookup and fc_retrieve on the
    queries it did not serve (one launch, fc_retrieve_cached) -> insert.

Every call is asynchronous on the current stream and allocates nothing, so
steps can be captured once into a CUDA graph and replayed (lengths ping-pong
between two buffers, so a graph holds an even number of consecutive steps).
PipelinedStepLoop runs the step over sub-batches of the sequences on streams
of their own, through the native step executor (fc_pipeline_step): one C call
enqueues every sub-batch's kernels.
"""
from __future__ import annotations

import contextlib

import numpy as np
import torch

from . import fastcoder as fc


class StepLoop:
    def __init__(self, sources, ctx, ctx_len, p, node_budget, n_pad, src_weight, H, Hkv, D, kv_cap, kv_len0, vocab,
                 cache_capacity=1 << 14, device="cuda", k_cache=None, v_cache=None, seq_cache=None,
                 rope_base=None, decoder=None):
        """seq_cache: None, or a dict with capacity, min_size, chunk, ctx_keep
        (the CACHE), missing_capacity (M) and weight (the CACHE slot's tree
        weight); it replaces the replay cache.  rope_base: None (q and the
        tree keys arrive rotated), or the RoPE base: step() then takes them
        unrotated, the tree keys are rotated once by their node positions
        (fc_rope) for the attention and the cache append, and the queries are
        rotated inside the attention kernel (fc_tree_attn_rope).  decoder: None,
        or a decoder.TreeDecoder: the verification is then its forward over the
        tree (step()'s q, k_tree, v_tree, plen and rtok are unused), greedy
        acceptance from its logits (fc_argmax_accept), and the accepted path
        appended to every layer's cache."""
        self.sources, self.p, self.node_budget, self.n_pad = sources, p, node_budget, n_pad
        self.src_weight = list(src_weight)
        self.H, self.Hkv, self.D, self.kv_cap, self.vocab = H, Hkv, D, kv_cap, vocab
        ctx = torch.as_tensor(np.ascontiguousarray(ctx).view(np.int32)) if isinstance(ctx, np.ndarray) else ctx
        ctx_len = torch.as_tensor(np.asarray(ctx_len, np.int32)) if isinstance(ctx_len, np.ndarray) else ctx_len
        self.B = ctx.shape[0]
        B = self.B
        self.ctx = ctx.to(device=device, dtype=torch.int32).contiguous()
        self.ctx_len = [ctx_len.to(device=device, dtype=torch.int32).clone(), torch.empty(B, dtype=torch.int32, device=device)]
        kv0 = torch.as_tensor(np.broadcast_to(np.asarray(kv_len0, np.int32), (B,)).copy())
        self.kv_len = [kv0.to(device), torch.empty(B, dtype=torch.int32, device=device)]
        cl = self.ctx_len[0].long()
        self.root = self.ctx.gather(1, (cl - 1).clamp(min=0).view(B, 1)).view(B).contiguous()
        self.cur = 0
        self._init = (self.ctx.clone(), self.ctx_len[0].clone(), self.kv_len[0].clone(), self.root.clone())
        S = len(sources)
        self.seq = dict(seq_cache) if seq_cache else None
        n_slots = S + 1 if self.seq else S
        self.res = fc.retrieve_outputs(n_slots, B, p, device)
        self.skip = torch.zeros(B, dtype=torch.int32, device=device)
        self.tree = fc.tree_outputs(B, n_pad, device)
        self.argmax = torch.empty((B, n_pad), dtype=torch.int32, device=device)
        self.path_cap = p.draft_len + 2
        self.acc = dict(acc_len=torch.empty(B, dtype=torch.int32, device=device),
                        path=torch.empty((B, self.path_cap), dtype=torch.int32, device=device),
                        bonus=torch.empty(B, dtype=torch.int32, device=device))
        shape = (B, Hkv, kv_cap, D)
        self.k_cache = k_cache if k_cache is not None else torch.zeros(shape, dtype=torch.bfloat16, device=device)
        self.v_cache = v_cache if v_cache is not None else torch.zeros(shape, dtype=torch.bfloat16, device=device)
        self.attn_out = torch.empty((B, n_pad, H, D), dtype=torch.bfloat16, device=device)
        # optional: a stream of its own for the attention launch (the step's other
        # work waits for it through an event)
        self.attn_stream = None
        self._ev_pre, self._ev_post = torch.cuda.Event(), torch.cuda.Event()
        # the attention's own workspace (KV-split partials and counters): loops whose
        # steps overlap on different streams must not share one
        self.attn_ws = torch.empty(max(int(fc.LIB.fc_tree_attn_workspace(B, n_pad, H, Hkv)), 16), dtype=torch.uint8,
                                   device=device)
        self.rope_base = rope_base
        self.decoder = decoder
        self.k_tree_rot = (torch.empty((B, Hkv, n_pad, D), dtype=torch.bfloat16, device=device)
                           if rope_base is not None else None)
        self.cache = fc.RetrievalCache(cache_capacity, S, p, device) if cache_capacity and not self.seq else None
        if self.seq:
            q = self.seq
            self.seq_cache = fc.SequenceCache(B, q.get("capacity", 8192), q.get("min_size", 50), q.get("chunk", 20),
                                              q.get("ctx_keep", p.n_max), device)
            self.missing = fc.MissingTable(q.get("missing_capacity", 1 << 16), p.n_min, device)
            self.tree_weight = self.src_weight + [int(q.get("weight", 1))]
            self.seq_cache.init(self.ctx_len[0])
        else:
            self.tree_weight = self.src_weight

    def step(self, q, k_tree, v_tree, want_hit, plen, rtok, attention=True, events=None):
        """Enqueue one step.  q [B, Np, H, D], k_tree/v_tree [B, Hkv, Np, D]
        (bf16); want_hit [B], plen [B], rtok [B, Np] (int32).  ``events``
        optionally maps "retrieve" / "tree" / "attn" / "tail" (and, with the
        CACHE, "cache_search" / "cache_update") to (start, end) CUDA events
        recorded around those stages on the current stream."""
        c, n = self.cur, 1 - self.cur
        ev = events or {}
        if "retrieve" in ev:
            ev["retrieve"][0].record()
        S = len(self.sources)
        if self.seq:
            if "cache_search" in ev:
                ev["cache_search"][0].record()
            fc.fc_cache_search(self.seq_cache, self.missing, self.ctx, self.ctx_len[c], self.p, S, self.res, self.skip)
            if "cache_search" in ev:
                ev["cache_search"][1].record()
            fc.fc_retrieve(self.sources, self.ctx, self.ctx_len[c], self.p, skip=self.skip, out=self.res)
            fc.fc_missing_insert(self.missing, self.ctx, self.ctx_len[c], self.skip, self.res["n_drafts"], S)
        elif self.cache is not None:
            fc.fc_retrieve_cached(self.sources, self.cache, self.ctx, self.ctx_len[c], want_hit, self.skip, self.p,
                                  self.res)
            fc.fc_rcache_insert(self.cache, self.ctx, self.ctx_len[c], self.skip, self.res)
        else:
            fc.fc_retrieve(self.sources, self.ctx, self.ctx_len[c], self.p, out=self.res)
        if "retrieve" in ev:
            ev["retrieve"][1].record()
        if "tree" in ev:
            ev["tree"][0].record()
        fc.fc_build_tree(self.res, self.tree_weight, self.root, self.kv_len[c], self.node_budget, self.n_pad,
                         out=self.tree)
        if "tree" in ev:
            ev["tree"][1].record()
        if self.decoder is not None:
            self._verify_with_decoder(c, n, ev)
            self.cur = n
            return
        if self.rope_base is not None:
            k_tree = fc.fc_rope(k_tree, self.tree["pos"], self.rope_base, layout=1, out=self.k_tree_rot)
        if attention:
            side = self.attn_stream
            if side is not None:  # the attention on its own stream, ordered by events
                self._ev_pre.record()
                side.wait_event(self._ev_pre)
            with torch.cuda.stream(side) if side is not None else contextlib.nullcontext():
                if "attn" in ev:
                    ev["attn"][0].record()
                if self.rope_base is not None:
                    fc.fc_tree_attn_rope(q, self.k_cache, self.v_cache, self.kv_len[c], k_tree, v_tree,
                                         self.tree["mask"], self.tree["n_nodes"], self.tree["pos"], self.rope_base,
                                         out=self.attn_out, workspace=self.attn_ws)
                else:
                    fc.fc_tree_attn(q, self.k_cache, self.v_cache, self.kv_len[c], k_tree, v_tree, self.tree["mask"],
                                    self.tree["n_nodes"], out=self.attn_out, workspace=self.attn_ws)
                if "attn" in ev:
                    ev["attn"][1].record()
                if side is not None:
                    self._ev_post.record(side)
            if side is not None:
                torch.cuda.current_stream().wait_event(self._ev_post)
        if "tail" in ev:
            ev["tail"][0].record()
        fc.fc_synth_argmax(self.tree["tok"], self.tree["parent"], self.tree["n_nodes"], plen, rtok, self.vocab,
                           out=self.argmax)
        fc.fc_accept(self.tree["tok"], self.tree["parent"], self.tree["n_nodes"], self.argmax, self.path_cap,
                     out=self.acc)
        fc.fc_kv_append(self.acc, self.tree["tok"], k_tree, v_tree, self.k_cache, self.v_cache, self.kv_len[c],
                        self.kv_len[n], self.ctx, self.ctx_len[c], self.ctx_len[n], self.root)
        if self.seq:
            if "cache_update" in ev:
                ev["cache_update"][0].record()
            fc.fc_cache_update(self.seq_cache, self.ctx, self.ctx_len[c], self.ctx_len[n], self.acc["acc_len"])
            if "cache_update" in ev:
                ev["cache_update"][1].record()
        if "tail" in ev:
            ev["tail"][1].record()
        self.cur = n

    def _verify_with_decoder(self, c, n, ev):
        t = self.tree
        if "attn" in ev:
            ev["attn"][0].record()
        logits = self.decoder.forward(t["tok"], t["n_nodes"], t["mask"], t["pos"], self.kv_len[c])
        if "attn" in ev:
            ev["attn"][1].record()
        if "tail" in ev:
            ev["tail"][0].record()
        fc.fc_argmax_accept(logits, t["tok"], t["parent"], t["n_nodes"], self.path_cap,
                            out=dict(self.acc, argmax=self.argmax))
        self.decoder.append(self.acc, t["tok"], self.kv_len[c], self.kv_len[n], self.ctx, self.ctx_len[c],
                            self.ctx_len[n], self.root)
        if self.seq:
            fc.fc_cache_update(self.seq_cache, self.ctx, self.ctx_len[c], self.ctx_len[n], self.acc["acc_len"])
        if "tail" in ev:
            ev["tail"][1].record()

    def capture(self, inputs, attention=True):
        """Capture consecutive steps into a CUDA graph.  ``inputs`` holds an
        even number of tuples (q, k_tree, v_tree, want_hit, plen, rtok) of
        device tensors, one per step, that the graph reads at every replay
        (update them in place between replays).  Call with the loop at an even
        step, after one eager pair of steps so that lazily made workspaces and
        kernel attributes exist.  Each replay advances the loop by
        len(inputs) steps."""
        if self.cur != 0:
            raise RuntimeError("capture at an even step")
        if len(inputs) < 2 or len(inputs) % 2:
            raise ValueError("capture an even number of steps (the lengths alternate between two buffers)")
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, capture_error_mode="thread_local"):
            for ins in inputs:
                self.step(*ins, attention=attention)
        return g

    def reset(self):
        """Back to the initial contexts and cache lengths.  The replay cache
        keeps its entries (a replay of the same trajectory then hits it); the
        CACHE and the missing table start empty again, as for a new
        generation."""
        ctx0, cl0, kv0, root0 = self._init
        self.ctx.copy_(ctx0)
        self.ctx_len[0].copy_(cl0)
        self.kv_len[0].copy_(kv0)
        self.root.copy_(root0)
        self.cur = 0
        if self.seq:
            self.seq_cache.init(self.ctx_len[0])
            self.missing.clear()

    @property
    def kv_len_now(self):
        return self.kv_len[self.cur]

    @property
    def ctx_len_now(self):
        return self.ctx_len[self.cur]


def sub_batch_slices(B, n_split):
    """The sub-batches of a batch of B sequences: n_split contiguous slices, the
    h-th ending at floor(B (h + 1) / n_split), so their sizes differ by at most
    one."""
    if not 1 <= n_split <= B:
        raise ValueError("n_split must be between 1 and the batch size")
    edges = [B * h // n_split for h in range(n_split + 1)]
    return [slice(edges[h], edges[h + 1]) for h in range(n_split)]


class PipelinedStepLoop:
    """The step loop over sub-batches of the sequences, each on CUDA streams
    of its own, issued by the native step executor (fc_pipeline).

    The sequences of a batch are independent, so sub-batch h can run step
    s + 1 while sub-batch h' is still in step s. Then one sub-batch's small,
    latency-bound kernels (retrieval, tree build, acceptance, append) run on
    the SMs that the other's attention launch leaves idle in its last wave;
    an SM that holds an attention CTA has no room for any other CTA.  Each
    sub-batch owns the buffers of a StepLoop over a slice of the sequences.
    They share the datastores and slices of one pair of KV caches, and every
    per-sequence result is the single loop's.  The replay cache is per
    sub-batch; it replays deterministic retrieval results, so that changes no
    output.  One fc_pipeline_step call enqueues a step of every sub-batch:
    the host cost of a step no longer grows by a Python call per kernel.

    step() makes every sub-batch wait for the work already enqueued on the
    caller's stream, so inputs written there are visible.  It does not make
    the caller's stream wait for the sub-batches, or they could not overlap;
    join() does that, and must precede any read of the results on the
    caller's stream.

    With ``seq_cache`` (Algorithm 1, as StepLoop's) every sub-batch keeps a
    CACHE and a missing table M of its own.  The CACHE is per sequence in
    any case.  M only lets a query skip a datastore search that would find
    nothing (its keys are contexts whose search found no continuation in any
    source), so a per-sub-batch M changes no draft: each sub-batch is
    exactly the single loop over its slice of the sequences."""

    def __init__(self, n_split, sources, ctx, ctx_len, p, node_budget, n_pad, src_weight, H, Hkv, D, kv_cap,
                 kv_len0, vocab, cache_capacity=1 << 14, device="cuda", k_cache=None, v_cache=None, rope_base=None,
                 seq_cache=None):
        B = ctx.shape[0]
        self.slices = sub_batch_slices(B, n_split)
        self.B = B
        shape = (B, Hkv, kv_cap, D)
        self.k_cache = k_cache if k_cache is not None else torch.zeros(shape, dtype=torch.bfloat16, device=device)
        self.v_cache = v_cache if v_cache is not None else torch.zeros(shape, dtype=torch.bfloat16, device=device)
        kv0 = np.broadcast_to(np.asarray(kv_len0, np.int32), (B,))
        # the StepLoops hold each sub-batch's buffers and initial state
        self.loops = [StepLoop(sources, ctx[sl], ctx_len[sl], p, node_budget, n_pad, src_weight, H, Hkv, D, kv_cap,
                               kv0[sl], vocab, cache_capacity=cache_capacity, device=device,
                               k_cache=self.k_cache[sl], v_cache=self.v_cache[sl], rope_base=rope_base,
                               seq_cache=seq_cache)
                      for sl in self.slices]
        # every sub-batch records its device errors in a word of its own
        self.err_words = torch.zeros((len(self.slices), 1), dtype=torch.int32, device=device)
        parts = [fc.pipeline_part(sl.stop - sl.start, sl.start, lp.ctx, lp.ctx_len, lp.kv_len, lp.root, lp.cache,
                                  lp.skip, lp.res, lp.tree, lp.k_cache, lp.v_cache, lp.k_tree_rot, lp.attn_out,
                                  lp.attn_ws, lp.argmax, lp.acc, err=self.err_words[h],
                                  seq_cache=lp.seq_cache if lp.seq else None, missing=lp.missing if lp.seq else None)
                 for h, (lp, sl) in enumerate(zip(self.loops, self.slices))]
        lp0 = self.loops[0]
        self.pipe = fc.Pipeline(sources, p, lp0.tree_weight, node_budget, n_pad, H, Hkv, D, kv_cap, lp0.path_cap,
                                vocab, parts, rope_base=rope_base)
        self.streams = self.pipe.streams  # each sub-batch's chain stream (lookup .. append)

    def step(self, q, k_tree, v_tree, want_hit, plen, rtok, attention=True, events=None):
        """Enqueue one step of every sub-batch (arguments as StepLoop.step,
        for the whole batch); ``events``: None or one StepLoop events dict per
        sub-batch, recorded on its streams."""
        self.pipe.step(self.loops[0].cur, q, k_tree, v_tree, want_hit, plen, rtok, attention=attention,
                       events=events)
        for lp in self.loops:
            lp.cur = 1 - lp.cur

    def join(self):
        """The caller's current stream waits for everything enqueued so far."""
        self.pipe.join()

    def errors(self):
        """Each sub-batch's device errors since the last call (status names;
        waits for the sub-batches and clears their words).  The sub-batches'
        kernels report here, not through fc_get_error."""
        return [self.pipe.error(h) for h in range(len(self.loops))]

    def capture(self, inputs, attention=True):
        """An even number of steps of every sub-batch in one CUDA graph (fork
        and join inside it); as StepLoop.capture.  The sub-batches rejoin only
        at the end of the graph."""
        if any(lp.cur != 0 for lp in self.loops):
            raise RuntimeError("capture at an even step")
        if len(inputs) < 2 or len(inputs) % 2:
            raise ValueError("capture an even number of steps (the lengths alternate between two buffers)")
        self.join()  # no eager work may still be pending on the streams the graph forks to
        torch.cuda.current_stream().synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, capture_error_mode="thread_local"):
            for ins in inputs:
                self.step(*ins, attention=attention)
            self.join()
        return g

    def capture_parts(self, inputs, attention=True):
        """One CUDA graph per sub-batch, each holding an even number of steps
        of that sub-batch alone (inputs as capture).  Replay them on streams of
        their own: the sub-batches then never join, as in the eager loop.  A
        sub-batch reads only its slice of the inputs, so each may copy its
        slice of the next inputs on its own stream before its replay."""
        if any(lp.cur != 0 for lp in self.loops):
            raise RuntimeError("capture at an even step")
        if len(inputs) < 2 or len(inputs) % 2:
            raise ValueError("capture an even number of steps (the lengths alternate between two buffers)")
        self.join()
        torch.cuda.current_stream().synchronize()
        graphs = []
        for h in range(len(self.loops)):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, capture_error_mode="thread_local"):
                for t, ins in enumerate(inputs):
                    self.pipe.step(t & 1, *ins, attention=attention, part=h)
                self.pipe.join(part=h)
            graphs.append(g)
        return graphs

    def capture_native(self, inputs, attention=True):
        """As capture_parts, through the executor's own capture
        (fc_pipeline_capture_part): one graph per sub-batch whose kernels keep
        the priorities of the eager step's streams (the chain's above the
        attention's), which a graph captured through torch loses.  Returns one
        fc.PipelineGraph per sub-batch; launch each into a stream of its own
        (graph.launch() on the current stream)."""
        if any(lp.cur != 0 for lp in self.loops):
            raise RuntimeError("capture at an even step")
        if len(inputs) < 2 or len(inputs) % 2:
            raise ValueError("capture an even number of steps (the lengths alternate between two buffers)")
        return [self.pipe.capture(h, inputs, 0, attention) for h in range(len(self.loops))]

    def reset(self):
        self.join()
        for lp in self.loops:
            lp.reset()

    # gathered copies over the whole batch (they allocate; call after join())
    def _cat(self, get):
        return torch.cat([get(lp) for lp in self.loops])

    @property
    def kv_len_now(self):
        return self._cat(lambda lp: lp.kv_len_now)

    @property
    def ctx_len_now(self):
        return self._cat(lambda lp: lp.ctx_len_now)

    @property
    def ctx(self):
        return self._cat(lambda lp: lp.ctx)

    @property
    def acc(self):
        return {k: self._cat(lambda lp, k=k: lp.acc[k]) for k in self.loops[0].acc}

    @property
    def tree(self):
        return {k: self._cat(lambda lp, k=k: lp.tree[k]) for k in self.loops[0].tree}

    @property
    def skip(self):
        return self._cat(lambda lp: lp.skip)

    @property
    def attn_out(self):
        return self._cat(lambda lp: lp.attn_out)
