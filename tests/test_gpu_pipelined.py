"""The step loop over sub-batches on separate streams (PipelinedStepLoop):
every per-sequence result equals the single loop's (contexts, lengths, trees,
acceptance and cache rows bit-exact, attention within max-abs 2e-2), for two
and three sub-batches of unequal size, and a CUDA graph of two pipelined steps
(fork and join inside the graph) replays the eager pipelined trajectory."""
import numpy as np
import pytest
import torch

import paper_2502_17139_gb300.synth as synth

pytestmark = pytest.mark.gpu
ATOL = 2e-2


@pytest.fixture(scope="module")
def fc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2502_17139_gb300 import build
    build.build()
    import paper_2502_17139_gb300.fastcoder as fcm
    return fcm


def dev(a):
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint32:
        a = a.view(np.int32)
    return torch.from_numpy(a.copy()).cuda()


@pytest.fixture(scope="module")
def setup(fc):
    rng = synth.rng_for(77)
    Tr, _ = synth.make_corpus(rng, 200_000, 1.3, synth.VOCAB, n_grams=500, len_range=(8, 64))
    Tc, _ = synth.make_corpus(rng, 1_000_000, 1.1, synth.VOCAB)
    B, steps, n_pad, H, Hkv, D, kv0 = 9, 10, 128, 8, 2, 128, 100
    stride = 128 + steps * 12
    ctx, cl, _ = synth.make_contexts(rng, B, 128, 16, [Tr, Tc, None], [0.5, 0.25, 0.25], 1.1, ctx_stride=stride)
    hits = synth.cache_hit_pattern(rng, steps, B)
    draws = [synth.argmax_draws(rng, B, n_pad) for _ in range(steps)]
    srcs = [fc.fc_datastore_build(dev(Tr), synth.VOCAB), fc.fc_datastore_build(dev(Tc), synth.VOCAB)]
    ins = [(synth.randn_bf16((B, n_pad, H, D), 10 + s, "cuda"), synth.randn_bf16((B, Hkv, n_pad, D), 40 + s, "cuda"),
            synth.randn_bf16((B, Hkv, n_pad, D), 70 + s, "cuda"), dev(hits[s]), dev(draws[s][0]), dev(draws[s][1]))
           for s in range(steps)]
    args = (srcs, ctx, cl, fc.params(16, 2, 64, 10, 4096), n_pad, n_pad, [1, 1], H, Hkv, D)
    kw = dict(kv_cap=kv0 + steps * 12, kv_len0=kv0, vocab=synth.VOCAB)
    return dict(args=args, kw=kw, ins=ins, steps=steps)


def state(loop):
    s = dict(ctx=loop.ctx, cl=loop.ctx_len_now, kv=loop.kv_len_now, kc=loop.k_cache, vc=loop.v_cache)
    s.update({"acc_" + k: v for k, v in loop.acc.items()})
    s.update({"tree_" + k: v for k, v in loop.tree.items()})
    out = {k: v.cpu().clone() for k, v in s.items()}
    out["attn"] = loop.attn_out.float().cpu().clone()
    return out


def same(a, b):
    for k in a:
        if k == "attn":
            assert (a[k] - b[k]).abs().max().item() <= ATOL, k
        else:
            assert torch.equal(a[k], b[k]), k


@pytest.mark.parametrize("n_split", [2, 3])
def test_pipelined_matches_single_loop(fc, setup, n_split):
    from paper_2502_17139_gb300.step import PipelinedStepLoop, StepLoop
    single = StepLoop(*setup["args"], **setup["kw"])
    piped = PipelinedStepLoop(n_split, *setup["args"], **setup["kw"])
    assert [sl.stop - sl.start for sl in piped.slices] == ([4, 5] if n_split == 2 else [3, 3, 3])
    for s in range(setup["steps"]):
        single.step(*setup["ins"][s])
        piped.step(*setup["ins"][s])
        piped.join()
        same(state(single), state(piped))
    assert fc.fc_get_error() == "FC_OK" and piped.errors() == ["FC_OK"] * n_split
    # reset replays the same trajectory
    piped.reset()
    for s in range(2):
        piped.step(*setup["ins"][s])
    piped.join()
    single.reset()
    for s in range(2):
        single.step(*setup["ins"][s])
    same(state(single), state(piped))


def test_pipelined_graph_replay(fc, setup):
    from paper_2502_17139_gb300.step import PipelinedStepLoop
    ins, steps = setup["ins"], setup["steps"]
    eager = PipelinedStepLoop(2, *setup["args"], **setup["kw"])
    want = []
    for s in range(steps):
        eager.step(*ins[s])
        if s % 2 == 1:
            eager.join()
            want.append(state(eager))
    graphed = PipelinedStepLoop(2, *setup["args"], **setup["kw"])
    graphed.step(*ins[0])
    graphed.step(*ins[1])
    graphed.join()
    static = [tuple(t.clone() for t in ins[2]), tuple(t.clone() for t in ins[3])]
    g = graphed.capture(static)
    got = []
    for s in range(2, steps, 2):
        for j in range(2):
            for dst, src in zip(static[j], ins[s + j]):
                dst.copy_(src)
        g.replay()
        got.append(state(graphed))
    torch.cuda.synchronize()
    assert fc.fc_get_error() == "FC_OK"
    for w, gt in zip(want[1:], got):
        same(w, gt)


def test_pipelined_one_sequence_per_sub_batch(fc, setup):
    """As many sub-batches as sequences (nine streams of one sequence each), and
    the bounds of n_split."""
    from paper_2502_17139_gb300.step import PipelinedStepLoop, StepLoop
    B = setup["args"][1].shape[0]
    with pytest.raises(ValueError):
        PipelinedStepLoop(0, *setup["args"], **setup["kw"])
    with pytest.raises(ValueError):
        PipelinedStepLoop(B + 1, *setup["args"], **setup["kw"])
    single = StepLoop(*setup["args"], **setup["kw"])
    piped = PipelinedStepLoop(B, *setup["args"], **setup["kw"])
    for s in range(4):
        single.step(*setup["ins"][s])
        piped.step(*setup["ins"][s])
    piped.join()
    same(state(single), state(piped))
    assert fc.fc_get_error() == "FC_OK"


def test_pipelined_kv_split_workspaces(fc):
    """Two sub-batches whose attention launches both split their last wave's
    KV blocks over several CTAs (10 sequences x 8 kv heads x 2 row chunks =
    160 units on 152 SMs) while they overlap: each sub-batch has its own
    workspace, so the results equal the single loop's."""
    from paper_2502_17139_gb300.step import PipelinedStepLoop, StepLoop
    rng = synth.rng_for(78)
    Tr, _ = synth.make_corpus(rng, 200_000, 1.3, synth.VOCAB, n_grams=500, len_range=(8, 64))
    Tc, _ = synth.make_corpus(rng, 1_000_000, 1.1, synth.VOCAB)
    B, steps, n_pad, H, Hkv, D, kv0 = 20, 4, 128, 32, 8, 128, 4000
    ctx, cl, _ = synth.make_contexts(rng, B, 128, 16, [Tr, Tc, None], [0.5, 0.25, 0.25], 1.1, ctx_stride=128 + 60)
    hits = synth.cache_hit_pattern(rng, steps, B)
    draws = [synth.argmax_draws(rng, B, n_pad) for _ in range(steps)]
    srcs = [fc.fc_datastore_build(dev(Tr), synth.VOCAB), fc.fc_datastore_build(dev(Tc), synth.VOCAB)]
    ins = [(synth.randn_bf16((B, n_pad, H, D), 110 + s, "cuda"), synth.randn_bf16((B, Hkv, n_pad, D), 140 + s, "cuda"),
            synth.randn_bf16((B, Hkv, n_pad, D), 170 + s, "cuda"), dev(hits[s]), dev(draws[s][0]), dev(draws[s][1]))
           for s in range(steps)]
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    cap = kv0 + steps * 12
    assert fc.LIB.fc_tree_attn_parts(B // 2, n_pad, H, Hkv, cap, int(fc.LIB.fc_tree_attn_workspace(B // 2, n_pad, H, Hkv))) > 1 \
        or (B // 2) * Hkv * 2 <= sms  # the split is active on a 152-SM part
    args = (srcs, ctx, cl, fc.params(16, 2, 64, 10, 4096), n_pad, n_pad, [1, 1], H, Hkv, D)
    kw = dict(kv_cap=cap, kv_len0=kv0, vocab=synth.VOCAB)
    kc0 = synth.randn_bf16((B, Hkv, cap, D), 200, "cuda")
    vc0 = synth.randn_bf16((B, Hkv, cap, D), 201, "cuda")
    single = StepLoop(*args, **kw, k_cache=kc0.clone(), v_cache=vc0.clone())
    piped = PipelinedStepLoop(2, *args, **kw, k_cache=kc0.clone(), v_cache=vc0.clone())
    for s in range(steps):
        single.step(*ins[s])
        piped.step(*ins[s])
        piped.join()
        same(state(single), state(piped))
    assert fc.fc_get_error() == "FC_OK"


def test_pipelined_rope_matches_single_loop(fc, setup):
    """The executor's RoPE path (tree keys rotated by fc_rope, queries inside
    the attention kernel) against the single loop's."""
    from paper_2502_17139_gb300.step import PipelinedStepLoop, StepLoop
    single = StepLoop(*setup["args"], **setup["kw"], rope_base=10000.0)
    piped = PipelinedStepLoop(2, *setup["args"], **setup["kw"], rope_base=10000.0)
    for s in range(4):
        single.step(*setup["ins"][s])
        piped.step(*setup["ins"][s])
        piped.join()
        same(state(single), state(piped))
    assert fc.fc_get_error() == "FC_OK"


def test_pipelined_without_attention(fc, setup):
    """A step without the attention launch follows the same trajectory (the
    synthetic predictions do not read the attention output) and leaves the
    output untouched."""
    from paper_2502_17139_gb300.step import PipelinedStepLoop
    full = PipelinedStepLoop(3, *setup["args"], **setup["kw"])
    bare = PipelinedStepLoop(3, *setup["args"], **setup["kw"])
    for lp in bare.loops:
        lp.attn_out.fill_(float("nan"))
    for s in range(4):
        full.step(*setup["ins"][s])
        q, kt, vt, h, p, r = setup["ins"][s]
        bare.step(None, kt, vt, h, p, r, attention=False)
    full.join()
    bare.join()
    a, b = state(full), state(bare)
    assert torch.isnan(b.pop("attn")).all()
    a.pop("attn")
    same(a, b)


def test_pipelined_stage_events_and_streams(fc, setup):
    """Stage events land in order on each sub-batch's streams, and work the
    caller enqueues on a sub-batch's exposed stream follows its step."""
    from paper_2502_17139_gb300.step import PipelinedStepLoop
    piped = PipelinedStepLoop(2, *setup["args"], **setup["kw"])
    mk = lambda: (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
    evs = [dict(retrieve=mk(), tree=mk(), attn=mk(), tail=mk()) for _ in piped.loops]
    piped.step(*setup["ins"][0], events=evs)
    outs = []
    for lp, st in zip(piped.loops, piped.streams):
        with torch.cuda.stream(st):
            outs.append(lp.acc["acc_len"].clone())
    piped.join()
    torch.cuda.synchronize()
    for e in evs:
        t = {k: a.elapsed_time(b) for k, (a, b) in e.items()}
        assert all(v >= 0 for v in t.values()), t
        assert e["retrieve"][1].elapsed_time(e["tree"][0]) >= 0
        assert e["tree"][1].elapsed_time(e["attn"][0]) >= 0
        assert e["attn"][1].elapsed_time(e["tail"][0]) >= 0
    for lp, o in zip(piped.loops, outs):
        assert torch.equal(o, lp.acc["acc_len"])


def test_pipelined_errors_attributed_to_their_sub_batch(fc, setup):
    """A context token outside the vocabulary in one sequence of sub-batch 1:
    its retrieval records FC_ERR_INVALID_ARG in sub-batch 1's own error word;
    sub-batch 0's word and the library-wide words stay clean, and the word
    reads clean again after it was taken."""
    from paper_2502_17139_gb300.step import PipelinedStepLoop
    srcs, ctx, cl = setup["args"][:3]
    bad = np.array(ctx, copy=True)
    b = 6  # in the second sub-batch (sequences 4..8)
    bad[b, int(cl[b]) - 3] = synth.VOCAB + 5
    piped = PipelinedStepLoop(2, srcs, bad, cl, *setup["args"][3:], **setup["kw"])
    piped.step(*setup["ins"][0])
    piped.join()
    assert piped.errors() == ["FC_OK", "FC_ERR_INVALID_ARG"]
    assert fc.fc_get_error() == "FC_OK"
    assert piped.errors() == ["FC_OK", "FC_OK"]


def test_pipelined_part_graphs(fc, setup):
    """One CUDA graph per sub-batch (fc_pipeline_step_part), each replayed on a
    stream of its own, follows the eager pipelined trajectory."""
    from paper_2502_17139_gb300.step import PipelinedStepLoop
    ins, steps = setup["ins"], setup["steps"]
    eager = PipelinedStepLoop(3, *setup["args"], **setup["kw"])
    want = []
    for s in range(steps):
        eager.step(*ins[s])
        if s % 2 == 1:
            eager.join()
            want.append(state(eager))
    graphed = PipelinedStepLoop(3, *setup["args"], **setup["kw"])
    graphed.step(*ins[0])
    graphed.step(*ins[1])
    graphed.join()
    static = [tuple(t.clone() for t in ins[2]), tuple(t.clone() for t in ins[3])]
    graphs = graphed.capture_parts(static)
    assert len(graphs) == 3
    streams = [torch.cuda.Stream() for _ in graphs]
    got = []
    main = torch.cuda.current_stream()
    for s in range(2, steps, 2):
        for j in range(2):
            for dst, src in zip(static[j], ins[s + j]):
                dst.copy_(src)
        ready = torch.cuda.Event()
        ready.record(main)
        for g, st in zip(graphs, streams):
            st.wait_event(ready)
            with torch.cuda.stream(st):
                g.replay()
        for st in streams:
            main.wait_stream(st)
        got.append(state(graphed))
    torch.cuda.synchronize()
    assert fc.fc_get_error() == "FC_OK" and graphed.errors() == ["FC_OK"] * 3
    for w, gt in zip(want[1:], got):
        same(w, gt)


SEQ = dict(capacity=2048, min_size=3, chunk=8, ctx_keep=16, missing_capacity=1 << 10, weight=2)


def seq_state(lp):
    """A StepLoop's CACHE words and meta, missing table and search states."""
    return dict(words=lp.seq_cache.words.cpu().clone(), meta=lp.seq_cache.meta.cpu().clone(),
                missing=lp.missing.table.cpu().clone(), skip=lp.skip.cpu().clone())


def test_pipelined_algorithm1_matches_slice_loops(fc, setup):
    """Algorithm 1 through the executor (CACHE search -> retrieval -> missing
    insert ... append -> CACHE update per sub-batch), against a StepLoop over
    each sub-batch's slice of the sequences: every result bit-exact, the
    attention within 2e-2, and the CACHE stores, missing tables and search
    states byte for byte; against the single loop over the whole batch (one
    missing table): the same trees, acceptance, contexts and CACHE stores.
    The CACHE slot's tree weight is 2, so a wrong slot weight shows in the
    trees."""
    from paper_2502_17139_gb300.step import PipelinedStepLoop, StepLoop
    srcs, ctx, cl = setup["args"][:3]
    rest, kw, ins = setup["args"][3:], setup["kw"], setup["ins"]
    piped = PipelinedStepLoop(2, *setup["args"], **kw, seq_cache=SEQ)
    slices = piped.slices
    per = [StepLoop(srcs, ctx[sl], cl[sl], *rest, **kw, seq_cache=SEQ) for sl in slices]
    whole = StepLoop(*setup["args"], **kw, seq_cache=SEQ)
    codes = []
    for s in range(setup["steps"]):
        piped.step(*ins[s])
        for lp, sl in zip(per, slices):
            lp.step(*[t[sl] for t in ins[s]])
        whole.step(*ins[s])
        piped.join()
        torch.cuda.synchronize()
        for h, (lp, sl) in enumerate(zip(per, slices)):
            a, b = state(lp), state(piped.loops[h])
            same(a, b)
            sa, sb = seq_state(lp), seq_state(piped.loops[h])
            for k in sa:
                assert torch.equal(sa[k], sb[k]), (s, h, k)
        a, b = state(whole), state(piped)
        same(a, b)
        assert torch.equal(whole.seq_cache.words.cpu(), torch.cat([lp.seq_cache.words for lp in piped.loops]).cpu())
        assert torch.equal(whole.seq_cache.meta.cpu(), torch.cat([lp.seq_cache.meta for lp in piped.loops]).cpu())
        codes.append(piped.skip.cpu().numpy())
    codes = np.stack(codes)
    assert (codes == 1).any() and (codes == 0).any()  # the CACHE served some queries, the datastores others
    assert sum(int(lp.missing.table[0].item()) for lp in piped.loops) > 0  # M took keys
    assert fc.fc_get_error() == "FC_OK" and piped.errors() == ["FC_OK", "FC_OK"]
    # reset empties the CACHE and M and replays the same trajectory
    piped.reset()
    for lp in per:
        lp.reset()
    for s in range(2):
        piped.step(*ins[s])
        for lp, sl in zip(per, slices):
            lp.step(*[t[sl] for t in ins[s]])
    piped.join()
    for h, lp in enumerate(per):
        same(state(lp), state(piped.loops[h]))
        sa, sb = seq_state(lp), seq_state(piped.loops[h])
        for k in sa:
            assert torch.equal(sa[k], sb[k]), (h, k)


@pytest.mark.parametrize("algorithm1", [False, True], ids=["replay_cache", "algorithm1"])
def test_pipelined_native_graphs(fc, setup, algorithm1):
    """The executor's own capture (fc_pipeline_capture_part): one graph of two
    steps per sub-batch, launched into a stream of its own, follows the eager
    pipelined trajectory (with the replay cache, and with Algorithm 1's CACHE
    and missing table), and its kernel nodes carry the eager streams'
    priorities: per step one attention node and the chain's six (eight with
    the CACHE) above it."""
    from paper_2502_17139_gb300.step import PipelinedStepLoop
    ins, steps = setup["ins"], setup["steps"]
    kw = dict(setup["kw"], seq_cache=SEQ) if algorithm1 else setup["kw"]
    eager = PipelinedStepLoop(3, *setup["args"], **kw)
    want = []
    for s in range(steps):
        eager.step(*ins[s])
        if s % 2 == 1:
            eager.join()
            want.append(state(eager))
    graphed = PipelinedStepLoop(3, *setup["args"], **kw)
    graphed.step(*ins[0])
    graphed.step(*ins[1])
    graphed.join()
    static = [tuple(t.clone() for t in ins[2]), tuple(t.clone() for t in ins[3])]
    graphs = graphed.capture_native(static)
    assert len(graphs) == 3
    for g in graphs:
        assert g.kernels() == ((8 if algorithm1 else 6) * 2, 2)
    streams = [torch.cuda.Stream() for _ in graphs]
    got = []
    main = torch.cuda.current_stream()
    for s in range(2, steps, 2):
        for j in range(2):
            for dst, src in zip(static[j], ins[s + j]):
                dst.copy_(src)
        ready = torch.cuda.Event()
        ready.record(main)
        for g, st in zip(graphs, streams):
            st.wait_event(ready)
            with torch.cuda.stream(st):
                g.launch()
        for st in streams:
            main.wait_stream(st)
        got.append(state(graphed))
    torch.cuda.synchronize()
    assert fc.fc_get_error() == "FC_OK" and graphed.errors() == ["FC_OK"] * 3
    for w, gt in zip(want[1:], got):
        same(w, gt)
    for g in graphs:
        g.close()


def test_pipelined_native_graphs_rope_and_no_attention(fc, setup):
    """The executor's own graphs with RoPE (the tree keys rotated by fc_rope on
    the chain: seven chain nodes a step, the attention rotating the queries)
    follow the eager pipelined trajectory; graphs captured without the
    attention launch hold only the chain's six nodes a step and follow the
    eager trajectory without attention."""
    from paper_2502_17139_gb300.step import PipelinedStepLoop
    ins, steps = setup["ins"], 6
    for rope, attention in ((10000.0, True), (None, False)):
        kw = dict(setup["kw"], rope_base=rope)
        eager = PipelinedStepLoop(2, *setup["args"], **kw)
        want = []
        for s in range(steps):
            eager.step(*ins[s], attention=attention)
            if s % 2 == 1:
                eager.join()
                want.append(state(eager))
        graphed = PipelinedStepLoop(2, *setup["args"], **kw)
        graphed.step(*ins[0], attention=attention)
        graphed.step(*ins[1], attention=attention)
        graphed.join()
        windows = {s: graphed.capture_native([ins[s], ins[s + 1]], attention=attention) for s in range(2, steps, 2)}
        for gs in windows.values():
            for g in gs:
                assert g.kernels() == ((7 if rope else 6) * 2, 2 if attention else 0)
        streams = [torch.cuda.Stream() for _ in graphed.loops]
        main = torch.cuda.current_stream()
        got = []
        for s in range(2, steps, 2):
            ready = torch.cuda.Event()
            ready.record(main)
            for g, st in zip(windows[s], streams):
                st.wait_event(ready)
                with torch.cuda.stream(st):
                    g.launch()
            for st in streams:
                main.wait_stream(st)
            got.append(state(graphed))
        torch.cuda.synchronize()
        assert fc.fc_get_error() == "FC_OK" and graphed.errors() == ["FC_OK"] * 2
        for w, gt in zip(want[1:], got):
            if not attention:
                w.pop("attn")
                gt.pop("attn")
            same(w, gt)
