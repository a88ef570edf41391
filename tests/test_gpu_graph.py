"""CUDA-graph replay of the step loop: two consecutive steps captured once
and replayed with inputs updated in place give the same trajectory as eager
steps (integer outputs bit-exact, attention within the step's max-abs 2e-2),
for the replay-cache loop and for the loop with Algorithm 1's CACHE."""
import numpy as np
import pytest
import torch

import paper_2502_17139_gb300.synth as synth

pytestmark = pytest.mark.gpu


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


@pytest.mark.parametrize("seq_cache", [None, dict(capacity=2048, min_size=3, chunk=8, missing_capacity=1 << 10)],
                         ids=["replay_cache", "algorithm1"])
def test_graph_replay_matches_eager(fc, seq_cache):
    from paper_2502_17139_gb300.step import StepLoop
    rng = synth.rng_for(76)
    Tr, _ = synth.make_corpus(rng, 200_000, 1.3, synth.VOCAB, n_grams=500, len_range=(8, 64))
    Tc, _ = synth.make_corpus(rng, 1_000_000, 1.1, synth.VOCAB)
    B, steps, n_pad, H, Hkv, D, kv0 = 8, 12, 128, 8, 2, 128, 100
    stride = 128 + steps * 12
    ctx, cl, _ = synth.make_contexts(rng, B, 128, 16, [Tr, Tc, None], [0.5, 0.25, 0.25], 1.1, ctx_stride=stride)
    hits = synth.cache_hit_pattern(rng, steps, B)
    plen = np.stack([synth.argmax_draws(rng, B, n_pad)[0] for _ in range(steps)])
    rtok = np.stack([synth.argmax_draws(rng, B, n_pad)[1] for _ in range(steps)])
    srcs = [fc.fc_datastore_build(dev(Tr), synth.VOCAB), fc.fc_datastore_build(dev(Tc), synth.VOCAB)]
    qs = [synth.randn_bf16((B, n_pad, H, D), 10 + s, "cuda") for s in range(steps)]
    ks = [synth.randn_bf16((B, Hkv, n_pad, D), 40 + s, "cuda") for s in range(steps)]
    vs = [synth.randn_bf16((B, Hkv, n_pad, D), 70 + s, "cuda") for s in range(steps)]
    ins = [(qs[s], ks[s], vs[s], dev(hits[s]), dev(plen[s]), dev(rtok[s])) for s in range(steps)]

    def make():
        return StepLoop(srcs, ctx, cl, fc.params(16, 2, 64, 10, 4096), n_pad, n_pad, [1, 1], H, Hkv, D,
                        kv_cap=kv0 + steps * 12, kv_len0=kv0, vocab=synth.VOCAB, seq_cache=seq_cache)

    def state(loop):
        return dict(ctx=loop.ctx.cpu().clone(), cl=loop.ctx_len_now.cpu().clone(), kv=loop.kv_len_now.cpu().clone(),
                    acc=loop.acc["acc_len"].cpu().clone(), nn=loop.tree["n_nodes"].cpu().clone(),
                    kc=loop.k_cache.cpu().clone(), attn=loop.attn_out.float().cpu().clone())

    eager = make()
    want = []
    for s in range(steps):
        eager.step(*ins[s])
        if s % 2 == 1:
            want.append(state(eager))
    torch.cuda.synchronize()
    assert fc.fc_get_error() == "FC_OK"

    graphed = make()
    graphed.step(*ins[0])
    graphed.step(*ins[1])
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
        for name in ("ctx", "cl", "kv", "acc", "nn", "kc"):
            assert torch.equal(w[name], gt[name]), name
        assert (w["attn"] - gt["attn"]).abs().max().item() <= 2e-2
