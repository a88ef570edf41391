"""Datastore files on the GPU: a store built on the device, saved, loaded
into new device buffers and searched gives the same retrieval results bit
for bit; a file written from the oracle's host arrays loads onto the device
and retrieves like the store built there."""
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
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int32)).cuda()


def test_save_load_retrieve(fc, orc, tmp_path):
    rng = synth.rng_for(95)
    Tr, _ = synth.make_corpus(rng, 300_000, 1.3, synth.VOCAB, n_grams=1000, len_range=(8, 40))
    Tc, _ = synth.make_corpus(rng, 2_000_000, 1.1, synth.VOCAB)
    ctx, cl, _ = synth.make_contexts(rng, 64, 128, 16, [Tr, Tc, None], [0.5, 0.25, 0.25], 1.1)
    built = [fc.fc_datastore_build(dev(T), synth.VOCAB) for T in (Tr, Tc)]
    paths = [str(tmp_path / f"s{i}.fcds") for i in range(2)]
    for ds, path in zip(built, paths):
        fc.fc_datastore_save(ds, path)
    loaded = [fc.fc_datastore_load(path) for path in paths]
    for a, b in zip(built, loaded):
        for name in ("tokens", "sa", "bucket", "lcp"):
            assert torch.equal(getattr(a, name), getattr(b, name)), name
    p = fc.params(16, 2, 64, 10, 4096)
    g0 = fc.fc_retrieve(built, dev(ctx), dev(cl), p)
    g1 = fc.fc_retrieve(loaded, dev(ctx), dev(cl), p)
    torch.cuda.synchronize()
    for k in g0:
        assert torch.equal(g0[k], g1[k]), k
    # the oracle's arrays, written on the host, read onto the device
    sa = orc.suffix_array(Tr)
    hp = str(tmp_path / "oracle.fcds")
    fc.datastore_save_host(hp, Tr, sa, orc.bucket(Tr, sa, synth.VOCAB), orc.lcp(Tr, sa))
    from_oracle = fc.fc_datastore_load(hp)
    g2 = fc.fc_retrieve([from_oracle], dev(ctx), dev(cl), p)
    g3 = fc.fc_retrieve([built[0]], dev(ctx), dev(cl), p)
    torch.cuda.synchronize()
    for k in g2:
        assert torch.equal(g2[k], g3[k]), k
    assert fc.fc_get_error() == "FC_OK"
