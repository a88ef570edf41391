"""The FC_DEBUG build (libfastcoder_debug.so, loaded when FC_DEBUG=1): its
kernels bounds-check the indexes their gathers take from data.  On valid
inputs it gives the release build's results bit for bit; given a datastore
whose suffix array holds out-of-range entries, retrieval reports
FC_ERR_INTERNAL and skips those gathers instead of reading past the corpus.
Each case runs in a fresh process, since the binding picks the library at
import."""
import json
import os
import subprocess
import sys

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CASE = r"""
import json, sys
import numpy as np, torch
sys.path.insert(0, sys.argv[1])
import paper_2502_17139_gb300.fastcoder as fc
import paper_2502_17139_gb300.synth as synth
rng = synth.rng_for(97)
T, _ = synth.make_corpus(rng, 200_000, 1.2, 2000, n_grams=400, len_range=(8, 40))
ctx, cl, _ = synth.make_contexts(rng, 24, 48, 16, [T, None], [0.8, 0.2], 1.1, 2000)
dev = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int32)).cuda()
ds = fc.fc_datastore_build(dev(T), 2000)
p = fc.params(16, 2, 16, 8, 4096)
out = {"lib": fc._build.LIB_DEBUG if "debug" in sys.argv[2] else fc._build.LIB}
g = fc.fc_retrieve([ds], dev(ctx), dev(cl), p)
tree = fc.fc_build_tree(g, [1], dev(ctx[np.arange(24), cl - 1]), dev(np.full(24, 100, np.int32)), 64, 64)
out["status"] = fc.fc_get_error()
out["retrieve"] = {k: v.cpu().numpy().tolist() for k, v in g.items()}
out["tree"] = {k: v.cpu().numpy().tolist() for k, v in tree.items()}
if sys.argv[2] == "debug_bad_sa":
    ds.sa.fill_(-268435456)  # 0xF0000000: every suffix-array entry past the corpus end
    bad = fc.Datastore(ds.tokens, ds.sa, ds.bucket, ds.lcp, ds.vocab)
    fc.fc_retrieve([bad], dev(ctx), dev(cl), p)
    out["bad_status"] = fc.fc_get_error()
    fc.fc_retrieve([fc.fc_datastore_build(dev(T), 2000)], dev(ctx), dev(cl), p)
    out["after_status"] = fc.fc_get_error()
print(json.dumps(out))
"""


def run_case(kind):
    env = dict(os.environ, FC_DEBUG="1" if kind.startswith("debug") else "0")
    r = subprocess.run([sys.executable, "-c", CASE, ROOT, kind], capture_output=True, text=True, env=env, timeout=600)
    assert r.returncode == 0, r.stderr[-3000:]
    return json.loads(r.stdout.strip().splitlines()[-1])


@pytest.fixture(scope="module")
def built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2502_17139_gb300 import build
    build.build()
    build.build(debug=True)


def test_debug_build_matches_release(built):
    rel, dbg = run_case("release"), run_case("debug")
    assert rel["status"] == dbg["status"] == "FC_OK"
    assert rel["retrieve"] == dbg["retrieve"] and rel["tree"] == dbg["tree"]
    assert max(max(x) for x in dbg["retrieve"]["match_len"]) > 0


def test_debug_build_reports_bad_suffix_array(built):
    got = run_case("debug_bad_sa")
    assert got["status"] == "FC_OK"
    assert got["bad_status"] == "FC_ERR_INTERNAL"
    assert got["after_status"] == "FC_OK"  # the context keeps working
