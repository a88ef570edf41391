"""The allocation-free datastore build, checked against the regular one.

Some callers cannot call cudaMalloc (a serving process whose memory manager
holds all free device memory for its KV cache, a plugin inside an application
that owns every device allocation).  fc_datastore_build_noalloc serves them with
scratch space compiled into the library.  This test calls it through the C ABI
twice in a row (the second corpus is smaller, so leftovers of the first call
stay in the shared scratch array) and compares each suffix array and bucket
table with fc_datastore_build's, which must agree exactly (integer outputs).
It also checks the property the entry point exists for: once a first call
has placed the library's scratch array on the device, a call changes the
device's free memory by nothing.  A fresh process measures what that first
call places.  The file is named so that pytest collects it after every other
test.
"""
import ctypes as C
import json
import os
import subprocess
import sys

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def fc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2502_17139_gb300 import build
    build.build()
    import paper_2502_17139_gb300.fastcoder as fcm
    return fcm


def _corpus(seed, n, vocab):
    rng = np.random.default_rng(seed)
    T = rng.integers(0, vocab, n).astype(np.int32)
    T[n // 2:n // 2 + 200] = T[:200]  # a long repeat: several doubling rounds
    return torch.from_numpy(T).cuda()


def _noalloc_call(fc, tokens, vocab):
    """Through the C ABI: only the caller's output buffers exist."""
    n = tokens.numel()
    sa = torch.full((n,), -5, dtype=torch.int32, device="cuda")
    bucket = torch.full((vocab + 1,), -5, dtype=torch.int32, device="cuda")
    lcp = torch.full((n,), 7, dtype=torch.uint8, device="cuda")
    view = fc.fc_datastore()
    rc = fc.LIB.fc_datastore_build_noalloc(C.c_void_p(tokens.data_ptr()), n, vocab, C.c_void_p(sa.data_ptr()),
                                           C.c_void_p(bucket.data_ptr()), C.c_void_p(lcp.data_ptr()),
                                           C.c_void_p(torch.cuda.current_stream().cuda_stream), C.byref(view))
    assert rc == 0, fc.STATUS.get(rc, rc)
    assert view.n_tokens == n and view.vocab == vocab and view.sa == sa.data_ptr() and view.lcp == lcp.data_ptr()
    return sa, bucket, lcp


def test_noalloc_build_matches_regular_build(fc):
    for seed, n, vocab in ((1, 1 << 20, 32256), (2, 300_001, 7)):
        tokens = _corpus(seed, n, vocab)
        sa, bucket, lcp = _noalloc_call(fc, tokens, vocab)
        ref = fc.fc_datastore_build(tokens, vocab)
        torch.cuda.synchronize()
        assert torch.equal(sa, ref.sa), (seed, n)
        assert torch.equal(bucket, ref.bucket), (seed, n)
        assert torch.equal(lcp, ref.lcp), (seed, n)
    assert fc.fc_get_error() == "FC_OK"


def test_noalloc_rejects_oversized_corpus(fc):
    n = fc.NOALLOC_MAX_TOKENS + 1
    tokens = torch.zeros(n, dtype=torch.int32, device="cuda")
    rc = fc.LIB.fc_datastore_build_noalloc(C.c_void_p(tokens.data_ptr()), n, 4, C.c_void_p(tokens.data_ptr()),
                                           C.c_void_p(tokens.data_ptr()), C.c_void_p(tokens.data_ptr()), None, None)
    assert fc.STATUS[rc] == "FC_ERR_CAPACITY"


def test_noalloc_call_allocates_nothing(fc):
    tokens = _corpus(3, 200_000, 1000)
    _noalloc_call(fc, tokens, 1000)  # the first call on this device places the scratch array
    torch.cuda.synchronize()
    sa = torch.empty(tokens.numel(), dtype=torch.int32, device="cuda")
    bucket = torch.empty(1001, dtype=torch.int32, device="cuda")
    lcp = torch.empty(tokens.numel(), dtype=torch.uint8, device="cuda")
    torch.cuda.synchronize()
    for _ in range(2):
        free0 = torch.cuda.mem_get_info()[0]
        rc = fc.LIB.fc_datastore_build_noalloc(C.c_void_p(tokens.data_ptr()), tokens.numel(), 1000,
                                               C.c_void_p(sa.data_ptr()), C.c_void_p(bucket.data_ptr()),
                                               C.c_void_p(lcp.data_ptr()),
                                               C.c_void_p(torch.cuda.current_stream().cuda_stream), None)
        torch.cuda.synchronize()
        assert rc == 0
        assert torch.cuda.mem_get_info()[0] == free0


_FIRST_CALL = r"""
import ctypes as C, json, sys
import torch
sys.path.insert(0, sys.argv[1])
import paper_2502_17139_gb300.fastcoder as fc
n = 100_000
tokens = torch.randint(0, 50, (n,), dtype=torch.int32, device="cuda")
sa = torch.empty(n, dtype=torch.int32, device="cuda")
bucket = torch.empty(51, dtype=torch.int32, device="cuda")
lcp = torch.empty(n, dtype=torch.uint8, device="cuda")
torch.cuda.synchronize()
free = [torch.cuda.mem_get_info()[0]]
for _ in range(2):
    rc = fc.LIB.fc_datastore_build_noalloc(C.c_void_p(tokens.data_ptr()), n, 50, C.c_void_p(sa.data_ptr()),
                                           C.c_void_p(bucket.data_ptr()), C.c_void_p(lcp.data_ptr()), None, None)
    torch.cuda.synchronize()
    assert rc == 0, rc
    free.append(torch.cuda.mem_get_info()[0])
print(json.dumps({"first_call_bytes": free[0] - free[1], "second_call_bytes": free[1] - free[2]}))
"""


def test_noalloc_first_call_in_fresh_process(fc):
    """In a fresh process the first call loads the library's datastore-build
    module on the device, which places the 30 MiB scratch array (and the
    module's code); the second call places nothing."""
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    r = subprocess.run([sys.executable, "-c", _FIRST_CALL, root], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    got = json.loads(r.stdout.strip().splitlines()[-1])
    print("fc_datastore_build_noalloc in a fresh process:", got)
    assert got["second_call_bytes"] == 0
    assert 30 << 20 <= got["first_call_bytes"] <= 64 << 20, got
