"""The allocation-free datastore build, checked against the regular one.

Some callers cannot call cudaMalloc (a serving process whose memory manager
holds all free device memory for its KV cache, a plugin inside an application
that owns every device allocation).  fc_datastore_build_noalloc serves them with
scratch space compiled into the library.  This test calls it through the C ABI
twice in a row (the second corpus is smaller, so leftovers of the first call
stay in the shared scratch array) and compares each suffix array and bucket
table with fc_datastore_build's, which must agree exactly (integer outputs).
It lives in its own file so that pytest collects it after every other test.
"""
import ctypes as C

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
