"""The C-ABI library builds, loads and exports every entry point that
include/fastcoder.h declares; host-side argument validation rejects bad calls
before anything reaches a GPU (these calls launch nothing)."""
import ctypes as C
import os
import re
import subprocess

import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "fastcoder.h")


def declared():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(fc_[a-z0-9_]+)\s*\(", src)))


@pytest.fixture(scope="module")
def lib():
    from paper_2502_17139_gb300 import build
    path = build.build()
    return path


def test_exports_match_header(lib):
    names = declared()
    assert "fc_tree_attn" in names and "fc_retrieve" in names and len(names) >= 15
    out = subprocess.run(["nm", "-D", "--defined-only", lib], capture_output=True, text=True, check=True).stdout
    exported = set(re.findall(r"\bT (fc_[a-z0-9_]+)", out))
    missing = [n for n in names if n not in exported]
    assert not missing, missing


def test_binding_names_match_header(lib):
    import paper_2502_17139_gb300.fastcoder as fc
    for n in declared():
        assert hasattr(fc.LIB, n)
    assert fc.version() == "0.1.0"
    assert fc.LIB.fc_status_string(5) == b"FC_ERR_TIMEOUT"


def test_host_validation_without_gpu(lib):
    import paper_2502_17139_gb300.fastcoder as fc
    L = fc.LIB
    p = fc.params(16, 2, 16, 8)
    nul = None
    # no sources
    assert L.fc_retrieve(nul, 0, nul, 64, nul, 4, nul, p, nul, nul, nul, nul, nul, nul) == 1
    # parameters beyond what the kernels support
    views = (fc.fc_datastore * 1)(fc.fc_datastore(1, 1, 1, 1, 10, 5))
    assert L.fc_retrieve(views, 1, 1, 64, 1, 4, nul, fc.params(40, 2, 16, 8), 1, 1, 1, 1, 1, nul) == 2
    assert L.fc_retrieve(views, 1, 1, 64, 1, 4, nul, fc.params(16, 2, 16, 8, 0), 1, 1, 1, 1, 1, nul) == 2
    # empty batch is a no-op
    assert L.fc_retrieve(views, 1, nul, 64, nul, 0, nul, p, nul, nul, nul, nul, nul, nul) == 0
    # cached retrieval: no table, a capacity that is not a power of two, no skip output
    assert L.fc_retrieve_cached(views, 1, 16, 64, 16, 4, nul, 64, nul, 16, p, 16, 16, 16, 16, 16, nul) == 1
    assert L.fc_retrieve_cached(views, 1, 16, 64, 16, 4, 16, 60, nul, 16, p, 16, 16, 16, 16, 16, nul) == 1
    assert L.fc_retrieve_cached(views, 1, 16, 64, 16, 4, 16, 64, nul, nul, p, 16, 16, 16, 16, 16, nul) == 1
    # attention: head dim / tree padding / GQA ratio outside the supported set
    args = [1, 1, 1, 128, 1, 1, 1, 8, 1, 2]
    assert L.fc_tree_attn(*args, 64, 32, 8, 64, C.c_float(0.1), 1, nul, 0, nul) == 2
    assert L.fc_tree_attn(*args, 96, 32, 8, 128, C.c_float(0.1), 1, nul, 0, nul) == 2
    assert L.fc_tree_attn(*args, 64, 30, 8, 128, C.c_float(0.1), 1, nul, 0, nul) == 2
    assert L.fc_tree_attn(*args, 64, 32, 8, 128, C.c_float(-1.0), 1, nul, 0, nul) == 1
    # misaligned pointers (an operand, or the workspace)
    assert L.fc_tree_attn(3, 16, 16, 128, 16, 16, 16, 8, 16, 2, 64, 32, 8, 128, C.c_float(0.1), 16, nul, 0, nul) == 1
    assert L.fc_tree_attn(16, 16, 16, 128, 16, 16, 16, 8, 16, 2, 64, 32, 8, 128, C.c_float(0.1), 16, 8, 1 << 20,
                          nul) == 1
    # workspace query: positive, never shrinking with the batch (it is capped at
    # one wave of split units), 0 for an unsupported shape; no device, no split
    w1, w2 = L.fc_tree_attn_workspace(1, 128, 32, 8), L.fc_tree_attn_workspace(2, 128, 32, 8)
    assert 0 < w1 <= w2 and L.fc_tree_attn_workspace(1, 100, 32, 8) == 0
    if not torch.cuda.is_available():
        assert L.fc_tree_attn_parts(64, 128, 32, 8, 16384, 1 << 40) == 1
    # tree: budget larger than the padding, too many drafts
    w = (C.c_uint32 * 2)(1, 1)
    tree_ptrs = [1] * 6
    assert L.fc_build_tree(2, 1, 1, 1, 1, w, 64, 10, 1, 1, 4, 65, 64, *tree_ptrs, nul) == 1
    assert L.fc_build_tree(2, 1, 1, 1, 1, w, 300, 10, 1, 1, 4, 64, 64, *tree_ptrs, nul) == 2
    # datastore: empty corpus, short workspace
    assert L.fc_datastore_build(1, 0, 10, 1, 1, 1, 1, 1 << 20, nul, nul) == 1
    need = L.fc_datastore_build_workspace(1000, 10)
    assert need > 1000 * 28
    assert L.fc_datastore_build(1, 1000, 10, 1, 1, 1, 256, need - 1, nul, nul) == 3
    # kv append: aliasing in/out lengths
    assert L.fc_kv_append(1, 1, 1, 1, 16, 16, 2, 64, 8, 128, 12, 16, 16, 100, 8, 8, 1, 64, 4, 12, 1, nul) == 1
    # argmax + accept: an empty vocabulary, an odd logits address
    assert L.fc_argmax_accept(16, 0, 16, 16, 16, 2, 64, 16, 16, 16, 12, 16, nul) == 1
    assert L.fc_argmax_accept(17, 100, 16, 16, 16, 2, 64, 16, 16, 16, 12, 16, nul) == 1
    # cache: capacity must be a power of two
    assert L.fc_rcache_init(1, 1 << 30, 1000, 2, p, nul) == 1


def test_cache_host_validation_without_gpu(lib):
    import paper_2502_17139_gb300.fastcoder as fc
    L = fc.LIB
    p = fc.params(16, 2, 16, 8)
    nul = None
    good = fc.fc_cache(256, 256, 8192, 50, 20, 16)
    bad_cap = fc.fc_cache(256, 256, 8190, 50, 20, 16)      # not a multiple of 4
    big_cap = fc.fc_cache(256, 256, 32768, 50, 20, 16)     # beyond FC_CACHE_MAX_WORDS
    odd_words = fc.fc_cache(260, 256, 8192, 50, 20, 16)    # words not 16-byte aligned
    bad_keep = fc.fc_cache(256, 256, 8192, 50, 20, 40)     # ctx_keep > FC_MAX_NMAX
    zero_chunk = fc.fc_cache(256, 256, 8192, 50, 0, 16)
    outs = [16] * 5
    for c in (bad_cap, big_cap, odd_words, bad_keep, zero_chunk):
        assert L.fc_cache_search(C.byref(c), nul, 0, 16, 64, 16, 4, p, 2, *outs, 16, nul) == 1
        assert L.fc_cache_update(C.byref(c), 16, 64, 16, 16, 16, 4, nul) == 1
        assert L.fc_cache_init(C.byref(c), 4, 16, nul) == 1
    # the CACHE slot must fit next to the datastore slots
    assert L.fc_cache_search(C.byref(good), nul, 0, 16, 64, 16, 4, p, 4, *outs, 16, nul) == 1
    # a missing table whose capacity is not a power of two
    assert L.fc_cache_search(C.byref(good), 16, 1000, 16, 64, 16, 4, p, 2, *outs, 16, nul) == 1
    # unsupported retrieval parameters, missing state array, empty batch
    assert L.fc_cache_search(C.byref(good), nul, 0, 16, 64, 16, 4, fc.params(40, 2, 16, 8), 2, *outs, 16, nul) == 2
    assert L.fc_cache_search(C.byref(good), nul, 0, 16, 64, 16, 4, p, 2, *outs, nul, nul) == 1
    assert L.fc_cache_search(C.byref(good), nul, 0, nul, 64, nul, 0, p, 2, *([nul] * 5), nul, nul) == 0
    # missing table sizes: header + capacity slots of 1 + key_len words
    assert L.fc_missing_bytes(1024, 2) == 4 * (4 + 1024 * 3)
    assert L.fc_missing_bytes(1000, 2) == 0 and L.fc_missing_bytes(1024, 0) == 0 and L.fc_missing_bytes(1024, 33) == 0
    assert L.fc_missing_init(16, 4 * (4 + 1024 * 3) - 1, 1024, 2, nul) == 3
    assert L.fc_missing_insert(16, 1024, 0, 16, 64, 16, 4, 16, 16, 2, nul) == 1
    assert L.fc_missing_insert(nul, 1024, 2, 16, 64, 16, 4, 16, 16, 2, nul) == 1


def test_rope_host_validation_without_gpu(lib):
    import paper_2502_17139_gb300.fastcoder as fc
    L = fc.LIB
    nul = None
    f = C.c_float
    # head dims that are not a multiple of 16, a bad layout, a non-positive base, odd addresses
    assert L.fc_rope(16, 16, 2, 64, 4, 100, 0, 16, f(10000.0), nul) == 1
    assert L.fc_rope(16, 16, 2, 64, 4, 128, 2, 16, f(10000.0), nul) == 1
    assert L.fc_rope(16, 16, 2, 64, 4, 128, 0, 16, f(0.0), nul) == 1
    assert L.fc_rope(17, 16, 2, 64, 4, 128, 0, 16, f(10000.0), nul) == 1
    assert L.fc_rope(nul, nul, 0, 64, 4, 128, 0, nul, f(10000.0), nul) == 0
    # the rotated attention: missing positions, a non-positive base, then fc_tree_attn's own limits
    args = [16, 16, 16, 128, 16, 16, 16, 8, 16, 2, 64, 32, 8, 128, f(0.1)]
    assert L.fc_tree_attn_rope(*args, nul, f(10000.0), 16, nul, 0, nul) == 1
    assert L.fc_tree_attn_rope(*args, 16, f(-1.0), 16, nul, 0, nul) == 1
    bad_d = args[:13] + [96, f(0.1)]
    assert L.fc_tree_attn_rope(*bad_d, 16, f(10000.0), 16, nul, 0, nul) == 2


def test_selftest_validation_without_gpu(lib):
    import paper_2502_17139_gb300.fastcoder as fc
    L = fc.LIB
    # a wait limit of zero or beyond ~4e9 cycles is refused before any launch
    assert L.fc_selftest_wait(0, 0, None) == 1
    assert L.fc_selftest_wait(0, 5_000_000_000, None) == 1


def test_reversed_retrieval_validation_without_gpu(lib):
    import paper_2502_17139_gb300.fastcoder as fc
    L = fc.LIB
    nul = None
    p = fc.params(16, 2, 16, 8)
    views = (fc.fc_datastore * 1)(fc.fc_datastore(16, 16, 16, 16, 10, 5))
    # no reversed stores; a reversed store of another length or vocabulary
    assert L.fc_retrieve_rev(views, nul, 1, 16, 64, 16, 4, nul, p, 16, 16, 16, 16, 16, nul) == 1
    rv = (fc.fc_datastore * 1)(fc.fc_datastore(16, 16, 16, nul, 9, 5))
    assert L.fc_retrieve_rev(views, rv, 1, 16, 64, 16, 4, nul, p, 16, 16, 16, 16, 16, nul) == 1
    rv = (fc.fc_datastore * 1)(fc.fc_datastore(16, 16, 16, nul, 10, 6))
    assert L.fc_retrieve_rev(views, rv, 1, 16, 64, 16, 4, nul, p, 16, 16, 16, 16, 16, nul) == 1
    # reversal: empty is a no-op; overlapping buffers and null pointers are refused
    assert L.fc_reverse_tokens(nul, 0, nul, nul) == 0
    assert L.fc_reverse_tokens(4096, 100, 4096 + 200, nul) == 1
    assert L.fc_reverse_tokens(nul, 100, 4096, nul) == 1


def test_trie_all_validation_without_gpu(lib):
    import paper_2502_17139_gb300.fastcoder as fc
    L = fc.LIB
    nul = None
    w = (C.c_uint32 * 2)(1, 1)
    # workspace size: zero for unsupported shapes (more than 8192 drafts, long drafts)
    assert L.fc_build_tree_all_workspace(2, 4096, 10, 32) > 0
    assert L.fc_build_tree_all_workspace(3, 4096, 10, 32) == 0
    assert L.fc_build_tree_all_workspace(2, 64, 17, 32) == 0
    args = [16, 16, 16, 16, w, 4096, 10, 16, 16, 32, 128, 128]
    outs = [16, 16, 16, 16, 16, 16, nul]
    assert L.fc_build_tree_all(2, *args, 256, 1000, *outs) == 3          # FC_ERR_WORKSPACE
    assert L.fc_build_tree_all(3, *args, 256, 1 << 40, *outs) == 2       # too many drafts: FC_ERR_UNSUPPORTED
    assert L.fc_build_tree_all(2, *args[:10], 128, 96, 256, 1 << 40, *outs) == 2  # n_pad 96
    assert L.fc_build_tree_all(2, *args[:10], 0, 128, 256, 1 << 40, *outs) == 1   # budget 0


def test_pipeline_host_validation(lib):
    """The native step executor rejects bad descriptions before it creates
    any stream (nothing here touches a GPU)."""
    import paper_2502_17139_gb300.fastcoder as fc
    L = fc.LIB
    h = C.c_void_p()
    assert L.fc_pipeline_create(None, C.byref(h)) == 1 and not h.value
    views = (fc.fc_datastore * 1)(fc.fc_datastore(16, 16, 16, 16, 10, 5))
    w = (C.c_uint32 * 1)(1)
    buf = [16 * (i + 1) for i in range(40)]
    part = fc.fc_pipeline_part(4, 0, buf[0], 64, (C.c_void_p * 2)(buf[1], buf[2]), (C.c_void_p * 2)(buf[3], buf[4]),
                               buf[5], None, 0, buf[6], buf[7], buf[8], buf[9], buf[10], buf[11], buf[12], buf[13],
                               buf[14], buf[15], buf[16], buf[17], buf[18], buf[19], None, buf[20], None, 0, buf[21],
                               buf[22], buf[23], buf[24])

    def desc(parts, n_parts=None, **kw):
        d = dict(node_budget=64, n_pad=128, H=32, Hkv=8, D=128, kv_cap=1024, path_cap=10, vocab=1000, scale=0.1,
                 rope_base=0.0)
        d.update(kw)
        arr = (fc.fc_pipeline_part * max(1, len(parts)))(*parts)
        return fc.fc_pipeline_desc(views, 1, fc.params(16, 2, 16, 8), w, d["node_budget"], d["n_pad"], d["H"],
                                   d["Hkv"], d["D"], d["kv_cap"], d["path_cap"], d["vocab"], d["scale"],
                                   d["rope_base"], len(parts) if n_parts is None else n_parts, arr)

    assert L.fc_pipeline_create(C.byref(desc([part], n_parts=0)), C.byref(h)) == 1
    assert L.fc_pipeline_create(C.byref(desc([part], scale=0.0)), C.byref(h)) == 1
    assert L.fc_pipeline_create(C.byref(desc([part], rope_base=1e4)), C.byref(h)) == 1  # RoPE needs k_tree_rot
    same = fc.fc_pipeline_part.from_buffer_copy(part)
    same.kv_len[1] = same.kv_len[0]  # the ping-pong buffers must differ
    assert L.fc_pipeline_create(C.byref(desc([same])), C.byref(h)) == 1
    missing = fc.fc_pipeline_part.from_buffer_copy(part)
    missing.mask = None
    assert L.fc_pipeline_create(C.byref(desc([missing])), C.byref(h)) == 1
    # Algorithm 1 parts: a CACHE view fc_cache_search would reject, a CACHE
    # beside a replay cache, a missing table without a CACHE or of a bad size
    def seq(cache=(buf[30], buf[31], 8192, 50, 20, 16), rcache=None, missing=buf[32], cap=1 << 10):
        q = fc.fc_pipeline_part.from_buffer_copy(part)
        q.seq_cache = fc.fc_cache(*cache) if cache else fc.fc_cache()
        q.rcache, q.rcache_capacity = rcache, 16 if rcache else 0
        q.missing, q.missing_capacity = missing, cap
        return q
    for bad in (seq(rcache=buf[33]), seq(cache=None), seq(cap=3), seq(cap=1 << 25), seq(cap=1),
                seq(cache=(buf[30], buf[31], 8190, 50, 20, 16)), seq(cache=(buf[30], buf[31], 8, 50, 20, 16)),
                seq(cache=(buf[30] + 8, buf[31], 8192, 50, 20, 16)), seq(cache=(buf[30], None, 8192, 50, 20, 16)),
                seq(cache=(buf[30], buf[31], 8192, -1, 20, 16)), seq(cache=(buf[30], buf[31], 8192, 50, 0, 16)),
                seq(cache=(buf[30], buf[31], 8192, 50, 20, 33))):
        assert L.fc_pipeline_create(C.byref(desc([part, bad])), C.byref(h)) == 1
    assert not h.value
    nul = None
    assert L.fc_pipeline_step(nul, 0, 0, 16, 16, 16, nul, 16, 16, nul, nul) == 1
    assert L.fc_pipeline_step_part(nul, 0, 0, 0, 16, 16, 16, nul, 16, 16, nul, nul) == 1
    assert L.fc_pipeline_join(nul, nul) == 1
    assert L.fc_pipeline_join_part(nul, 0, nul) == 1
    assert L.fc_pipeline_error(nul, 0) == 1
    assert L.fc_pipeline_stream(nul, 0) is None
    g = C.c_void_p(7)
    arr = (C.c_void_p * 2)(16, 16)
    assert L.fc_pipeline_capture_part(nul, 0, 2, 0, 0, arr, arr, arr, None, arr, arr, C.byref(g)) == 1
    assert not g.value  # cleared on failure
    assert L.fc_pipeline_capture_part(nul, 0, 2, 0, 0, arr, arr, arr, None, arr, arr, None) == 1
    assert L.fc_pipeline_graph_launch(nul, nul) == 1
    a, b = C.c_int(), C.c_int()
    assert L.fc_pipeline_graph_kernels(nul, C.byref(a), C.byref(b)) == 1
    L.fc_pipeline_graph_destroy(nul)
    L.fc_pipeline_destroy(nul)
