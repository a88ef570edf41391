"""Python binding of libfastcoder.so: argument marshalling only.

Every function here checks tensor dtypes, devices and shapes, passes raw
device pointers and the current CUDA stream to the C ABI of the same name
(include/fastcoder.h), and raises FastCoderError on a non-OK status.  All
computation happens in the CUDA kernels behind that ABI; if the library
cannot be loaded, importing this module raises (there is no fallback).

Tensor conventions: uint32 token ids travel in int32 tensors (same bits),
uint64 mask words in int64 tensors, bf16 tensors as torch.bfloat16.
"""
from __future__ import annotations

import atexit
import ctypes as C
import os
import weakref

import numpy as np
import torch

from . import build as _build

PAD = 0xFFFFFFFF
PAD_I32 = -1  # FC_PAD_TOKEN seen through an int32 tensor
MAX_OCC = 4096
MAX_NODES = 128

STATUS = {0: "FC_OK", 1: "FC_ERR_INVALID_ARG", 2: "FC_ERR_UNSUPPORTED", 3: "FC_ERR_WORKSPACE",
          4: "FC_ERR_CAPACITY", 5: "FC_ERR_TIMEOUT", 6: "FC_ERR_CUDA", 7: "FC_ERR_INTERNAL", 8: "FC_ERR_IO"}


class FastCoderError(RuntimeError):
    def __init__(self, fn: str, code: int):
        super().__init__(f"{fn} returned {STATUS.get(code, code)}")
        self.code = code
        self.status = STATUS.get(code, str(code))


class fc_datastore(C.Structure):
    _fields_ = [("tokens", C.c_void_p), ("sa", C.c_void_p), ("bucket", C.c_void_p), ("lcp", C.c_void_p),
                ("n_tokens", C.c_uint64), ("vocab", C.c_uint32), ("keys", C.c_void_p)]


class fc_retrieve_params(C.Structure):
    _fields_ = [("n_max", C.c_int32), ("n_min", C.c_int32), ("top_k", C.c_int32),
                ("draft_len", C.c_int32), ("max_occ", C.c_uint32)]


class fc_cache(C.Structure):
    _fields_ = [("d_words", C.c_void_p), ("d_meta", C.c_void_p), ("capacity", C.c_int32), ("min_size", C.c_int32),
                ("chunk", C.c_int32), ("ctx_keep", C.c_int32)]


class fc_pipeline_part(C.Structure):
    _fields_ = [("batch", C.c_int32), ("first", C.c_int32), ("ctx", C.c_void_p), ("ctx_stride", C.c_int32),
                ("ctx_len", C.c_void_p * 2), ("kv_len", C.c_void_p * 2), ("root", C.c_void_p),
                ("rcache", C.c_void_p), ("rcache_capacity", C.c_int32), ("skip", C.c_void_p),
                ("drafts", C.c_void_p), ("draft_len", C.c_void_p), ("count", C.c_void_p), ("n_drafts", C.c_void_p),
                ("match_len", C.c_void_p), ("tok", C.c_void_p), ("parent", C.c_void_p), ("depth", C.c_void_p),
                ("pos", C.c_void_p), ("mask", C.c_void_p), ("n_nodes", C.c_void_p), ("k_cache", C.c_void_p),
                ("v_cache", C.c_void_p), ("k_tree_rot", C.c_void_p), ("attn_out", C.c_void_p),
                ("attn_ws", C.c_void_p), ("attn_ws_bytes", C.c_size_t), ("argmax", C.c_void_p),
                ("acc_len", C.c_void_p), ("path", C.c_void_p), ("bonus", C.c_void_p), ("err", C.c_void_p),
                ("seq_cache", fc_cache), ("missing", C.c_void_p), ("missing_capacity", C.c_int32)]


class fc_pipeline_desc(C.Structure):
    _fields_ = [("sources", C.POINTER(fc_datastore)), ("n_sources", C.c_int32), ("p", fc_retrieve_params),
                ("src_weight", C.POINTER(C.c_uint32)), ("node_budget", C.c_int32), ("n_pad", C.c_int32),
                ("H", C.c_int32), ("Hkv", C.c_int32), ("D", C.c_int32), ("kv_cap", C.c_int32),
                ("path_cap", C.c_int32), ("vocab", C.c_uint32), ("scale", C.c_float), ("rope_base", C.c_float),
                ("n_parts", C.c_int32), ("parts", C.POINTER(fc_pipeline_part)), ("cache_weight", C.c_uint32)]


EXPORTS = ["fc_status_string", "fc_version", "fc_get_error", "fc_datastore_build_workspace", "fc_datastore_build",
           "fc_datastore_build_noalloc", "fc_datastore_keys", "fc_datastore_save", "fc_datastore_file_info", "fc_datastore_load",
           "fc_retrieve", "fc_retrieve_all", "fc_retrieve_rev", "fc_reverse_tokens", "fc_rcache_bytes", "fc_rcache_init", "fc_rcache_lookup", "fc_rcache_insert", "fc_retrieve_cached",
           "fc_cache_init", "fc_cache_search", "fc_cache_update", "fc_missing_bytes", "fc_missing_init",
           "fc_missing_insert", "fc_build_tree", "fc_build_tree_all_workspace", "fc_build_tree_all", "fc_tree_mask", "fc_tree_attn", "fc_tree_attn_workspace", "fc_tree_attn_parts", "fc_tree_attn_streamed", "fc_rope", "fc_tree_attn_rope", "fc_gemm_workspace", "fc_gemm_bf16", "fc_gemm_kv_heads", "fc_gemm_silu_mul", "fc_interleave_gate_up", "fc_embed",
           "fc_add_rmsnorm", "fc_silu_mul", "fc_rope_heads", "fc_selftest_wait", "fc_accept", "fc_argmax_accept", "fc_kv_append", "fc_synth_argmax",
           "fc_pipeline_create", "fc_pipeline_step", "fc_pipeline_step_part", "fc_pipeline_join_part", "fc_pipeline_stream", "fc_pipeline_error", "fc_pipeline_join",
           "fc_pipeline_capture_part", "fc_pipeline_graph_launch", "fc_pipeline_graph_kernels", "fc_pipeline_graph_destroy",
           "fc_pipeline_destroy"]


def _load():
    # FC_DEBUG=1 loads the bounds-checking debug build (build(debug=True))
    path = _build.LIB_DEBUG if os.environ.get("FC_DEBUG", "0") not in ("", "0") else _build.LIB
    if not os.path.exists(path):
        raise ImportError(f"libfastcoder.so is not built ({path}); run __graft_entry__.build()")
    lib = C.CDLL(path)
    vp, i32, u32, u64, sz = C.c_void_p, C.c_int, C.c_uint32, C.c_uint64, C.c_size_t
    sig = {
        "fc_status_string": (C.c_char_p, [C.c_int]),
        "fc_version": (C.c_char_p, []),
        "fc_get_error": (C.c_int, [vp]),
        "fc_datastore_build_workspace": (sz, [u64, u32]),
        "fc_datastore_build": (C.c_int, [vp, u64, u32, vp, vp, vp, vp, sz, vp, C.POINTER(fc_datastore)]),
        "fc_datastore_build_noalloc": (C.c_int, [vp, u64, u32, vp, vp, vp, vp, C.POINTER(fc_datastore)]),
        "fc_datastore_keys": (C.c_int, [C.POINTER(fc_datastore), vp, vp]),
        "fc_datastore_save": (C.c_int, [C.c_char_p, C.POINTER(fc_datastore), i32, vp]),
        "fc_datastore_file_info": (C.c_int, [C.c_char_p, C.POINTER(C.c_uint64), C.POINTER(C.c_uint32)]),
        "fc_datastore_load": (C.c_int, [C.c_char_p, vp, vp, vp, vp, u64, u32, i32, vp, C.POINTER(fc_datastore)]),
        "fc_retrieve": (C.c_int, [C.POINTER(fc_datastore), i32, vp, i32, vp, i32, vp, fc_retrieve_params,
                                  vp, vp, vp, vp, vp, vp]),
        "fc_retrieve_all": (C.c_int, [C.POINTER(fc_datastore), i32, vp, i32, vp, i32, vp, fc_retrieve_params,
                                      vp, vp, vp, vp, vp, vp]),
        "fc_retrieve_rev": (C.c_int, [C.POINTER(fc_datastore), C.POINTER(fc_datastore), i32, vp, i32, vp, i32, vp,
                                      fc_retrieve_params, vp, vp, vp, vp, vp, vp]),
        "fc_reverse_tokens": (C.c_int, [vp, u64, vp, vp]),
        "fc_rcache_bytes": (sz, [i32, i32, fc_retrieve_params]),
        "fc_rcache_init": (C.c_int, [vp, sz, i32, i32, fc_retrieve_params, vp]),
        "fc_rcache_lookup": (C.c_int, [vp, i32, i32, fc_retrieve_params, vp, i32, vp, i32, vp, vp,
                                       vp, vp, vp, vp, vp, vp]),
        "fc_rcache_insert": (C.c_int, [vp, i32, i32, fc_retrieve_params, vp, i32, vp, i32, vp,
                                       vp, vp, vp, vp, vp, vp]),
        "fc_retrieve_cached": (C.c_int, [C.POINTER(fc_datastore), i32, vp, i32, vp, i32, vp, i32, vp, vp,
                                         fc_retrieve_params, vp, vp, vp, vp, vp, vp]),
        "fc_cache_init": (C.c_int, [C.POINTER(fc_cache), i32, vp, vp]),
        "fc_cache_search": (C.c_int, [C.POINTER(fc_cache), vp, i32, vp, i32, vp, i32, fc_retrieve_params, i32,
                                      vp, vp, vp, vp, vp, vp, vp]),
        "fc_cache_update": (C.c_int, [C.POINTER(fc_cache), vp, i32, vp, vp, vp, i32, vp]),
        "fc_missing_bytes": (sz, [i32, i32]),
        "fc_missing_init": (C.c_int, [vp, sz, i32, i32, vp]),
        "fc_missing_insert": (C.c_int, [vp, i32, i32, vp, i32, vp, i32, vp, vp, i32, vp]),
        "fc_build_tree": (C.c_int, [i32, vp, vp, vp, vp, C.POINTER(C.c_uint32), i32, i32, vp, vp, i32, i32, i32,
                                    vp, vp, vp, vp, vp, vp, vp]),
        "fc_build_tree_all_workspace": (sz, [i32, i32, i32, i32]),
        "fc_build_tree_all": (C.c_int, [i32, vp, vp, vp, vp, C.POINTER(C.c_uint32), i32, i32, vp, vp, i32, i32, i32,
                                        vp, sz, vp, vp, vp, vp, vp, vp, vp]),
        "fc_tree_mask": (C.c_int, [vp, vp, vp, i32, i32, vp, vp, vp, vp]),
        "fc_tree_attn": (C.c_int, [vp, vp, vp, i32, vp, vp, vp, vp, vp, i32, i32, i32, i32, i32, C.c_float, vp, vp, sz,
                                   vp]),
        "fc_tree_attn_workspace": (sz, [i32, i32, i32, i32]),
        "fc_rope": (C.c_int, [vp, vp, i32, i32, i32, i32, i32, vp, C.c_float, vp]),
        "fc_gemm_workspace": (sz, []),
        "fc_selftest_wait": (C.c_int, [i32, C.c_ulonglong, vp]),
        "fc_gemm_bf16": (C.c_int, [vp, vp, vp, i32, i32, i32, vp, sz, vp]),
        "fc_gemm_kv_heads": (C.c_int, [vp, vp, i32, i32, i32, i32, i32, i32, vp, C.c_float, vp, vp, vp]),
        "fc_gemm_silu_mul": (C.c_int, [vp, vp, i32, i32, i32, vp, vp]),
        "fc_interleave_gate_up": (C.c_int, [vp, vp, i32, i32, vp]),
        "fc_embed": (C.c_int, [vp, i32, vp, i32, i32, vp, vp]),
        "fc_add_rmsnorm": (C.c_int, [vp, vp, vp, vp, i32, i32, C.c_float, vp]),
        "fc_silu_mul": (C.c_int, [vp, vp, i32, i32, vp]),
        "fc_rope_heads": (C.c_int, [vp, i32, vp, i32, i32, i32, i32, vp, C.c_float, vp]),
        "fc_tree_attn_rope": (C.c_int, [vp, vp, vp, i32, vp, vp, vp, vp, vp, i32, i32, i32, i32, i32, C.c_float, vp,
                                        C.c_float, vp, vp, sz, vp]),
        "fc_tree_attn_parts": (C.c_int, [i32, i32, i32, i32, i32, sz]),
        "fc_tree_attn_streamed": (C.c_int, [i32, i32, i32, i32, i32]),
        "fc_accept": (C.c_int, [vp, vp, vp, vp, i32, i32, vp, vp, i32, vp, vp]),
        "fc_argmax_accept": (C.c_int, [vp, i32, vp, vp, vp, i32, i32, vp, vp, vp, i32, vp, vp]),
        "fc_kv_append": (C.c_int, [vp, vp, vp, vp, vp, vp, i32, i32, i32, i32, i32, vp, vp, i32, vp, vp, vp, i32,
                                   vp, vp, vp, vp]),
        "fc_synth_argmax": (C.c_int, [vp, vp, vp, i32, i32, vp, vp, u32, vp, vp]),
        "fc_pipeline_create": (C.c_int, [C.POINTER(fc_pipeline_desc), C.POINTER(vp)]),
        "fc_pipeline_step": (C.c_int, [vp, i32, i32, vp, vp, vp, vp, vp, vp, vp, vp]),
        "fc_pipeline_join": (C.c_int, [vp, vp]),
        "fc_pipeline_step_part": (C.c_int, [vp, i32, i32, i32, vp, vp, vp, vp, vp, vp, vp, vp]),
        "fc_pipeline_join_part": (C.c_int, [vp, i32, vp]),
        "fc_pipeline_stream": (vp, [vp, i32]),
        "fc_pipeline_error": (C.c_int, [vp, i32]),
        "fc_pipeline_destroy": (None, [vp]),
        "fc_pipeline_capture_part": (C.c_int, [vp, i32, i32, i32, i32, vp, vp, vp, vp, vp, vp, vp]),
        "fc_pipeline_graph_launch": (C.c_int, [vp, vp]),
        "fc_pipeline_graph_kernels": (C.c_int, [vp, C.POINTER(C.c_int), C.POINTER(C.c_int)]),
        "fc_pipeline_graph_destroy": (None, [vp]),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    return lib


LIB = _load()


def _stream():
    return C.c_void_p(torch.cuda.current_stream().cuda_stream)


def _ptr(t):
    return None if t is None else C.c_void_p(t.data_ptr())


def _check(fn, code):
    if code != 0:
        raise FastCoderError(fn, code)


def _need(t, dtype, name, shape=None):
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_cuda:
        raise ValueError(f"{name} must be on a CUDA device")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} must have shape {tuple(shape)}, got {tuple(t.shape)}")
    return t


def version() -> str:
    return LIB.fc_version().decode()


def fc_selftest_wait(arrive: bool, limit_cycles: int = 2_000_000):
    """Bounded-wait self-test: with arrive=False the wait runs out and
    fc_get_error() then reports FC_ERR_TIMEOUT."""
    _check("fc_selftest_wait", LIB.fc_selftest_wait(1 if arrive else 0, int(limit_cycles), _stream()))


def fc_get_error(stream=None) -> str:
    s = C.c_void_p(stream.cuda_stream) if stream is not None else _stream()
    return STATUS.get(LIB.fc_get_error(s), "?")


# --------------------------------------------------------------- datastore
class Datastore:
    """A built datastore: the token corpus, its suffix array, bucket table and
    LCP array (device tensors owned here), optionally its suffix keys
    (fc_datastore_keys), plus the C view struct."""

    def __init__(self, tokens, sa, bucket, lcp, vocab, keys=None):
        self.tokens, self.sa, self.bucket, self.lcp, self.vocab = tokens, sa, bucket, lcp, int(vocab)
        self.keys = keys
        self.view = fc_datastore(tokens.data_ptr(), sa.data_ptr(), bucket.data_ptr(), lcp.data_ptr(),
                                 tokens.numel(), int(vocab), None if keys is None else keys.data_ptr())

    @property
    def n_tokens(self):
        return self.tokens.numel()

    def without_keys(self):
        """The same store viewed without its suffix keys (the search then reads
        the suffix array and the corpus)."""
        return Datastore(self.tokens, self.sa, self.bucket, self.lcp, self.vocab)


def fc_datastore_keys(ds: Datastore) -> Datastore:
    """Builds the suffix keys of a datastore (32 bytes per token) and returns
    the store with them in its view."""
    keys = torch.empty((ds.n_tokens, 8), dtype=torch.int32, device=ds.tokens.device)
    _check("fc_datastore_keys", LIB.fc_datastore_keys(C.byref(ds.view), _ptr(keys), _stream()))
    return Datastore(ds.tokens, ds.sa, ds.bucket, ds.lcp, ds.vocab, keys)


def fc_datastore_build_workspace(n_tokens: int, vocab: int) -> int:
    return int(LIB.fc_datastore_build_workspace(n_tokens, vocab))


def fc_datastore_build(tokens: torch.Tensor, vocab: int, workspace: torch.Tensor | None = None,
                       keys: bool = True) -> Datastore:
    """tokens: int32 [N] on the GPU (uint32 ids < vocab).  Synchronous.  With
    ``keys`` the suffix keys are built too (fc_datastore_keys)."""
    _need(tokens, torch.int32, "tokens")
    n = tokens.numel()
    sa = torch.empty(n, dtype=torch.int32, device=tokens.device)
    bucket = torch.empty(vocab + 1, dtype=torch.int32, device=tokens.device)
    lcp = torch.empty(n, dtype=torch.uint8, device=tokens.device)
    need = fc_datastore_build_workspace(n, vocab)
    ws = workspace if workspace is not None else torch.empty(need, dtype=torch.uint8, device=tokens.device)
    if ws.numel() < need:
        raise ValueError("workspace too small")
    _check("fc_datastore_build", LIB.fc_datastore_build(_ptr(tokens), n, vocab, _ptr(sa), _ptr(bucket), _ptr(lcp),
                                                        _ptr(ws), ws.numel(), _stream(), None))
    ds = Datastore(tokens, sa, bucket, lcp, vocab)
    return fc_datastore_keys(ds) if keys else ds


def _np_ptr(a):
    return C.c_void_p(a.ctypes.data)


def fc_datastore_save(ds: Datastore, path: str) -> None:
    """Writes a device datastore to ``path`` (synchronous)."""
    _check("fc_datastore_save", LIB.fc_datastore_save(os.fsencode(path), C.byref(ds.view), 0, _stream()))


def fc_datastore_file_info(path: str):
    """(n_tokens, vocab) from a datastore file's header."""
    n, v = C.c_uint64(0), C.c_uint32(0)
    _check("fc_datastore_file_info", LIB.fc_datastore_file_info(os.fsencode(path), C.byref(n), C.byref(v)))
    return int(n.value), int(v.value)


def fc_datastore_load(path: str, device="cuda") -> Datastore:
    """Reads a datastore file into new device tensors (synchronous)."""
    n, vocab = fc_datastore_file_info(path)
    tokens = torch.empty(n, dtype=torch.int32, device=device)
    sa = torch.empty(n, dtype=torch.int32, device=device)
    bucket = torch.empty(vocab + 1, dtype=torch.int32, device=device)
    lcp = torch.empty(n, dtype=torch.uint8, device=device)
    _check("fc_datastore_load", LIB.fc_datastore_load(os.fsencode(path), _ptr(tokens), _ptr(sa), _ptr(bucket),
                                                      _ptr(lcp), n, vocab, 0, _stream(), None))
    return fc_datastore_keys(Datastore(tokens, sa, bucket, lcp, vocab))


def datastore_save_host(path: str, tokens, sa, bucket, lcp) -> None:
    """The same file from host arrays (numpy uint32 tokens / sa / bucket,
    uint8 lcp); no CUDA call is made."""
    arrs = [np.ascontiguousarray(tokens, np.uint32), np.ascontiguousarray(sa, np.uint32),
            np.ascontiguousarray(bucket, np.uint32), np.ascontiguousarray(lcp, np.uint8)]
    view = fc_datastore(arrs[0].ctypes.data, arrs[1].ctypes.data, arrs[2].ctypes.data, arrs[3].ctypes.data,
                        len(arrs[0]), len(arrs[2]) - 1)
    _check("fc_datastore_save", LIB.fc_datastore_save(os.fsencode(path), C.byref(view), 1, None))


def datastore_load_host(path: str):
    """A datastore file into host arrays: dict(tokens, sa, bucket, lcp)."""
    n, vocab = fc_datastore_file_info(path)
    out = dict(tokens=np.empty(n, np.uint32), sa=np.empty(n, np.uint32), bucket=np.empty(vocab + 1, np.uint32),
               lcp=np.empty(n, np.uint8))
    _check("fc_datastore_load", LIB.fc_datastore_load(os.fsencode(path), _np_ptr(out["tokens"]), _np_ptr(out["sa"]),
                                                      _np_ptr(out["bucket"]), _np_ptr(out["lcp"]), n, vocab, 1, None,
                                                      None))
    return out


NOALLOC_MAX_TOKENS = 1 << 20


def fc_datastore_build_noalloc(tokens: torch.Tensor, vocab: int, sa: torch.Tensor, bucket: torch.Tensor,
                               lcp: torch.Tensor) -> Datastore:
    """The datastore build for callers that cannot allocate device memory:
    scratch comes from a fixed array inside the library, and the outputs go
    to the caller's sa [N] (int32), bucket [vocab + 1] (int32) and lcp [N]
    (uint8).  N is at most NOALLOC_MAX_TOKENS.  This wrapper allocates
    nothing either."""
    _need(tokens, torch.int32, "tokens")
    n = tokens.numel()
    _need(sa, torch.int32, "sa", (n,))
    _need(bucket, torch.int32, "bucket", (vocab + 1,))
    _need(lcp, torch.uint8, "lcp", (n,))
    _check("fc_datastore_build_noalloc", LIB.fc_datastore_build_noalloc(_ptr(tokens), n, vocab, _ptr(sa),
                                                                        _ptr(bucket), _ptr(lcp), _stream(), None))
    return Datastore(tokens, sa, bucket, lcp, vocab)


def datastore_from_parts(tokens, sa, bucket, lcp, vocab) -> Datastore:
    for t, nm in ((tokens, "tokens"), (sa, "sa"), (bucket, "bucket")):
        _need(t, torch.int32, nm)
    _need(lcp, torch.uint8, "lcp")
    return Datastore(tokens, sa, bucket, lcp, vocab)


# --------------------------------------------------------------- retrieval
def params(n_max, n_min, top_k, draft_len, max_occ=MAX_OCC) -> fc_retrieve_params:
    return fc_retrieve_params(n_max, n_min, top_k, draft_len, max_occ)


def retrieve_outputs(n_sources, batch, p: fc_retrieve_params, device="cuda", slots=None):
    S, B, k, d = n_sources, batch, (p.top_k if slots is None else slots), p.draft_len
    return dict(drafts=torch.empty((S, B, k, d), dtype=torch.int32, device=device),
                draft_len=torch.empty((S, B, k), dtype=torch.int32, device=device),
                count=torch.empty((S, B, k), dtype=torch.int32, device=device),
                n_drafts=torch.empty((S, B), dtype=torch.int32, device=device),
                match_len=torch.empty((S, B), dtype=torch.int32, device=device))


def fc_retrieve(sources, ctx, ctx_len, p: fc_retrieve_params, skip=None, out=None):
    """ctx: int32 [B, stride]; ctx_len: int32 [B]; returns dict of outputs
    shaped [S, B, ...] (see include/fastcoder.h)."""
    S = len(sources)
    _need(ctx, torch.int32, "ctx")
    B, stride = ctx.shape
    _need(ctx_len, torch.int32, "ctx_len", (B,))
    if skip is not None:
        _need(skip, torch.int32, "skip", (B,))
    o = out if out is not None else retrieve_outputs(S, B, p, ctx.device)
    views = (fc_datastore * S)(*[s.view for s in sources])
    _check("fc_retrieve", LIB.fc_retrieve(views, S, _ptr(ctx), stride, _ptr(ctx_len), B, _ptr(skip), p,
                                          _ptr(o["drafts"]), _ptr(o["draft_len"]), _ptr(o["count"]),
                                          _ptr(o["n_drafts"]), _ptr(o["match_len"]), _stream()))
    return o


def fc_retrieve_all(sources, ctx, ctx_len, p: fc_retrieve_params, skip=None, out=None):
    """Every distinct continuation (no top-k), in ascending token order:
    outputs shaped [S, B, p.max_occ, ...]."""
    S = len(sources)
    _need(ctx, torch.int32, "ctx")
    B, stride = ctx.shape
    _need(ctx_len, torch.int32, "ctx_len", (B,))
    if skip is not None:
        _need(skip, torch.int32, "skip", (B,))
    o = out if out is not None else retrieve_outputs(S, B, p, ctx.device, slots=int(p.max_occ))
    views = (fc_datastore * S)(*[s.view for s in sources])
    _check("fc_retrieve_all", LIB.fc_retrieve_all(views, S, _ptr(ctx), stride, _ptr(ctx_len), B, _ptr(skip), p,
                                                  _ptr(o["drafts"]), _ptr(o["draft_len"]), _ptr(o["count"]),
                                                  _ptr(o["n_drafts"]), _ptr(o["match_len"]), _stream()))
    return o


def fc_reverse_tokens(tokens: torch.Tensor, out: torch.Tensor | None = None) -> torch.Tensor:
    """The reversed corpus (int32 [N] on the GPU); asynchronous."""
    _need(tokens, torch.int32, "tokens")
    o = out if out is not None else torch.empty_like(tokens)
    _need(o, torch.int32, "out", tuple(tokens.shape))
    _check("fc_reverse_tokens", LIB.fc_reverse_tokens(_ptr(tokens), tokens.numel(), _ptr(o), _stream()))
    return o


def fc_datastore_build_reversed(tokens: torch.Tensor, vocab: int) -> Datastore:
    """The datastore of the reversed corpus, for fc_retrieve_rev (its narrowing
    search reads the reversed suffix array directly; no suffix keys)."""
    return fc_datastore_build(fc_reverse_tokens(tokens), vocab, keys=False)


def fc_retrieve_rev(sources, rev_sources, ctx, ctx_len, p: fc_retrieve_params, skip=None, out=None):
    """fc_retrieve with n* found in the reversed corpora (same outputs)."""
    S = len(sources)
    if len(rev_sources) != S:
        raise ValueError("one reversed datastore per source")
    _need(ctx, torch.int32, "ctx")
    B, stride = ctx.shape
    _need(ctx_len, torch.int32, "ctx_len", (B,))
    if skip is not None:
        _need(skip, torch.int32, "skip", (B,))
    o = out if out is not None else retrieve_outputs(S, B, p, ctx.device)
    views = (fc_datastore * S)(*[s.view for s in sources])
    rviews = (fc_datastore * S)(*[s.view for s in rev_sources])
    _check("fc_retrieve_rev", LIB.fc_retrieve_rev(views, rviews, S, _ptr(ctx), stride, _ptr(ctx_len), B, _ptr(skip),
                                                  p, _ptr(o["drafts"]), _ptr(o["draft_len"]), _ptr(o["count"]),
                                                  _ptr(o["n_drafts"]), _ptr(o["match_len"]), _stream()))
    return o


class RetrievalCache:
    """Context-keyed replay cache in caller-owned device memory."""

    def __init__(self, capacity, n_sources, p: fc_retrieve_params, device="cuda"):
        self.capacity, self.n_sources, self.p = capacity, n_sources, p
        nbytes = int(LIB.fc_rcache_bytes(capacity, n_sources, p))
        if nbytes == 0:
            raise ValueError("bad cache parameters")
        self.table = torch.empty(nbytes, dtype=torch.uint8, device=device)
        _check("fc_rcache_init", LIB.fc_rcache_init(_ptr(self.table), nbytes, capacity, n_sources, p, _stream()))


def fc_rcache_lookup(cache: RetrievalCache, ctx, ctx_len, want_hit, skip, out):
    B, stride = ctx.shape
    _check("fc_rcache_lookup", LIB.fc_rcache_lookup(
        _ptr(cache.table), cache.capacity, cache.n_sources, cache.p, _ptr(ctx), stride, _ptr(ctx_len), B,
        _ptr(want_hit), _ptr(skip), _ptr(out["drafts"]), _ptr(out["draft_len"]), _ptr(out["count"]),
        _ptr(out["n_drafts"]), _ptr(out["match_len"]), _stream()))


def fc_retrieve_cached(sources, cache: RetrievalCache, ctx, ctx_len, want_hit, skip, p: fc_retrieve_params, out):
    """fc_rcache_lookup + fc_retrieve of the queries it did not serve, in one
    launch (skip [B] written: 1 = served)."""
    S = len(sources)
    _need(ctx, torch.int32, "ctx")
    B, stride = ctx.shape
    _need(ctx_len, torch.int32, "ctx_len", (B,))
    _need(skip, torch.int32, "skip", (B,))
    if want_hit is not None:
        _need(want_hit, torch.int32, "want_hit", (B,))
    views = (fc_datastore * S)(*[s.view for s in sources])
    _check("fc_retrieve_cached", LIB.fc_retrieve_cached(
        views, S, _ptr(ctx), stride, _ptr(ctx_len), B, _ptr(cache.table), cache.capacity, _ptr(want_hit), _ptr(skip),
        p, _ptr(out["drafts"]), _ptr(out["draft_len"]), _ptr(out["count"]), _ptr(out["n_drafts"]),
        _ptr(out["match_len"]), _stream()))
    return out


def fc_rcache_insert(cache: RetrievalCache, ctx, ctx_len, skip, res):
    B, stride = ctx.shape
    _check("fc_rcache_insert", LIB.fc_rcache_insert(
        _ptr(cache.table), cache.capacity, cache.n_sources, cache.p, _ptr(ctx), stride, _ptr(ctx_len), B,
        _ptr(skip), _ptr(res["drafts"]), _ptr(res["draft_len"]), _ptr(res["count"]), _ptr(res["n_drafts"]),
        _ptr(res["match_len"]), _stream()))


# ------------------------------------------------- CACHE and missing table
SERVE_DATASTORE, SERVE_CACHE, SKIP_MISSING = 0, 1, 2
SEP_I32 = -2  # FC_SEP_TOKEN seen through an int32 tensor


class SequenceCache:
    """The CACHE of Section IV-B for a batch: per sequence, a store of
    verified retrievals and output pieces (words [B, capacity] int32, meta
    [B, 4] int32: words used, sequences stored, output mark, dropped)."""

    def __init__(self, batch, capacity=8192, min_size=50, chunk=20, ctx_keep=16, device="cuda"):
        self.batch = batch
        self.words = torch.zeros((batch, capacity), dtype=torch.int32, device=device)
        self.meta = torch.zeros((batch, 4), dtype=torch.int32, device=device)
        self.view = fc_cache(self.words.data_ptr(), self.meta.data_ptr(), capacity, min_size, chunk, ctx_keep)

    def init(self, prompt_len):
        _need(prompt_len, torch.int32, "prompt_len", (self.batch,))
        _check("fc_cache_init", LIB.fc_cache_init(C.byref(self.view), self.batch, _ptr(prompt_len), _stream()))


class MissingTable:
    """The missing table M of Algorithm 1 (keys of key_len tokens)."""

    def __init__(self, capacity, key_len, device="cuda"):
        self.capacity, self.key_len = capacity, key_len
        nbytes = int(LIB.fc_missing_bytes(capacity, key_len))
        if nbytes == 0:
            raise ValueError("bad missing-table parameters")
        self.table = torch.empty(nbytes // 4, dtype=torch.int32, device=device)
        self.clear()

    def clear(self):
        _check("fc_missing_init", LIB.fc_missing_init(_ptr(self.table), self.table.numel() * 4, self.capacity,
                                                      self.key_len, _stream()))


def fc_cache_search(cache: SequenceCache, missing, ctx, ctx_len, p: fc_retrieve_params, n_sources, out, state):
    """out: retrieve_outputs(n_sources + 1, B, p); slot n_sources gets the
    CACHE's result.  state: int32 [B]."""
    _need(ctx, torch.int32, "ctx")
    B, stride = ctx.shape
    _need(ctx_len, torch.int32, "ctx_len", (B,))
    _need(state, torch.int32, "state", (B,))
    if out["n_drafts"].shape != (n_sources + 1, B):
        raise ValueError("out must hold n_sources + 1 result slots")
    tab = None if missing is None else missing.table
    cap = 0 if missing is None else missing.capacity
    _check("fc_cache_search", LIB.fc_cache_search(
        C.byref(cache.view), _ptr(tab), cap, _ptr(ctx), stride, _ptr(ctx_len), B, p, n_sources,
        _ptr(out["drafts"]), _ptr(out["draft_len"]), _ptr(out["count"]), _ptr(out["n_drafts"]),
        _ptr(out["match_len"]), _ptr(state), _stream()))


def fc_missing_insert(missing: MissingTable, ctx, ctx_len, state, n_drafts, n_sources):
    """n_drafts: the [>= n_sources, B] retrieval counts (datastore slots first)."""
    B, stride = ctx.shape
    _need(n_drafts, torch.int32, "n_drafts")
    _check("fc_missing_insert", LIB.fc_missing_insert(
        _ptr(missing.table), missing.capacity, missing.key_len, _ptr(ctx), stride, _ptr(ctx_len), B, _ptr(state),
        _ptr(n_drafts), n_sources, _stream()))


def fc_cache_update(cache: SequenceCache, ctx, ctx_len_old, ctx_len_new, acc_len):
    B, stride = ctx.shape
    for t, nm in ((ctx_len_old, "ctx_len_old"), (ctx_len_new, "ctx_len_new"), (acc_len, "acc_len")):
        _need(t, torch.int32, nm, (B,))
    _check("fc_cache_update", LIB.fc_cache_update(C.byref(cache.view), _ptr(ctx), stride, _ptr(ctx_len_old),
                                                  _ptr(ctx_len_new), _ptr(acc_len), B, _stream()))


# -------------------------------------------------------------------- tree
def tree_outputs(batch, n_pad, device="cuda"):
    return dict(tok=torch.empty((batch, n_pad), dtype=torch.int32, device=device),
                parent=torch.empty((batch, n_pad), dtype=torch.int32, device=device),
                depth=torch.empty((batch, n_pad), dtype=torch.int32, device=device),
                pos=torch.empty((batch, n_pad), dtype=torch.int32, device=device),
                mask=torch.empty((batch, n_pad, n_pad // 64), dtype=torch.int64, device=device),
                n_nodes=torch.empty(batch, dtype=torch.int32, device=device))


def fc_build_tree(res, src_weight, root_tok, kv_len, node_budget, n_pad, out=None):
    """res: fc_retrieve outputs ([S, B, ...]); src_weight: S ints."""
    S, B, k, d = res["drafts"].shape
    _need(root_tok, torch.int32, "root_tok", (B,))
    _need(kv_len, torch.int32, "kv_len", (B,))
    w = (C.c_uint32 * S)(*[int(x) for x in src_weight])
    o = out if out is not None else tree_outputs(B, n_pad, root_tok.device)
    _check("fc_build_tree", LIB.fc_build_tree(S, _ptr(res["drafts"]), _ptr(res["draft_len"]), _ptr(res["count"]),
                                              _ptr(res["n_drafts"]), w, k, d, _ptr(root_tok), _ptr(kv_len), B,
                                              node_budget, n_pad, _ptr(o["tok"]), _ptr(o["parent"]),
                                              _ptr(o["depth"]), _ptr(o["pos"]), _ptr(o["mask"]), _ptr(o["n_nodes"]),
                                              _stream()))
    return o


def fc_build_tree_all(res, src_weight, root_tok, kv_len, node_budget, n_pad, workspace=None, out=None):
    """The all-occurrence trie over fc_retrieve_all's outputs ([S, B, slots, ...])."""
    S, B, k, d = res["drafts"].shape
    _need(root_tok, torch.int32, "root_tok", (B,))
    _need(kv_len, torch.int32, "kv_len", (B,))
    need = int(LIB.fc_build_tree_all_workspace(S, k, d, B))
    if need == 0:
        raise ValueError("unsupported shape for the all-occurrence trie")
    ws = workspace if workspace is not None else torch.empty(need, dtype=torch.uint8, device=root_tok.device)
    w = (C.c_uint32 * S)(*[int(x) for x in src_weight])
    o = out if out is not None else tree_outputs(B, n_pad, root_tok.device)
    _check("fc_build_tree_all", LIB.fc_build_tree_all(
        S, _ptr(res["drafts"]), _ptr(res["draft_len"]), _ptr(res["count"]), _ptr(res["n_drafts"]), w, k, d,
        _ptr(root_tok), _ptr(kv_len), B, node_budget, n_pad, _ptr(ws), ws.numel(), _ptr(o["tok"]), _ptr(o["parent"]),
        _ptr(o["depth"]), _ptr(o["pos"]), _ptr(o["mask"]), _ptr(o["n_nodes"]), _stream()))
    return o


def fc_tree_mask(parent, n_nodes, kv_len):
    _need(parent, torch.int32, "parent")
    B, n_pad = parent.shape
    _need(n_nodes, torch.int32, "n_nodes", (B,))
    _need(kv_len, torch.int32, "kv_len", (B,))
    dev = parent.device
    o = dict(depth=torch.empty((B, n_pad), dtype=torch.int32, device=dev),
             pos=torch.empty((B, n_pad), dtype=torch.int32, device=dev),
             mask=torch.empty((B, n_pad, n_pad // 64), dtype=torch.int64, device=dev))
    _check("fc_tree_mask", LIB.fc_tree_mask(_ptr(parent), _ptr(n_nodes), _ptr(kv_len), B, n_pad, _ptr(o["depth"]),
                                            _ptr(o["pos"]), _ptr(o["mask"]), _stream()))
    return o


# --------------------------------------------------------------- attention
_ATTN_WS = {}


def attn_workspace(B, Np, H, Hkv, device):
    """A cached device workspace of fc_tree_attn_workspace() bytes for this shape."""
    n = int(LIB.fc_tree_attn_workspace(B, Np, H, Hkv))
    key = (str(device), n)
    if key not in _ATTN_WS:
        _ATTN_WS[key] = torch.empty(max(n, 16), dtype=torch.uint8, device=device)
    return _ATTN_WS[key]


def fc_tree_attn(q, k_cache, v_cache, kv_len, k_tree, v_tree, mask, n_nodes, scale=None, out=None, workspace="auto"):
    """q [B, Np, H, D]; caches [B, Hkv, cap, D]; tree K/V [B, Hkv, Np, D] (bf16).

    ``workspace``: "auto" (a cached one of the full size, shared by every call
    with that size: calls that may overlap on different streams must each pass
    their own), None (no key split) or a uint8 device tensor."""
    _need(q, torch.bfloat16, "q")
    B, Np, H, D = q.shape
    _need(k_cache, torch.bfloat16, "k_cache")
    Hkv, cap = k_cache.shape[1], k_cache.shape[2]
    _need(v_cache, torch.bfloat16, "v_cache", k_cache.shape)
    _need(k_tree, torch.bfloat16, "k_tree", (B, Hkv, Np, D))
    _need(v_tree, torch.bfloat16, "v_tree", (B, Hkv, Np, D))
    _need(mask, torch.int64, "mask", (B, Np, Np // 64))
    _need(kv_len, torch.int32, "kv_len", (B,))
    _need(n_nodes, torch.int32, "n_nodes", (B,))
    o = out if out is not None else torch.empty_like(q)
    sc = float(scale) if scale is not None else D ** -0.5
    if isinstance(workspace, str):
        workspace = attn_workspace(B, Np, H, Hkv, q.device)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check("fc_tree_attn", LIB.fc_tree_attn(_ptr(q), _ptr(k_cache), _ptr(v_cache), cap, _ptr(kv_len), _ptr(k_tree),
                                            _ptr(v_tree), _ptr(mask), _ptr(n_nodes), B, Np, H, Hkv, D, sc, _ptr(o),
                                            _ptr(workspace), ws_bytes, _stream()))
    return o


def fc_rope(x, pos, base=10000.0, layout=None, out=None):
    """bf16 x [B, Np, heads, D] (layout 0, queries) or [B, heads, Np, D]
    (layout 1, tree keys; pass layout=1); pos int32 [B, Np].  Returns the
    rotated rows (``out`` may be ``x``)."""
    _need(x, torch.bfloat16, "x")
    B = x.shape[0]
    layout = 0 if layout is None else layout
    if layout == 0:
        _, Np, heads, D = x.shape
    else:
        _, heads, Np, D = x.shape
    _need(pos, torch.int32, "pos", (B, Np))
    o = out if out is not None else torch.empty_like(x)
    _check("fc_rope", LIB.fc_rope(_ptr(x), _ptr(o), B, Np, heads, D, layout, _ptr(pos), C.c_float(base), _stream()))
    return o


def fc_tree_attn_rope(q, k_cache, v_cache, kv_len, k_tree_rot, v_tree, mask, n_nodes, pos, rope_base=10000.0,
                      scale=None, out=None, workspace="auto"):
    """fc_tree_attn with unrotated q (rotated in the kernel by pos [B, Np]);
    k_tree_rot: the tree keys rotated by fc_rope(..., layout=1)."""
    _need(q, torch.bfloat16, "q")
    B, Np, H, D = q.shape
    _need(k_cache, torch.bfloat16, "k_cache")
    Hkv, cap = k_cache.shape[1], k_cache.shape[2]
    _need(v_cache, torch.bfloat16, "v_cache", k_cache.shape)
    _need(k_tree_rot, torch.bfloat16, "k_tree_rot", (B, Hkv, Np, D))
    _need(v_tree, torch.bfloat16, "v_tree", (B, Hkv, Np, D))
    _need(mask, torch.int64, "mask", (B, Np, Np // 64))
    _need(kv_len, torch.int32, "kv_len", (B,))
    _need(n_nodes, torch.int32, "n_nodes", (B,))
    _need(pos, torch.int32, "pos", (B, Np))
    o = out if out is not None else torch.empty_like(q)
    sc = float(scale) if scale is not None else D ** -0.5
    if isinstance(workspace, str):
        workspace = attn_workspace(B, Np, H, Hkv, q.device)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check("fc_tree_attn_rope", LIB.fc_tree_attn_rope(
        _ptr(q), _ptr(k_cache), _ptr(v_cache), cap, _ptr(kv_len), _ptr(k_tree_rot), _ptr(v_tree), _ptr(mask),
        _ptr(n_nodes), B, Np, H, Hkv, D, sc, _ptr(pos), C.c_float(rope_base), _ptr(o), _ptr(workspace), ws_bytes,
        _stream()))
    return o


# ------------------------------------------------------- decoder blocks
def fc_gemm_bf16(a, b, out=None):
    """a [M, K] @ b [K, N] (bf16, row-major) -> [M, N] bf16 (the library's
    tcgen05 GEMM; it needs no workspace)."""
    _need(a, torch.bfloat16, "a")
    _need(b, torch.bfloat16, "b")
    M, K = a.shape
    K2, N = b.shape
    if K != K2:
        raise ValueError("inner dimensions differ")
    o = out if out is not None else torch.empty((M, N), dtype=torch.bfloat16, device=a.device)
    _need(o, torch.bfloat16, "out")
    if tuple(o.shape) != (M, N):
        raise ValueError("out must be [M, N]")
    _check("fc_gemm_bf16", LIB.fc_gemm_bf16(_ptr(a), _ptr(b), _ptr(o), M, N, K, None, 0, _stream()))
    return o


def fc_gemm_kv_heads(a, wkv, batch, n_pad, Hkv, pos, rope_base, k_rot, v_heads):
    """kv = a [batch * n_pad, K] @ wkv [K, 2 * Hkv * 128]; key heads rotated by
    pos [batch, n_pad] into k_rot, value heads into v_heads (both
    [batch, Hkv, n_pad, 128], bf16)."""
    _need(a, torch.bfloat16, "a")
    _need(wkv, torch.bfloat16, "wkv")
    _need(pos, torch.int32, "pos", (batch, n_pad))
    M, K = a.shape
    D = 128
    if tuple(wkv.shape) != (K, 2 * Hkv * D):
        raise ValueError("wkv must be [K, 2 * Hkv * 128]")
    for t, name in ((k_rot, "k_rot"), (v_heads, "v_heads")):
        _need(t, torch.bfloat16, name, (batch, Hkv, n_pad, D))
    _check("fc_gemm_kv_heads", LIB.fc_gemm_kv_heads(_ptr(a), _ptr(wkv), M, K, Hkv, D, batch, n_pad, _ptr(pos),
                                                    C.c_float(rope_base), _ptr(k_rot), _ptr(v_heads), _stream()))


def fc_interleave_gate_up(wgu, out=None):
    """[K, 2 * inter] gate|up weights -> 128-column blocks interleaved, for
    fc_gemm_silu_mul."""
    _need(wgu, torch.bfloat16, "wgu")
    K, n2 = wgu.shape
    o = out if out is not None else torch.empty_like(wgu)
    _check("fc_interleave_gate_up", LIB.fc_interleave_gate_up(_ptr(wgu), _ptr(o), K, n2 // 2, _stream()))
    return o


def fc_gemm_silu_mul(a, wgu_interleaved, out):
    """out [M, inter] = silu(a @ Wg) * (a @ Wu), with the weights interleaved by
    fc_interleave_gate_up."""
    _need(a, torch.bfloat16, "a")
    _need(wgu_interleaved, torch.bfloat16, "wgu_interleaved")
    M, K = a.shape
    inter = wgu_interleaved.shape[1] // 2
    _need(out, torch.bfloat16, "out", (M, inter))
    _check("fc_gemm_silu_mul", LIB.fc_gemm_silu_mul(_ptr(a), _ptr(wgu_interleaved), M, K, inter, _ptr(out),
                                                    _stream()))
    return out


def fc_embed(tok, table, out):
    _need(tok, torch.int32, "tok")
    vocab, hidden = table.shape
    _check("fc_embed", LIB.fc_embed(_ptr(tok), tok.numel(), _ptr(table), vocab, hidden, _ptr(out), _stream()))
    return out


def fc_add_rmsnorm(x, r, w, out, eps=1e-6):
    """x += r (if r is not None), out = rmsnorm(x) * w; x, r, out [rows, dim]."""
    rows, dim = x.shape
    _check("fc_add_rmsnorm", LIB.fc_add_rmsnorm(_ptr(x), _ptr(r), _ptr(w), _ptr(out), rows, dim, C.c_float(eps),
                                                _stream()))
    return out


def fc_silu_mul(gu, out):
    rows, two_inter = gu.shape
    _check("fc_silu_mul", LIB.fc_silu_mul(_ptr(gu), _ptr(out), rows, two_inter // 2, _stream()))
    return out


def fc_rope_heads(x, col0, stride, out, B, n_pad, heads, D, pos, base):
    """Node-major rows of x (row stride ``stride`` elements, head h at column
    col0 + h*D) -> head-major out [B, heads, n_pad, D], rotated by pos when
    base > 0."""
    ptr = C.c_void_p(x.data_ptr() + col0 * x.element_size())
    _check("fc_rope_heads", LIB.fc_rope_heads(ptr, stride, _ptr(out), B, n_pad, heads, D, _ptr(pos), C.c_float(base),
                                              _stream()))
    return out


# ---------------------------------------------------------- accept / append
def fc_accept(tok, parent, n_nodes, argmax, path_cap, out=None):
    B, Np = tok.shape
    for t, nm in ((tok, "tok"), (parent, "parent"), (argmax, "argmax")):
        _need(t, torch.int32, nm, (B, Np))
    _need(n_nodes, torch.int32, "n_nodes", (B,))
    dev = tok.device
    o = out if out is not None else dict(acc_len=torch.empty(B, dtype=torch.int32, device=dev),
                                         path=torch.empty((B, path_cap), dtype=torch.int32, device=dev),
                                         bonus=torch.empty(B, dtype=torch.int32, device=dev))
    _check("fc_accept", LIB.fc_accept(_ptr(tok), _ptr(parent), _ptr(n_nodes), _ptr(argmax), B, Np, _ptr(o["acc_len"]),
                                      _ptr(o["path"]), path_cap, _ptr(o["bonus"]), _stream()))
    return o


def fc_argmax_accept(logits, tok, parent, n_nodes, path_cap, out=None):
    """logits bf16 [B, Np, V]; returns dict(argmax [B, Np], acc_len, path, bonus) (int32)."""
    _need(logits, torch.bfloat16, "logits")
    B, Np, V = logits.shape
    for t, nm in ((tok, "tok"), (parent, "parent")):
        _need(t, torch.int32, nm, (B, Np))
    _need(n_nodes, torch.int32, "n_nodes", (B,))
    dev = tok.device
    o = out if out is not None else dict(argmax=torch.empty((B, Np), dtype=torch.int32, device=dev),
                                         acc_len=torch.empty(B, dtype=torch.int32, device=dev),
                                         path=torch.empty((B, path_cap), dtype=torch.int32, device=dev),
                                         bonus=torch.empty(B, dtype=torch.int32, device=dev))
    _check("fc_argmax_accept", LIB.fc_argmax_accept(_ptr(logits), V, _ptr(tok), _ptr(parent), _ptr(n_nodes), B, Np,
                                                    _ptr(o["argmax"]), _ptr(o["acc_len"]), _ptr(o["path"]), path_cap,
                                                    _ptr(o["bonus"]), _stream()))
    return o


def fc_kv_append(acc, tok, k_tree, v_tree, k_cache, v_cache, kv_len_in, kv_len_out, ctx, ctx_len_in, ctx_len_out,
                 root_out):
    B, Hkv, Np, D = k_tree.shape
    cap = k_cache.shape[2]
    _need(ctx, torch.int32, "ctx")
    _check("fc_kv_append", LIB.fc_kv_append(
        _ptr(acc["path"]), _ptr(acc["acc_len"]), _ptr(acc["bonus"]), _ptr(tok), _ptr(k_tree), _ptr(v_tree), B, Np, Hkv,
        D, acc["path"].shape[1], _ptr(k_cache), _ptr(v_cache), cap, _ptr(kv_len_in), _ptr(kv_len_out), _ptr(ctx),
        ctx.shape[1], _ptr(ctx_len_in), _ptr(ctx_len_out), _ptr(root_out), _stream()))


def fc_synth_argmax(tok, parent, n_nodes, plen, rtok, vocab, out=None):
    B, Np = tok.shape
    o = out if out is not None else torch.empty((B, Np), dtype=torch.int32, device=tok.device)
    _check("fc_synth_argmax", LIB.fc_synth_argmax(_ptr(tok), _ptr(parent), _ptr(n_nodes), B, Np, _ptr(plen),
                                                  _ptr(rtok), vocab, _ptr(o), _stream()))
    return o


# ------------------------------------------------------ native step executor
PIPELINE_NO_ATTENTION = 1
_PIPELINES = weakref.WeakSet()
_GRAPHS = weakref.WeakSet()


@atexit.register
def _close_pipelines():
    # before the CUDA runtime shuts down: destroying graphs and streams later is unsafe
    for g in list(_GRAPHS):
        g.close()
    for pl in list(_PIPELINES):
        pl.close()


def pipeline_part(batch, first, ctx, ctx_len, kv_len, root, rcache, skip, res, tree, k_cache, v_cache, k_tree_rot,
                  attn_out, attn_ws, argmax, acc, err=None, seq_cache=None, missing=None) -> fc_pipeline_part:
    """One sub-batch's buffers (device tensors the caller keeps alive):
    ctx_len and kv_len are pairs (the ping-pong lengths), rcache a
    RetrievalCache or None, res/tree/acc the dicts of retrieve_outputs,
    tree_outputs and fc_accept's outputs, err None or a zeroed one-element
    int32 tensor: the sub-batch's own error word.  seq_cache / missing: a
    SequenceCache and MissingTable (Algorithm 1, in place of rcache); res
    then holds one more slot, the CACHE's."""
    if err is not None:
        _need(err, torch.int32, "err", (1,))
    if seq_cache is not None and seq_cache.batch != batch:
        raise ValueError("the CACHE must cover the sub-batch")
    _need(ctx, torch.int32, "ctx", (batch, ctx.shape[1]))
    for t in (*ctx_len, *kv_len, root, skip):
        _need(t, torch.int32, "length", (batch,))
    _need(k_cache, torch.bfloat16, "k_cache")
    _need(v_cache, torch.bfloat16, "v_cache", tuple(k_cache.shape))
    return fc_pipeline_part(
        batch, first, _ptr(ctx), ctx.shape[1], (C.c_void_p * 2)(*[t.data_ptr() for t in ctx_len]),
        (C.c_void_p * 2)(*[t.data_ptr() for t in kv_len]), _ptr(root), _ptr(rcache.table) if rcache else None,
        rcache.capacity if rcache else 0, _ptr(skip), _ptr(res["drafts"]), _ptr(res["draft_len"]), _ptr(res["count"]),
        _ptr(res["n_drafts"]), _ptr(res["match_len"]), _ptr(tree["tok"]), _ptr(tree["parent"]), _ptr(tree["depth"]),
        _ptr(tree["pos"]), _ptr(tree["mask"]), _ptr(tree["n_nodes"]), _ptr(k_cache), _ptr(v_cache), _ptr(k_tree_rot),
        _ptr(attn_out), _ptr(attn_ws), 0 if attn_ws is None else attn_ws.numel() * attn_ws.element_size(),
        _ptr(argmax), _ptr(acc["acc_len"]), _ptr(acc["path"]), _ptr(acc["bonus"]), _ptr(err),
        seq_cache.view if seq_cache is not None else fc_cache(), _ptr(missing.table) if missing else None,
        missing.capacity if missing else 0)


class PipelineGraph:
    """fc_pipeline_graph: captured steps of one sub-batch (Pipeline.capture).
    It keeps its executor and input tensors alive."""

    def __init__(self, handle, pipe, inputs):
        self.handle, self._pipe, self._inputs = handle, pipe, inputs
        self._destroy = LIB.fc_pipeline_graph_destroy
        _GRAPHS.add(self)

    def launch(self):
        """Launch into the current stream."""
        _check("fc_pipeline_graph_launch", LIB.fc_pipeline_graph_launch(self.handle, _stream()))

    def kernels(self):
        """(kernel nodes at the chain stream's priority, at the attention stream's)."""
        a, b = C.c_int(), C.c_int()
        _check("fc_pipeline_graph_kernels", LIB.fc_pipeline_graph_kernels(self.handle, C.byref(a), C.byref(b)))
        return a.value, b.value

    def close(self):
        if getattr(self, "handle", None):
            self._destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class Pipeline:
    """fc_pipeline: the native step executor over sub-batches.  ``parts`` are
    pipeline_part() descriptions; their tensors must outlive this object."""

    def __init__(self, sources, p: fc_retrieve_params, src_weight, node_budget, n_pad, H, Hkv, D, kv_cap, path_cap,
                 vocab, parts, scale=None, rope_base=None):
        S = len(sources)
        if len(src_weight) not in (S, S + 1):
            raise ValueError("one tree weight per source, and optionally the CACHE slot's")
        self.B = sum(pt.batch for pt in parts)
        self.shapes = ((self.B, n_pad, H, D), (self.B, Hkv, n_pad, D), (self.B,), (self.B, n_pad))
        views = (fc_datastore * S)(*[s.view for s in sources])
        w = (C.c_uint32 * S)(*[int(x) for x in src_weight[:S]])
        arr = (fc_pipeline_part * len(parts))(*parts)
        desc = fc_pipeline_desc(views, S, p, w, node_budget, n_pad, H, Hkv, D, kv_cap, path_cap, vocab,
                                float(scale) if scale is not None else D ** -0.5,
                                0.0 if rope_base is None else float(rope_base), len(parts), arr,
                                int(src_weight[S]) if len(src_weight) > S else 1)
        h = C.c_void_p()
        _check("fc_pipeline_create", LIB.fc_pipeline_create(C.byref(desc), C.byref(h)))
        self.handle = h
        self.n_parts = len(parts)
        self._destroy = LIB.fc_pipeline_destroy
        # each sub-batch's chain stream, for work that must follow its steps
        self.streams = [torch.cuda.ExternalStream(LIB.fc_pipeline_stream(h, i)) for i in range(len(parts))]
        _PIPELINES.add(self)

    def step(self, phase, q, k_tree, v_tree, want_hit, plen, rtok, attention=True, events=None, part=None):
        """Enqueue one step of every sub-batch (or of sub-batch ``part``
        alone) after the work on the current stream (inputs batch-wide, as
        fc_pipeline_step); ``events``: None or, per sub-batch, a dict mapping
        "retrieve" / "tree" / "attn" / "tail" to a (start, end) pair of
        torch.cuda.Event."""
        qs, ks, bs, rs = self.shapes
        if attention:
            _need(q, torch.bfloat16, "q", qs)
        _need(k_tree, torch.bfloat16, "k_tree", ks)
        _need(v_tree, torch.bfloat16, "v_tree", ks)
        _need(plen, torch.int32, "plen", bs)
        _need(rtok, torch.int32, "rtok", rs)
        if want_hit is not None:
            _need(want_hit, torch.int32, "want_hit", bs)
        ev = None
        if events is not None:
            ev = (C.c_void_p * (8 * self.n_parts))()
            for h, e in enumerate(events):
                for j, nm in enumerate(("retrieve", "tree", "attn", "tail")):
                    for k in range(2):
                        if e and nm in e:
                            t = e[nm][k]
                            if not t.cuda_event:  # torch creates its events at the first record
                                t.record()
                            ev[8 * h + 2 * j + k] = t.cuda_event
        args = (phase, 0 if attention else PIPELINE_NO_ATTENTION, _ptr(q) if attention else None, _ptr(k_tree),
                _ptr(v_tree), _ptr(want_hit), _ptr(plen), _ptr(rtok), _stream(), ev)
        if part is None:
            _check("fc_pipeline_step", LIB.fc_pipeline_step(self.handle, *args))
        else:
            _check("fc_pipeline_step_part", LIB.fc_pipeline_step_part(self.handle, part, *args))

    def join(self, part=None):
        """The current stream waits for everything enqueued on the sub-batches
        (or on sub-batch ``part``)."""
        if part is None:
            _check("fc_pipeline_join", LIB.fc_pipeline_join(self.handle, _stream()))
        else:
            _check("fc_pipeline_join_part", LIB.fc_pipeline_join_part(self.handle, part, _stream()))

    def capture(self, part, inputs, phase0=0, attention=True):
        """A CUDA graph of len(inputs) steps of sub-batch ``part`` (inputs:
        tuples (q, k_tree, v_tree, want_hit, plen, rtok) of batch-wide device
        tensors, read at every launch; q may be None without attention),
        whose kernels keep their streams' priorities (fc_pipeline_capture_part).
        Returns a PipelineGraph; launching it advances the sub-batch."""
        qs, ks, bs, rs = self.shapes
        n = len(inputs)
        arrs = [(C.c_void_p * n)() for _ in range(6)]
        for t, (q, kt, vt, wh, pl, rt) in enumerate(inputs):
            if attention:
                _need(q, torch.bfloat16, "q", qs)
            _need(kt, torch.bfloat16, "k_tree", ks)
            _need(vt, torch.bfloat16, "v_tree", ks)
            _need(pl, torch.int32, "plen", bs)
            _need(rt, torch.int32, "rtok", rs)
            if wh is not None:
                _need(wh, torch.int32, "want_hit", bs)
            for a, x in zip(arrs, (q if attention else None, kt, vt, wh, pl, rt)):
                a[t] = _ptr(x)
        g = C.c_void_p()
        want = None if all(w is None for _, _, _, w, _, _ in inputs) else arrs[3]
        _check("fc_pipeline_capture_part", LIB.fc_pipeline_capture_part(
            self.handle, part, n, phase0, 0 if attention else PIPELINE_NO_ATTENTION, arrs[0] if attention else None,
            arrs[1], arrs[2], want, arrs[4], arrs[5], C.byref(g)))
        return PipelineGraph(g, self, inputs)

    def error(self, part):
        """Sub-batch ``part``'s device errors since the last call (a status
        name; waits for its work, clears its word)."""
        code = LIB.fc_pipeline_error(self.handle, part)
        return STATUS.get(code, str(code))

    def close(self):
        if getattr(self, "handle", None):
            self._destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
