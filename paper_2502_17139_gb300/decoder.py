"""The target model's forward over a draft tree (Section IV-D: one forward
verifies every draft, each token attending to the cached context and to its
tree ancestors at position kv_len + depth), for a LLaMA-family decoder like
the paper's models, composed from the C-ABI calls (argument marshalling
only; every step runs in the library's kernels).

Per layer: add + RMSNorm -> Q projection -> the K/V projection, whose GEMM
epilogue rotates the key heads and writes both head-major (fc_gemm_kv_heads)
-> tree attention with the queries rotated inside the kernel
(fc_tree_attn_rope) over the layer's rotated cache -> output projection ->
add + RMSNorm -> the gate/up projection, whose GEMM epilogue applies SiLU *
up (fc_gemm_silu_mul, weights interleaved once at construction) -> down
projection.  The residual adds are fused into the next norm; after the last
layer the final norm feeds the LM head.  The tree's rotated keys and values
of every layer stay in buffers until the accepted path is appended to the
caches.
"""
from __future__ import annotations

import dataclasses

import torch

from . import fastcoder as fc


@dataclasses.dataclass
class DecoderShape:
    hidden: int
    layers: int
    H: int
    Hkv: int
    inter: int
    vocab: int
    D: int = 128
    eps: float = 1e-6
    rope_base: float = 10000.0


# DeepSeek-Coder 1.3B, one of the paper's models (Section V-A)
DEEPSEEK_CODER_1_3B = DecoderShape(hidden=2048, layers=24, H=16, Hkv=16, inter=5504, vocab=32256)


class TreeDecoder:
    """Weights W (synth.decoder_weights layout, bf16 on the device), per-layer
    KV caches [B, Hkv, kv_cap, D] and the step's buffers."""

    def __init__(self, shape: DecoderShape, W, B, n_pad, kv_cap, device="cuda", caches=None):
        self.s, self.W, self.B, self.n_pad, self.kv_cap = shape, W, B, n_pad, kv_cap
        s = shape
        T = B * n_pad
        bf = dict(dtype=torch.bfloat16, device=device)
        if caches is None:
            caches = [(torch.zeros((B, s.Hkv, kv_cap, s.D), **bf), torch.zeros((B, s.Hkv, kv_cap, s.D), **bf))
                      for _ in range(s.layers)]
        self.k_cache = [c[0] for c in caches]
        self.v_cache = [c[1] for c in caches]
        self.x = torch.empty((T, s.hidden), **bf)
        self.h = torch.empty((T, s.hidden), **bf)
        self.q = torch.empty((T, s.H * s.D), **bf)
        # the gate/up weights in the 128-column interleave fc_gemm_silu_mul reads
        self.wgu = [fc.fc_interleave_gate_up(Lw["wgu"]) for Lw in W["layers"]]
        self.k_rot = [torch.empty((B, s.Hkv, n_pad, s.D), **bf) for _ in range(s.layers)]
        self.v_heads = [torch.empty((B, s.Hkv, n_pad, s.D), **bf) for _ in range(s.layers)]
        self.attn = torch.empty((T, s.H * s.D), **bf)
        self.o = torch.empty((T, s.hidden), **bf)
        self.act = torch.empty((T, s.inter), **bf)
        self.logits = torch.empty((T, s.vocab), **bf)

    def forward(self, tok, n_nodes, mask, pos, kv_len, events=None):
        """tok [B, n_pad] (int32; padding >= vocab), n_nodes [B], mask
        [B, n_pad, n_pad/64], pos [B, n_pad], kv_len [B].  Returns the logits
        [B, n_pad, vocab] (rows past a tree's node count are not meaningful).
        ``events`` optionally maps "attn" to a list that receives one
        (start, end) CUDA-event pair per layer around the attention."""
        s, W, B, n_pad = self.s, self.W, self.B, self.n_pad
        fc.fc_embed(tok.reshape(-1), W["embed"], self.x)
        r = None
        for l, Lw in enumerate(W["layers"]):
            fc.fc_add_rmsnorm(self.x, r, Lw["attn_norm"], self.h, s.eps)
            fc.fc_gemm_bf16(self.h, Lw["wq"], out=self.q)
            fc.fc_gemm_kv_heads(self.h, Lw["wkv"], B, n_pad, s.Hkv, pos, s.rope_base, self.k_rot[l], self.v_heads[l])
            ev = None
            if events is not None and "attn" in events:
                ev = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                events["attn"].append(ev)
                ev[0].record()
            fc.fc_tree_attn_rope(self.q.view(B, n_pad, s.H, s.D), self.k_cache[l], self.v_cache[l], kv_len,
                                 self.k_rot[l], self.v_heads[l], mask, n_nodes, pos, s.rope_base,
                                 out=self.attn.view(B, n_pad, s.H, s.D))
            if ev is not None:
                ev[1].record()
            fc.fc_gemm_bf16(self.attn, Lw["wo"], out=self.o)
            fc.fc_add_rmsnorm(self.x, self.o, Lw["mlp_norm"], self.h, s.eps)
            fc.fc_gemm_silu_mul(self.h, self.wgu[l], self.act)
            fc.fc_gemm_bf16(self.act, Lw["wd"], out=self.o)
            r = self.o
        fc.fc_add_rmsnorm(self.x, r, W["final_norm"], self.h, s.eps)
        fc.fc_gemm_bf16(self.h, W["lm_head"], out=self.logits)
        return self.logits.view(B, n_pad, s.vocab)

    def append(self, acc, tok, kv_len_in, kv_len_out, ctx, ctx_len_in, ctx_len_out, root):
        """The accepted path's rotated keys and values into every layer's cache
        (the context update repeats per layer and writes the same tokens)."""
        for l in range(self.s.layers):
            fc.fc_kv_append(acc, tok, self.k_rot[l], self.v_heads[l], self.k_cache[l], self.v_cache[l], kv_len_in,
                            kv_len_out, ctx, ctx_len_in, ctx_len_out, root)
