"""The target model's forward over a draft tree (Section IV-D: one forward
verifies every draft, each token attending to the cached context and to its
own tree ancestors, at position kv_len + depth), for a LLaMA-family decoder
like the paper's models (DeepSeek-Coder, CodeLlama): RMSNorm, rotary
position embedding (O12), grouped-query attention, a SiLU-gated MLP, a final
RMSNorm and the LM head.

TEST INFRASTRUCTURE ONLY: imported by tests/, never by the product package.
Plain numpy in float64: matmuls are library primitives, every other step is
written out.  Weights arrive as bf16 bit patterns (uint16) from the seeded
generator and are widened exactly.

Layout and conventions (shared with the GPU path as interface facts):
  * a layer's weights: attn_norm [hidden], wq [hidden][H*D], wkv
    [hidden][2*Hkv*D] (the K columns, then the V columns), wo [H*D][hidden],
    mlp_norm [hidden], wgu [hidden][2*inter] (gate, then up), wd
    [inter][hidden]; globals embed [vocab][hidden], final_norm [hidden],
    lm_head [hidden][vocab].  A projection is x @ W.
  * RMSNorm(x) = x / sqrt(mean(x^2) + eps) * w.
  * MLP(x) = (silu(x Wg) * (x Wu)) Wd, silu(z) = z / (1 + exp(-z)).
  * attention scale 1/sqrt(D); query head h uses kv head h // (H / Hkv).
  * cached keys are stored rotated (at their own positions); a token with id
    >= vocab (tree padding) embeds as zeros.
"""
from __future__ import annotations

import dataclasses

import numpy as np

from . import oracle as O


@dataclasses.dataclass
class DecoderConfig:
    hidden: int
    layers: int
    H: int
    Hkv: int
    inter: int
    vocab: int
    D: int = 128
    eps: float = 1e-6
    rope_base: float = 10000.0


def widen(b16):
    """bf16 bit patterns (uint16) -> float64, exactly."""
    b16 = np.ascontiguousarray(b16, np.uint16)
    return (b16.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def round_bf16(x):
    """Nearest bf16 value (ties to even) of each element, as float64.  Used
    only by forward(..., store_bf16=True)."""
    f = np.ascontiguousarray(x, np.float64).astype(np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    lsb = (u >> 16) & 1
    r = ((u + 0x7FFF + lsb) >> 16) << 16
    return r.astype(np.uint32).view(np.float32).astype(np.float64)


def rmsnorm(x, w, eps):
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * w


def silu(z):
    return z / (1.0 + np.exp(-z))


def tree_attention(q, k_cache, v_cache, kv_len, k_tree, v_tree, ancestors, n_nodes, pos, cfg):
    """One sequence: q [n, H, D] (unrotated), k_cache/v_cache [Hkv, L, D]
    (cached keys rotated), k_tree/v_tree [n, Hkv, D] (unrotated keys),
    ancestors[i] = the nodes node i attends to (its ancestors and itself),
    pos [n].  Returns [n, H, D]."""
    G = cfg.H // cfg.Hkv
    out = np.zeros((n_nodes, cfg.H, cfg.D))
    qr = O.rope(q[:n_nodes], np.repeat(pos[:n_nodes, None], cfg.H, 1), cfg.rope_base)
    kr = O.rope(k_tree[:n_nodes], np.repeat(pos[:n_nodes, None], cfg.Hkv, 1), cfg.rope_base)
    scale = 1.0 / np.sqrt(cfg.D)
    for i in range(n_nodes):
        anc = ancestors[i]
        for h in range(cfg.H):
            g = h // G
            keys = np.concatenate([k_cache[g, :kv_len], kr[anc, g]], 0)
            vals = np.concatenate([v_cache[g, :kv_len], v_tree[anc, g]], 0)
            s = keys @ qr[i, h] * scale
            p = np.exp(s - s.max())
            out[i, h] = (p / p.sum()) @ vals
    return out


def ancestors_of(parent, n):
    """ancestors[i]: node i and every node on its path to the root (ascending)."""
    res = []
    for i in range(n):
        path, j = [], i
        while j >= 0:
            path.append(j)
            j = int(parent[j])
        res.append(sorted(path))
    return res


def forward(cfg, W, tokens, parent, n_nodes, kv_len, k_caches, v_caches, pos, store_bf16=False):
    """The tree forward for a batch.  W: dict of float64 weights (widened),
    with W["layers"][l] a dict per layer.  tokens/parent/pos [B][n_pad];
    k_caches/v_caches [L][B][Hkv][cap][D] (float64, keys rotated).  Returns
    (logits [B][n_pad][vocab] with padding rows zero, k_new [L][B][n_pad][Hkv][D]
    rotated tree keys, v_new [L][B][n_pad][Hkv][D]).

    store_bf16: round every intermediate to bf16 where a bf16 forward stores
    it (the residual stream after each add, each norm's output, the query,
    output and down projections, the rotated keys and the values, the
    attention output, the MLP activation and the logits), fp64 otherwise;
    the key/value and gate/up projections are consumed unrounded by the
    rotation and by SiLU * up.  The paper states no precision; this
    variant measures how far bf16 storage alone moves the result, which sizes
    the tolerance of a bf16 forward against the fp64 one."""
    rb = round_bf16 if store_bf16 else (lambda a: a)
    B, n_pad = tokens.shape
    logits = np.zeros((B, n_pad, cfg.vocab))
    k_new = np.zeros((cfg.layers, B, n_pad, cfg.Hkv, cfg.D))
    v_new = np.zeros((cfg.layers, B, n_pad, cfg.Hkv, cfg.D))
    for b in range(B):
        n = int(n_nodes[b])
        anc = ancestors_of(parent[b], n)
        ids = np.asarray(tokens[b, :n], np.int64)
        x = np.zeros((n, cfg.hidden))
        ok = ids < cfg.vocab
        x[ok] = W["embed"][ids[ok]]
        for l, Lw in enumerate(W["layers"]):
            h = rb(rmsnorm(x, Lw["attn_norm"], cfg.eps))
            q = rb(h @ Lw["wq"]).reshape(n, cfg.H, cfg.D)
            kv = (h @ Lw["wkv"]).reshape(n, 2, cfg.Hkv, cfg.D)
            k, v = kv[:, 0], rb(kv[:, 1])
            k_new[l, b, :n] = rb(O.rope(k, np.repeat(pos[b, :n, None], cfg.Hkv, 1), cfg.rope_base))
            v_new[l, b, :n] = v
            a = rb(tree_attention(q, k_caches[l][b], v_caches[l][b], int(kv_len[b]), k, v, anc, n, pos[b], cfg))
            x = rb(x + rb(a.reshape(n, cfg.H * cfg.D) @ Lw["wo"]))
            h = rb(rmsnorm(x, Lw["mlp_norm"], cfg.eps))
            gu = h @ Lw["wgu"]
            x = rb(x + rb(rb(silu(gu[:, :cfg.inter]) * gu[:, cfg.inter:]) @ Lw["wd"]))
        logits[b, :n] = rb(rb(rmsnorm(x, W["final_norm"], cfg.eps)) @ W["lm_head"])
    return logits, k_new, v_new


def widen_weights(Wb):
    """The generator's bf16 weights (uint16 arrays) -> float64, same structure."""
    out = {k: widen(v) for k, v in Wb.items() if k != "layers"}
    out["layers"] = [{k: widen(v) for k, v in Lw.items()} for Lw in Wb["layers"]]
    return out
