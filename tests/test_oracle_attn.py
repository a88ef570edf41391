"""Pins for the oracle's tree attention (O6, Section IV-D Eq. 4).

* a chain tree (mask = lower-triangular ones) equals ordinary causal
  attention over [cache; chain], computed here by a separate plain loop;
* a single node equals one-token decode attention;
* kv_len = 0 leaves only the tree keys;
* torch.nn.functional.scaled_dot_product_attention in float64 on the CPU,
  with the boolean tree mask and GQA by repeated K/V heads, agrees to 1e-12;
* rows at or beyond n_nodes are zero and the sampled-row mode equals the
  full mode.
"""
import numpy as np
import pytest
import torch


def bf16_bits(x: torch.Tensor) -> np.ndarray:
    return x.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def bits_to_f64(a: np.ndarray) -> np.ndarray:
    return (a.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def _case(seed, B, n_pad, H, Hkv, D, cap):
    g = torch.Generator().manual_seed(seed)
    q = torch.randn(B, n_pad, H, D, generator=g)
    kc = torch.randn(B, Hkv, cap, D, generator=g)
    vc = torch.randn(B, Hkv, cap, D, generator=g)
    kt = torch.randn(B, Hkv, n_pad, D, generator=g)
    vt = torch.randn(B, Hkv, n_pad, D, generator=g)
    return [bf16_bits(x) for x in (q, kc, vc, kt, vt)]


def _chain_mask(B, n_pad, n):
    nw = (n_pad + 63) // 64
    m = np.zeros((B, n_pad, nw), np.uint64)
    for i in range(n):
        for j in range(i + 1):
            m[:, i, j // 64] |= np.uint64(1) << np.uint64(j % 64)
    return m


def test_chain_equals_causal_attention(orc):
    B, n_pad, H, D, cap, L, n = 2, 64, 2, 16, 40, 33, 64
    q, kc, vc, kt, vt = _case(1, B, n_pad, H, H, D, cap)
    mask = _chain_mask(B, n_pad, n)
    out = orc.tree_attn(q, kc, vc, np.full(B, L, np.int32), kt, vt, mask, np.full(B, n, np.int32))
    Q, K, V = bits_to_f64(q), np.concatenate([bits_to_f64(kc)[:, :, :L], bits_to_f64(kt)], 2), \
        np.concatenate([bits_to_f64(vc)[:, :, :L], bits_to_f64(vt)], 2)
    scale = 1.0 / np.sqrt(D)
    for b in range(B):
        for h in range(H):
            for i in range(n):
                # causal attention of position L + i over positions 0..L+i
                s = [scale * sum(Q[b, i, h, x] * K[b, h, j, x] for x in range(D)) for j in range(L + i + 1)]
                mx = max(s)
                e = [np.exp(v - mx) for v in s]
                tot = sum(e)
                ref = [sum(e[j] * V[b, h, j, x] for j in range(L + i + 1)) / tot for x in range(D)]
                assert np.allclose(out[b, i, h], ref, rtol=0, atol=1e-12)


def test_single_node_is_decode_attention(orc):
    B, n_pad, H, D, cap, L = 3, 64, 4, 32, 50, 50
    q, kc, vc, kt, vt = _case(2, B, n_pad, H, H, D, cap)
    mask = _chain_mask(B, n_pad, 1)
    out = orc.tree_attn(q, kc, vc, np.full(B, L, np.int32), kt, vt, mask, np.ones(B, np.int32))
    Q, K, V = bits_to_f64(q), bits_to_f64(kc), bits_to_f64(vc)
    Kt, Vt = bits_to_f64(kt), bits_to_f64(vt)
    for b in range(B):
        for h in range(H):
            Kall = np.concatenate([K[b, h, :L], Kt[b, h, :1]])
            Vall = np.concatenate([V[b, h, :L], Vt[b, h, :1]])
            s = Kall @ Q[b, 0, h] / np.sqrt(D)
            p = np.exp(s - s.max())
            np.testing.assert_allclose(out[b, 0, h], p @ Vall / p.sum(), rtol=0, atol=1e-12)
    assert (out[:, 1:] == 0).all()


def _tree_inputs(orc, seed, B, n_pad, kvl):
    import paper_2502_17139_gb300.synth as synth
    rng = synth.rng_for(94, seed)
    par = np.full((B, n_pad), -1, np.int32)
    nn = rng.integers(1, n_pad + 1, B).astype(np.int32)
    for b in range(B):
        _, p = synth.random_tree(rng, int(nn[b]), 10, 4, 1000)
        par[b, :nn[b]] = p
    return orc.tree_mask(par, nn, kvl, n_pad)["mask"], nn


@pytest.mark.parametrize("H,Hkv,n_pad", [(4, 4, 64), (8, 2, 64), (4, 1, 128)])
def test_sdpa_fp64_library_pin(orc, H, Hkv, n_pad):
    B, D, cap = 3, 32, 70
    kvl = np.array([0, 17, 70], np.int32)
    q, kc, vc, kt, vt = _case(3, B, n_pad, H, Hkv, D, cap)
    mask, nn = _tree_inputs(orc, H, B, n_pad, kvl)
    out = orc.tree_attn(q, kc, vc, kvl, kt, vt, mask, nn)
    G = H // Hkv
    Q, K, V, Kt, Vt = (torch.from_numpy(bits_to_f64(a)) for a in (q, kc, vc, kt, vt))
    for b in range(B):
        L = int(kvl[b])
        keys = torch.cat([K[b, :, :L], Kt[b]], 1).repeat_interleave(G, 0)   # [H, L+Np, D]
        vals = torch.cat([V[b, :, :L], Vt[b]], 1).repeat_interleave(G, 0)
        allow = torch.zeros(n_pad, L + n_pad, dtype=torch.bool)
        allow[:, :L] = True
        for i in range(n_pad):
            for j in range(n_pad):
                allow[i, L + j] = bool((int(mask[b, i, j // 64]) >> (j % 64)) & 1)
        n = int(nn[b])
        ref = torch.nn.functional.scaled_dot_product_attention(
            Q[b, :n].transpose(0, 1), keys, vals, attn_mask=allow[:n])  # [H, n, D]
        np.testing.assert_allclose(out[b, :n], ref.transpose(0, 1).numpy(), rtol=0, atol=1e-12)
        assert (out[b, n:] == 0).all()


def test_rows_mode_matches_full(orc):
    B, n_pad, H, Hkv, D, cap = 2, 64, 4, 2, 16, 20
    kvl = np.array([20, 5], np.int32)
    q, kc, vc, kt, vt = _case(4, B, n_pad, H, Hkv, D, cap)
    mask, nn = _tree_inputs(orc, 9, B, n_pad, kvl)
    full = orc.tree_attn(q, kc, vc, kvl, kt, vt, mask, nn)
    rows = np.array([[0, 0, 0], [1, 3, 2], [0, 63, 3], [1, 0, 1]], np.int32)
    part = orc.tree_attn(q, kc, vc, kvl, kt, vt, mask, nn, rows=rows)
    for r, (b, i, h) in enumerate(rows):
        assert np.array_equal(part[r], full[b, i, h])
