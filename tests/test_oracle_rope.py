"""Pins for the oracle's rotary position embedding (O12) and the attention
that applies it to the queries and the tree keys.

RoPE is checked against hand-worked values that fix the pairing convention
(tests/golden/rope_handmade.json), and against properties a wrong sign, pair
or frequency breaks: the identity at position 0, norm preservation per pair,
composition of rotations, and dot products that depend only on the position
difference.  The rotated attention is checked by shift invariance (a tree
without cached keys gives the same output when every position moves by the
same amount) and by the case where all positions are equal, where the
rotations cancel and the plain attention (O6) must come out.
"""
import json
import os

import numpy as np
import pytest

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_rope_handmade_golden(orc):
    g = json.load(open(os.path.join(GOLDEN, "rope_handmade.json")))
    x = np.array([g["x"]], np.float64)
    for case in g["cases"]:
        y = orc.rope(x, [case["pos"]], g["base"])
        assert np.allclose(y[0], case["y"], rtol=0, atol=1e-12), case


def test_rope_properties(orc):
    rng = np.random.default_rng(31)
    D = 128
    x = rng.standard_normal((50, D))
    pos = rng.integers(0, 40000, 50)
    assert np.array_equal(orc.rope(x, np.zeros(50, np.int32)), x)
    y = orc.rope(x, pos)
    h = D // 2
    assert np.allclose(y[:, :h] ** 2 + y[:, h:] ** 2, x[:, :h] ** 2 + x[:, h:] ** 2, rtol=1e-10)
    a, b = rng.integers(0, 20000, 50), rng.integers(0, 20000, 50)
    assert np.allclose(orc.rope(orc.rope(x, a), b), orc.rope(x, a + b), atol=1e-8)
    q, k = rng.standard_normal((50, D)), rng.standard_normal((50, D))
    m, n, t = rng.integers(0, 20000, 50), rng.integers(0, 20000, 50), rng.integers(0, 10000, 50)
    d1 = (orc.rope(q, m) * orc.rope(k, n)).sum(1)
    d2 = (orc.rope(q, m + t) * orc.rope(k, n + t)).sum(1)
    assert np.allclose(d1, d2, atol=1e-8)
    # a different base changes every pair but the first
    y2 = orc.rope(x, pos, 500000.0)
    assert np.allclose(y2[:, 0], y[:, 0]) and not np.allclose(y2[:, 1:h], y[:, 1:h])


def _tree_case(orc, rng, B, n_pad, H, Hkv, D, kv):
    import paper_2502_17139_gb300.synth as synth
    bits = lambda a: a.astype(np.float32).view(np.uint32).__rshift__(16).astype(np.uint16)
    par = np.full((B, n_pad), -1, np.int32)
    nn = rng.integers(1, n_pad + 1, B).astype(np.int32)
    for b in range(B):
        _, p = synth.random_tree(rng, int(nn[b]), 10, 4, 100)
        par[b, :nn[b]] = p
    kvl = np.full(B, kv, np.int32)
    m = orc.tree_mask(par, nn, kvl, n_pad)
    q = bits(rng.standard_normal((B, n_pad, H, D)))
    kc = bits(rng.standard_normal((B, Hkv, max(kv, 1), D)))
    vc = bits(rng.standard_normal((B, Hkv, max(kv, 1), D)))
    kt = bits(rng.standard_normal((B, Hkv, n_pad, D)))
    vt = bits(rng.standard_normal((B, Hkv, n_pad, D)))
    return q, kc, vc, kvl, kt, vt, m, nn


def test_rope_attention_shift_invariance(orc):
    rng = np.random.default_rng(32)
    B, n_pad, H, Hkv, D = 3, 64, 4, 2, 16
    q, kc, vc, kvl, kt, vt, m, nn = _tree_case(orc, rng, B, n_pad, H, Hkv, D, 0)
    pos = m["pos"] + rng.integers(0, 1000, (B, 1)).astype(np.int32)
    o1 = orc.tree_attn(q, kc, vc, kvl, kt, vt, m["mask"], nn, pos=pos)
    o2 = orc.tree_attn(q, kc, vc, kvl, kt, vt, m["mask"], nn, pos=pos + 12345)
    assert np.allclose(o1, o2, atol=1e-9)
    # positions do matter once they differ between nodes
    o3 = orc.tree_attn(q, kc, vc, kvl, kt, vt, m["mask"], nn, pos=pos * 7)
    assert not np.allclose(o1, o3, atol=1e-3)


def test_rope_attention_equal_positions_cancel(orc):
    rng = np.random.default_rng(33)
    B, n_pad, H, Hkv, D = 3, 64, 4, 1, 32
    q, kc, vc, kvl, kt, vt, m, nn = _tree_case(orc, rng, B, n_pad, H, Hkv, D, 0)
    for p in (0, 5, 4321):
        pos = np.full((B, n_pad), p, np.int32)
        o_rope = orc.tree_attn(q, kc, vc, kvl, kt, vt, m["mask"], nn, pos=pos)
        o_plain = orc.tree_attn(q, kc, vc, kvl, kt, vt, m["mask"], nn)
        assert np.allclose(o_rope, o_plain, atol=1e-9), p


def test_rope_attention_cache_keys_not_rotated(orc):
    # cached keys are taken as rotated already: a single-node tree at position
    # p attends to them with the rotated query, so moving p changes the output
    rng = np.random.default_rng(34)
    B, n_pad, H, Hkv, D = 2, 64, 2, 2, 16
    q, kc, vc, kvl, kt, vt, m, nn = _tree_case(orc, rng, B, n_pad, H, Hkv, D, 40)
    nn[:] = 1
    m = orc.tree_mask(np.full((B, n_pad), -1, np.int32), nn, kvl, n_pad)
    o1 = orc.tree_attn(q, kc, vc, kvl, kt, vt, m["mask"], nn, pos=np.full((B, n_pad), 40, np.int32))
    o2 = orc.tree_attn(q, kc, vc, kvl, kt, vt, m["mask"], nn, pos=np.full((B, n_pad), 90, np.int32))
    assert not np.allclose(o1[:, 0], o2[:, 0], atol=1e-3)
