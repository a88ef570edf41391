"""Pins for the oracle's greedy prediction at every tree node (O10): the
argmax of each logits row, checked against numpy.argmax (an independent
library routine with the same tie and NaN conventions) and hand-made rows."""
import numpy as np
import pytest


def bf16_bits(x):
    """float32 -> bf16 bit patterns by truncation (every value used here is exact in bf16)."""
    return (np.asarray(x, np.float32).view(np.uint32) >> 16).astype(np.uint16)


def bits_to_f32(h):
    return (h.astype(np.uint32) << 16).view(np.float32)


def test_argmax_hand_cases(orc):
    rows = [
        [1.0, 1.0, 1.0, 1.0],            # all equal: the first
        [0.0, -1.0, 2.0, 2.0],           # tie at the top: the first of them
        [-0.0, 0.0, -1.0, -2.0],         # -0 == +0: the first
        [-np.inf, -np.inf, -5.0, -np.inf],
        [1.0, np.nan, 3.0, np.nan],      # NaN beats numbers, the first NaN wins
        [5.0, 4.0, 3.0, np.inf],
    ]
    want = [0, 2, 0, 2, 1, 3]
    logits = bf16_bits(np.array(rows, np.float32))[None]
    got = orc.argmax_rows(logits, np.array([len(rows)], np.int32))
    assert got[0].tolist() == want


@pytest.mark.parametrize("seed", range(4))
def test_argmax_matches_numpy(orc, seed):
    rng = np.random.default_rng(70 + seed)
    B, Np, V = 3, 5, [1, 7, 1000, 32256][seed]
    x = rng.standard_normal((B, Np, V)).astype(np.float32)
    x = bits_to_f32(bf16_bits(x))                 # exact bf16 values
    # planted ties, signed zeros, infinities and NaNs
    x[0, 0, :] = 0.5
    if V > 4:
        x[0, 1, [1, V - 1]] = 9.0
        x[1, 0, [0, 2]] = [-0.0, 0.0]
        x[1, 0, 1:] = np.minimum(x[1, 0, 1:], -1.0)
        x[1, 0, 2] = 0.0
        x[2, 2, V // 2] = np.inf
        x[2, 3, [3, V - 2]] = np.nan
    n_nodes = np.array([Np, Np - 1, Np], np.int32)
    got = orc.argmax_rows(bf16_bits(x), n_nodes)
    for b in range(B):
        for i in range(Np):
            want = int(np.argmax(x[b, i])) if i < n_nodes[b] else 0
            assert got[b, i] == want, (b, i)
