"""Pins of the oracle's LM head with the top-1 epilogue (Section 6.7): final
RMSNorm, INT4 lm_head projection, greedy token and its softmax probability.
Checked against an independent numpy formulation (dense matrix built without
the oracle, numpy's fp16 rounding, scipy's softmax), closed forms for uniform
and single-row logits, the lowest-id tie rule and the norm's scale
invariance.  No GPU."""
import numpy as np
import pytest
from scipy.special import softmax

import oracle
import synth


def _pack_exact(D: np.ndarray, z: np.ndarray, s: np.ndarray, group: int) -> synth.PackedMatrix:
    """Codes q = D + z per group in the boundary format; W = D * s exactly."""
    rows, cols = D.shape
    G = -(-cols // group)
    q = D + np.repeat(z, group, axis=1)[:, :cols]
    assert q.min() >= 0 and q.max() <= 15
    codes = np.zeros((rows, (cols + 1) // 2), dtype=np.uint8)
    for c in range(cols):
        codes[:, c // 2] |= (q[:, c].astype(np.uint8) << (4 * (c % 2))).astype(np.uint8)
    zeros = np.zeros((rows, (G + 1) // 2), dtype=np.uint8)
    for g in range(G):
        zeros[:, g // 2] |= (z[:, g].astype(np.uint8) << (4 * (g % 2))).astype(np.uint8)
    scales = np.ascontiguousarray(s.astype(np.float16).view(np.uint16))
    return synth.PackedMatrix(rows, cols, group, codes, scales, zeros)


def _random_exact(rows, cols, group, rng):
    G = -(-cols // group)
    z = rng.integers(0, 16, (rows, G))
    zz = np.repeat(z, group, axis=1)[:, :cols]
    D = rng.integers(-zz, 16 - zz)
    s = 2.0 ** rng.integers(-7, -3, (rows, G)).astype(np.float64)
    return _pack_exact(D, z, s, group), D * np.repeat(s, group, axis=1)[:, :cols]


def _norm16(H, rng):
    return (1.0 + 0.1 * rng.standard_normal(H)).astype(np.float16)


@pytest.mark.parametrize("V,H,group", [(97, 64, 32), (300, 160, 32), (64, 256, 128)])
def test_head_matches_independent_numpy_formulation(V, H, group):
    rng = np.random.default_rng(V + H)
    w, Wd = _random_exact(V, H, group, rng)
    nw = _norm16(H, rng)
    h = rng.standard_normal((3, H)).astype(np.float16)
    eps = 1e-5
    tok, p, margin, lg = oracle.head_top1(h.view(np.uint16), nw.view(np.uint16), w, eps)
    hd = h.astype(np.float64)
    x = hd / np.sqrt((hd * hd).mean(axis=1, keepdims=True) + eps) * nw.astype(np.float64)
    x = x.astype(np.float16).astype(np.float64)  # the projection's fp16 operand
    ref = x @ Wd.T
    assert np.allclose(lg, ref, rtol=1e-12, atol=1e-12)
    assert np.array_equal(tok, ref.argmax(axis=1))
    assert np.allclose(p, softmax(ref, axis=1).max(axis=1), rtol=1e-12)
    srt = np.sort(ref, axis=1)
    assert np.allclose(margin, srt[:, -1] - srt[:, -2], rtol=1e-9, atol=1e-12)


def test_head_zero_weights_give_uniform_probability_and_token_zero():
    V, H, g = 50, 64, 32
    w = _pack_exact(np.zeros((V, H), np.int64), np.full((V, H // g), 3), np.ones((V, H // g)), g)
    h = np.random.default_rng(1).standard_normal((2, H)).astype(np.float16)
    tok, p, margin, lg = oracle.head_top1(h.view(np.uint16), np.ones(H, np.float16).view(np.uint16), w, 1e-5)
    assert np.all(lg == 0.0)
    assert np.array_equal(tok, [0, 0])          # every logit ties: the lowest id
    assert np.array_equal(p, [1.0 / V, 1.0 / V])
    assert np.array_equal(margin, [0.0, 0.0])


@pytest.mark.parametrize("v_star,sign", [(7, 1), (0, 1), (7, -1)])
def test_head_single_live_row_closed_form(v_star, sign):
    # only row v* has weights: its logit L, every other logit 0
    V, H, g = 40, 32, 32
    D = np.zeros((V, H), np.int64)
    D[v_star] = sign * np.where(np.arange(H) % 3 == 0, 5, 2)
    w = _pack_exact(D, np.full((V, 1), 8), np.full((V, 1), 0.125), g)
    h = np.abs(np.random.default_rng(2).standard_normal((1, H))).astype(np.float16) + np.float16(0.25)
    tok, p, margin, lg = oracle.head_top1(h.view(np.uint16), np.ones(H, np.float16).view(np.uint16), w, 1e-5)
    L = lg[0, v_star]
    assert sign * L > 0 and np.all(np.delete(lg[0], v_star) == 0.0)
    if sign > 0:
        assert tok[0] == v_star
        assert np.isclose(p[0], 1.0 / (1.0 + (V - 1) * np.exp(-L)), rtol=1e-13)
        assert np.isclose(margin[0], L, rtol=1e-13)
    else:
        assert tok[0] == (1 if v_star == 0 else 0)  # the lowest id among the zero logits
        assert np.isclose(p[0], 1.0 / ((V - 1) + np.exp(L)), rtol=1e-13)
        assert margin[0] == 0.0


def test_head_equal_rows_pick_the_lowest_id():
    rng = np.random.default_rng(5)
    V, H, g = 30, 64, 32
    w, Wd = _random_exact(V, H, g, rng)
    h = rng.standard_normal((1, H)).astype(np.float16)
    nw = np.ones(H, np.float16).view(np.uint16)
    tok0, _, _, lg0 = oracle.head_top1(h.view(np.uint16), nw, w, 1e-5)
    best = int(tok0[0])
    lo, hi = (3, 20) if best not in (3, 20) else (4, 21)
    for a in (w.codes, w.scales, w.zeros):   # rows lo and hi become copies of the best row
        a[lo] = a[best]
        a[hi] = a[best]
    tok, p, margin, lg = oracle.head_top1(h.view(np.uint16), nw, w, 1e-5)
    assert lg[0, lo] == lg[0, hi] == lg[0].max()
    assert tok[0] == min(lo, best)
    assert margin[0] == 0.0
    assert np.isclose(p[0], softmax(lg[0]).max(), rtol=1e-12)


def test_head_norm_is_scale_invariant():
    # without eps, doubling the hidden row is exact and leaves x bit-identical
    rng = np.random.default_rng(8)
    V, H, g = 80, 128, 64
    w, _ = _random_exact(V, H, g, rng)
    h = rng.standard_normal((2, H)).astype(np.float16)
    nw = _norm16(H, rng).view(np.uint16)
    a = oracle.head_top1(h.view(np.uint16), nw, w, 0.0)
    b = oracle.head_top1((h * np.float16(2)).view(np.uint16), nw, w, 0.0)
    for u, v in zip(a, b):
        assert np.array_equal(u, v)


def test_head_probability_bounds_on_a_seeded_head():
    hw = synth.make_head(256, 512, 32, 3)
    h = synth.hidden_in(synth.TINY, 3, 0, 4)
    tok, p, margin, lg = oracle.head_top1(h, hw.norm, hw.lm_head, hw.rms_eps)
    assert np.all((p > 1.0 / 512) & (p <= 1.0))
    assert np.all(margin >= 0)
    assert np.array_equal(tok, lg.argmax(axis=1))
