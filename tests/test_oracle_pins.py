"""Pins for the oracle's building blocks, each against something other than
the oracle itself: numpy's fp16 conversion, exact integer arithmetic, numpy
matmul on an independently built matrix, closed forms and invariants.
No GPU."""
import math
from fractions import Fraction

import numpy as np
import pytest

import oracle
import synth


# ----------------------------------------------------------------------------
# fp16 rounding (rounding points R1-R3)
# ----------------------------------------------------------------------------

def test_f16_rounding_matches_numpy():
    rng = np.random.default_rng(1)
    vals = np.concatenate([
        rng.standard_normal(20000) * 10.0 ** rng.integers(-9, 6, 20000),
        # exact ties between fp16 neighbours (round half to even)
        (np.arange(2048) + 0.5) * 2.0 ** -10 + 1.0,
        (np.arange(64) + 0.5) * 2.0 ** -24,
        np.array([0.0, -0.0, 65504.0, 65519.0, 65520.0, 2.0 ** -24, 2.0 ** -25, 2.0 ** -14]),
    ])
    with np.errstate(over="ignore"):
        ref = vals.astype(np.float16)
    got = np.array([oracle.f64_to_f16_bits(v) for v in vals], dtype=np.uint16)
    assert np.array_equal(got, ref.view(np.uint16))
    back = np.array([oracle.f16_bits_to_f64(h) for h in got[:3000]])
    assert np.array_equal(back, ref[:3000].astype(np.float64))


# ----------------------------------------------------------------------------
# INT4 dequantisation and projections
# ----------------------------------------------------------------------------

def _pack_exact(D: np.ndarray, z: np.ndarray, s16: np.ndarray, group: int) -> synth.PackedMatrix:
    """Packs codes q = D + z (D integer, per-group z) in the boundary format."""
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
    scales = np.ascontiguousarray(s16.astype(np.float16).view(np.uint16))
    return synth.PackedMatrix(rows, cols, group, codes, scales, zeros)


@pytest.mark.parametrize("rows,cols,group", [(16, 64, 32), (9, 688, 32), (5, 256, 128), (7, 50, 16)])
def test_dequant_matches_independent_construction(rows, cols, group):
    rng = np.random.default_rng(rows + cols)
    G = -(-cols // group)
    z = rng.integers(0, 16, (rows, G))
    lo, hi = -np.repeat(z, group, axis=1)[:, :cols], 15 - np.repeat(z, group, axis=1)[:, :cols]
    D = rng.integers(lo, hi + 1)
    s = (2.0 ** rng.integers(-12, -2, (rows, G))) * rng.choice([1.0, 1.5, 1.25], (rows, G))
    m = _pack_exact(D, z, s, group)
    W = oracle.dequant(m)
    assert np.array_equal(W, D * np.repeat(s, group, axis=1)[:, :cols])


def test_gemv_symmetric_case_equals_numpy_matmul():
    # z = 8 for every group: a symmetric code; W is built independently of the oracle
    rng = np.random.default_rng(7)
    rows, cols, group = 33, 256, 64
    D = rng.integers(-8, 8, (rows, cols))
    z = np.full((rows, cols // group), 8)
    s = rng.uniform(0.001, 0.05, (rows, cols // group)).astype(np.float16).astype(np.float64)
    m = _pack_exact(D, z, s, group)
    Wd = D * np.repeat(s, group, axis=1)
    x = rng.standard_normal((3, cols))
    y = oracle.gemv(m, x)
    ref = x @ Wd.T
    assert np.allclose(y, ref, rtol=1e-13, atol=1e-13)


def test_gemv_integer_inputs_exact():
    # integer codes, power-of-two scales and integer activations: the exact
    # result is a rational number representable in fp64, computed here with
    # Python Fractions.
    rng = np.random.default_rng(9)
    rows, cols, group = 12, 96, 32
    G = cols // group
    z = rng.integers(0, 16, (rows, G))
    D = rng.integers(-np.repeat(z, group, axis=1), 16 - np.repeat(z, group, axis=1))
    e = rng.integers(-8, 0, (rows, G))
    s = 2.0 ** e
    m = _pack_exact(D, z, s, group)
    x = rng.integers(-20, 21, (4, cols)).astype(np.float64)
    y = oracle.gemv(m, x)
    for t in range(4):
        for o in range(rows):
            exact = sum(Fraction(int(D[o, i])) * Fraction(2) ** int(e[o, i // group]) * int(x[t, i])
                        for i in range(cols))
            assert Fraction(y[t, o]) == exact


def test_gemv_ragged_last_group():
    # 688 = 21.5 groups of 32: the last group has 16 columns
    rng = np.random.default_rng(11)
    w = (rng.standard_normal((4, 688)) * 0.02).astype(np.float32)
    m = synth.quantize(w, 32)
    W = oracle.dequant(m)
    # the last group's dequantised values only depend on its 16 columns
    w2 = w.copy()
    w2[:, 672:] *= 1.7
    W2 = oracle.dequant(synth.quantize(w2, 32))
    assert np.array_equal(W[:, :672], W2[:, :672])
    assert not np.array_equal(W[:, 672:], W2[:, 672:])
    assert np.max(np.abs(W - w)) < 0.02


# ----------------------------------------------------------------------------
# RMSNorm, RoPE, SiLU
# ----------------------------------------------------------------------------

def test_rmsnorm_closed_forms():
    n = 64
    w16 = np.full(n, 0x3C00, dtype=np.uint16)  # weights 1.0
    for c in (3.0, -0.5, 1e-3):
        out = oracle.rmsnorm(np.full(n, c), w16, 1e-5)
        assert np.allclose(out, c / math.sqrt(c * c + 1e-5), rtol=1e-14)
    rng = np.random.default_rng(2)
    x = rng.standard_normal(n)
    a = oracle.rmsnorm(x, w16, 0.0)
    b = oracle.rmsnorm(7.25 * x, w16, 0.0)
    assert np.allclose(a, b, rtol=1e-14)
    assert abs(np.mean(a * a) - 1.0) < 1e-12
    # per-channel weights multiply elementwise
    w = rng.uniform(0.5, 1.5, n).astype(np.float16)
    c2 = oracle.rmsnorm(x, w.view(np.uint16), 0.0)
    assert np.allclose(c2, a * w.astype(np.float64), rtol=1e-14)


@pytest.mark.parametrize("d", [64, 128])
def test_rope_properties(d):
    theta = 500000.0
    rng = np.random.default_rng(d)
    v = rng.standard_normal(d)
    assert np.array_equal(oracle.rope(v, 0, theta), v)  # position 0 is the identity
    h = d // 2
    r = oracle.rope(v, 37, theta)
    # each (i, i + d/2) pair keeps its norm
    assert np.allclose(v[:h] ** 2 + v[h:] ** 2, r[:h] ** 2 + r[h:] ** 2, rtol=1e-13)
    # the first pair has frequency theta^0 = 1: e_0 at position p -> (cos p, sin p) at dims (0, d/2)
    e0 = np.zeros(d)
    e0[0] = 1.0
    p = 5
    r0 = oracle.rope(e0, p, theta)
    assert abs(r0[0] - math.cos(p)) < 1e-15 and abs(r0[h] - math.sin(p)) < 1e-15
    assert np.count_nonzero(r0) == 2
    # frequencies are geometric with ratio theta^(-2/d) between neighbouring pairs
    angles = []
    for i in range(h):
        e = np.zeros(d)
        e[i] = 1.0
        ri = oracle.rope(e, 1, theta)
        angles.append(math.atan2(ri[i + h], ri[i]))
    ratios = np.array(angles[1:]) / np.array(angles[:-1])
    assert np.allclose(ratios, theta ** (-2.0 / d), rtol=1e-10)
    # rotations compose: the score of rotated q, k depends only on the distance
    q, k = rng.standard_normal(d), rng.standard_normal(d)
    s1 = oracle.rope(q, 100, theta) @ oracle.rope(k, 90, theta)
    s2 = oracle.rope(q, 1010, theta) @ oracle.rope(k, 1000, theta)
    assert abs(s1 - s2) < 1e-10


def test_silu_identities():
    assert oracle.silu(0.0) == 0.0
    for x in (0.3, 1.7, 5.0, -2.2):
        assert abs(oracle.silu(x) - oracle.silu(-x) - x) < 1e-15   # x*sig(x) + x*sig(-x) = x
    assert abs(oracle.silu(40.0) - 40.0) < 1e-12
    assert abs(oracle.silu(1.0) - 1.0 / (1.0 + math.exp(-1.0))) < 1e-16


# ----------------------------------------------------------------------------
# Attention
# ----------------------------------------------------------------------------

def test_attend_single_visible_entry_returns_its_value_row():
    rng = np.random.default_rng(4)
    K, V = rng.standard_normal((9, 64)), rng.standard_normal((9, 64))
    q = rng.standard_normal(64)
    vis = np.zeros(9, dtype=np.uint8)
    vis[6] = 1
    assert np.array_equal(oracle.attend(q, K, V, vis), V[6])


def test_attend_equal_keys_give_mean_of_values():
    rng = np.random.default_rng(5)
    k = rng.standard_normal(64)
    K = np.tile(k, (10, 1))
    V = rng.standard_normal((10, 64))
    vis = np.array([1, 0, 1, 1, 0, 1, 1, 1, 0, 1], dtype=np.uint8)
    out = oracle.attend(rng.standard_normal(64), K, V, vis)
    assert np.allclose(out, V[vis == 1].mean(axis=0), rtol=1e-13, atol=1e-14)


def test_attend_masked_entries_have_no_effect_and_order_does_not_matter():
    rng = np.random.default_rng(6)
    K, V = rng.standard_normal((12, 32)), rng.standard_normal((12, 32))
    q = rng.standard_normal(32)
    vis = (rng.random(12) < 0.6).astype(np.uint8)
    vis[0] = 1
    a = oracle.attend(q, K, V, vis)
    K2, V2 = K.copy(), V.copy()
    K2[vis == 0] = 1e6
    V2[vis == 0] = -1e6
    assert np.array_equal(oracle.attend(q, K2, V2, vis), a)
    # the masked result equals attention over the kept rows only (a physical trim)
    keep = vis == 1
    assert np.array_equal(oracle.attend(q, K[keep], V[keep], np.ones(keep.sum(), np.uint8)), a)
    perm = rng.permutation(12)
    assert np.allclose(oracle.attend(q, K[perm], V[perm], vis[perm]), a, rtol=1e-13, atol=1e-14)


def test_attend_two_entries_closed_form():
    # two visible entries: p_1 = 1 / (1 + exp(s_0 - s_1)) (logistic of the score gap)
    d = 4
    q = np.array([1.0, 0.0, 0.0, 0.0])
    K = np.array([[0.0, 0, 0, 0], [2.0, 0, 0, 0]])
    V = np.array([[1.0, 0, 0, 0], [0.0, 1, 0, 0]])
    out = oracle.attend(q, K, V, np.ones(2, np.uint8))
    p1 = 1.0 / (1.0 + math.exp(-2.0 / math.sqrt(d)))
    assert abs(out[0] - (1 - p1)) < 1e-15 and abs(out[1] - p1) < 1e-15
