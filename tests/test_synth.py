"""Input generator checks: Philox known answers, fp16 encoding, the uint4
quantiser's defining property (nearest code), packing, and the workload
recipes.  No GPU."""
import json
import os

import numpy as np
import pytest

import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_philox_known_answers():
    kat = json.load(open(os.path.join(GOLDEN, "philox4x32_10_kat.json")))
    for v in kat["vectors"]:
        ctr = [int(x, 16) for x in v["ctr"]]
        key = [int(x, 16) for x in v["key"]]
        out = [int(x, 16) for x in v["out"]]
        assert list(synth.philox4x32_10(ctr, key)) == out


def test_f16_encoding_matches_numpy():
    rng = np.random.default_rng(0)
    vals = np.concatenate([
        rng.standard_normal(20000) * 10.0 ** rng.integers(-9, 6, 20000),
        np.array([0.0, -0.0, 65504.0, 65519.99, 65520.0, 1e9, -1e9, 2.0 ** -24, 2.0 ** -25, 3 * 2.0 ** -26,
                  2.0 ** -14, 2.0 ** -14 - 2.0 ** -25, 1.0 + 2.0 ** -11, 1.0 + 3 * 2.0 ** -11]),
    ])
    with np.errstate(over="ignore"):  # values beyond fp16's range round to infinity on purpose
        ref = vals.astype(np.float16).view(np.uint16)
    got = np.array([synth.f64_to_f16_bits(v) for v in vals], dtype=np.uint16)
    assert np.array_equal(got, ref)


def _unpack(m: synth.PackedMatrix):
    q = np.zeros((m.rows, m.cols), dtype=np.int64)
    q[:, 0::2] = (m.codes & 15)[:, : (m.cols + 1) // 2]
    q[:, 1::2] = (m.codes >> 4)[:, : m.cols // 2]
    G = m.n_groups
    z = np.zeros((m.rows, G), dtype=np.int64)
    z[:, 0::2] = (m.zeros & 15)[:, : (G + 1) // 2]
    z[:, 1::2] = (m.zeros >> 4)[:, : G // 2]
    s = m.scales.view(np.float16).astype(np.float64)
    return q, z, s


@pytest.mark.parametrize("rows,cols,group", [(3, 64, 32), (5, 50, 16), (4, 688, 32), (2, 256, 128), (3, 7, 4)])
def test_quantizer_nearest_code(rows, cols, group):
    rng = np.random.default_rng(rows * 1000 + cols)
    w = (rng.standard_normal((rows, cols)) * 0.02).astype(np.float32)
    m = synth.quantize(w, group)
    q, z, s = _unpack(m)
    G = m.n_groups
    for r in range(rows):
        for g in range(G):
            c0, c1 = g * group, min(cols, (g + 1) * group)
            seg = w[r, c0:c1].astype(np.float64)
            mn, mx = seg.min(), seg.max()
            # scale: fp16 rounding of (max - min) / 15, computed from this group's elements only
            s16 = np.float16((mx - mn) / 15.0).astype(np.float64)
            if s16 == 0:
                s16 = 1.0
            assert s[r, g] == s16
            assert 0 <= z[r, g] <= 15
            for c in range(c0, c1):
                # brute force over all 16 codes: q is the code nearest to w
                errs = np.abs(seg[c - c0] - (np.arange(16) - z[r, g]) * s16)
                best = errs.min()
                assert errs[q[r, c]] == best
                # unclamped codes reconstruct within half a step
                if 0 < q[r, c] < 15:
                    assert abs(seg[c - c0] - (q[r, c] - z[r, g]) * s16) <= s16 / 2 + 1e-12


def test_quantizer_constant_group_and_symmetric_case():
    w = np.zeros((1, 64), dtype=np.float32)
    w[0, 32:] = 0.5  # second group constant positive
    m = synth.quantize(w, 32)
    q, z, s = _unpack(m)
    assert s[0, 0] == 1.0 and s[0, 1] == 1.0  # zero range -> scale 1
    assert (q[0, :32] - z[0, 0] == 0).all()
    # exactly representable symmetric grid: w = (c - 8) * 2^-6 with min -8 and max +7 steps
    c = np.tile(np.arange(16), 4)
    w = ((c - 8) * 2.0 ** -6).astype(np.float32).reshape(1, 64)
    m = synth.quantize(w, 64)
    q, z, s = _unpack(m)
    assert s[0, 0] == 2.0 ** -6 and z[0, 0] == 8
    assert np.array_equal(q[0], c)


def test_pack_layout_round_trip():
    rng = np.random.default_rng(3)
    w = (rng.standard_normal((6, 37)) * 0.02).astype(np.float32)
    m = synth.quantize(w, 8)
    assert m.codes.shape == (6, 19) and m.scales.shape == (6, 5) and m.zeros.shape == (6, 3)
    q, z, s = _unpack(m)
    # padding nibbles are zero
    assert ((m.codes[:, -1] >> 4) == 0).all()
    assert ((m.zeros[:, -1] >> 4) == 0).all()
    s_el = np.repeat(s, 8, axis=1)[:, :37]
    deq = (q - np.repeat(z, 8, axis=1)[:, :37]) * s_el
    # Groups whose range contains 0 reconstruct within half a step (plus the fp16
    # rounding of the step at the range ends); a group of one sign may clamp z.
    gmin = np.minimum.reduceat(w, np.arange(0, 37, 8), axis=1)
    gmax = np.maximum.reduceat(w, np.arange(0, 37, 8), axis=1)
    straddle = np.repeat((gmin <= 0) & (gmax >= 0), 8, axis=1)[:, :37]
    assert straddle.sum() > 150
    assert (np.abs(deq - w)[straddle] <= (s_el * (0.5 + 16 * 2.0 ** -11))[straddle]).all()


def test_quant_matrix_deterministic_and_thread_independent():
    a = synth.quant_matrix(64, 256, 32, 0.02, seed=5, stream=1, tag=1, threads=1)
    b = synth.quant_matrix(64, 256, 32, 0.02, seed=5, stream=1, tag=1, threads=7)
    c = synth.quant_matrix(64, 256, 32, 0.02, seed=6, stream=1, tag=1, threads=7)
    assert np.array_equal(a.codes, b.codes) and np.array_equal(a.scales, b.scales)
    assert not np.array_equal(a.codes, c.codes)


def test_normals_moments():
    x = synth.normal(400000, seed=11, stream=3, tag=9, dtype=np.float64)
    assert abs(x.mean()) < 0.01 and abs(x.std() - 1.0) < 0.01
    h = synth.normal(1000, seed=11, stream=3, tag=9, dtype=np.uint16)
    assert np.array_equal(h, x[:1000].astype(np.float16).view(np.uint16))


def test_recipe_helpers():
    claims = json.load(open(os.path.join(GOLDEN, "paper_claims.json")))
    acc = [synth.accepted_drafts(seed=1, step=s) for s in range(4000)]
    assert all(0 <= a <= 4 for a in acc)
    assert abs(np.mean(acc) - claims["expected_accepted_drafts_k4_p06"]["value"]) < 0.06
    for s in range(5):
        p = synth.permutation(seed=2, step=s, n=8)
        assert sorted(p.tolist()) == list(range(8))
    L = synth.lengths(seed=3, n=1000, lo=128, hi=2048)
    assert L.min() >= 128 and L.max() <= 2048
    t = synth.token_ids(synth.TINY, seed=1, step=0, M=1000)
    assert t.min() >= 0 and t.max() < synth.TINY.vocab


def test_shape_byte_counts():
    s = synth.LLAMA8B_STAGE
    assert s.params_per_layer() * s.n_layers == 3_489_660_928
    assert s.packed_bytes_per_layer() * s.n_layers == 1_812_987_904
    s70 = synth.LLAMA70B_STAGE
    assert s70.params_per_layer() * s70.n_layers == 17_112_760_320
    assert synth.TINY.params_per_layer() * synth.TINY.n_layers == 1_449_984
