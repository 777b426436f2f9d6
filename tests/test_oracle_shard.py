"""Shard-level pins for the oracle: the paper's own claims (masked rewind
equals a physical trim, Section 5.2; the beam_idx gather is a reorder,
Section 4; speculative greedy decoding emits the target's greedy tokens,
Section 5.3) plus structural special cases (zero weights pass the residual
through, GQA with duplicated KV heads equals MHA, causality inside the verify
block, batch-composition invariance) and an independent numpy formulation of
one layer.  No GPU."""
import json
import math
import os

import numpy as np
import pytest

import oracle
import synth
from scenarios import (MaskedRequest, OracleEngine, f16, greedy_decode, prefill, spec_decode,
                       tiny_steps_masked_vs_trim)

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
CLAIMS = json.load(open(os.path.join(GOLDEN, "paper_claims.json")))
TINY = synth.TINY
SEED = 20260802


@pytest.fixture(scope="module")
def tiny_weights():
    return synth.make_weights(TINY, SEED)


def test_masked_rewind_equals_physical_trim(tiny_weights):
    out = tiny_steps_masked_vs_trim(lambda cap: OracleEngine(TINY, tiny_weights, 1, cap), TINY, tiny_weights)
    for s in ("A", "B", "C"):
        diff = np.max(np.abs(f16(out[("mask", s)]) - f16(out[("trim", s)])))
        assert diff == CLAIMS["mask_vs_trim"]["max_abs_diff"]
    # and the un-rounded residual streams agree bit for bit
    assert np.array_equal(out[("mask", "engine")].last_f64, out[("trim", "engine")].last_f64)
    # the masked cache, compacted to its live entries, is the trimmed cache
    em, et, rm = out[("mask", "engine")], out[("trim", "engine")], out[("mask", "req")]
    live = np.flatnonzero(np.array(rm.valid))
    for layer in range(TINY.n_layers):
        km, vm = em.read(0, layer, 0, em.length(0))
        kt, vt = et.read(0, layer, 0, et.length(0))
        assert np.array_equal(km[live], kt) and np.array_equal(vm[live], vt)


def test_step_outputs_are_finite_and_move(tiny_weights):
    eng = OracleEngine(TINY, tiny_weights, 1, 96)
    prefill(eng, TINY, SEED, 0, 72)
    h = synth.hidden_in(TINY, SEED, 0, 1)
    o = eng.step([1], np.array([72], np.int32), np.ones(73, np.uint8), hidden_in=h)
    assert np.isfinite(f16(o)).all()
    assert np.abs(f16(o) - f16(h)).max() > 0.05   # the layers do something
    assert eng.length(0) == 73


def _zero_weights(shape, like):
    """Weights whose codes equal their zero points, so every W = 0."""
    layers = []
    for lw in like.layers:
        mats = []
        for m in lw.matrices:
            z = np.zeros_like(m.zeros)
            z[:] = 0x55  # zero point 5 in both nibbles
            codes = np.full_like(m.codes, 0x55)
            if m.cols % 2:
                codes[:, -1] = 0x05
            mats.append(synth.PackedMatrix(m.rows, m.cols, m.group, codes, m.scales.copy(), z))
        layers.append(synth.LayerWeights(mats, lw.attn_norm, lw.ffn_norm))
    return synth.ShardWeights(shape, 0, layers, like.embedding)


def test_zero_weights_pass_the_residual_through(tiny_weights):
    zw = _zero_weights(TINY, tiny_weights)
    eng = OracleEngine(TINY, zw, 1, 96)
    prefill(eng, TINY, SEED, 0, 10)
    h = synth.hidden_in(TINY, SEED, 3, 3)
    o = eng.step([3], np.arange(10, 13, dtype=np.int32), np.ones(13, np.uint8), hidden_in=h)
    assert np.array_equal(o, h)
    k, v = eng.read(0, 0, 10, 3)
    assert (f16(k) == 0).all() and (f16(v) == 0).all()


def test_beam_gather_equals_physically_reordered_cache(tiny_weights):
    B = 3
    lens = [20, 33, 27]
    perm = np.array([2, 0, 2], dtype=np.int32)  # with a duplicate: a Gather, not only a permutation
    a = OracleEngine(TINY, tiny_weights, B, 64)
    b = OracleEngine(TINY, tiny_weights, B, 64)
    for r in range(B):
        prefill(a, TINY, SEED + r, r, lens[r])
    # b holds the gathered rows physically
    for r in range(B):
        for layer in range(TINY.n_layers):
            k, v = a.read(int(perm[r]), layer, 0, lens[perm[r]])
            b.load(r, layer, k, v)
    n_new = [1, 2, 1]
    M = sum(n_new)
    h = synth.hidden_in(TINY, SEED, 9, M)
    new_len = [lens[p] for p in perm]
    pos = np.concatenate([np.arange(L, L + n, dtype=np.int32) for L, n in zip(new_len, n_new)])
    stride = max(L + n for L, n in zip(new_len, n_new))
    mask = np.zeros((B, stride), np.uint8)
    for r in range(B):
        mask[r, : new_len[r] + n_new[r]] = 1
    mask[1, 5] = 0  # a hole inside a gathered history
    oa = a.step(n_new, pos, mask, hidden_in=h, beam_idx=perm)
    ob = b.step(n_new, pos, mask, hidden_in=h)
    assert np.array_equal(oa, ob)
    for r in range(B):
        assert a.length(r) == b.length(r) == new_len[r] + n_new[r]
        for layer in range(TINY.n_layers):
            assert all(np.array_equal(x, y) for x, y in zip(a.read(r, layer, 0, a.length(r)),
                                                            b.read(r, layer, 0, b.length(r))))
    # identity beam_idx changes nothing (Section 4: the runtime value is the identity)
    c = OracleEngine(TINY, tiny_weights, 1, 96)
    d = OracleEngine(TINY, tiny_weights, 1, 96)
    prefill(c, TINY, SEED, 0, 40)
    prefill(d, TINY, SEED, 0, 40)
    h1 = synth.hidden_in(TINY, SEED, 4, 1)
    oc = c.step([1], np.array([40], np.int32), np.ones(41, np.uint8), hidden_in=h1, beam_idx=np.array([0], np.int32))
    od = d.step([1], np.array([40], np.int32), np.ones(41, np.uint8), hidden_in=h1)
    assert np.array_equal(oc, od) == (not CLAIMS["beam_idx_identity"]["identity_changes_output"])


def test_gqa_equals_mha_with_duplicated_kv_heads(tiny_weights):
    shape = TINY
    grp = shape.n_heads // shape.n_kv_heads
    d = shape.head_dim
    mha_shape = synth.ShardShape("tiny-mha", shape.n_layers, shape.hidden, shape.n_heads, shape.n_heads, d,
                                 shape.ffn, shape.group, shape.weight_sigma, shape.vocab, shape.rms_eps,
                                 shape.rope_theta, shape.max_position)
    layers = []
    rows = np.concatenate([np.arange(h // grp * d, h // grp * d + d) for h in range(shape.n_heads)])
    for lw in tiny_weights.layers:
        mats = list(lw.matrices)
        for mi in (1, 2):
            m = mats[mi]
            mats[mi] = synth.PackedMatrix(m.rows * grp, m.cols, m.group, np.ascontiguousarray(m.codes[rows]),
                                          np.ascontiguousarray(m.scales[rows]), np.ascontiguousarray(m.zeros[rows]))
        layers.append(synth.LayerWeights(mats, lw.attn_norm, lw.ffn_norm))
    mw = synth.ShardWeights(mha_shape, 0, layers, tiny_weights.embedding)
    g = OracleEngine(shape, tiny_weights, 1, 64)
    m = OracleEngine(mha_shape, mw, 1, 64)
    for layer in range(shape.n_layers):
        k, v = synth.kv_prefill(shape, SEED, 0, 30, layer)
        g.load(0, layer, k, v)
        heads = [h // grp for h in range(shape.n_heads)]
        m.load(0, layer, np.ascontiguousarray(k[:, heads]), np.ascontiguousarray(v[:, heads]))
    h = synth.hidden_in(shape, SEED, 5, 2)
    pos = np.array([30, 31], np.int32)
    assert np.array_equal(g.step([2], pos, np.ones(32, np.uint8), hidden_in=h),
                          m.step([2], pos, np.ones(32, np.uint8), hidden_in=h))


def test_verify_block_is_causal(tiny_weights):
    outs = []
    for variant in range(2):
        eng = OracleEngine(TINY, tiny_weights, 1, 96)
        prefill(eng, TINY, SEED, 0, 50)
        h = synth.hidden_in(TINY, SEED, 6, 5).copy()
        if variant:
            h[3:] = synth.hidden_in(TINY, SEED, 7, 2)  # change the later tokens only
        outs.append(eng.step([5], np.arange(50, 55, dtype=np.int32), np.ones(55, np.uint8), hidden_in=h))
    assert np.array_equal(outs[0][:3], outs[1][:3])
    assert not np.array_equal(outs[0][3:], outs[1][3:])


def test_batch_composition_invariance(tiny_weights):
    lens = [40, 61, 25]
    n_new = [1, 3, 2]
    B = 3
    hs = [synth.hidden_in(TINY, SEED + 10 + r, 0, n_new[r]) for r in range(B)]
    batch = OracleEngine(TINY, tiny_weights, B, 80)
    for r in range(B):
        prefill(batch, TINY, SEED + r, r, lens[r])
    stride = max(L + n for L, n in zip(lens, n_new))
    mask = np.zeros((B, stride), np.uint8)
    for r in range(B):
        mask[r, : lens[r] + n_new[r]] = 1
    pos = np.concatenate([np.arange(L, L + n, dtype=np.int32) for L, n in zip(lens, n_new)])
    ob = batch.step(n_new, pos, mask, hidden_in=np.concatenate(hs))
    t = 0
    for r in range(B):
        alone = OracleEngine(TINY, tiny_weights, 1, 80)
        prefill(alone, TINY, SEED + r, 0, lens[r], src_row=r)
        oa = alone.step([n_new[r]], np.arange(lens[r], lens[r] + n_new[r], dtype=np.int32),
                        np.ones(lens[r] + n_new[r], np.uint8), hidden_in=hs[r])
        assert np.array_equal(oa, ob[t: t + n_new[r]])
        t += n_new[r]
    # "the check has teeth": changing request 1's input moves only request 1's rows
    hs2 = list(hs)
    hs2[1] = synth.hidden_in(TINY, SEED + 99, 0, n_new[1])
    batch2 = OracleEngine(TINY, tiny_weights, B, 80)
    for r in range(B):
        prefill(batch2, TINY, SEED + r, r, lens[r])
    ob2 = batch2.step(n_new, pos, mask, hidden_in=np.concatenate(hs2))
    assert np.array_equal(ob2[0:1], ob[0:1]) and np.array_equal(ob2[4:], ob[4:])
    assert np.abs(f16(ob2[1:4]) - f16(ob[1:4])).max() > 0.1


def test_speculative_greedy_equals_target_greedy(tiny_weights):
    n = 24
    target, margins = greedy_decode(OracleEngine(TINY, tiny_weights, 1, 256), TINY, tiny_weights, SEED, n)
    spec, smargins, req = spec_decode(OracleEngine(TINY, tiny_weights, 1, 256), TINY, tiny_weights, SEED, n, target)
    mism = sum(1 for a, b in zip(target, spec) if a != b)
    assert mism == CLAIMS["spec_vs_target_greedy"]["token_mismatches"]
    assert len(req.valid) > req.pos  # rejected drafts really stayed in the cache, masked


def test_error_codes(tiny_weights):
    st = oracle.OracleShard(TINY, tiny_weights).state(2, 16)
    k, v = synth.kv_prefill(TINY, SEED, 0, 15, 0)
    assert st.load(0, 0, k, v) == 0
    h = synth.hidden_in(TINY, SEED, 0, 2)
    # capacity: 15 + 2 > 16
    rc, _, _ = st.step([2], np.array([15, 16], np.int32), np.ones(17, np.uint8), hidden_in=h)
    assert rc == oracle.ECAP
    st2 = oracle.OracleShard(TINY, tiny_weights).state(1, 64)
    # a zero in the mask at a new entry
    m = np.ones(2, np.uint8)
    m[1] = 0
    rc, _, _ = st2.step([2], np.array([0, 1], np.int32), m, hidden_in=h)
    assert rc == oracle.EINVAL
    # beam_idx out of range
    rc, _, _ = st2.step([1], np.array([0], np.int32), np.ones(1, np.uint8), hidden_in=h[:1],
                        beam_idx=np.array([1], np.int32))
    assert rc == oracle.EINVAL


# ----------------------------------------------------------------------------
# One layer against an independent numpy formulation (dense matrices built
# without the oracle, RoPE as complex rotation, softmax with numpy)
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("round_points", [False, True])
def test_one_layer_matches_independent_numpy_formulation(round_points):
    shape = synth.ShardShape("one-layer", 1, 64, 4, 2, 16, 96, 32, 0.02, 0, 1e-5, 10000.0, 128)
    rng = np.random.default_rng(12)
    mats, dense = [], []
    for name in synth.MATRIX_NAMES:
        r, c = shape.matrix_shape(name)
        G = c // 32
        z = rng.integers(0, 16, (r, G))
        zz = np.repeat(z, 32, axis=1)
        D = rng.integers(-zz, 16 - zz)
        s = (2.0 ** rng.integers(-8, -4, (r, G))).astype(np.float64)
        codes = np.zeros((r, c // 2), np.uint8)
        q = D + zz
        codes[:] = (q[:, 0::2] | (q[:, 1::2] << 4)).astype(np.uint8)
        zeros = (z[:, 0::2] | (z[:, 1::2] << 4)).astype(np.uint8)
        mats.append(synth.PackedMatrix(r, c, 32, codes, s.astype(np.float16).view(np.uint16), zeros))
        dense.append(D * np.repeat(s, 32, axis=1))
    an = (1 + 0.1 * rng.standard_normal(64)).astype(np.float16)
    fn = (1 + 0.1 * rng.standard_normal(64)).astype(np.float16)
    w = synth.ShardWeights(shape, 0, [synth.LayerWeights(mats, an.view(np.uint16), fn.view(np.uint16))], None)
    eng = OracleEngine(shape, w, 1, 32, round_points=round_points)
    P = 7
    k0 = rng.standard_normal((P, 2, 16)).astype(np.float16)
    v0 = rng.standard_normal((P, 2, 16)).astype(np.float16)
    eng.load(0, 0, k0.view(np.uint16), v0.view(np.uint16))
    x16 = rng.standard_normal((3, 64)).astype(np.float16)
    pos = np.array([11, 12, 13], np.int32)
    mask = np.ones(P + 3, np.uint8)
    mask[2] = 0
    out16 = eng.step([3], pos, mask, hidden_in=x16.view(np.uint16))
    got = eng.last_f64
    # fp16 rounding at the W4A16 storage points, done with numpy's conversion
    r16 = (lambda a: a.astype(np.float16).astype(np.float64)) if round_points else (lambda a: a)

    Wq, Wk, Wv, Wo, Wg, Wu, Wd = dense
    x = x16.astype(np.float64)

    def norm(a, g):
        return a / np.sqrt((a * a).mean(axis=1, keepdims=True) + 1e-5) * g.astype(np.float64)

    def rot(vecs, p):  # complex-number form of rotate-half RoPE
        h = vecs.shape[-1] // 2
        z = vecs[..., :h] + 1j * vecs[..., h:]
        ang = p * 10000.0 ** (-np.arange(h) * 2.0 / vecs.shape[-1])
        z = z * np.exp(1j * ang)
        return np.concatenate([z.real, z.imag], axis=-1)

    xn = r16(norm(x, an))
    q = (xn @ Wq.T).reshape(3, 4, 16)
    k = (xn @ Wk.T).reshape(3, 2, 16)
    v = (xn @ Wv.T).reshape(3, 2, 16)
    q = np.stack([rot(q[t], pos[t]) for t in range(3)])
    k = np.stack([rot(k[t], pos[t]) for t in range(3)])
    K = np.concatenate([k0.astype(np.float64), r16(k)])
    V = np.concatenate([v0.astype(np.float64), r16(v)])
    att = np.zeros((3, 4, 16))
    for t in range(3):
        vis = np.flatnonzero(mask[: P + t + 1])
        for hh in range(4):
            sc = K[vis, hh // 2] @ q[t, hh] / math.sqrt(16)
            p_ = np.exp(sc - sc.max())
            p_ /= p_.sum()
            att[t, hh] = p_ @ V[vis, hh // 2]
    x = x + r16(att.reshape(3, 64)) @ Wo.T
    xn = r16(norm(x, fn))
    g, u = xn @ Wg.T, xn @ Wu.T
    hmid = r16(g / (1 + np.exp(-g)) * u)
    x = x + hmid @ Wd.T
    assert np.allclose(got, x, rtol=1e-11, atol=1e-11)
    assert np.array_equal(out16, x.astype(np.float16).view(np.uint16)) or \
        np.abs(f16(out16) - x).max() <= np.abs(x).max() * 2.0 ** -11
    k_new, v_new = eng.read(0, 0, P, 3)
    assert np.allclose(f16(k_new), r16(k).astype(np.float16).astype(np.float64), rtol=2.0 ** -10, atol=1e-6)


def test_logits_head_closed_form():
    # embedding rows e_v = unit vectors: logits are the un-weighted RMSNorm of h
    H, V = 16, 16
    E = np.eye(V, H).astype(np.float16).view(np.uint16)
    h = np.random.default_rng(3).standard_normal((2, H))
    lg = oracle.logits(h, E, 1e-5)
    ref = h / np.sqrt((h * h).mean(axis=1, keepdims=True) + 1e-5)
    assert np.allclose(lg, ref, rtol=1e-14)
