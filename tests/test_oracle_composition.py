"""The oracle's whole shard against an independent numpy model, over several
steps: two layers, two requests, a decode and a verify row in one step, a
rejected draft left masked in the cache (Section 5.2), a beam_idx gather
that swaps the requests' histories and one with a duplicate parent
(Section 4).

The numpy model keeps its own cache, a list of K and V arrays per request
and layer.  It appends each step's rounded K and V in token order and
copies whole histories for a gather.  Its matrices are exactly
representable integers times powers of two, built without the oracle.  RoPE
is a complex rotation and the softmax is numpy's.  It shares nothing with
the oracle but the seeded inputs.  Agreement pins what the one-layer
formulation cannot: the layers' order and their residual hand-off, each
layer's K/V going to its own cache at the right positions, state carried
from step to step, the per-request causal bound inside a multi-token row,
and gather lineage with unequal lengths.
"""
import copy
import math

import numpy as np
import pytest

import synth
from scenarios import OracleEngine, f16

H, HQ, HKV, D, F, G, L = 64, 4, 2, 16, 96, 32, 2
THETA = 10000.0
SHAPE = synth.ShardShape("composition", L, H, HQ, HKV, D, F, G, 0.02, 0, 1e-5, THETA, 128)


def _weights(rng):
    layers, dense = [], []
    for _ in range(L):
        mats, dl = [], []
        for name in synth.MATRIX_NAMES:
            r, c = SHAPE.matrix_shape(name)
            n_g = c // G
            z = rng.integers(0, 16, (r, n_g))
            zz = np.repeat(z, G, axis=1)
            Dq = rng.integers(-zz, 16 - zz)       # q - z, with q in [0, 15]
            s = 2.0 ** rng.integers(-8, -4, (r, n_g)).astype(np.float64)
            q = Dq + zz
            codes = (q[:, 0::2] | (q[:, 1::2] << 4)).astype(np.uint8)
            zeros = (z[:, 0::2] | (z[:, 1::2] << 4)).astype(np.uint8)
            mats.append(synth.PackedMatrix(r, c, G, codes, s.astype(np.float16).view(np.uint16), zeros))
            dl.append(Dq * np.repeat(s, G, axis=1))
        an = (1 + 0.1 * rng.standard_normal(H)).astype(np.float16)
        fn = (1 + 0.1 * rng.standard_normal(H)).astype(np.float16)
        layers.append(synth.LayerWeights(mats, an.view(np.uint16), fn.view(np.uint16)))
        dense.append((dl, an.astype(np.float64), fn.astype(np.float64)))
    return synth.ShardWeights(SHAPE, 0, layers, None), dense


def _r16(a):
    return a.astype(np.float16).astype(np.float64)


def _norm(a, g):
    return a / np.sqrt((a * a).mean(axis=1, keepdims=True) + 1e-5) * g


def _rot(vecs, p):
    h = vecs.shape[-1] // 2
    z = (vecs[..., :h] + 1j * vecs[..., h:]) * np.exp(1j * p * THETA ** (-np.arange(h) * 2.0 / vecs.shape[-1]))
    return np.concatenate([z.real, z.imag], axis=-1)


class Model:
    """Independent numpy shard with its own per-request, per-layer cache."""

    def __init__(self, dense, caches):
        self.dense = dense
        self.cache = caches  # [request][layer] -> (K [n][HKV][D], V [n][HKV][D]) as float64

    def step(self, n_new, pos, mask, x16, beam=None):
        if beam is not None:
            self.cache = [copy.deepcopy(self.cache[p]) for p in beam]
        x = x16.astype(np.float64)
        M = x.shape[0]
        for layer, (W, an, fn) in enumerate(self.dense):
            Wq, Wk, Wv, Wo, Wg, Wu, Wd = W
            xn = _r16(_norm(x, an))
            q = (xn @ Wq.T).reshape(M, HQ, D)
            k = (xn @ Wk.T).reshape(M, HKV, D)
            v = (xn @ Wv.T).reshape(M, HKV, D)
            att = np.zeros((M, HQ, D))
            t0 = 0
            for b, n in enumerate(n_new):
                Kc, Vc = self.cache[b][layer]
                P = Kc.shape[0]
                kb = np.stack([_r16(_rot(k[t0 + i], pos[t0 + i])) for i in range(n)])
                Kc = np.concatenate([Kc, kb])
                Vc = np.concatenate([Vc, _r16(v[t0:t0 + n])])
                self.cache[b][layer] = (Kc, Vc)
                for i in range(n):
                    qi = _rot(q[t0 + i], pos[t0 + i])
                    vis = np.flatnonzero(mask[b][: P + i + 1])
                    for h in range(HQ):
                        sc = Kc[vis, h // (HQ // HKV)] @ qi[h] / math.sqrt(D)
                        p_ = np.exp(sc - sc.max())
                        att[t0 + i, h] = (p_ / p_.sum()) @ Vc[vis, h // (HQ // HKV)]
                t0 += n
            x = x + _r16(att.reshape(M, H)) @ Wo.T
            xn = _r16(_norm(x, fn))
            g, u = xn @ Wg.T, xn @ Wu.T
            x = x + _r16(g / (1 + np.exp(-g)) * u) @ Wd.T
        return x


def _mask(rows, stride):
    m = np.zeros((len(rows), stride), np.uint8)
    for b, r in enumerate(rows):
        m[b, : len(r)] = r
    return m


def test_whole_shard_over_steps_matches_independent_model():
    rng = np.random.default_rng(2026)
    w, dense = _weights(rng)
    lens = [5, 9]
    eng = OracleEngine(SHAPE, w, 2, 32)
    caches = []
    for b, P in enumerate(lens):
        per = []
        for layer in range(L):
            k = rng.standard_normal((P, HKV, D)).astype(np.float16)
            v = rng.standard_normal((P, HKV, D)).astype(np.float16)
            eng.load(b, layer, k.view(np.uint16), v.view(np.uint16))
            per.append((k.astype(np.float64), v.astype(np.float64)))
        caches.append(per)
    model = Model(dense, caches)
    valid = [[1] * 5, [1] * 9]
    logical = [5, 9]

    def run(n_new, beam=None, rejected=None):
        nonlocal valid, logical
        if beam is not None:
            valid = [list(valid[p]) for p in beam]
            logical = [logical[p] for p in beam]
        pos = np.concatenate([np.arange(logical[b], logical[b] + n, dtype=np.int32) for b, n in enumerate(n_new)])
        rows = [valid[b] + [1] * n for b, n in enumerate(n_new)]
        mask = _mask(rows, max(len(r) for r in rows))
        x16 = rng.standard_normal((sum(n_new), H)).astype(np.float16)
        out16 = eng.step(n_new, pos, mask, hidden_in=x16.view(np.uint16),
                         beam_idx=None if beam is None else np.array(beam, np.int32))
        want = model.step(n_new, pos, mask, x16, beam)
        assert np.allclose(eng.last_f64, want, rtol=1e-11, atol=1e-11)
        assert np.abs(f16(out16) - want).max() <= np.abs(want).max() * 2.0 ** -11
        for b, n in enumerate(n_new):
            keep = n if rejected is None else n - rejected[b]
            valid[b] = valid[b] + [1] * keep + [0] * (n - keep)
            logical[b] += keep

    run([1, 3], rejected=[0, 1])     # request 1 verifies 3 tokens; its last draft is rejected
    run([2, 1], beam=[1, 0])         # the histories swap rows; the hole travels with request 1
    run([1, 1], beam=[0, 0])         # both rows continue the same history
    # the caches agree entry by entry, holes included
    for b in range(2):
        for layer in range(L):
            n = eng.length(b)
            k16, v16 = eng.read(b, layer, 0, n)
            K, V = model.cache[b][layer]
            assert n == K.shape[0]
            assert np.allclose(f16(k16), K, rtol=2.0 ** -10, atol=1e-6)
            assert np.array_equal(f16(v16), V)
