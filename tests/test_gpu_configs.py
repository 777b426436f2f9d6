"""GPU parity of the Llama-3.1-8B stage's micro-batch and speculative
workloads at their stated sizes, through the C ABI.

* Micro-batch: 8 requests with caches of U{128..2048} entries, a fresh
  random beam_idx permutation every step, one new token per request (M = 8).
  Layer by layer (as in test_gpu_layers.py), every layer's output is within
  the fixed bar of the one-layer oracle, and the beam-table reads
  (Gather(ReadValue, beam_idx), Section 4) are bit-exact against a second GPU
  state whose rows were physically gathered on the host before the step:
  same outputs, bit for bit, and the same appended K/V.
* Speculative decoding at full depth: greedy speculative decoding with
  mask-based rewind gives the same tokens as plain greedy decoding on the GPU
  (Section 5.3), and both give the oracle's tokens wherever its top-2 margin
  exceeds 1e-2.
"""
import numpy as np
import pytest

import synth
from gpu_engine import GpuEngine, GpuShard
from scenarios import OracleEngine, greedy_decode, spec_decode
from test_gpu_layers import assert_fixed_bar, one_layer

pytestmark = pytest.mark.gpu
SEED = 20261204


def _gather_rows_on_host(eng, shape, perm, lens):
    """Rebuilds eng so that row b holds what row perm[b] held (a physical
    gather, no beam table): export every row, reset, import permuted."""
    import paper_2608_19147_gb300 as pkg
    rows = [pkg.kv_state_export(eng.st, r, lens[r], 1, shape.n_kv_heads, shape.head_dim) for r in range(len(lens))]
    pkg.kv_state_reset(eng.st, -1)
    for b, src in enumerate(perm):
        pkg.kv_state_import(eng.st, b, *rows[src])


def test_8b_microbatch_every_layer_indirect_equals_gathered():
    shape = synth.LLAMA8B_STAGE
    B, n_steps = 8, 3
    lens0 = synth.lengths(SEED, B, 128, 2048).astype(int).tolist()
    cap = max(lens0) + n_steps + 8
    perms = [synth.permutation(SEED, s, B).astype(np.int32) for s in range(n_steps)]
    assert all(not np.array_equal(p, np.arange(B)) for p in perms)
    inputs = [synth.hidden_in(shape, SEED, 400 + s, B) for s in range(n_steps)]
    for layer in range(shape.n_layers):
        s1 = one_layer(shape, layer)
        w1 = synth.ShardWeights(s1, SEED, [synth.layer_weights(shape, SEED, layer)],
                                synth.embedding(shape, SEED) if s1.vocab else None)
        sh = GpuShard(s1, w1)
        ga, gb = GpuEngine(sh, B, cap), GpuEngine(sh, B, cap)
        o = OracleEngine(s1, w1, B, cap)
        for r in range(B):
            k, v = synth.kv_prefill(shape, SEED + 11, r, lens0[r], layer)
            for e in (ga, gb, o):
                e.load(r, 0, k, v)
        lens = list(lens0)
        outs = []
        for s in range(n_steps):
            perm = perms[s]
            new = [lens[p] for p in perm]
            mask = np.zeros((B, cap), np.uint8)
            for b in range(B):
                mask[b, : new[b] + 1] = 1
            pos = np.array(new, np.int32)
            _gather_rows_on_host(gb, shape, perm, lens)
            oa = ga.step([1] * B, pos, mask, hidden_in=inputs[s], beam_idx=perm)
            ob = gb.step([1] * B, pos, mask, hidden_in=inputs[s])
            oo = o.step([1] * B, pos, mask, hidden_in=inputs[s], beam_idx=perm)
            what = "8b micro-batch layer %d step %d" % (layer, s)
            assert np.array_equal(oa, ob), what + ": indirect != gathered"
            assert_fixed_bar(oa, oo, what)
            lens = [x + 1 for x in new]
            for r in range(B):
                assert ga.length(r) == gb.length(r) == o.length(r) == lens[r]
            outs.append(oa)
        for r in (0, 3, 7):
            ka, va = ga.read(r, 0, 0, lens[r])
            kb, vb = gb.read(r, 0, 0, lens[r])
            assert np.array_equal(ka, kb) and np.array_equal(va, vb), (layer, r)
        ga.close()
        gb.close()
        sh.close()
        inputs = outs


def test_8b_speculative_greedy_equals_plain_greedy_full_depth():
    shape = synth.LLAMA8B_STAGE
    w = synth.make_weights(shape, SEED)
    sh = GpuShard(shape, w)
    n, cap = 16, 256
    try:
        plain, pm = greedy_decode(GpuEngine(sh, 1, cap), shape, w, SEED, n)
        truth, margins = greedy_decode(OracleEngine(shape, w, 1, cap), shape, w, SEED, 8)
        spec, _, req = spec_decode(GpuEngine(sh, 1, cap), shape, w, SEED, n, plain)
    finally:
        sh.close()
    assert len(req.valid) > req.pos, "no draft was rejected"
    sure = n if all(m > 1e-2 for m in pm) else int(np.argmin(np.array(pm) > 1e-2))
    assert sure >= 8, pm
    assert spec[:sure] == plain[:sure], (spec, plain)
    for i in range(8):
        if margins[i] <= 1e-2:
            break
        assert plain[i] == truth[i], (i, plain, truth)
