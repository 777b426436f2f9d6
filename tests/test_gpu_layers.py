"""Layer-by-layer GPU parity at the fixed tolerance, at full width and depth.

Each layer of the Llama-3.1-8B stage (16 layers) and of the Llama-3.1-70B
stage (20 layers, 4096-entry cache) runs as a one-layer GPU shard through
the C ABI, and the same layer runs as a one-layer fp64 oracle shard.  Layer
l of both gets the GPU's fp16 output of layer l - 1 as its input, so every
layer is checked on its own, and a small bias that compounds over depth
cannot hide behind the drift that the fp16 rounding points cause between any
two correct implementations at full depth.

The steps follow the speculative-verify workloads: token or hidden-state
decode steps, then 1 + 4 verify steps whose rejected drafts (seeded
Bernoulli(0.6), longest accepted prefix, Section 5.2) stay in the cache
with attention_mask = 0, so masked holes accumulate mid-cache.  Every layer
also runs a second GPU state that physically trims the rejected entries
after each step (kv_trim): mask-based rewind must equal the trim.

Bar, per layer and step, on the fp16 hidden output: relative L2 <= 1e-3,
and max-abs <= 2e-2 -- except at elements whose oracle value is so large
that one fp16 ulp exceeds 2e-2 (|h| >= 32), where two correct
implementations may round to adjacent fp16 values: there the bound is one
ulp.  The appended K/V entries must match the oracle's within the same
per-element bound.
"""
import dataclasses

import numpy as np
import pytest

import synth
from gpu_engine import GpuEngine, GpuShard, TOL_MAX_ABS, TOL_REL_L2
from scenarios import MaskedRequest, OracleEngine, f16

pytestmark = pytest.mark.gpu


def fp16_ulp(x: np.ndarray) -> np.ndarray:
    """Spacing of fp16 values at |x| (normal range)."""
    a = np.maximum(np.abs(x), 2.0 ** -14)
    return 2.0 ** (np.floor(np.log2(a)) - 10)


def assert_fixed_bar(got16, want16, what):
    g, w = f16(got16), f16(want16)
    assert np.isfinite(g).all(), what + ": non-finite GPU output"
    r = np.linalg.norm(g - w) / np.linalg.norm(w)
    bound = np.maximum(TOL_MAX_ABS, fp16_ulp(w))
    err = np.abs(g - w)
    worst = int(np.argmax(err - bound))
    assert r <= TOL_REL_L2 and (err <= bound).all(), (
        "%s: relL2 %.3e (tol %.1e); max-abs %.3e at |h| = %.3g (bound %.3e)"
        % (what, r, TOL_REL_L2, err.flat[worst], abs(w.flat[worst]), bound.flat[worst]))
    return r, float(err.max())


def one_layer(shape, layer):
    return dataclasses.replace(shape, name="%s-layer%d" % (shape.name, layer), n_layers=1,
                               vocab=shape.vocab if layer == 0 else 0)


def _load_prefill(engine, shape, seed, layer, length):
    k, v = synth.kv_prefill(shape, seed, 0, length, layer)
    engine.load(0, 0, k, v)


def run_layer_chain(shape, seed, L0, plan, first_layer_input):
    """Runs `plan` (a list of (n_fed, n_kept) steps) layer by layer.

    first_layer_input(step, n) gives layer 0's input as ("token_ids" |
    "hidden_in", array).  Returns the per-(layer, step) (relL2, max-abs)
    of GPU vs oracle and of GPU trimmed vs GPU masked."""
    cap = L0 + sum(n for n, _ in plan) + 8
    inputs = [first_layer_input(s, n) for s, (n, _) in enumerate(plan)]
    report = []
    for layer in range(shape.n_layers):
        s1 = one_layer(shape, layer)
        lw = synth.layer_weights(shape, seed, layer)
        w1 = synth.ShardWeights(s1, seed, [lw], synth.embedding(shape, seed) if s1.vocab else None)
        sh = GpuShard(s1, w1)
        g, gt = GpuEngine(sh, 1, cap), GpuEngine(sh, 1, cap)
        o = OracleEngine(s1, w1, 1, cap)
        for e in (g, gt, o):
            _load_prefill(e, shape, seed + 7, layer, L0)
        req, req_t = MaskedRequest(L0), MaskedRequest(L0)
        outs = []
        for s, (n, kept) in enumerate(plan):
            kind, x = inputs[s]
            kw = {kind: x}
            args = ([n], req.positions(n), req.mask_for(n))
            og, oo = g.step(*args, **kw), o.step(*args, **kw)
            assert np.array_equal(req_t.positions(n), req.positions(n))
            ot = gt.step([n], req_t.positions(n), req_t.mask_for(n), **kw)
            what = "%s layer %d step %d (M=%d)" % (shape.name, layer, s, n)
            rep = assert_fixed_bar(og, oo, what)
            rept = assert_fixed_bar(ot, og, what + " trimmed vs masked")
            report.append((layer, s, rep, rept))
            outs.append(("hidden_in", og))
            req.commit(n, kept)
            # the physical-trim rerun drops the rejected entries at once
            gt.trim(0, np.array([1] * (gt.length(0) - (n - kept)) + [0] * (n - kept), np.uint8))
            req_t.valid = [1] * gt.length(0)
            req_t.pos = req.pos
        # the entries this layer appended, masked ones included, against the oracle's
        n_app = g.length(0) - L0
        kg, vg = g.read(0, 0, L0, n_app)
        ko, vo = o.read(0, 0, L0, n_app)
        for a, b, nm in ((kg, ko, "K"), (vg, vo, "V")):
            a, b = f16(a), f16(b)
            bound = np.maximum(TOL_MAX_ABS, fp16_ulp(b))
            assert (np.abs(a - b) <= bound).all(), "%s layer %d appended %s" % (shape.name, layer, nm)
        g.close()
        gt.close()
        sh.close()
        inputs = outs
    return report


def verify_plan(seed, n_decode, n_verify):
    plan = [(1, 1)] * n_decode
    for s in range(n_verify):
        plan.append((5, 1 + synth.accepted_drafts(seed, 100 + s)))
    return plan


def test_8b_every_layer_fixed_bar_decode_and_16_verify_steps():
    shape = synth.LLAMA8B_STAGE
    seed = 20261202
    plan = verify_plan(seed, 2, 16)
    assert any(k < 5 for n, k in plan if n == 5), "the accept pattern must reject some drafts"

    def first(s, n):
        if n == 1:
            return "token_ids", synth.token_ids(shape, seed, s, 1)
        return "hidden_in", synth.hidden_in(shape, seed, 100 + s, n)

    rep = run_layer_chain(shape, seed, 512, plan, first)
    worst = max(r[2][0] for r in rep)
    print("8b per-layer worst relL2 %.3e" % worst)


def test_70b_every_layer_fixed_bar_4096_cache():
    shape = synth.LLAMA70B_STAGE
    seed = 20261203
    plan = verify_plan(seed, 2, 2)

    def first(s, n):
        return "hidden_in", synth.hidden_in(shape, seed, 300 + s, n)

    rep = run_layer_chain(shape, seed, 4096, plan, first)
    worst = max(r[2][0] for r in rep)
    print("70b per-layer worst relL2 %.3e" % worst)
