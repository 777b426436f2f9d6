"""GPU parity of whole shard steps on the tiny workload (2 layers, hidden
256, 4q/2kv heads, head_dim 64, FFN 688, group 32), through the C ABI,
against the CPU oracle: decode, a 1+4 verify with mask rewind versus a
physical trim, beam_idx gathers versus physically reordered caches, greedy
speculative decoding versus target-only decoding, batch-composition
invariance, determinism, and the error paths."""
import numpy as np
import pytest
import torch

import paper_2608_19147_gb300 as pkg
import synth
from gpu_engine import GpuEngine, GpuShard, assert_close
from scenarios import (MaskedRequest, OracleEngine, f16, greedy_decode, prefill, spec_decode,
                       tiny_steps_masked_vs_trim)

pytestmark = pytest.mark.gpu
TINY = synth.TINY
SEED = 20260802


@pytest.fixture(scope="module")
def tiny():
    w = synth.make_weights(TINY, SEED)
    sh = GpuShard(TINY, w)
    yield w, sh
    sh.close()


def test_decode_and_verify_match_oracle_and_trim(tiny):
    w, sh = tiny
    gpu = tiny_steps_masked_vs_trim(lambda cap: GpuEngine(sh, 1, cap), TINY, w)
    ora = tiny_steps_masked_vs_trim(lambda cap: OracleEngine(TINY, w, 1, cap), TINY, w)
    for mode in ("mask", "trim"):
        for s in ("A", "B", "C"):
            assert_close(gpu[(mode, s)], ora[(mode, s)], what="%s step %s" % (mode, s))
    # the mask rewind and the physical trim agree on the GPU too (different
    # split-KV chunking, so within rounding rather than bit for bit)
    assert_close(gpu[("mask", "C")], gpu[("trim", "C")], rel=2e-4, mx=4e-3, what="mask vs trim on GPU")
    # appended K/V entries: positions written where the oracle writes them
    em, eo = gpu[("mask", "engine")], ora[("mask", "engine")]
    assert em.length(0) == eo.length(0) == 72 + 1 + 5 + 1
    for layer in range(TINY.n_layers):
        kg, vg = em.read(0, layer, 0, em.length(0))
        ko, vo = eo.read(0, layer, 0, eo.length(0))
        assert np.array_equal(kg[:72], ko[:72]) and np.array_equal(vg[:72], vo[:72])  # prefill untouched
        assert np.abs(f16(kg) - f16(ko)).max() < 2e-2 and np.abs(f16(vg) - f16(vo)).max() < 2e-2
    for e in (gpu[("mask", "engine")], gpu[("trim", "engine")]):
        e.close()


def test_steps_are_deterministic(tiny):
    # two shards, same inputs: bit-identical outputs and caches
    w, _ = tiny
    outs, caches = [], []
    for _rep in range(2):
        sh = GpuShard(TINY, w)
        eng = GpuEngine(sh, 1, 96)
        prefill(eng, TINY, SEED, 0, 72)
        req = MaskedRequest(72)
        o = []
        for step in range(3):
            n = 5 if step == 1 else 1
            o.append(eng.step([n], req.positions(n), req.mask_for(n), hidden_in=synth.hidden_in(TINY, SEED, step, n)))
            req.commit(n, n - 2 if n == 5 else 1)
        outs.append(o)
        caches.append(eng.read(0, 1, 0, eng.length(0)))
        eng.close()
        sh.close()
    for a, b in zip(outs[0], outs[1]):
        assert np.array_equal(a, b)
    assert all(np.array_equal(x, y) for x, y in zip(caches[0], caches[1]))


def test_phase_times_cover_the_step(tiny):
    w, sh = tiny
    eng = GpuEngine(sh, 1, 96)
    prefill(eng, TINY, SEED, 0, 40)
    eng.step([1], np.array([40], np.int32), np.ones(41, np.uint8), hidden_in=synth.hidden_in(TINY, SEED, 0, 1))
    t = pkg.shard_debug_phase_times(sh.h, TINY.n_layers)
    assert len(t) == len(pkg.PHASES) * TINY.n_layers + 1 and all(x >= 0 for x in t) and sum(t) > 0
    eng.close()


def test_beam_gather_steps_match_oracle(tiny):
    # several steps with permutations and a duplicate (a Gather, not only a
    # permutation); rows of unequal length; a hole in a gathered history
    w, sh = tiny
    B, lens = 4, [20, 33, 27, 41]
    a = GpuEngine(sh, B, 64)
    ref = OracleEngine(TINY, w, B, 64)
    for r in range(B):
        prefill(a, TINY, SEED + r, r, lens[r])
        prefill(ref, TINY, SEED + r, r, lens[r])
    cur = list(lens)
    for step, perm in enumerate([[2, 0, 3, 1], [1, 1, 0, 3], [3, 2, 1, 0]]):
        perm = np.array(perm, np.int32)
        n_new = [1, 2, 1, 1]
        new_len = [cur[p] for p in perm]
        stride = max(L + n for L, n in zip(new_len, n_new)) + 3
        mask = np.zeros((B, stride), np.uint8)
        for r in range(B):
            mask[r, : new_len[r] + n_new[r]] = 1
        mask[1, 3] = 0
        pos = np.concatenate([np.arange(L, L + n, dtype=np.int32) for L, n in zip(new_len, n_new)])
        h = synth.hidden_in(TINY, SEED, 40 + step, sum(n_new))
        og = a.step(n_new, pos, mask, hidden_in=h, beam_idx=perm)
        oo = ref.step(n_new, pos, mask, hidden_in=h, beam_idx=perm)
        assert_close(og, oo, what="beam step %d" % step)
        cur = [L + n for L, n in zip(new_len, n_new)]
        for r in range(B):
            assert a.length(r) == ref.length(r) == cur[r]
    a.close()


def test_indirect_reads_bit_exact_against_gathered_cache(tiny):
    w, sh = tiny
    B, lens = 3, [30, 18, 25]
    perm = np.array([2, 2, 0], np.int32)
    a, b = GpuEngine(sh, B, 64), GpuEngine(sh, B, 64)
    for r in range(B):
        prefill(a, TINY, SEED + r, r, lens[r])
    for r in range(B):
        for layer in range(TINY.n_layers):
            k, v = a.read(int(perm[r]), layer, 0, lens[perm[r]])
            b.load(r, layer, k, v)
    new_len = [lens[p] for p in perm]
    n_new = [1, 1, 2]
    stride = max(L + n for L, n in zip(new_len, n_new))
    mask = np.zeros((B, stride), np.uint8)
    for r in range(B):
        mask[r, : new_len[r] + n_new[r]] = 1
    pos = np.concatenate([np.arange(L, L + n, dtype=np.int32) for L, n in zip(new_len, n_new)])
    h = synth.hidden_in(TINY, SEED, 77, sum(n_new))
    oa = a.step(n_new, pos, mask, hidden_in=h, beam_idx=perm)
    ob = b.step(n_new, pos, mask, hidden_in=h)
    assert np.array_equal(oa, ob)
    for r in range(B):
        L = a.length(r)
        assert L == b.length(r)
        for layer in range(TINY.n_layers):
            ka, va = a.read(r, layer, 0, L)
            kb, vb = b.read(r, layer, 0, L)
            assert np.array_equal(ka, kb) and np.array_equal(va, vb)
    a.close()
    b.close()


def test_batch_composition_invariance_bitwise(tiny):
    w, sh = tiny
    lens, n_new, B = [40, 61, 25, 33], [1, 3, 2, 1], 4
    hs = [synth.hidden_in(TINY, SEED + 10 + r, 0, n_new[r]) for r in range(B)]
    batch = GpuEngine(sh, B, 80)
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
        alone = GpuEngine(sh, 1, 80)
        prefill(alone, TINY, SEED + r, 0, lens[r], src_row=r)
        oa = alone.step([n_new[r]], np.arange(lens[r], lens[r] + n_new[r], dtype=np.int32),
                        np.ones(lens[r] + n_new[r], np.uint8), hidden_in=hs[r])
        assert np.array_equal(oa, ob[t: t + n_new[r]]), r
        t += n_new[r]
        alone.close()
    batch.close()


def test_speculative_greedy_equals_target_greedy(tiny):
    w, sh = tiny
    n = 20
    target, margins = greedy_decode(OracleEngine(TINY, w, 1, 256), TINY, w, SEED, n)
    g_target, g_margins = greedy_decode(GpuEngine(sh, 1, 256), TINY, w, SEED, n)
    g_spec, s_margins, req = spec_decode(GpuEngine(sh, 1, 256), TINY, w, SEED, n, target)
    # tokens agree wherever the oracle's top-2 margin is decisive
    for i in range(n):
        if margins[i] <= 1e-2:
            break
        assert g_target[i] == target[i], i
        assert g_spec[i] == target[i], i
    assert len(req.valid) > req.pos  # rejected drafts stayed in the cache, masked


def test_token_ids_path_matches_oracle(tiny):
    w, sh = tiny
    g, o = GpuEngine(sh, 1, 96), OracleEngine(TINY, w, 1, 96)
    for e in (g, o):
        prefill(e, TINY, SEED, 0, 10)
    tok = synth.token_ids(TINY, SEED, 3, 4)
    args = ([4], np.arange(10, 14, dtype=np.int32), np.ones(14, np.uint8))
    assert_close(g.step(*args, token_ids=tok), o.step(*args, token_ids=tok), what="token ids")
    g.close()


def test_step_host_equals_device_step(tiny):
    w, sh = tiny
    a, b = GpuEngine(sh, 1, 96), GpuEngine(sh, 1, 96)
    for e in (a, b):
        prefill(e, TINY, SEED, 0, 50)
    h = synth.hidden_in(TINY, SEED, 8, 3)
    pos = np.arange(50, 53, dtype=np.int32)
    mask = np.ones((1, 53), np.uint8)
    oa = a.step([3], pos, mask, hidden_in=h)
    ob = np.empty((3, TINY.hidden), np.uint16)
    pkg.shard_step_host(sh.h, b.st, h, None, [3], pos, mask, None, ob)
    assert np.array_equal(oa, ob)
    a.close()
    b.close()


def test_error_paths(tiny):
    w, sh = tiny
    e = GpuEngine(sh, 2, 16)
    for r in range(2):
        prefill(e, TINY, SEED, r, 10)
    h = synth.hidden_in(TINY, SEED, 0, 17)
    one = np.ones((2, 16), np.uint8)
    # host-side: too many tokens, B mismatch, capacity
    rc, _ = e.step_raw([9, 8], np.arange(17, dtype=np.int32), one, hidden_in=h, check=False)
    assert rc == pkg.SHARD_EINVAL
    rc, _ = e.step_raw([1], np.array([10], np.int32), one[:1], hidden_in=h[:1], check=False)
    assert rc == pkg.SHARD_EINVAL
    rc, _ = e.step_raw([7, 1], np.arange(8, dtype=np.int32), one, hidden_in=h[:8], check=False)
    assert rc == pkg.SHARD_ECAPACITY
    # device-side: beam_idx out of range is reported, nothing is written
    rc, _ = e.step_raw([1, 1], np.array([10, 10], np.int32), one, hidden_in=h[:2],
                       beam_idx=np.array([0, 5], np.int32), check=False)
    assert rc == pkg.SHARD_EINVAL and "beam_idx" in pkg.shard_last_error()
    # the state is frozen until reset
    rc, _ = e.step_raw([1, 1], np.array([10, 10], np.int32), one, hidden_in=h[:2], check=False)
    assert rc == pkg.SHARD_EINVAL
    pkg.kv_state_reset(e.st, -1)
    assert e.length(0) == 0
    # a zero mask at a new entry
    rc, _ = e.step_raw([1, 1], np.array([0, 0], np.int32), np.zeros((2, 16), np.uint8), hidden_in=h[:2], check=False)
    assert rc == pkg.SHARD_EINVAL and "mask" in pkg.shard_last_error()
    pkg.kv_state_reset(e.st, -1)
    # position outside the rotary table
    rc, _ = e.step_raw([1, 1], np.array([0, TINY.max_position], np.int32), one, hidden_in=h[:2], check=False)
    assert rc == pkg.SHARD_EINVAL and "position" in pkg.shard_last_error()
    pkg.kv_state_reset(e.st, -1)
    # the state works again after the reset
    rc, out = e.step_raw([1, 1], np.array([0, 0], np.int32), one, hidden_in=h[:2], check=False)
    assert rc == 0 and np.isfinite(out.view(np.float16)).all()
    e.close()
