"""Edge cases of the oracle's shard step, each pinned by what it must equal.

- Empty cache (a stateful cache that starts a new sequence, Section 3.4): a
  request's first token sees only its own new entry, softmax over one entry
  is exactly 1, so the step's output cannot depend on the q or k projections
  of any layer.  With one cached entry in front it must depend on them: the
  check has teeth.
- A verify block on an empty cache (causality inside the block): its first
  token is independent of q and k as above, its second token is not.
- The largest step, 16 new tokens, both as 16 requests of one token (with a
  beam_idx gather among them) and as one request of 16 tokens, equals the
  same requests run one at a time, bit for bit (Section 8.6's
  batch-composition invariance at the size limit).
- Arbitrary hole patterns (Section 5.2): holes anywhere in the cache and any
  subset of each step's new entries rejected give the same bits as a cache
  with exactly those entries deleted.
"""
import dataclasses

import numpy as np
import pytest

import synth
from scenarios import OracleEngine, f16, prefill

TINY = synth.TINY
SEED = 20260803


@pytest.fixture(scope="module")
def weights():
    return synth.make_weights(TINY, SEED)


@pytest.fixture(scope="module")
def weights_other_qk(weights):
    """The same shard with every layer's q and k matrices replaced."""
    other = synth.make_weights(TINY, SEED + 1)
    layers = []
    for lw, lo in zip(weights.layers, other.layers):
        mats = list(lw.matrices)
        mats[0], mats[1] = lo.matrices[0], lo.matrices[1]
        layers.append(dataclasses.replace(lw, matrices=mats))
    return dataclasses.replace(weights, layers=layers)


def _step(w, cache_len, n, seed=5):
    e = OracleEngine(TINY, w, 1, 64)
    if cache_len:
        prefill(e, TINY, SEED, 0, cache_len)
    h = synth.hidden_in(TINY, seed, 0, n)
    return e.step([n], np.arange(cache_len, cache_len + n, dtype=np.int32), np.ones(cache_len + n, np.uint8),
                  hidden_in=h)


def test_first_token_on_an_empty_cache_ignores_q_and_k(weights, weights_other_qk):
    a = _step(weights, 0, 1)
    b = _step(weights_other_qk, 0, 1)
    assert np.array_equal(a, b)
    # teeth: with one cached entry the scores matter
    a1 = _step(weights, 1, 1)
    b1 = _step(weights_other_qk, 1, 1)
    assert np.abs(f16(a1) - f16(b1)).max() > 1e-3


def test_verify_block_on_an_empty_cache(weights, weights_other_qk):
    a = _step(weights, 0, 2)
    b = _step(weights_other_qk, 0, 2)
    assert np.array_equal(a[0], b[0])                     # sees only itself
    assert np.abs(f16(a[1]) - f16(b[1])).max() > 1e-3    # sees itself and token 0


def test_sixteen_requests_of_one_token_equal_each_alone(weights):
    B = 16
    lens = synth.lengths(SEED, B, 1, 40).tolist()
    beam = np.array([(3 * b + 1) % B for b in range(B)], np.int32)
    beam[5] = beam[6]  # a Gather, with a duplicate parent
    batch = OracleEngine(TINY, weights, B, 64)
    for r in range(B):
        prefill(batch, TINY, SEED + r, r, lens[r])
    new_len = [lens[p] for p in beam]
    h = synth.hidden_in(TINY, SEED, 3, B)
    stride = max(new_len) + 1
    mask = np.zeros((B, stride), np.uint8)
    for r in range(B):
        mask[r, :new_len[r] + 1] = 1
    out = batch.step([1] * B, np.array(new_len, np.int32), mask, hidden_in=h, beam_idx=beam)
    for r in range(B):
        alone = OracleEngine(TINY, weights, 1, 64)
        prefill(alone, TINY, SEED + int(beam[r]), 0, lens[beam[r]], src_row=int(beam[r]))
        o = alone.step([1], np.array([new_len[r]], np.int32), np.ones(new_len[r] + 1, np.uint8),
                       hidden_in=h[r:r + 1])
        assert np.array_equal(o[0], out[r]), r


def test_one_request_of_sixteen_tokens_equals_sixteen_single_steps(weights):
    # the 16-token block computes each token against the cache and the block's
    # earlier tokens: the same as feeding them one per step
    P, n = 20, 16
    h = synth.hidden_in(TINY, SEED, 7, n)
    block = OracleEngine(TINY, weights, 1, 64)
    prefill(block, TINY, SEED, 0, P)
    ob = block.step([n], np.arange(P, P + n, dtype=np.int32), np.ones(P + n, np.uint8), hidden_in=h)
    one = OracleEngine(TINY, weights, 1, 64)
    prefill(one, TINY, SEED, 0, P)
    for t in range(n):
        o = one.step([1], np.array([P + t], np.int32), np.ones(P + t + 1, np.uint8), hidden_in=h[t:t + 1])
        assert np.array_equal(o[0], ob[t]), t
    for layer in range(TINY.n_layers):
        ka, va = block.read(0, layer, 0, P + n)
        kb, vb = one.read(0, layer, 0, P + n)
        assert np.array_equal(ka, kb) and np.array_equal(va, vb)


@pytest.mark.parametrize("seed", range(6))
def test_arbitrary_holes_equal_physical_trim(weights, seed):
    # holes anywhere in the cache -- not only rejected-draft suffixes -- and
    # any subset of each step's new entries rejected afterwards: the masked
    # run equals a run whose cache had exactly those entries deleted, bit for
    # bit in fp64 and in fp16 (Section 5.2's exactness, for every hole pattern)
    rng = np.random.default_rng(seed)
    P = int(rng.integers(8, 40))
    keep = rng.random(P) >= 0.3
    keep[rng.integers(P)] = False  # at least one hole
    masked = OracleEngine(TINY, weights, 1, 96)
    trimmed = OracleEngine(TINY, weights, 1, 96)
    prefill(masked, TINY, SEED + seed, 0, P)
    prefill(trimmed, TINY, SEED + seed, 0, P)
    trimmed.trim(0, keep.astype(np.uint8))
    valid = keep.astype(np.uint8).tolist()
    pos = P
    for step in range(4):
        n = int(rng.integers(1, 5))
        h = synth.hidden_in(TINY, SEED + seed, step, n)
        positions = np.arange(pos, pos + n, dtype=np.int32)
        om = masked.step([n], positions, np.array(valid + [1] * n, np.uint8), hidden_in=h)
        ot = trimmed.step([n], positions, np.ones(sum(valid) + n, np.uint8), hidden_in=h)
        assert np.array_equal(om, ot), step
        assert np.array_equal(masked.last_f64, trimmed.last_f64), step
        new_keep = (rng.random(n) >= 0.4).astype(np.uint8)
        valid += new_keep.tolist()
        trimmed.trim(0, np.concatenate([np.ones(trimmed.length(0) - n, np.uint8), new_keep]))
        pos += n
    assert masked.length(0) == len(valid) and trimmed.length(0) == sum(valid)
    assert sum(valid) < len(valid)
