"""Pins of the oracle's packed step (Section 8.6: continuous batching through
the mask layout).  S query rows share one cache row partitioned into a
shared prefix and one region per slot; each row carries its own mask.  The
pins reduce it to the (separately pinned) per-request step: a plan with two
decode rows and a two-row causal chunk must give, bit for bit, what three
separate requests give on caches holding the prefix and their own region,
and the K/V it appends must be theirs.  Isolation has teeth: other slots'
inputs and regions do not move a slot's output, its own input does.  An
idle row that opens only its own entry changes nothing for the others.
No GPU."""
import numpy as np
import pytest

import oracle
import synth

SHAPE = synth.TINY
SEED = 2468
LP = 8                      # shared prefix entries
REGION = 24                 # entries per slot region
FILL = [10, 15, 7, 0]       # used entries per slot (slot 3 free)
ROWS = [0, 1, 2, 2]         # slot of each query row: two decodes, a 2-row chunk on slot 2


@pytest.fixture(scope="module")
def shard():
    return oracle.OracleShard(SHAPE, synth.make_weights(SHAPE, SEED))


def _kv(row, n, layer, seed=SEED):
    if n == 0:
        z = np.zeros((0, SHAPE.n_kv_heads, SHAPE.head_dim), np.uint16)
        return z, z
    return synth.kv_prefill(SHAPE, seed, row, n, layer)


def _window(layer, noise_seed=SEED + 1, other_seed=SEED):
    """[prefix | region 0 | region 1 | region 2 | region 3] K and V; the
    unused tail of each region holds unrelated entries (masked out)."""
    ks, vs = [], []
    k, v = _kv(100, LP, layer)
    ks.append(k)
    vs.append(v)
    for s in range(4):
        k, v = _kv(s, FILL[s], layer, SEED if s == 0 else other_seed)
        nk, nv = _kv(200 + s, REGION - FILL[s], layer, noise_seed)
        ks += [k, nk]
        vs += [v, nv]
    return np.concatenate(ks), np.concatenate(vs)


P = LP + 4 * REGION


def _start(s):
    return LP + s * REGION


def _plan(rows):
    S = len(rows)
    mask = np.zeros((S, P + S), np.uint8)
    pos = np.zeros(S, np.int32)
    for t, s in enumerate(rows):
        if s < 0:                      # idle row: its own new entry only
            mask[t, P + t] = 1
            continue
        mask[t, :LP] = 1
        mask[t, _start(s):_start(s) + FILL[s]] = 1
        before = [u for u in range(t + 1) if rows[u] == s]
        for u in before:
            mask[t, P + u] = 1
        pos[t] = LP + FILL[s] + len(before) - 1
    return pos, mask


def _packed(shard, rows, hidden, noise_seed=SEED + 1, other_seed=SEED):
    st = shard.state(1, P + 16)
    for layer in range(SHAPE.n_layers):
        k, v = _window(layer, noise_seed, other_seed)
        assert st.load(0, layer, k, v) == 0
    pos, mask = _plan(rows)
    rc, out16, out64 = st.step_packed(pos, mask, hidden_in=hidden, want_f64=True)
    assert rc == 0
    return st, out64


def _separate(shard, slot, hidden_rows):
    st = shard.state(1, 64)
    for layer in range(SHAPE.n_layers):
        pk, pv = _kv(100, LP, layer)
        k, v = _kv(slot, FILL[slot], layer)
        assert st.load(0, layer, np.concatenate([pk, k]), np.concatenate([pv, v])) == 0
    n = hidden_rows.shape[0]
    L = LP + FILL[slot]
    pos = np.arange(L, L + n, dtype=np.int32)
    rc, out16, out64 = st.step([n], pos, np.ones(L + n, np.uint8), hidden_in=hidden_rows, want_f64=True)
    assert rc == 0
    return st, out64


def test_packed_plan_equals_separate_requests_bit_for_bit(shard):
    h = synth.hidden_in(SHAPE, SEED, 0, 4)
    st, got = _packed(shard, ROWS, h)
    for slot, idx in ((0, [0]), (1, [1]), (2, [2, 3])):
        ref_st, want = _separate(shard, slot, h[idx])
        assert np.array_equal(got[idx], want), slot
        # the appended K/V: token t of the plan sits at P + t
        L = LP + FILL[slot]
        for layer in range(SHAPE.n_layers):
            kg, vg = st.read(0, layer, P + idx[0], len(idx), f64=True)
            kw, vw = ref_st.read(0, layer, L, len(idx), f64=True)
            assert np.array_equal(kg, kw) and np.array_equal(vg, vw)


def test_slots_are_isolated_and_the_check_has_teeth(shard):
    h = synth.hidden_in(SHAPE, SEED, 0, 4)
    _, base = _packed(shard, ROWS, h)
    # other slots' inputs, their region contents and the unused entries change
    h2 = h.copy()
    h2[1:] = synth.hidden_in(SHAPE, SEED, 9, 3)
    _, other = _packed(shard, ROWS, h2, noise_seed=SEED + 5, other_seed=SEED + 6)
    assert np.array_equal(other[0], base[0])
    assert not np.array_equal(other[1], base[1])
    # the slot's own input moves its output
    h3 = h.copy()
    h3[0] = synth.hidden_in(SHAPE, SEED, 10, 1)[0]
    _, own = _packed(shard, ROWS, h3)
    assert np.abs(own[0] - base[0]).max() > 1e-3
    assert np.array_equal(own[1:], base[1:])


def test_idle_row_changes_nothing_for_the_others(shard):
    h = synth.hidden_in(SHAPE, SEED, 0, 5)
    _, base = _packed(shard, ROWS, h[:4])
    _, with_idle = _packed(shard, ROWS + [-1], h)
    assert np.array_equal(with_idle[:4], base)
    assert np.isfinite(with_idle[4]).all()


def test_a_row_must_open_its_own_entry(shard):
    st = shard.state(1, P + 16)
    for layer in range(SHAPE.n_layers):
        k, v = _window(layer)
        assert st.load(0, layer, k, v) == 0
    pos, mask = _plan(ROWS)
    mask[1, P + 1] = 0
    rc, _, _ = st.step_packed(pos, mask, hidden_in=synth.hidden_in(SHAPE, SEED, 0, 4))
    assert rc == -1
