"""GPU tests of prefix capture and warm resume (kv_state_export /
kv_state_import; Section 8.4): the export is pure data movement, so it must
be bit-exact -- the kept entries of the row, in cache order, through the
beam table -- and a state resumed from a compacted export must continue
exactly like the original state with its rejected entries masked (up to
the split of attention into chunks, which moves with the cache length)."""
import numpy as np
import pytest

import paper_2608_19147_gb300 as pkg
import synth
from gpu_engine import GpuEngine, GpuShard, assert_close
from paper_2608_19147_gb300.spec import MaskedRequest
from scenarios import prefill

pytestmark = pytest.mark.gpu
SHAPE = synth.TINY
SEED = 777


@pytest.fixture(scope="module")
def shard():
    sh = GpuShard(SHAPE, synth.make_weights(SHAPE, SEED))
    yield sh
    sh.close()


def _dims():
    return SHAPE.n_layers, SHAPE.n_kv_heads, SHAPE.head_dim


def _with_rejections(eng, req, steps, seed):
    """Verify steps of 1 + 4 tokens keeping 1 + a of them."""
    outs = []
    for t in range(steps):
        h = synth.hidden_in(SHAPE, seed, t, 5)
        pos, mask = req.inputs(5)
        outs.append(eng.step([5], pos, mask, hidden_in=h))
        req.commit(5, 1 + synth.accepted_drafts(seed, t))
    return outs


def test_export_is_the_kept_entries_bit_exact(shard):
    eng = GpuEngine(shard, 1, 128)
    prefill(eng, SHAPE, SEED, 0, 40)
    req = MaskedRequest(40)
    _with_rejections(eng, req, 4, SEED)
    L = req.physical
    keep = np.array(req.valid, np.uint8)
    assert 0 < keep.sum() < L
    k, v = pkg.kv_state_export(eng.st, 0, L, *_dims(), keep=keep)
    assert k.shape == (SHAPE.n_layers, int(keep.sum()), SHAPE.n_kv_heads, SHAPE.head_dim)
    idx = np.nonzero(keep)[0]
    for layer in range(SHAPE.n_layers):
        kr, vr = eng.read(0, layer, 0, L)
        assert np.array_equal(k[layer], kr[idx]) and np.array_equal(v[layer], vr[idx])
    ka, va = pkg.kv_state_export(eng.st, 0, L, *_dims())   # keep = NULL: every entry
    assert ka.shape[1] == L and np.array_equal(ka[:, idx], k) and np.array_equal(va[:, idx], v)
    eng.close()


def test_export_reads_through_the_beam_table(shard):
    eng = GpuEngine(shard, 2, 96)
    for r, n in ((0, 30), (1, 50)):
        prefill(eng, SHAPE, SEED + r, r, n)
    mask = np.zeros((2, 64), np.uint8)
    mask[0, :51] = 1   # row 0 continues row 1's 50 entries
    mask[1, :31] = 1
    eng.step([1, 1], np.array([50, 30], np.int32), mask, hidden_in=synth.hidden_in(SHAPE, SEED, 9, 2),
             beam_idx=np.array([1, 0], np.int32))
    for row, n in ((0, 51), (1, 31)):
        k, v = pkg.kv_state_export(eng.st, row, n, *_dims())
        for layer in range(SHAPE.n_layers):
            kr, vr = eng.read(row, layer, 0, n)
            assert np.array_equal(k[layer], kr) and np.array_equal(v[layer], vr)
    eng.close()


def test_resumed_state_continues_like_the_masked_one(shard):
    a = GpuEngine(shard, 1, 160)
    prefill(a, SHAPE, SEED, 0, 48)
    ra = MaskedRequest(48)
    _with_rejections(a, ra, 5, SEED + 1)
    keep = np.array(ra.valid, np.uint8)
    k, v = pkg.kv_state_export(a.st, 0, ra.physical, *_dims(), keep=keep)
    b = GpuEngine(shard, 1, 160)
    pkg.kv_state_import(b.st, 0, k, v)
    assert pkg.kv_state_length(b.st, 0) == ra.position    # compacted: the logical length
    rb = MaskedRequest(ra.position)
    for t in range(3):
        h = synth.hidden_in(SHAPE, SEED + 2, t, 5)
        pa, ma = ra.inputs(5)
        pb, mb = rb.inputs(5)
        assert np.array_equal(pa, pb)                       # same logical positions
        oa = a.step([5], pa, ma, hidden_in=h)
        ob = b.step([5], pb, mb, hidden_in=h)
        assert_close(ob, oa, what="resumed vs masked, step %d" % t)
        n_keep = 1 + synth.accepted_drafts(SEED + 2, t)
        ra.commit(5, n_keep)
        rb.commit(5, n_keep)
    a.close()
    b.close()


def test_export_import_errors(shard):
    eng = GpuEngine(shard, 1, 64)
    prefill(eng, SHAPE, SEED, 0, 20)
    with pytest.raises(pkg.ShardError) as e:
        pkg.kv_state_export(eng.st, 0, 19, *_dims())       # len must be the row's length
    assert e.value.code == pkg.SHARD_EINVAL
    big = np.zeros((SHAPE.n_layers, 65, SHAPE.n_kv_heads, SHAPE.head_dim), np.uint16)
    with pytest.raises(pkg.ShardError) as e:
        pkg.kv_state_import(eng.st, 0, big, big)
    assert e.value.code == pkg.SHARD_ECAPACITY
    eng.close()
