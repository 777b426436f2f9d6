"""GPU parity of the packed step (shard_step_packed; Section 8.6) against the
oracle's packed step, through the C ABI: the plan of tests/test_oracle_packed
(a shared prefix, four slot regions, two decode rows and a two-row causal
chunk) within the fixed tolerance; appended K/V; slot isolation bit for bit
on the GPU (other slots' inputs and regions change, the slot's own output
does not); an idle row changes nothing; a row that does not open its own
entry is rejected by the device guard."""
import numpy as np
import pytest
import torch

import oracle
import paper_2608_19147_gb300 as pkg
import synth
from gpu_engine import GpuShard, assert_close, to_dev
from test_oracle_packed import LP, P, ROWS, SEED, SHAPE, _plan, _window

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def shards():
    w = synth.make_weights(SHAPE, SEED)
    g = GpuShard(SHAPE, w)
    yield g, oracle.OracleShard(SHAPE, w)
    g.close()


def _gpu_packed(g, rows, hidden, noise_seed=SEED + 1, other_seed=SEED, mask_override=None):
    st = pkg.kv_state_alloc(g.h, 1, P + 16)
    for layer in range(SHAPE.n_layers):
        k, v = _window(layer, noise_seed, other_seed)
        pkg.kv_state_load(st, 0, layer, k, v)
    pos, mask = _plan(rows)
    if mask_override is not None:
        mask = mask_override(mask)
    S = len(rows)
    d_h, d_pos, d_mask = to_dev(hidden), to_dev(pos), to_dev(mask)
    out = torch.empty((S, SHAPE.hidden), dtype=torch.int16, device="cuda")
    s = torch.cuda.current_stream().cuda_stream
    pkg.shard_step_packed(g.h, st, d_h.data_ptr(), None, S, d_pos.data_ptr(), d_mask.data_ptr(), mask.shape[1],
                          out.data_ptr(), s)
    rc = pkg.shard_sync_status(g.h, s, check=False)
    return st, rc, out.cpu().numpy().view(np.uint16)


def test_packed_matches_the_oracle(shards):
    g, o = shards
    h = synth.hidden_in(SHAPE, SEED, 0, 4)
    st, rc, got = _gpu_packed(g, ROWS, h)
    assert rc == 0
    ost = o.state(1, P + 16)
    for layer in range(SHAPE.n_layers):
        k, v = _window(layer)
        assert ost.load(0, layer, k, v) == 0
    pos, mask = _plan(ROWS)
    orc, want, _ = ost.step_packed(pos, mask, hidden_in=h)
    assert orc == 0
    assert_close(got, want, what="packed step")
    for layer in range(SHAPE.n_layers):
        kg, vg = pkg.kv_state_read(st, 0, layer, P, 4, SHAPE.n_kv_heads, SHAPE.head_dim)
        ko, vo = ost.read(0, layer, P, 4)
        assert np.abs(kg.view(np.float16).astype(float) - ko.view(np.float16).astype(float)).max() < 2e-2
    pkg.kv_state_free(st)


def test_packed_slots_isolated_on_the_gpu(shards):
    g, _ = shards
    h = synth.hidden_in(SHAPE, SEED, 0, 4)
    st, _, base = _gpu_packed(g, ROWS, h)
    pkg.kv_state_free(st)
    h2 = h.copy()
    h2[1:] = synth.hidden_in(SHAPE, SEED, 9, 3)
    st, _, other = _gpu_packed(g, ROWS, h2, noise_seed=SEED + 5, other_seed=SEED + 6)
    pkg.kv_state_free(st)
    assert np.array_equal(other[0], base[0])
    assert not np.array_equal(other[1], base[1])


def test_packed_idle_row_and_own_entry_rule(shards):
    g, _ = shards
    h = synth.hidden_in(SHAPE, SEED, 0, 5)
    st, _, base = _gpu_packed(g, ROWS, h[:4])
    pkg.kv_state_free(st)
    st, _, idle = _gpu_packed(g, ROWS + [-1], h)
    pkg.kv_state_free(st)
    assert_close(idle[:4], base, what="idle row added")   # the cache length, hence the chunking, moved

    def drop_own(mask):
        mask[1, P + 1] = 0
        return mask

    st, rc, _ = _gpu_packed(g, ROWS, h[:4], mask_override=drop_own)
    assert rc == pkg.SHARD_EINVAL
    pkg.kv_state_free(st)
