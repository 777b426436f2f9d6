"""GPU parity of shard_prefill (Section 3.4: a prompt fills the stateful
cache by running through the stage) against the fp64 oracle, through the C
ABI.  The oracle's reference is its decode step with all S prompt tokens as
the new tokens of one request -- the method's definition; the GPU computes
it with the projections on the tensor cores (tcgen05), in chunks of 256
tokens.  Checked at the fixed bar (relative L2 1e-3, max-abs 2e-2 with one
fp16 ulp where that is larger):

* the tiny shard: a prompt after a short cache, a prompt of two chunks on an
  empty row, token-id and hidden-state inputs, a prompt with masked holes in
  the row's cache, and a second row of a two-row state;
* two layers of the Llama-3.1-8B stage: a 200-token prompt on a 72-entry
  cache;
* after the prefill, the appended K/V entries match the oracle's, and decode
  steps (shard_step) continue from the prefilled state like the oracle's.
"""
import dataclasses

import numpy as np
import pytest
import torch

import paper_2608_19147_gb300 as pkg
import synth
from gpu_engine import GpuEngine, GpuShard, to_dev
from scenarios import OracleEngine, f16, prefill
from test_gpu_layers import assert_fixed_bar, fp16_ulp

pytestmark = pytest.mark.gpu
SEED = 31337


def _gpu_prefill(g, row, S, pos, mask, hidden_in=None, token_ids=None):
    d_pos, d_mask = to_dev(np.asarray(pos, np.int32)), to_dev(np.asarray(mask, np.uint8))
    d_h = to_dev(hidden_in) if hidden_in is not None else None
    d_t = to_dev(np.asarray(token_ids, np.int32)) if token_ids is not None else None
    out = torch.empty((S, g.shape.hidden), dtype=torch.int16, device="cuda")
    s = torch.cuda.current_stream().cuda_stream
    pkg.shard_prefill(g.shard.h, g.st, row, d_h.data_ptr() if d_h is not None else None,
                      d_t.data_ptr() if d_t is not None else None, S, d_pos.data_ptr(), d_mask.data_ptr(), mask.size,
                      out.data_ptr(), s)
    pkg.shard_sync_status(g.shard.h, s)
    return out.cpu().numpy().view(np.uint16)


def _appended_close(g, o, shape, row, start, n, what):
    for layer in range(shape.n_layers):
        kg, vg = g.read(row, layer, start, n)
        ko, vo = o.read(row, layer, start, n)
        for a, b, nm in ((kg, ko, "K"), (vg, vo, "V")):
            a, b = f16(a), f16(b)
            assert (np.abs(a - b) <= np.maximum(2e-2, fp16_ulp(b))).all(), (what, layer, nm)


@pytest.fixture(scope="module")
def tiny():
    w = synth.make_weights(synth.TINY, SEED)
    sh = GpuShard(synth.TINY, w)
    yield w, sh
    sh.close()


@pytest.mark.parametrize("P,S,use_tokens", [(10, 37, True), (0, 300, False), (72, 16, False)])
def test_tiny_prefill_matches_oracle_and_decoding_continues(tiny, P, S, use_tokens):
    w, sh = tiny
    shape = synth.TINY
    cap = P + S + 8
    g, o = GpuEngine(sh, 1, cap), OracleEngine(shape, w, 1, cap)
    if P:
        for e in (g, o):
            prefill(e, shape, SEED, 0, P)
    pos = np.arange(P, P + S, dtype=np.int32)
    mask = np.ones(P + S, np.uint8)
    kw = {"token_ids": synth.token_ids(shape, SEED, 1, S)} if use_tokens else {"hidden_in": synth.hidden_in(shape, SEED, 1, S)}
    got = _gpu_prefill(g, 0, S, pos, mask, **kw)
    want = o.step([S], pos, mask, **kw)
    assert_fixed_bar(got, want, "tiny prefill P=%d S=%d" % (P, S))
    assert g.length(0) == o.length(0) == P + S
    _appended_close(g, o, shape, 0, P, S, "tiny prefill")
    # decoding continues from the prefilled state
    for step in range(2):
        L = P + S + step
        h = synth.hidden_in(shape, SEED, 50 + step, 1)
        args = ([1], np.array([L], np.int32), np.ones(L + 1, np.uint8))
        assert_fixed_bar(g.step(*args, hidden_in=h), o.step(*args, hidden_in=h), "decode after prefill %d" % step)
    g.close()


def test_tiny_prefill_with_masked_holes_and_second_row(tiny):
    w, sh = tiny
    shape = synth.TINY
    B, cap = 2, 160
    g, o = GpuEngine(sh, B, cap), OracleEngine(shape, w, B, cap)
    for e in (g, o):
        prefill(e, shape, SEED, 0, 30)
        prefill(e, shape, SEED + 1, 1, 50)
    S = 40
    mask = np.ones(50 + S, np.uint8)
    mask[[3, 17, 18, 41]] = 0    # rejected entries of earlier steps stay masked
    pos = np.arange(46, 46 + S, dtype=np.int32)
    h = synth.hidden_in(shape, SEED, 7, S)
    got = _gpu_prefill(g, 1, S, pos, mask, hidden_in=h)
    # the oracle's step for request 1 alone: row 0 takes no new token, so
    # run it on a one-row copy of row 1
    o1 = OracleEngine(shape, w, 1, cap)
    prefill(o1, shape, SEED + 1, 0, 50, src_row=1)
    want = o1.step([S], pos, mask, hidden_in=h)
    assert_fixed_bar(got, want, "tiny prefill row 1 with holes")
    assert g.length(1) == 50 + S and g.length(0) == 30
    for layer in range(shape.n_layers):
        kg, _ = g.read(1, layer, 50, S)
        ko, _ = o1.read(0, layer, 50, S)
        assert (np.abs(f16(kg) - f16(ko)) <= np.maximum(2e-2, fp16_ulp(f16(ko)))).all()
    g.close()


def test_8b_two_layers_prefill_matches_oracle():
    shape = dataclasses.replace(synth.LLAMA8B_STAGE, name="llama3.1-8b-2L", n_layers=2)
    w = synth.make_weights(shape, SEED)
    sh = GpuShard(shape, w)
    P, S = 72, 200
    cap = P + S + 8
    g, o = GpuEngine(sh, 1, cap), OracleEngine(shape, w, 1, cap)
    for e in (g, o):
        prefill(e, shape, SEED, 0, P)
    pos = np.arange(P, P + S, dtype=np.int32)
    mask = np.ones(P + S, np.uint8)
    tok = synth.token_ids(shape, SEED, 3, S)
    got = _gpu_prefill(g, 0, S, pos, mask, token_ids=tok)
    want = o.step([S], pos, mask, token_ids=tok)
    assert_fixed_bar(got, want, "8b 2-layer prefill")
    _appended_close(g, o, shape, 0, P, S, "8b prefill")
    g.close()
    sh.close()
