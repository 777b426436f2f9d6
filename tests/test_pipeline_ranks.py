"""The multi-stage pipeline (paper_2608_19147_gb300.pipeline; Sections 3.3,
6.2 and 7) on CPU ranks: two gloo processes, each driving one stage of the
tiny shard (one layer each), the fp16 hidden state handed from rank to rank
with point-to-point messages, two request streams interleaved, greedy
decoding closing the loop (the next token comes from the last stage's
output).  The stages here are the fp64 oracle -- what crosses ranks, and in
which order, is the subject, not the stage arithmetic.  No GPU.

* The pipelined, interleaved run gives every stream exactly the outputs of
  running that stream alone through both stages in one process.
* A rank that leaves between steps (its process exits) is detected by the
  coordinator at its next receive: with "abort" it returns the completed
  prefix and where it stopped; with "restore" it rebuilds the lost stage
  locally by replaying the inputs it logged for it, and the finished run
  equals the run without a failure.
"""
import dataclasses
import datetime
import os
import socket

import numpy as np
import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

import oracle
import synth
from paper_2608_19147_gb300 import pipeline as pl
from scenarios import OracleEngine

SHAPE = synth.TINY
SEED = 777
STREAMS = (0, 1)
N_STEPS = 6
PREFILL = {0: 24, 1: 40}
CAP = 96


def _stages():
    w = synth.make_weights(SHAPE, SEED)
    s0 = dataclasses.replace(SHAPE, name="tiny-stage0", n_layers=1)
    s1 = dataclasses.replace(SHAPE, name="tiny-stage1", n_layers=1, vocab=0)
    return w, [(s0, synth.ShardWeights(s0, SEED, [w.layers[0]], w.embedding), 0),
               (s1, synth.ShardWeights(s1, SEED, [w.layers[1]], None), 1)]


class OracleStage:
    """One stage on the oracle, one KV state per stream, prefilled with the
    stream's seeded cache for the stage's layer of the whole shard."""

    def __init__(self, shape, weights, layer):
        self.eng = {}
        for s in STREAMS:
            e = OracleEngine(shape, weights, 1, CAP)
            k, v = synth.kv_prefill(SHAPE, SEED + s, 0, PREFILL[s], layer)
            e.load(0, 0, k, v)
            self.eng[s] = e

    def __call__(self, s, x, kind, n_new, pos, mask):
        kw = {"token_ids": x} if kind == pl.KIND_TOKENS else {"hidden_in": x}
        return self.eng[s].step([n_new], pos, mask, **kw)


def _inputs(embedding):
    """Greedy decoding: the next token is the test head's argmax of the last
    stage's output (tied embedding after an RMSNorm)."""
    def next_input(s, step, last):
        if step >= N_STEPS:
            return None
        if last is None:
            tok = int(synth.token_ids(SHAPE, SEED, 100 + s, 1)[0])
        else:
            lg = oracle.logits(last.view(np.float16).astype(np.float64), embedding, SHAPE.rms_eps)
            tok = int(lg.argmax(axis=1)[0])
        P = PREFILL[s] + step
        return np.array([tok], np.int32), pl.KIND_TOKENS, np.array([P], np.int32), np.ones(P + 1, np.uint8)
    return next_input


def _reference():
    """Each stream alone, both stages in one process."""
    w, st = _stages()
    stages = [OracleStage(sh, ww, layer) for sh, ww, layer in st]
    nxt = _inputs(w.embedding)
    outs = {}
    for s in STREAMS:
        outs[s], last, step = [], None, 0
        while True:
            inp = nxt(s, step, last)
            if inp is None:
                break
            x, kind, pos, mask = inp
            for stg in stages:
                x = stg(s, x, kind, len(pos), pos, mask)
                kind = pl.KIND_HIDDEN
            outs[s].append(x)
            last, step = x, step + 1
    return outs


def _free_port():
    with socket.socket() as so:
        so.bind(("127.0.0.1", 0))
        return so.getsockname()[1]


def _rank(rank, world, port, out_dir, mode, leave_after):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world, timeout=datetime.timedelta(seconds=30))
    w, st = _stages()
    sh, ww, layer = st[rank]
    stage = OracleStage(sh, ww, layer)
    if rank == 0:
        lost = (lambda: [OracleStage(st[1][0], st[1][1], st[1][2])]) if mode == "restore" else None
        res = pl.coordinate(stage, _inputs(w.embedding), STREAMS, SHAPE.hidden, on_failure=mode,
                            make_lost_stages=lost)
        np.savez(os.path.join(out_dir, "out.npz"), status=res.status,
                 failed=np.array(res.failed_at if res.failed_at else (-1, -1)),
                 **{"s%d_%d" % (s, i): o for s in STREAMS for i, o in enumerate(res.outputs[s])})
        if res.status == "ok":
            dist.destroy_process_group()
        return
    if leave_after is None:
        pl.run_stage_rank(stage, SHAPE.hidden)
        dist.destroy_process_group()
        return
    # leave between steps: serve `leave_after` steps, then exit at once
    served = [0]

    def counting(*a):
        out = stage(*a)
        served[0] += 1
        return out

    sends = pl._Sends()
    while served[0] < leave_after:
        msg = pl._recv(0, SHAPE.hidden)
        out = counting(msg.stream, msg.x, msg.kind, msg.n_new, msg.positions, msg.mask)
        pl._send(pl._Msg(msg.stream, msg.step, pl.KIND_HIDDEN, msg.n_new, msg.positions, msg.mask, out), 0, sends)
    sends.finish()
    os._exit(0)


def _run(tmp_path, mode, leave_after):
    mp.spawn(_rank, args=(2, _free_port(), str(tmp_path), mode, leave_after), nprocs=2, join=True)
    z = np.load(tmp_path / "out.npz")
    outs = {s: [] for s in STREAMS}
    for s in STREAMS:
        i = 0
        while "s%d_%d" % (s, i) in z:
            outs[s].append(z["s%d_%d" % (s, i)])
            i += 1
    return str(z["status"]), tuple(int(v) for v in z["failed"]), outs


@pytest.fixture(scope="module")
def reference():
    return _reference()


def test_interleaved_pipeline_equals_each_stream_alone(tmp_path, reference):
    status, _, outs = _run(tmp_path, "abort", None)
    assert status == "ok"
    for s in STREAMS:
        assert len(outs[s]) == N_STEPS
        for a, b in zip(outs[s], reference[s]):
            assert np.array_equal(a, b)
    # the streams really are different requests
    assert not np.array_equal(outs[0][0], outs[1][0])


def test_a_rank_that_leaves_is_detected_and_the_run_aborts(tmp_path, reference):
    status, failed, outs = _run(tmp_path, "abort", 5)
    assert status == "aborted" and failed != (-1, -1)
    done = sum(len(outs[s]) for s in STREAMS)
    assert done == 5
    for s in STREAMS:
        for a, b in zip(outs[s], reference[s]):
            assert np.array_equal(a, b)


def test_a_rank_that_leaves_is_restored_by_replay(tmp_path, reference):
    status, failed, outs = _run(tmp_path, "restore", 5)
    assert status == "restored" and failed != (-1, -1)
    for s in STREAMS:
        assert len(outs[s]) == N_STEPS
        for a, b in zip(outs[s], reference[s]):
            assert np.array_equal(a, b)
