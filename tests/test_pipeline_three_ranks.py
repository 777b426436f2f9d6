"""A three-stage pipeline on CPU ranks (Section 3.3's relay through a middle
stage; Section 7's three-node, three-stream runs): three gloo processes,
one layer of a 3-layer tiny shard each, three request streams interleaved,
greedy decoding closing the loop.  The stages are the fp64 oracle.  No GPU.

* Rank 1 receives from rank 0 and forwards to rank 2, which returns to rank
  0: the interleaved run gives every stream exactly the outputs of running
  it alone through the three stages in one process.
* The middle rank leaves between steps.  Its downstream peer loses its
  input, delivers what it had computed and stops; the coordinator detects
  the loss at its next receive.  With "abort" it returns a correct prefix of
  every stream and where it stopped; with "restore" it rebuilds stages 1 and
  2 locally by replaying the inputs it logged, and the finished run equals
  the run without a failure.
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

SHAPE = dataclasses.replace(synth.TINY, name="tiny-3L", n_layers=3)
SEED = 778
STREAMS = (0, 1, 2)
N_STEPS = 5
PREFILL = {0: 20, 1: 33, 2: 47}
CAP = 96
WORLD = 3


def _stages():
    w = synth.make_weights(SHAPE, SEED)
    out = []
    for layer in range(WORLD):
        s = dataclasses.replace(SHAPE, name="tiny-3L-stage%d" % layer, n_layers=1,
                                vocab=SHAPE.vocab if layer == 0 else 0)
        out.append((s, synth.ShardWeights(s, SEED, [w.layers[layer]], w.embedding if layer == 0 else None), layer))
    return w, out


class OracleStage:
    """One stage on the oracle: one KV state per stream, prefilled with the
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
    def next_input(s, step, last):
        if step >= N_STEPS:
            return None
        if last is None:
            tok = int(synth.token_ids(SHAPE, SEED, 200 + s, 1)[0])
        else:
            lg = oracle.logits(last.view(np.float16).astype(np.float64), embedding, SHAPE.rms_eps)
            tok = int(lg.argmax(axis=1)[0])
        P = PREFILL[s] + step
        return np.array([tok], np.int32), pl.KIND_TOKENS, np.array([P], np.int32), np.ones(P + 1, np.uint8)
    return next_input


def _reference():
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


def _rank(rank, port, out_dir, mode, leave_after):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=WORLD, timeout=datetime.timedelta(seconds=30))
    w, st = _stages()
    stage = OracleStage(*st[rank])
    if rank == 0:
        lost = (lambda: [OracleStage(*st[1]), OracleStage(*st[2])]) if mode == "restore" else None
        res = pl.coordinate(stage, _inputs(w.embedding), STREAMS, SHAPE.hidden, on_failure=mode,
                            make_lost_stages=lost)
        np.savez(os.path.join(out_dir, "out.npz"), status=res.status,
                 failed=np.array(res.failed_at if res.failed_at else (-1, -1)),
                 **{"s%d_%d" % (s, i): o for s in STREAMS for i, o in enumerate(res.outputs[s])})
        if res.status == "ok":
            dist.destroy_process_group()
        return
    if rank == 1 and leave_after is not None:
        # the middle stage serves `leave_after` steps, then its process exits
        sends = pl._Sends()
        for _ in range(leave_after):
            msg = pl._recv(0, SHAPE.hidden)
            out = stage(msg.stream, msg.x, msg.kind, msg.n_new, msg.positions, msg.mask)
            pl._send(pl._Msg(msg.stream, msg.step, pl.KIND_HIDDEN, msg.n_new, msg.positions, msg.mask, out), 2,
                     sends)
        sends.finish()
        os._exit(0)
    try:
        pl.run_stage_rank(stage, SHAPE.hidden)
    except pl.PeerLost:
        os._exit(0)  # lost its upstream peer: the coordinator handles the run
    dist.destroy_process_group()


def _run(tmp_path, mode, leave_after):
    mp.spawn(_rank, args=(_free_port(), str(tmp_path), mode, leave_after), nprocs=WORLD, join=True)
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


def test_three_stage_interleaved_pipeline_equals_each_stream_alone(tmp_path, reference):
    status, _, outs = _run(tmp_path, "abort", None)
    assert status == "ok"
    for s in STREAMS:
        assert len(outs[s]) == N_STEPS
        for a, b in zip(outs[s], reference[s]):
            assert np.array_equal(a, b)
    assert not np.array_equal(outs[0][0], outs[1][0]) and not np.array_equal(outs[1][0], outs[2][0])


def test_middle_rank_that_leaves_is_detected_and_the_run_aborts(tmp_path, reference):
    status, failed, outs = _run(tmp_path, "abort", 7)
    assert status == "aborted" and failed != (-1, -1)
    done = sum(len(outs[s]) for s in STREAMS)
    assert 1 <= done <= 7
    for s in STREAMS:
        for a, b in zip(outs[s], reference[s]):
            assert np.array_equal(a, b)


def test_middle_rank_that_leaves_is_restored_by_replay(tmp_path, reference):
    status, failed, outs = _run(tmp_path, "restore", 7)
    assert status == "restored" and failed != (-1, -1)
    for s in STREAMS:
        assert len(outs[s]) == N_STEPS
        for a, b in zip(outs[s], reference[s]):
            assert np.array_equal(a, b)
