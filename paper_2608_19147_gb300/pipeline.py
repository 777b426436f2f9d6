"""A pipeline of shard stages across ranks, with interleaved request streams.

The paper splits a model by layer range into stages, one per machine, relays
the hidden state of each step from stage to stage (Section 3.3, "TCP
Activation Relay") and fills the pipeline's bubbles by interleaving the
decode steps of several independent requests, each with its own KV state
(Section 7, "Multi-User Throughput via Micro-Batching"; Section 6.2,
"Progressive Optimization").  This module is that orchestration over
torch.distributed point-to-point messages:

* rank r runs stage r; rank 0 also coordinates: it makes each stream's next
  input, runs stage 0 and sends the fp16 hidden state (with the step's
  positions and attention mask) to rank 1; every rank forwards to the next;
  the last rank sends its output back to rank 0;
* the coordinator keeps every stream in flight: it submits step 0 of all
  streams, then for each returned result computes that stream's next input
  and submits it, so while the last stage works on stream A, stage 0 works
  on stream B;
* a stage is any callable ``stage(stream, x, kind, n_new, positions, mask)
  -> fp16 hidden bits [M][H]`` -- on a GPU machine the C ABI's shard_step_host
  with one KV state per stream (GpuStage below), elsewhere anything with the
  same contract.

Failure handling is on the host: a peer that leaves between steps (its
process exits) makes the coordinator's next receive fail, and a peer that
stops answering makes it time out (the process group's timeout).  The
coordinator then either aborts -- returning what completed and where it
stopped -- or restores: it builds the lost stages locally (a factory the
caller gives), rebuilds their KV states by replaying the inputs it logged
for them, and finishes the run alone.  Stages are deterministic, so a
restored run gives the same outputs as one without a failure.

Messages: a header (int64 [8]: op, stream, step, kind, M, mask length, 0, 0),
then int32 positions [M], uint8 mask [mask length], and the payload (fp16
bits as int16 [M][H], or int32 token ids [M] for kind "tokens").
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import Callable, Dict, List, Optional, Sequence, Tuple

import numpy as np
import torch
import torch.distributed as dist

OP_FORWARD, OP_STOP = 1, 2
KIND_HIDDEN, KIND_TOKENS = 0, 1

# stage(stream, x, kind, n_new, positions, mask) -> fp16 bits [M][H]
StageFn = Callable[[int, np.ndarray, int, int, np.ndarray, np.ndarray], np.ndarray]
# next_input(stream, step, last_output or None) -> (x, kind, positions, mask), or None when the stream is done
InputFn = Callable[[int, int, Optional[np.ndarray]], Optional[Tuple[np.ndarray, int, np.ndarray, np.ndarray]]]


class PeerLost(RuntimeError):
    """A pipeline peer left or stopped answering."""


@dataclass
class PipelineResult:
    outputs: Dict[int, List[np.ndarray]]   # per stream, the last stage's output of every completed step
    status: str = "ok"                     # "ok", "restored" or "aborted"
    failed_at: Optional[Tuple[int, int]] = None  # (stream, step) whose result was lost
    detail: str = ""


@dataclass
class _Msg:
    stream: int
    step: int
    kind: int
    n_new: int
    positions: np.ndarray
    mask: np.ndarray
    x: np.ndarray


class _Sends:
    """Outstanding non-blocking sends.  A blocking send waits for the peer's
    matching receive, so two ranks sending to each other at once would wait
    for ever; sends are posted and finished later instead (the tensors stay
    referenced until then)."""

    def __init__(self):
        self.works = []

    def post(self, t: torch.Tensor, dst: int) -> None:
        self.works.append((dist.isend(t, dst), t))
        self.works = [(w, x) for w, x in self.works if not w.is_completed()]

    def finish(self) -> None:
        for w, _ in self.works:
            w.wait()
        self.works = []


def _send(msg: _Msg, dst: int, sends: _Sends) -> None:
    hdr = torch.tensor([OP_FORWARD, msg.stream, msg.step, msg.kind, msg.n_new, msg.mask.size, 0, 0], dtype=torch.int64)
    sends.post(hdr, dst)
    sends.post(torch.from_numpy(np.ascontiguousarray(msg.positions, dtype=np.int32)), dst)
    sends.post(torch.from_numpy(np.ascontiguousarray(msg.mask, dtype=np.uint8)), dst)
    if msg.kind == KIND_TOKENS:
        sends.post(torch.from_numpy(np.ascontiguousarray(msg.x, dtype=np.int32)), dst)
    else:
        sends.post(torch.from_numpy(np.ascontiguousarray(msg.x, dtype=np.uint16).view(np.int16)), dst)


def _send_stop(dst: int, sends: _Sends) -> None:
    sends.post(torch.tensor([OP_STOP, 0, 0, 0, 0, 0, 0, 0], dtype=torch.int64), dst)


def _recv(src: int, hidden: int) -> Optional[_Msg]:
    hdr = torch.empty(8, dtype=torch.int64)
    dist.recv(hdr, src)
    op, stream, step, kind, M, mlen = (int(v) for v in hdr[:6])
    if op == OP_STOP:
        return None
    pos = torch.empty(M, dtype=torch.int32)
    dist.recv(pos, src)
    mask = torch.empty(mlen, dtype=torch.uint8)
    dist.recv(mask, src)
    if kind == KIND_TOKENS:
        x = torch.empty(M, dtype=torch.int32)
        dist.recv(x, src)
        xs = x.numpy()
    else:
        x = torch.empty((M, hidden), dtype=torch.int16)
        dist.recv(x, src)
        xs = x.numpy().view(np.uint16)
    return _Msg(stream, step, kind, M, pos.numpy(), mask.numpy(), xs)


def _recv_from_peer(src: int, hidden: int) -> Optional[_Msg]:
    try:
        return _recv(src, hidden)
    except RuntimeError as e:  # gloo / NCCL: connection closed by the peer, or the timeout ran out
        raise PeerLost(str(e)) from e


def run_stage_rank(stage: StageFn, hidden: int) -> int:
    """Loop of a non-coordinating rank r > 0: receive from r - 1, run the
    stage, send to r + 1 (the last rank sends back to rank 0), until the
    coordinator's stop message comes through.  Returns the number of steps run.
    If the upstream peer is lost, the results already computed are still
    delivered downstream (as far as that peer is alive) before PeerLost
    propagates, so the coordinator keeps every step that completed."""
    rank, world = dist.get_rank(), dist.get_world_size()
    src, dst = rank - 1, (rank + 1) % world
    sends = _Sends()
    n = 0
    while True:
        try:
            msg = _recv_from_peer(src, hidden)
        except PeerLost:
            try:
                sends.finish()
            except RuntimeError:
                pass
            raise
        if msg is None:
            if dst != 0:
                _send_stop(dst, sends)
            sends.finish()
            return n
        out = stage(msg.stream, msg.x, msg.kind, msg.n_new, msg.positions, msg.mask)
        _send(_Msg(msg.stream, msg.step, KIND_HIDDEN, msg.n_new, msg.positions, msg.mask, out), dst, sends)
        n += 1


@dataclass
class _Flight:
    step: int
    msg_into_stage1: _Msg  # what stage 1 was sent (also in the replay log)


def coordinate(stage0: StageFn, next_input: InputFn, streams: Sequence[int], hidden: int,
               on_failure: str = "abort", make_lost_stages: Optional[Callable[[], List[StageFn]]] = None
               ) -> PipelineResult:
    """Rank 0: drives every stream through the pipeline, interleaved.

    on_failure: "abort" -- stop at the lost result and return what completed;
    "restore" -- build the stages of ranks 1.. locally with
    make_lost_stages(), rebuild their state by replaying the inputs logged for
    them (per stream, in order) and finish the run locally."""
    world = dist.get_world_size()
    last = world - 1
    res = PipelineResult(outputs={s: [] for s in streams})
    log: Dict[int, List[_Msg]] = {s: [] for s in streams}  # inputs sent into stage 1, per stream
    pending: List[Tuple[int, _Flight]] = []                # in submission order (results return in order)
    sends = _Sends()

    def submit(s: int, step: int, last_out: Optional[np.ndarray]) -> None:
        nxt = next_input(s, step, last_out)
        if nxt is None:
            return
        x, kind, pos, mask = nxt
        n_new = int(len(pos))
        h = stage0(s, x, kind, n_new, pos, mask)
        m = _Msg(s, step, KIND_HIDDEN, n_new, np.asarray(pos, np.int32), np.asarray(mask, np.uint8), h)
        log[s].append(m)
        _send(m, 1, sends)
        pending.append((s, _Flight(step, m)))

    where = (streams[0], 0)
    try:
        for s in streams:
            where = (s, 0)
            submit(s, 0, None)
        while pending:
            s, fl = pending.pop(0)
            where = (s, fl.step)
            msg = _recv_from_peer(last, hidden)
            assert msg is not None and msg.stream == s and msg.step == fl.step, "out-of-order result"
            res.outputs[s].append(msg.x)
            where = (s, fl.step + 1)
            submit(s, fl.step + 1, msg.x)
    except (PeerLost, RuntimeError) as e:  # a send to a peer that left fails too
        res.failed_at = where
        res.detail = "peer lost at stream %d step %d: %s" % (where[0], where[1], e)
        if on_failure != "restore" or make_lost_stages is None:
            res.status = "aborted"
            return res
        res.status = "restored"
        _restore_and_finish(stage0, next_input, streams, res, log, make_lost_stages())
        return res
    try:
        _send_stop(1, sends)
        sends.finish()
    except RuntimeError:
        pass
    return res


def _restore_and_finish(stage0: StageFn, next_input: InputFn, streams: Sequence[int], res: PipelineResult,
                        log: Dict[int, List[_Msg]], stages: List[StageFn]) -> None:
    """Rebuild the lost stages from the logged stage-1 inputs, then run every
    unfinished stream to the end locally (streams still interleaved)."""
    def rest(m: _Msg) -> np.ndarray:
        x, kind = m.x, m.kind
        for st in stages:
            x = st(m.stream, x, kind, m.n_new, m.positions, m.mask)
            kind = KIND_HIDDEN
        return x

    done = {s: len(res.outputs[s]) for s in streams}
    for s in streams:
        for i, m in enumerate(log[s]):
            out = rest(m)            # replays rebuild the lost stages' KV states
            if i >= done[s]:         # results that were in flight when the peer was lost
                res.outputs[s].append(out)
    active = list(streams)
    while active:
        for s in list(active):
            step = len(res.outputs[s])
            nxt = next_input(s, step, res.outputs[s][-1] if res.outputs[s] else None)
            if nxt is None:
                active.remove(s)
                continue
            x, kind, pos, mask = nxt
            h = stage0(s, x, kind, int(len(pos)), pos, mask)
            res.outputs[s].append(rest(_Msg(s, step, KIND_HIDDEN, int(len(pos)), np.asarray(pos, np.int32),
                                            np.asarray(mask, np.uint8), h)))


class GpuStage:
    """A stage on this process's GPU through the C ABI: one shard, one KV
    state (one row) per stream, shard_step_host per call.  `prefill` loads a
    stream's cache before the run (k, v per layer: fp16 bits [len][Hkv][d])."""

    def __init__(self, shard: int, hidden: int, streams: Sequence[int], capacity: int, stream: int = 0):
        from . import kv_state_alloc
        self.shard, self.hidden, self.cuda_stream = shard, hidden, stream
        self.states = {s: kv_state_alloc(shard, 1, capacity) for s in streams}

    def prefill(self, s: int, layer: int, k: np.ndarray, v: np.ndarray) -> None:
        from . import kv_state_load
        kv_state_load(self.states[s], 0, layer, k, v)

    def __call__(self, s: int, x: np.ndarray, kind: int, n_new: int, positions: np.ndarray,
                 mask: np.ndarray) -> np.ndarray:
        from . import shard_step_host
        hid = x if kind == KIND_HIDDEN else None
        tok = x if kind == KIND_TOKENS else None
        out = np.empty((n_new, self.hidden), np.uint16)
        shard_step_host(self.shard, self.states[s], hid, tok, [n_new], positions, mask.reshape(1, -1), None, out,
                        self.cuda_stream)
        return out

    def close(self) -> None:
        from . import kv_state_free
        for st in self.states.values():
            kv_state_free(st)
        self.states = {}
