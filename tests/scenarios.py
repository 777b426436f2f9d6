"""Workload drivers shared by the oracle tests and the GPU parity tests.

An *engine* is any object with
    step(n_new, position_ids, mask, hidden_in=None, token_ids=None, beam_idx=None) -> fp16 bits [M][H]
    load(row, layer, k16, v16), read(row, layer, start, n) -> (k16, v16), trim(row, keep)
    length(row)
(OracleEngine below; the GPU engine lives in the GPU tests).  Masks are
built the way the paper's coordinator builds them (Section 5.2): a tracked
valid-mask prefix followed by ones for the new tokens.
"""
from __future__ import annotations

from typing import List, Optional

import numpy as np

import oracle
import synth


class OracleEngine:
    def __init__(self, shape, weights, n_rows: int, capacity: int, round_points: bool = True):
        self.shape = shape
        self.shard = oracle.OracleShard(shape, weights)
        self.state = self.shard.state(n_rows, capacity)
        self.round_points = round_points
        self.last_f64 = None

    def step(self, n_new, position_ids, mask, hidden_in=None, token_ids=None, beam_idx=None):
        rc, out16, out64 = self.state.step(n_new, position_ids, mask, hidden_in=hidden_in, token_ids=token_ids,
                                           beam_idx=beam_idx, round_points=self.round_points, want_f64=True)
        if rc != 0:
            raise RuntimeError("oracle step failed: %d" % rc)
        self.last_f64 = out64
        return out16

    def load(self, row, layer, k16, v16):
        rc = self.state.load(row, layer, k16, v16)
        assert rc == 0, rc

    def read(self, row, layer, start, n):
        return self.state.read(row, layer, start, n)

    def trim(self, row, keep):
        rc = self.state.trim(row, keep)
        assert rc == 0, rc

    def length(self, row):
        return self.state.length(row)


def prefill(engine, shape, seed: int, row: int, length: int, src_row=None):
    """Loads the seeded prefill of stream row `src_row` (default: `row`) into `row`."""
    for layer in range(shape.n_layers):
        k, v = synth.kv_prefill(shape, seed, row if src_row is None else src_row, length, layer)
        engine.load(row, layer, k, v)


def f16(a: np.ndarray) -> np.ndarray:
    return a.view(np.float16).astype(np.float64)


class MaskedRequest:
    """Coordinator-side bookkeeping of one request under mask-based rewind:
    `valid` tracks which cache entries are live, `pos` the logical length."""

    def __init__(self, cache_len: int):
        self.valid: List[int] = [1] * cache_len
        self.pos = cache_len

    def mask_for(self, n: int, stride: Optional[int] = None) -> np.ndarray:
        m = np.array(self.valid + [1] * n, dtype=np.uint8)
        if stride is not None:
            m = np.concatenate([m, np.zeros(stride - m.size, np.uint8)])
        return m

    def positions(self, n: int) -> np.ndarray:
        return np.arange(self.pos, self.pos + n, dtype=np.int32)

    def commit(self, n_fed: int, n_kept: int):
        """n_fed entries were appended; the first n_kept of them stay live."""
        self.valid += [1] * n_kept + [0] * (n_fed - n_kept)
        self.pos += n_kept


def tiny_steps_masked_vs_trim(make_engine, shape, weights, seed: int = 1234, capacity: int = 96):
    """The tiny workload: 72-token prefill; step A decodes 1 token; step B
    verifies 1+4 tokens, rejects the last 2 through the mask and decodes one
    more.  The same sequence is run with a physical trim instead of the mask.
    Returns dict of outputs for both runs."""
    out = {}
    for mode in ("mask", "trim"):
        eng = make_engine(capacity)
        prefill(eng, shape, seed, 0, 72)
        req = MaskedRequest(72)
        # step A: one token
        h = synth.hidden_in(shape, seed, 0, 1)
        out[(mode, "A")] = eng.step([1], req.positions(1), req.mask_for(1), hidden_in=h)
        req.commit(1, 1)
        # step B: verify 1 + 4, keep 3 of the 5 new entries
        h = synth.hidden_in(shape, seed, 1, 5)
        out[(mode, "B")] = eng.step([5], req.positions(5), req.mask_for(5), hidden_in=h)
        if mode == "mask":
            req.commit(5, 3)
        else:
            keep = np.array([1] * (eng.length(0) - 2) + [0, 0], dtype=np.uint8)
            eng.trim(0, keep)
            req = MaskedRequest(eng.length(0))
            req.pos = 72 + 1 + 3
        # step C: one more token
        h = synth.hidden_in(shape, seed, 2, 1)
        out[(mode, "C")] = eng.step([1], req.positions(1), req.mask_for(1), hidden_in=h)
        req.commit(1, 1)
        out[(mode, "engine")] = eng
        out[(mode, "req")] = req
    return out


def greedy_token(engine_out16: np.ndarray, embedding: np.ndarray, eps: float):
    """Test head (tied embedding after RMSNorm) on fp16 hidden states, fp64
    on the host.  Returns (argmax tokens, top-2 margins)."""
    lg = oracle.logits(f16(engine_out16), embedding, eps)
    top2 = np.sort(lg, axis=1)[:, -2:]
    return lg.argmax(axis=1), top2[:, 1] - top2[:, 0]


def greedy_decode(engine, shape, weights, seed: int, n_tokens: int, prefill_len: int = 72):
    """Target-only greedy decode with token ids (one token per step)."""
    prefill(engine, shape, seed, 0, prefill_len)
    req = MaskedRequest(prefill_len)
    tok = int(synth.token_ids(shape, seed, 0, 1)[0])
    toks, margins = [], []
    for _ in range(n_tokens):
        o = engine.step([1], req.positions(1), req.mask_for(1), token_ids=np.array([tok], np.int32))
        req.commit(1, 1)
        t, mg = greedy_token(o, weights.embedding, shape.rms_eps)
        tok = int(t[0])
        toks.append(tok)
        margins.append(float(mg[0]))
    return toks, margins


def spec_decode(engine, shape, weights, seed: int, n_tokens: int, target_tokens: List[int], k: int = 4,
                p_accept: float = 0.6, prefill_len: int = 72):
    """Greedy speculative decoding with mask-based rewind (Section 5).  The
    draft proposes the target's own greedy token with probability p_accept,
    else a seeded wrong token.  Verify feeds [current, d1..dk] in one step;
    the longest prefix of drafts equal to the target's argmax is accepted,
    rejected entries are masked out on all later steps, and the target's
    token after the accepted prefix becomes the next current token."""
    prefill(engine, shape, seed, 0, prefill_len)
    req = MaskedRequest(prefill_len)
    cur = int(synth.token_ids(shape, seed, 0, 1)[0])
    emitted: List[int] = []
    margins: List[float] = []
    step = 0
    while len(emitted) < n_tokens:
        u = synth.uniform(k, seed=seed, stream=1000 + step, tag=synth.TAG_ACCEPT)
        wrong = synth.draft_tokens(seed, step, k, shape.vocab)
        drafts = []
        for j in range(k):
            idx = len(emitted) + j
            good = target_tokens[idx] if idx < len(target_tokens) else int(wrong[j])
            d = good if u[j] < p_accept else int(wrong[j])
            if d == good and u[j] >= p_accept:
                d = (d + 1) % shape.vocab
            drafts.append(d)
        feed = np.array([cur] + drafts, dtype=np.int32)
        o = engine.step([k + 1], req.positions(k + 1), req.mask_for(k + 1), token_ids=feed)
        g, mg = greedy_token(o, weights.embedding, shape.rms_eps)
        a = 0
        while a < k and drafts[a] == int(g[a]):
            a += 1
        new = drafts[:a] + [int(g[a])]
        emitted += new
        margins += [float(x) for x in mg[: a + 1]]
        req.commit(k + 1, a + 1)
        cur = int(g[a])
        step += 1
    return emitted[:n_tokens], margins[:n_tokens], req
