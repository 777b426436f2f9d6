"""Greedy speculative decoding over pipeline shards with mask-based KV rewind
(Section 5.2) and the final stage's top-1 head (Section 6.7).

Host orchestration only, as the paper's coordinator does it: every forward
runs in the library's kernels through the C ABI -- one `shard_step_host` per
pipeline stage (the hidden states are handed from stage to stage, Section
3.3) and `head_top1_host` on the last stage's output -- while the host keeps
the per-request rewind state (a valid bit per physical cache entry and the
logical position, Section 5.2) and makes the greedy acceptance decision, a
token-id comparison (Section 5.2, greedy decoding only).

A verify step feeds [current token, d_1 .. d_k]: the target's greedy token
after input i is targets[i]; the longest prefix of drafts with
d_{i+1} == targets[i] is accepted (a tokens), the emitted tokens are
d_1 .. d_a followed by the correction targets[a], the rejected entries
d_{a+1} .. d_k stay in the cache but are masked out on every later forward,
and the logical position advances by 1 + a.  The emitted sequence equals
plain greedy decoding's (Section 5.3, 5.4).
"""
from __future__ import annotations

from typing import Callable, List, Optional, Sequence, Tuple

import numpy as np

from . import (SHARD_MAX_TOKENS, head_top1_host, kv_state_alloc, kv_state_free, shard_step_host)

# forward(token_ids [n] int32, position_ids [n] int32, mask [L + n] uint8) -> greedy tokens [n] int32
Forward = Callable[[np.ndarray, np.ndarray, np.ndarray], np.ndarray]


def greedy_accept(drafts: Sequence[int], targets: Sequence[int]) -> Tuple[int, List[int]]:
    """Greedy acceptance of one verify block.  targets has one more entry
    than drafts (targets[i] is the target's token after input i of
    [current, d_1 .. d_k]).  Returns (a, emitted): a = the number of leading
    drafts the target agrees with, emitted = drafts[:a] + [targets[a]]."""
    k = len(drafts)
    if len(targets) != k + 1:
        raise ValueError("need len(targets) == len(drafts) + 1, got %d and %d" % (len(targets), k))
    a = 0
    while a < k and int(drafts[a]) == int(targets[a]):
        a += 1
    return a, [int(d) for d in drafts[:a]] + [int(targets[a])]


class MaskedRequest:
    """Rewind state of one request row (Section 5.2): cache entries are
    appended in order and never removed; `valid[j]` says whether entry j
    still takes part in attention, `position` is the logical length (the
    next position id, which RoPE uses)."""

    def __init__(self, cached: int = 0):
        self.valid: List[int] = [1] * cached
        self.position = cached

    @property
    def physical(self) -> int:
        return len(self.valid)

    def inputs(self, n: int) -> Tuple[np.ndarray, np.ndarray]:
        """position_ids and attention mask for n new entries (all visible)."""
        pos = np.arange(self.position, self.position + n, dtype=np.int32)
        mask = np.array(self.valid + [1] * n, dtype=np.uint8)
        return pos, mask

    def commit(self, n_fed: int, n_kept: int) -> None:
        """n_fed entries were appended; the first n_kept stay visible."""
        if not 0 <= n_kept <= n_fed:
            raise ValueError("kept %d of %d" % (n_kept, n_fed))
        self.valid += [1] * n_kept + [0] * (n_fed - n_kept)
        self.position += n_kept


class GreedySpecDecoder:
    """Greedy (speculative) decoding of one request over a forward function.

    `prefill(prompt)` feeds the prompt in blocks of at most
    SHARD_MAX_TOKENS tokens and returns the first generated token;
    `step(drafts)` runs one verify block and returns the emitted tokens
    (`step([])` is one plain greedy step)."""

    def __init__(self, forward: Forward, max_block: int = SHARD_MAX_TOKENS):
        self.forward = forward
        self.max_block = max_block
        self.req = MaskedRequest(0)
        self.current: Optional[int] = None
        self.accepted = 0
        self.proposed = 0
        self.steps = 0

    def prefill(self, prompt: Sequence[int]) -> int:
        prompt = [int(t) for t in prompt]
        if not prompt:
            raise ValueError("empty prompt")
        last = None
        for i in range(0, len(prompt), self.max_block):
            block = np.array(prompt[i:i + self.max_block], dtype=np.int32)
            pos, mask = self.req.inputs(block.size)
            out = np.asarray(self.forward(block, pos, mask))
            self.req.commit(block.size, block.size)
            last = int(out[-1])
        self.current = last
        return last

    def step(self, drafts: Sequence[int] = ()) -> List[int]:
        if self.current is None:
            raise RuntimeError("prefill first")
        drafts = [int(d) for d in drafts]
        if len(drafts) + 1 > self.max_block:
            raise ValueError("at most %d drafts per step" % (self.max_block - 1))
        feed = np.array([self.current] + drafts, dtype=np.int32)
        pos, mask = self.req.inputs(feed.size)
        targets = np.asarray(self.forward(feed, pos, mask))
        a, emitted = greedy_accept(drafts, targets)
        self.req.commit(feed.size, 1 + a)
        self.current = emitted[-1]
        self.accepted += a
        self.proposed += len(drafts)
        self.steps += 1
        return emitted


class ShardPipeline:
    """A forward function over pipeline stages and a top-1 head through the
    C ABI: stage 0 takes token ids (it owns the embedding), every later
    stage the previous stage's fp16 hidden states; the head returns the
    greedy tokens.  One request row per stage state.

    stages: shard handles in pipeline order; hidden: their hidden width;
    head: a head handle; capacity: cache entries per stage state (prompt,
    generated tokens and rejected drafts)."""

    def __init__(self, stages: Sequence[int], hidden: int, head: int, capacity: int, stream: int = 0):
        self.stages = list(stages)
        self.hidden = hidden
        self.head = head
        self.stream = stream
        self.states = [kv_state_alloc(s, 1, capacity) for s in self.stages]
        self.capacity = capacity

    def __call__(self, tokens: np.ndarray, positions: np.ndarray, mask: np.ndarray) -> np.ndarray:
        n = int(tokens.size)
        h = np.empty((n, self.hidden), dtype=np.uint16)
        for i, (sh, st) in enumerate(zip(self.stages, self.states)):
            out = np.empty((n, self.hidden), dtype=np.uint16)
            shard_step_host(sh, st, None if i == 0 else h, tokens if i == 0 else None, [n], positions,
                            mask.reshape(1, -1), None, out, self.stream)
            h = out
        tok, _ = head_top1_host(self.head, h, self.stream)
        return tok

    def close(self) -> None:
        for st in self.states:
            kv_state_free(st)
        self.states = []
